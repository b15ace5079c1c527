"""Device buffers and call sequence of one verify step.

``VerifyStep`` owns the device tensors of one workload (queries, proposal
K/V and prefix caches of every layer, hidden states, LM-head weight, tree
structure, outputs) and issues the three C-ABI calls of the step:
``pf_verify_attention`` once per layer, ``pf_lmhead_accept`` once, and
``pf_kv_commit`` once for all layers.  torch provides device memory and
streams only; nothing here computes any part of the step.

Layouts (row-major):
  q, attn_out     [L, T, Hq, D]
  tree_k, tree_v  [L, T, Hkv, D]
  cache_k/v       [L, B, Hkv, S, D] (contiguous) or [L, pages, Hkv, 16, D] (paged)
  mask            [T, 2] uint64 ancestor bitmaps (pf_tree_prepare)
  hidden          [T, H];  weight [V, H]
"""
from __future__ import annotations

import numpy as np
import torch

from . import binding as pb
from . import inputs as I


def _dev(arr: np.ndarray, dtype: str, device) -> torch.Tensor:
    """Host array (bf16 bit patterns or float32/ints) -> device tensor."""
    if dtype == "bf16":
        t = torch.from_numpy(np.ascontiguousarray(arr).view(np.int16)).view(torch.bfloat16)
    else:
        t = torch.from_numpy(np.ascontiguousarray(arr))
    return t.to(device)


def _torch_dtype(dtype: str):
    return torch.bfloat16 if dtype == "bf16" else torch.float32


def host_bits(t: torch.Tensor) -> np.ndarray:
    """Device tensor -> host numpy of the same bits (uint16 for bf16)."""
    t = t.detach().cpu().contiguous()
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).numpy().view(np.uint16)
    return t.numpy()


class VerifyStep:
    """One workload's device state.  ``layers`` may restrict the layer count
    (parity tests use a few layers of a full-size workload).  ``balanced``
    gives the attention calls a workspace, with which a batch of several
    sequences is dealt out to the SMs in proportion to their lengths.

    ``fill="host"`` (the default) uploads the seeded host generator's values,
    which the oracle also receives; ``fill="device"`` draws the bulk tensors
    (queries, proposal K/V, caches, hidden states, LM weight) with torch's
    seeded device generator instead -- the same shapes and distributions
    (N(0, 1), weight N(0, 0.02), bf16), minutes faster for the 32K-token
    cache, for measurements that are not compared with the oracle.
    ``weight_dev`` shares an LM-head weight already on the device."""

    def __init__(self, w: I.Workload, batch: I.Batch, tokens: np.ndarray, layers: int = None,
                 device: str = "cuda", weight: np.ndarray = None, hidden: np.ndarray = None,
                 balanced: bool = True, attn_launch: dict = None, fill: str = "host",
                 weight_dev: torch.Tensor = None):
        self.w, self.batch = w, batch
        self.balanced = balanced
        # pf_attn_desc launch fields (kernel, splits, rows_per_cta, stages):
        # empty = the library's automatic choice
        self.attn_launch = dict(attn_launch or {})
        self.L = layers if layers is not None else w.layers
        self.device = device
        td = _torch_dtype(w.dtype)
        T, B = batch.total_nodes, w.batch
        self.T = T
        self.max_nodes = max(len(p) for p in batch.parents)
        self.max_prefix = int(batch.prefix_lens.max())

        masks = []
        for p in batch.parents:
            _, m = pb.pf_tree_prepare(p)
            masks.append(m)
        mask = np.concatenate(masks, axis=0).astype(np.uint64)
        self.mask = torch.from_numpy(mask.view(np.int64)).to(device)
        self.cu_nodes = torch.from_numpy(batch.cu_nodes).to(device)
        self.prefix_len = torch.from_numpy(batch.prefix_lens.astype(np.int32)).to(device)
        # host copies for the launch plan (read by the attention call only)
        self.h_cu_nodes = np.array(batch.cu_nodes, dtype=np.int32)
        self.h_prefix_len = np.array(batch.prefix_lens, dtype=np.int32)
        self.parent = torch.from_numpy(batch.parent_flat).to(device)
        self.tokens = torch.from_numpy(np.asarray(tokens, dtype=np.int32)).to(device)
        self.page_table = (torch.from_numpy(batch.page_table).to(device)
                           if batch.page_table is not None else None)

        shp = I.cache_shape(w, batch)
        self.q = torch.empty((self.L, T, w.hq, w.d), dtype=td, device=device)
        self.tree_k = torch.empty((self.L, T, w.hkv, w.d), dtype=td, device=device)
        self.tree_v = torch.empty_like(self.tree_k)
        self.cache_k = torch.zeros((self.L,) + shp, dtype=td, device=device)
        self.cache_v = torch.zeros_like(self.cache_k)
        gen = None
        if fill == "device":
            gen = torch.Generator(device=device)
            gen.manual_seed(int(batch.seed) * 7919 + 17)
            for t in (self.q, self.tree_k, self.tree_v, self.cache_k, self.cache_v):
                t.normal_(0.0, 1.0, generator=gen)
        elif fill != "host":
            raise ValueError(f"fill must be 'host' or 'device', not {fill!r}")
        for l in (range(self.L) if fill == "host" else ()):
            self.q[l] = _dev(I.layer_q(w, batch, l), w.dtype, device)
            tk, tv = I.layer_tree_kv(w, batch, l)
            self.tree_k[l] = _dev(tk, w.dtype, device)
            self.tree_v[l] = _dev(tv, w.dtype, device)
            ck = np.zeros(shp, dtype=np.uint16 if w.dtype == "bf16" else np.float32)
            cv = np.zeros_like(ck)
            for s in range(B):
                pk, pv = I.layer_prefix_kv(w, batch, l, s)
                I.place_prefix(w, batch, ck, s, pk)
                I.place_prefix(w, batch, cv, s, pv)
            self.cache_k[l] = _dev(ck, w.dtype, device)
            self.cache_v[l] = _dev(cv, w.dtype, device)
        self.attn_out = torch.zeros_like(self.q)
        if fill == "device" and hidden is None:
            self.hidden = torch.empty((T, w.hidden), dtype=td, device=device)
            self.hidden.normal_(0.0, 1.0, generator=gen)
        else:
            self.hidden = _dev(I.hidden_states(w, batch) if hidden is None else hidden, w.dtype,
                               device)
        if weight_dev is not None:
            assert tuple(weight_dev.shape) == (w.vocab, w.hidden) and weight_dev.dtype == td
            self.weight = weight_dev
        elif fill == "device" and weight is None:
            self.weight = torch.empty((w.vocab, w.hidden), dtype=td, device=device)
            self.weight.normal_(0.0, 0.02, generator=gen)
        else:
            self.weight = _dev(I.lm_weight(w, batch.seed) if weight is None else weight, w.dtype,
                               device)

        i32 = dict(dtype=torch.int32, device=device)
        self.argmax = torch.full((T,), -1, **i32)
        self.max_logit = torch.zeros((T,), dtype=torch.float32, device=device)
        self.accept_len = torch.full((B,), -1, **i32)
        self.path = torch.full((B, self.max_nodes), -1, **i32)
        self.out_tokens = torch.full((B, self.max_nodes), -1, **i32)
        self.last_node = torch.full((B,), -1, **i32)
        self.new_len = torch.zeros((B,), **i32)
        self.err = torch.zeros((1,), **i32)
        self.ws_bytes = pb.pf_lmhead_accept_workspace_size()
        self.workspace = torch.zeros((self.ws_bytes,), dtype=torch.uint8, device=device)
        # A step's inputs and outputs each live in one contiguous arena (the
        # tensors above become views of it), so that a host round trip is
        # one copy each way.
        # (the ancestor bitmaps are derived on the device from the parent
        # array by pf_tree_prepare_device, so they are not among the inputs)
        self.in_arena = self._input_arena(device)
        self.out_arena = self._arena(("accept_len", "out_tokens", "new_len"), device)
        self._build_descs()

    def _input_arena(self, device) -> torch.Tensor:
        """The step's inputs in one 256-byte-aligned byte arena, in the order
        the step consumes them: the per-step arrays (tokens, parent array,
        cu_nodes, prefix lengths), then one block per layer holding that
        layer's q, proposal K and proposal V, then the hidden states.  q,
        tree_k and tree_v become [L, ...] views with the block as their layer
        stride, so a host copy can be issued layer by layer
        (input_segments) and the commit still sees one layer stride."""
        al = lambda x: (x + 255) // 256 * 256
        es = self.q.element_size()
        qb = self.q[0].numel() * es
        kb = self.tree_k[0].numel() * es
        q_o, k_o = 0, al(qb)
        v_o = al(k_o + kb)
        blk = al(v_o + kb)
        off, heads = 0, {}
        for n in ("tokens", "parent", "cu_nodes", "prefix_len"):
            t = getattr(self, n)
            off = al(off)
            heads[n] = off
            off += t.numel() * t.element_size()
        layers0 = al(off)
        hid_o = al(layers0 + self.L * blk)
        total = hid_o + self.hidden.numel() * self.hidden.element_size()
        arena = torch.empty(total, dtype=torch.uint8, device=device)
        for n, o in heads.items():
            t = getattr(self, n)
            v = arena[o:o + t.numel() * t.element_size()].view(t.dtype).view(t.shape)
            v.copy_(t)
            setattr(self, n, v)
        h = self.hidden
        hv = arena[hid_o:hid_o + h.numel() * h.element_size()].view(h.dtype).view(h.shape)
        hv.copy_(h)
        self.hidden = hv
        elems = arena[layers0:layers0 + self.L * blk].view(self.q.dtype)
        base = elems.storage_offset()
        for n, o in (("q", q_o), ("tree_k", k_o), ("tree_v", v_o)):
            t = getattr(self, n)
            stride = (blk // es,) + tuple(t[0].stride())
            v = torch.as_strided(elems, tuple(t.shape), stride, base + o // es)
            v.copy_(t)
            setattr(self, n, v)
        self._layers0, self._layer_block, self._hidden_off = layers0, blk, hid_o
        return arena

    def input_segments(self, boundaries) -> list:
        """Byte ranges (offset, nbytes, first layer, end layer) of the input
        arena for a layer-by-layer host copy: the first range holds the
        per-step arrays and layers [0, boundaries[0]), each next one the
        layers up to the next boundary, the last one also the hidden states
        (end layer = L + 1 marks it)."""
        cuts = [0] + [b for b in boundaries if 0 < b < self.L] + [self.L]
        segs = []
        for i in range(len(cuts) - 1):
            l0, l1 = cuts[i], cuts[i + 1]
            start = 0 if i == 0 else self._layers0 + l0 * self._layer_block
            end = self._layers0 + l1 * self._layer_block
            last = i == len(cuts) - 2
            if last:
                end = self.in_arena.numel()
            segs.append((start, end - start, l0, self.L + 1 if last else l1))
        return segs

    def _arena(self, names, device) -> torch.Tensor:
        """Move the named tensors into one 256-byte-aligned byte arena and
        replace each by a view of it; returns the arena."""
        layout, total = [], 0
        for n in names:
            t = getattr(self, n)
            total = (total + 255) // 256 * 256
            nbytes = t.numel() * t.element_size()
            layout.append((n, total, nbytes))
            total += nbytes
        arena = torch.empty(total, dtype=torch.uint8, device=device)
        for n, off, nbytes in layout:
            t = getattr(self, n)
            v = arena[off:off + nbytes].view(t.dtype).view(t.shape)
            v.copy_(t)
            setattr(self, n, v)
        return arena

    # ------------------------------------------------------------------ descs
    def _view(self, l: int) -> pb.pf_kv_view:
        w, b = self.w, self.batch
        v = pb.pf_kv_view()
        v.layout = pb.PF_KV_PAGED if w.layout == "paged" else pb.PF_KV_CONTIGUOUS
        v.k = self.cache_k[l].data_ptr()
        v.v = self.cache_v[l].data_ptr()
        v.max_seq = b.max_seq if w.layout == "contiguous" else 0
        if w.layout == "paged":
            v.num_pages = b.num_pages
            v.page_table = self.page_table.data_ptr()
            v.pages_per_seq = int(b.page_table.shape[1])
        return v

    def _build_descs(self):
        w = self.w
        dt = pb.PF_BF16 if w.dtype == "bf16" else pb.PF_F32
        self.attn_descs = []
        for l in range(self.L):
            d = pb.pf_attn_desc()
            d.dtype, d.batch = dt, w.batch
            d.n_q_heads, d.n_kv_heads, d.head_dim = w.hq, w.hkv, w.d
            d.scale = 0.0
            d.total_nodes, d.max_nodes, d.max_prefix_len = self.T, self.max_nodes, self.max_prefix
            d.cu_nodes, d.prefix_len = self.cu_nodes.data_ptr(), self.prefix_len.data_ptr()
            d.q = self.q[l].data_ptr()
            d.tree_k, d.tree_v = self.tree_k[l].data_ptr(), self.tree_v[l].data_ptr()
            d.mask = self.mask.data_ptr()
            d.cache = self._view(l)
            d.out = self.attn_out[l].data_ptr()
            d.error_flag = self.err.data_ptr()
            # Within one step only pf_kv_commit writes the cache, and it runs
            # after the last layer: every layer but the first may request its
            # cache tiles while the previous layer is still finishing.
            d.flags = pb.PF_ATTN_EARLY_PREFETCH if l > 0 else 0
            d.host_cu_nodes = self.h_cu_nodes.ctypes.data
            d.host_prefix_len = self.h_prefix_len.ctypes.data
            for k, v in self.attn_launch.items():
                setattr(d, k, int(v))
            self.attn_descs.append(d)
        # one attention workspace serves every layer (calls run in stream order)
        self.attn_ws_bytes = (pb.pf_verify_attention_workspace_size(self.attn_descs[0])
                              if self.balanced else 0)
        self.attn_ws = (torch.empty((self.attn_ws_bytes,), dtype=torch.uint8, device=self.device)
                        if self.attn_ws_bytes else None)
        for d in self.attn_descs:
            d.workspace = self.attn_ws.data_ptr() if self.attn_ws is not None else None
            d.workspace_bytes = self.attn_ws_bytes
        d = pb.pf_lm_desc()
        d.dtype, d.batch, d.hidden, d.vocab = dt, w.batch, w.hidden, w.vocab
        d.total_nodes, d.max_nodes = self.T, self.max_nodes
        d.cu_nodes = self.cu_nodes.data_ptr()
        d.hidden_states, d.weight = self.hidden.data_ptr(), self.weight.data_ptr()
        d.tokens, d.parent = self.tokens.data_ptr(), self.parent.data_ptr()
        d.argmax, d.max_logit = self.argmax.data_ptr(), self.max_logit.data_ptr()
        d.accept_len, d.path = self.accept_len.data_ptr(), self.path.data_ptr()
        d.out_tokens, d.last_node = self.out_tokens.data_ptr(), self.last_node.data_ptr()
        d.error_flag = self.err.data_ptr()
        d.flags = pb.PF_LM_EARLY_WEIGHT  # nothing in the step writes the weight
        self.lm_desc = d
        c = pb.pf_commit_desc()
        c.dtype, c.batch, c.n_layers = dt, w.batch, self.L
        c.n_kv_heads, c.head_dim = w.hkv, w.d
        c.total_nodes, c.max_nodes, c.max_prefix_len = self.T, self.max_nodes, self.max_prefix
        c.cu_nodes, c.prefix_len = self.cu_nodes.data_ptr(), self.prefix_len.data_ptr()
        c.accept_len, c.path = self.accept_len.data_ptr(), self.path.data_ptr()
        c.tree_k, c.tree_v = self.tree_k.data_ptr(), self.tree_v.data_ptr()
        c.tree_layer_stride = self.tree_k.stride(0)  # elements between layers' proposal K/V
        c.cache = self._view(0)
        c.cache_layer_stride = self.cache_k[0].numel()
        c.new_len = self.new_len.data_ptr()
        c.error_flag = self.err.data_ptr()
        self.commit_desc = c

    # ------------------------------------------------------------------ calls
    @staticmethod
    def _stream(stream):
        return torch.cuda.current_stream().cuda_stream if stream is None else int(stream)

    def attention(self, layer: int, stream=None):
        pb.pf_verify_attention(self.attn_descs[layer], self._stream(stream))

    def lmhead(self, stream=None):
        pb.pf_lmhead_accept(self.lm_desc, self.workspace.data_ptr(), self.ws_bytes,
                            self._stream(stream))

    def commit(self, stream=None):
        pb.pf_kv_commit(self.commit_desc, self._stream(stream))

    def tree_prepare(self, stream=None):
        """Ancestor bitmaps of this step's trees, on the device, from the
        parent array (pf_tree_prepare_device)."""
        pb.pf_tree_prepare_device(self.parent.data_ptr(), self.cu_nodes.data_ptr(), self.w.batch,
                                  self.T, self.max_nodes, 0, self.mask.data_ptr(),
                                  self.err.data_ptr(), self._stream(stream))

    def step(self, stream=None, tree_prepare: bool = False):
        """One verify step: (optionally the device tree bitmaps,) L attention
        calls, the LM head with acceptance, the commit."""
        s = self._stream(stream)
        if tree_prepare:
            self.tree_prepare(s)
        for l in range(self.L):
            pb.pf_verify_attention(self.attn_descs[l], s)
        pb.pf_lmhead_accept(self.lm_desc, self.workspace.data_ptr(), self.ws_bytes, s)
        pb.pf_kv_commit(self.commit_desc, s)

    def launches_per_step(self) -> int:
        # what each attention call launches (one kernel, or two with a separate
        # merge), the LM head, the commit
        return sum(pb.pf_verify_attention_launches(d) for d in self.attn_descs) + 2

    # ------------------------------------------------------------------ results
    def results(self) -> dict:
        torch.cuda.synchronize()
        return dict(argmax=self.argmax.cpu().numpy(), max_logit=self.max_logit.cpu().numpy(),
                    accept_len=self.accept_len.cpu().numpy(), path=self.path.cpu().numpy(),
                    out_tokens=self.out_tokens.cpu().numpy(),
                    last_node=self.last_node.cpu().numpy(), new_len=self.new_len.cpu().numpy(),
                    err=int(self.err.item()))
