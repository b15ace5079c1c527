"""Shared helpers of the GPU parity tests: build a case from the seeded
generator, plant tokens from the oracle's greedy predictions, run the CUDA
path through the C ABI and compare with the fp64 oracle.

Tolerances (fixed for the verify step):
  attention  max |gpu - oracle| <= 1e-4 (fp32) and <= 2e-2 (bf16)
  argmax     bit-exact except at nodes whose oracle top-2 margin < 1e-2
             (flagged); acceptance is then checked for self-consistency
  commit     bit-exact, every other cache byte unchanged
"""
from __future__ import annotations

import numpy as np
import torch

from oracle import accept as OAcc
from oracle import attention as OA
from oracle import commit as OC
from oracle import lmhead as OL
from paper_2609_32166_gb300 import inputs as I
from paper_2609_32166_gb300.step import VerifyStep, host_bits

ATTN_TOL = {"f32": 1e-4, "bf16": 2e-2}
MARGIN_FLAG = 1e-2


def values(x: np.ndarray, dtype: str) -> np.ndarray:
    """Exact float32 values of generated data (bf16 bits or float32)."""
    return I.bf16_bits_to_f32(x) if dtype == "bf16" else np.asarray(x, dtype=np.float32)


class Case:
    """A generated workload, the oracle's greedy predictions and a device step."""

    def __init__(self, w: I.Workload, seed: int = 0, layers: int = None, batch: I.Batch = None,
                 balanced: bool = True, attn_launch: dict = None):
        self.w = w
        self.batch = batch if batch is not None else I.make_batch(w, seed)
        self.L = layers if layers is not None else w.layers
        self.hidden = I.hidden_states(w, self.batch)
        self.weight = I.lm_weight(w, self.batch.seed)
        lg = OL.logits(values(self.hidden, w.dtype), values(self.weight, w.dtype))
        self.o_argmax, self.o_margin, self.o_top = OL.greedy(lg)
        del lg
        self.tokens = I.plant_tokens(self.batch, self.o_argmax)
        self.vs = VerifyStep(w, self.batch, self.tokens, layers=self.L,
                             weight=self.weight, hidden=self.hidden, balanced=balanced,
                             attn_launch=attn_launch)

    # --------------------------------------------------------------- attention
    def oracle_attention(self, layer: int, seq: int, nodes=None) -> np.ndarray:
        w, b = self.w, self.batch
        c0, c1 = int(b.cu_nodes[seq]), int(b.cu_nodes[seq + 1])
        q = values(I.layer_q(w, b, layer), w.dtype)[c0:c1]
        tk, tv = (values(x, w.dtype)[c0:c1] for x in I.layer_tree_kv(w, b, layer))
        pk, pv = (values(x, w.dtype) for x in I.layer_prefix_kv(w, b, layer, seq))
        return OA.tree_attention(q, pk, pv, tk, tv, b.parents[seq], nodes=nodes)

    def check_attention(self, layer: int, seq: int, nodes=None) -> float:
        ref = self.oracle_attention(layer, seq, nodes)
        c0, c1 = int(self.batch.cu_nodes[seq]), int(self.batch.cu_nodes[seq + 1])
        got = self.vs.attn_out[layer, c0:c1].float().cpu().numpy().astype(np.float64)
        sel = range(c1 - c0) if nodes is None else nodes
        err = max(float(np.abs(got[n] - ref[n]).max()) for n in sel)
        assert np.isfinite(got[list(sel)]).all()
        assert err <= ATTN_TOL[self.w.dtype], (layer, seq, err)
        return err

    def compare_attention(self, layer: int, seq: int, ref: dict) -> float:
        """Max error against precomputed oracle rows {node: [Hq, D]}."""
        c0 = int(self.batch.cu_nodes[seq])
        got = self.vs.attn_out[layer].float().cpu().numpy().astype(np.float64)
        err = 0.0
        for n, r in ref.items():
            g = got[c0 + n]
            assert np.isfinite(g).all(), (layer, seq, n)
            err = max(err, float(np.abs(g - r).max()))
        assert err <= ATTN_TOL[self.w.dtype], (layer, seq, err)
        return err

    # --------------------------------------------------------------- LM head
    def check_lmhead(self, res: dict) -> int:
        """Returns the number of flagged (near-tie) nodes."""
        flagged = self.o_margin < MARGIN_FLAG
        mism = res["argmax"] != self.o_argmax
        assert not np.any(mism & ~flagged), np.nonzero(mism & ~flagged)
        # the reported maximum logit matches the oracle's top logit
        tol = 1e-5 if self.w.dtype == "f32" else 2e-3
        assert np.allclose(res["max_logit"], self.o_top, rtol=0, atol=tol * (1 + np.abs(self.o_top)).max())
        b = self.batch
        for s, parent in enumerate(b.parents):
            c0, c1 = int(b.cu_nodes[s]), int(b.cu_nodes[s + 1])
            tok = self.tokens[c0:c1]
            # the GPU's walk is exactly the greedy descent over the GPU's argmax
            a, path, out_tokens, last = OAcc.accept_walk(parent, tok, res["argmax"][c0:c1])
            assert res["accept_len"][s] == a
            assert list(res["path"][s, :a + 1]) == path
            assert list(res["out_tokens"][s, :a + 1]) == out_tokens
            assert res["last_node"][s] == last
            # ... and, with no near-tie on the oracle's path, equals the oracle's
            oa, opath, otok, olast = OAcc.accept_walk(parent, tok, self.o_argmax[c0:c1])
            if not any(flagged[c0 + n] for n in opath):
                assert (a, path, out_tokens, last) == (oa, opath, otok, olast)
                assert opath == I.root_path(parent, int(b.forced_end[s]))
        return int(flagged.sum())

    # --------------------------------------------------------------- commit
    def check_commit(self, res: dict, layers=None) -> None:
        w, b = self.w, self.batch
        assert list(res["new_len"]) == [int(b.prefix_lens[s]) + int(res["accept_len"][s]) + 1
                                        for s in range(w.batch)]
        for l in (range(self.L) if layers is None else layers):
            tk_all, tv_all = I.layer_tree_kv(w, b, l)
            for kv, (gpu, tree_all) in enumerate(((self.vs.cache_k, tk_all), (self.vs.cache_v, tv_all))):
                got = host_bits(gpu[l])
                expect = np.zeros_like(got)
                for s in range(w.batch):
                    pre = I.layer_prefix_kv(w, b, l, s)[kv]
                    I.place_prefix(w, b, expect, s, pre)
                for s in range(w.batch):
                    P = int(b.prefix_lens[s])
                    a = int(res["accept_len"][s])
                    path = [int(x) for x in res["path"][s, :a + 1]]
                    c0, c1 = int(b.cu_nodes[s]), int(b.cu_nodes[s + 1])
                    rows = I.cache_rows(w, b, expect, s, 0, P + len(path))
                    full = np.zeros((w.hkv, P + len(path), w.d), dtype=rows.dtype)
                    full[:, :P] = rows[:, :P]
                    new, n1 = OC.commit_rows(full, P, path, tree_all[c0:c1])
                    assert n1 == P + a + 1
                    # write the committed rows back into the expected layout
                    for k in range(len(path)):
                        one = np.zeros((w.hkv, 1, w.d), dtype=rows.dtype)
                        one[:, 0] = new[:, P + k]
                        _place_rows(w, b, expect, s, P + k, one)
                assert np.array_equal(got, expect), (l, kv)


def _place_rows(w, b, cache, seq, start, rows):
    if w.layout == "contiguous":
        cache[seq, :, start:start + rows.shape[1], :] = rows
        return
    for i in range(rows.shape[1]):
        pos = start + i
        cache[b.page_table[seq][pos // I.PAGE_SIZE], :, pos % I.PAGE_SIZE, :] = rows[:, i]
