"""ctypes binding of libpfverify.so (include/pf_verify.h).

Argument marshalling only: every step of the verify path runs in the CUDA
library.  The functions carry the C names; descriptors are the C structs.
Tensors are passed as raw device pointers (``tensor.data_ptr()``); torch is
used by callers for device memory and streams only.

There is no fallback: if the library is missing or fails to load, every
entry point raises ``PfLibraryMissing``.
"""
from __future__ import annotations

import ctypes as C
import os
import re

import numpy as np

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libpfverify.so")
HEADER = os.path.join(os.path.dirname(_PKG), "include", "pf_verify.h")

PF_OK, PF_ERR_NULL, PF_ERR_SHAPE, PF_ERR_DTYPE, PF_ERR_TREE = 0, 1, 2, 3, 4
PF_ERR_CAPACITY, PF_ERR_ALIGN, PF_ERR_CUDA, PF_ERR_WORKSPACE = 5, 6, 7, 8
PF_F32, PF_BF16 = 0, 1
PF_KV_CONTIGUOUS, PF_KV_PAGED = 0, 1
PF_MAX_NODES, PF_MASK_WORDS, PF_PAGE_SIZE, PF_MAX_LM_ROWS = 128, 2, 16, 256
PF_DEVERR_TIMEOUT, PF_DEVERR_CAPACITY, PF_DEVERR_BOUNDS, PF_DEVERR_TREE = 1, 2, 4, 8
PF_ATTN_EARLY_PREFETCH, PF_ATTN_NO_PDL = 1, 2
PF_LM_EARLY_WEIGHT, PF_LM_NO_PDL = 1, 2
(PF_ATTN_KERNEL_AUTO, PF_ATTN_KERNEL_MMA, PF_ATTN_KERNEL_TC64, PF_ATTN_KERNEL_TC128,
 PF_ATTN_KERNEL_PAIR, PF_ATTN_KERNEL_STREAM, PF_ATTN_KERNEL_BATCH,
 PF_ATTN_KERNEL_TWO_BLOCK) = 0, 1, 2, 3, 4, 5, 6, 7

STATUS_NAMES = {0: "PF_OK", 1: "PF_ERR_NULL", 2: "PF_ERR_SHAPE", 3: "PF_ERR_DTYPE",
                4: "PF_ERR_TREE", 5: "PF_ERR_CAPACITY", 6: "PF_ERR_ALIGN", 7: "PF_ERR_CUDA",
                8: "PF_ERR_WORKSPACE"}


class PfLibraryMissing(RuntimeError):
    pass


class PfError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"{STATUS_NAMES.get(status, status)}: {message}")
        self.status = status


class pf_kv_view(C.Structure):
    _fields_ = [("layout", C.c_int32), ("k", C.c_void_p), ("v", C.c_void_p),
                ("max_seq", C.c_int32), ("num_pages", C.c_int32),
                ("page_table", C.c_void_p), ("pages_per_seq", C.c_int32)]


class pf_attn_desc(C.Structure):
    _fields_ = [("dtype", C.c_int32), ("batch", C.c_int32), ("n_q_heads", C.c_int32),
                ("n_kv_heads", C.c_int32), ("head_dim", C.c_int32), ("scale", C.c_float),
                ("total_nodes", C.c_int32), ("max_nodes", C.c_int32),
                ("max_prefix_len", C.c_int32), ("cu_nodes", C.c_void_p),
                ("prefix_len", C.c_void_p), ("q", C.c_void_p), ("tree_k", C.c_void_p),
                ("tree_v", C.c_void_p), ("mask", C.c_void_p), ("cache", pf_kv_view),
                ("out", C.c_void_p), ("error_flag", C.c_void_p), ("flags", C.c_int32),
                ("workspace", C.c_void_p), ("workspace_bytes", C.c_size_t),
                ("kernel", C.c_int32), ("splits", C.c_int32), ("rows_per_cta", C.c_int32),
                ("stages", C.c_int32), ("host_cu_nodes", C.c_void_p),
                ("host_prefix_len", C.c_void_p)]


class pf_lm_desc(C.Structure):
    _fields_ = [("dtype", C.c_int32), ("batch", C.c_int32), ("hidden", C.c_int32),
                ("vocab", C.c_int32), ("total_nodes", C.c_int32), ("max_nodes", C.c_int32),
                ("cu_nodes", C.c_void_p), ("hidden_states", C.c_void_p),
                ("weight", C.c_void_p), ("tokens", C.c_void_p), ("parent", C.c_void_p),
                ("argmax", C.c_void_p), ("max_logit", C.c_void_p),
                ("accept_len", C.c_void_p), ("path", C.c_void_p),
                ("out_tokens", C.c_void_p), ("last_node", C.c_void_p),
                ("error_flag", C.c_void_p), ("flags", C.c_int32), ("stages", C.c_int32)]


class pf_commit_desc(C.Structure):
    _fields_ = [("dtype", C.c_int32), ("batch", C.c_int32), ("n_layers", C.c_int32),
                ("n_kv_heads", C.c_int32), ("head_dim", C.c_int32),
                ("total_nodes", C.c_int32), ("max_nodes", C.c_int32),
                ("max_prefix_len", C.c_int32), ("cu_nodes", C.c_void_p),
                ("prefix_len", C.c_void_p), ("accept_len", C.c_void_p), ("path", C.c_void_p),
                ("tree_k", C.c_void_p), ("tree_v", C.c_void_p),
                ("tree_layer_stride", C.c_int64), ("cache", pf_kv_view),
                ("cache_layer_stride", C.c_int64), ("new_len", C.c_void_p),
                ("error_flag", C.c_void_p)]


class pf_shift_desc(C.Structure):
    _fields_ = [("dtype", C.c_int32), ("n_layers", C.c_int32), ("n_kv_heads", C.c_int32),
                ("head_dim", C.c_int32), ("seq", C.c_int32), ("batch", C.c_int32),
                ("src", C.c_int32), ("dst", C.c_int32), ("count", C.c_int32),
                ("rope_base", C.c_float), ("cache", pf_kv_view),
                ("cache_layer_stride", C.c_int64), ("error_flag", C.c_void_p)]


class pf_key_desc(C.Structure):
    _fields_ = [("dtype", C.c_int32), ("hidden", C.c_int32), ("hidden_state", C.c_void_p),
                ("projection", C.c_void_p), ("key_out", C.c_void_p),
                ("error_flag", C.c_void_p)]


class pf_retrieval_desc(C.Structure):
    _fields_ = [("n_entries", C.c_int32), ("lo", C.c_int32), ("hi", C.c_int32),
                ("token", C.c_int32), ("query_key", C.c_void_p), ("keys", C.c_void_p),
                ("entry_token", C.c_void_p), ("entry_pos", C.c_void_p),
                ("entry_bound", C.c_void_p), ("best", C.c_void_p),
                ("similarity", C.c_void_p), ("error_flag", C.c_void_p)]


class pf_prefix_desc(C.Structure):
    _fields_ = [("prev", C.c_void_p), ("n_prev", C.c_int32), ("next", C.c_void_p),
                ("n_next", C.c_int32), ("lcp", C.c_void_p), ("cache_len", C.c_void_p)]


class pf_length_controller(C.Structure):
    _fields_ = [("l_max", C.c_int32), ("n_latency", C.c_int32), ("lr", C.c_double),
                ("epsilon", C.c_double), ("w_first", C.c_double * 3), ("w_cont", C.c_double * 3),
                ("c", C.c_double * 3), ("P", C.c_double * 9)]


_lib = None


def lib() -> C.CDLL:
    """The loaded library; raises PfLibraryMissing if it is not built."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise PfLibraryMissing(
            f"{LIB_PATH} is not built; run __graft_entry__.build() (nvcc, sm_103a)")
    try:
        L = C.CDLL(LIB_PATH)
    except OSError as e:
        raise PfLibraryMissing(f"cannot load {LIB_PATH}: {e}") from e
    L.pf_last_error.restype = C.c_char_p
    L.pf_last_error.argtypes = []
    L.pf_version.restype = C.c_int32
    L.pf_tree_prepare.restype = C.c_int
    L.pf_tree_prepare.argtypes = [C.c_void_p, C.c_int32, C.c_void_p, C.c_void_p]
    L.pf_tree_prepare_device.restype = C.c_int
    L.pf_tree_prepare_device.argtypes = [C.c_void_p, C.c_void_p, C.c_int32, C.c_int32, C.c_int32,
                                         C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p]
    L.pf_verify_attention.restype = C.c_int
    L.pf_verify_attention.argtypes = [C.POINTER(pf_attn_desc), C.c_void_p]
    L.pf_verify_attention_workspace_size.restype = C.c_size_t
    L.pf_verify_attention_workspace_size.argtypes = [C.POINTER(pf_attn_desc)]
    L.pf_verify_attention_launches.restype = C.c_int32
    L.pf_verify_attention_launches.argtypes = [C.POINTER(pf_attn_desc)]
    L.pf_verify_attention_team_plan.restype = C.c_int32
    L.pf_verify_attention_team_plan.argtypes = [C.c_void_p, C.c_void_p] + [C.c_int32] * 6 + [
        C.c_void_p, C.c_int32, C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p]
    L.pf_lmhead_accept_workspace_size.restype = C.c_size_t
    L.pf_lmhead_accept_workspace_size.argtypes = [C.POINTER(pf_lm_desc)]
    L.pf_lmhead_accept.restype = C.c_int
    L.pf_lmhead_accept.argtypes = [C.POINTER(pf_lm_desc), C.c_void_p, C.c_size_t, C.c_void_p]
    L.pf_lmhead_accept_noalloc.restype = C.c_int
    L.pf_lmhead_accept_noalloc.argtypes = [C.POINTER(pf_lm_desc), C.c_void_p]
    L.pf_kv_commit.restype = C.c_int
    L.pf_kv_commit.argtypes = [C.POINTER(pf_commit_desc), C.c_void_p]
    L.pf_kv_shift.restype = C.c_int
    L.pf_kv_shift.argtypes = [C.POINTER(pf_shift_desc), C.c_void_p]
    L.pf_retrieval_workspace_size.restype = C.c_size_t
    L.pf_retrieval_workspace_size.argtypes = []
    L.pf_retrieval_key.restype = C.c_int
    L.pf_retrieval_key.argtypes = [C.POINTER(pf_key_desc), C.c_void_p, C.c_size_t, C.c_void_p]
    L.pf_retrieve.restype = C.c_int
    L.pf_retrieve.argtypes = [C.POINTER(pf_retrieval_desc), C.c_void_p, C.c_size_t,
                              C.c_void_p]
    L.pf_controller_init.restype = C.c_int
    L.pf_controller_init.argtypes = [C.POINTER(pf_length_controller), C.c_int32, C.c_double,
                                     C.c_double]
    L.pf_controller_observe.restype = C.c_int
    L.pf_controller_observe.argtypes = [C.POINTER(pf_length_controller), C.c_int32, C.c_double,
                                        C.c_int32, C.c_double]
    L.pf_controller_choose.restype = C.c_int
    L.pf_controller_choose.argtypes = [C.POINTER(pf_length_controller), C.c_double, C.c_double,
                                       C.c_double, C.POINTER(C.c_int32),
                                       C.POINTER(C.c_double)]
    L.pf_length_select.restype = C.c_int
    L.pf_length_select.argtypes = [C.c_void_p, C.c_void_p, C.c_void_p, C.c_int32,
                                   C.POINTER(C.c_int32), C.POINTER(C.c_double)]
    L.pf_selftest_wait.restype = C.c_int
    L.pf_selftest_wait.argtypes = [C.c_void_p, C.c_int64, C.c_int32, C.c_void_p, C.c_void_p]
    L.pf_prefix_match.restype = C.c_int
    L.pf_prefix_match.argtypes = [C.POINTER(pf_prefix_desc), C.c_void_p]
    _lib = L
    return L


def header_functions() -> list:
    """Names of the functions include/pf_verify.h declares."""
    src = open(HEADER).read()
    return re.findall(r"PF_API\s+[\w\s\*]+?\b(pf_\w+)\s*\(", src)


def _check(status: int) -> None:
    if status != PF_OK:
        raise PfError(status, lib().pf_last_error().decode())


def pf_version() -> int:
    return int(lib().pf_version())


def pf_last_error() -> str:
    return lib().pf_last_error().decode()


def pf_tree_prepare(parent) -> tuple:
    """Host call: returns (depth int32 [N], mask uint64 [N, 2])."""
    p = np.ascontiguousarray(parent, dtype=np.int32)
    n = int(p.shape[0])
    depth = np.zeros(max(n, 1), dtype=np.int32)
    mask = np.zeros((max(n, 1), PF_MASK_WORDS), dtype=np.uint64)
    _check(lib().pf_tree_prepare(p.ctypes.data, n, depth.ctypes.data, mask.ctypes.data))
    return depth[:n], mask[:n]


def pf_tree_prepare_device(parent: int, cu_nodes: int, batch: int, total_nodes: int,
                           max_nodes: int, depth_out: int, mask_out: int, error_flag: int = 0,
                           stream: int = 0) -> None:
    """Device call (pointers are device addresses; depth_out and error_flag
    may be 0): ancestor bitmaps and depths of a batch of trees."""
    _check(lib().pf_tree_prepare_device(C.c_void_p(parent), C.c_void_p(cu_nodes), batch,
                                        total_nodes, max_nodes, C.c_void_p(depth_out or None),
                                        C.c_void_p(mask_out), C.c_void_p(error_flag or None),
                                        C.c_void_p(stream)))


def pf_verify_attention_workspace_size(desc: pf_attn_desc) -> int:
    return int(lib().pf_verify_attention_workspace_size(C.byref(desc)))


def pf_verify_attention_launches(desc: pf_attn_desc) -> int:
    return int(lib().pf_verify_attention_launches(C.byref(desc)))


PF_TEAM_MAX_CTAS = 160


def pf_verify_attention_team_plan(cu_nodes, prefix_len, n_kv_heads: int, group: int,
                                  max_nodes: int, max_prefix_len: int, num_sms: int,
                                  max_clusters, uniform_splits: int):
    """The two-block kernel's team plan for host lengths: (status, entries
    [PF_TEAM_MAX_CTAS] uint32, cluster size, CTAs, longest piece in tiles)."""
    import numpy as np
    cu = np.ascontiguousarray(cu_nodes, dtype=np.int32)
    pl = np.ascontiguousarray(prefix_len, dtype=np.int32)
    mc = None if max_clusters is None else np.ascontiguousarray(max_clusters, dtype=np.int32)
    entries = np.zeros(PF_TEAM_MAX_CTAS, dtype=np.uint32)
    out = np.zeros(3, dtype=np.int32)
    st = lib().pf_verify_attention_team_plan(
        cu.ctypes.data, pl.ctypes.data, len(pl), n_kv_heads, group, max_nodes, max_prefix_len,
        num_sms, None if mc is None else mc.ctypes.data, uniform_splits, entries.ctypes.data,
        out[0:].ctypes.data, out[1:].ctypes.data, out[2:].ctypes.data)
    return int(st), entries, int(out[0]), int(out[1]), int(out[2])


def pf_verify_attention(desc: pf_attn_desc, stream: int = 0) -> None:
    _check(lib().pf_verify_attention(C.byref(desc), C.c_void_p(stream)))


def pf_lmhead_accept_workspace_size(desc: pf_lm_desc = None) -> int:
    return int(lib().pf_lmhead_accept_workspace_size(C.byref(desc) if desc else None))


def pf_lmhead_accept(desc: pf_lm_desc, workspace: int, workspace_bytes: int,
                     stream: int = 0) -> None:
    _check(lib().pf_lmhead_accept(C.byref(desc), C.c_void_p(workspace),
                                  C.c_size_t(workspace_bytes), C.c_void_p(stream)))


def pf_lmhead_accept_noalloc(desc: pf_lm_desc, stream: int = 0) -> None:
    """pf_lmhead_accept with the scratch in the library's fixed device array
    (for callers that cannot allocate; calls must not overlap on the GPU)."""
    _check(lib().pf_lmhead_accept_noalloc(C.byref(desc), C.c_void_p(stream)))


def pf_kv_commit(desc: pf_commit_desc, stream: int = 0) -> None:
    _check(lib().pf_kv_commit(C.byref(desc), C.c_void_p(stream)))


def pf_kv_shift(desc: pf_shift_desc, stream: int = 0) -> None:
    _check(lib().pf_kv_shift(C.byref(desc), C.c_void_p(stream)))


def pf_retrieval_workspace_size() -> int:
    return int(lib().pf_retrieval_workspace_size())


def pf_retrieval_key(desc: pf_key_desc, workspace: int, workspace_bytes: int,
                     stream: int = 0) -> None:
    _check(lib().pf_retrieval_key(C.byref(desc), C.c_void_p(workspace),
                                  C.c_size_t(workspace_bytes), C.c_void_p(stream)))


def pf_retrieve(desc: pf_retrieval_desc, workspace: int, workspace_bytes: int,
                stream: int = 0) -> None:
    _check(lib().pf_retrieve(C.byref(desc), C.c_void_p(workspace),
                             C.c_size_t(workspace_bytes), C.c_void_p(stream)))


def pf_prefix_match(desc: pf_prefix_desc, stream: int = 0) -> None:
    _check(lib().pf_prefix_match(C.byref(desc), C.c_void_p(stream)))


def pf_controller_init(l_max: int, lr: float, epsilon: float) -> pf_length_controller:
    c = pf_length_controller()
    _check(lib().pf_controller_init(C.byref(c), l_max, lr, epsilon))
    return c


def pf_controller_observe(c: pf_length_controller, ell: int, similarity: float, accepted: int,
                          latency_us: float) -> None:
    _check(lib().pf_controller_observe(C.byref(c), ell, similarity, accepted, latency_us))


def pf_controller_choose(c: pf_length_controller, similarity: float, u: float = 1.0,
                         u_dir: float = 0.0) -> tuple:
    ell, obj = C.c_int32(), C.c_double()
    _check(lib().pf_controller_choose(C.byref(c), similarity, u, u_dir, C.byref(ell),
                                      C.byref(obj)))
    return int(ell.value), float(obj.value)


def pf_length_select(t_hat, p_first, p_cont) -> tuple:
    """Eq. 1 over explicit float64 arrays of length l_max + 1 (host)."""
    t = np.ascontiguousarray(t_hat, dtype=np.float64)
    p1 = np.ascontiguousarray(p_first, dtype=np.float64)
    pc = np.ascontiguousarray(p_cont, dtype=np.float64)
    assert t.shape == p1.shape == pc.shape and t.ndim == 1
    ell, obj = C.c_int32(), C.c_double()
    _check(lib().pf_length_select(t.ctypes.data, p1.ctypes.data, pc.ctypes.data,
                                  int(t.shape[0]) - 1, C.byref(ell), C.byref(obj)))
    return int(ell.value), float(obj.value)


def pf_selftest_wait(error_flag: int, limit_ns: int, signal: bool, waited_ok: int,
                     stream: int = 0) -> None:
    _check(lib().pf_selftest_wait(C.c_void_p(error_flag), int(limit_ns), 1 if signal else 0,
                                  C.c_void_p(waited_ok), C.c_void_p(stream)))
