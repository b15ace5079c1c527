"""Host-side arithmetic of bench.py's roofline objects (no GPU)."""
import os

import pytest

from paper_2609_32166_gb300 import inputs

PEAKS = {"hbm_gbs": 6000.0, "bf16_tflops_sustained": 1500.0}   # ridge 250 FLOP/B


def _bench():
    import bench
    return bench


def test_attention_flops_counts_every_row_of_every_sequence():
    b = _bench()
    w = inputs.WORKLOADS["2b-bf16-chain16"]
    batch = inputs.make_batch(w, 0)
    assert b.attention_flops(w, batch) == 4 * 17 * 12 * (1800 + 17) * 128
    w8 = inputs.WORKLOADS["7b-bf16-batch8-paged"]
    b8 = inputs.make_batch(w8, 0)
    expect = sum(4 * 32 * 28 * (int(p) + 32) * 128 for p in b8.prefix_lens)
    assert b.attention_flops(w8, b8) == expect
    assert b.lmhead_flops(w, batch) == 2 * 17 * 151936 * 1536


def test_bound_follows_the_ridge():
    b = _bench()
    # 100 FLOP/B: below the ridge, HBM-bound; 1 MB in 1 us = 1000 GB/s.
    r = b.kernel_roofline("k", "bf16", 1e6, 1e8, 1e-6, 1, 1e-5, PEAKS, None)
    assert r["bound"] == "hbm" and r["unit"] == "GB/s"
    assert r["achieved"] == pytest.approx(1000.0)
    assert r["frac"] == pytest.approx(1000.0 / 6000.0)
    assert r["ridge_flop_per_byte"] == pytest.approx(250.0)
    # 1000 FLOP/B: above it, tensor-bound; 1 GFLOP in 1 us = 1000 TFLOP/s.
    r = b.kernel_roofline("k", "bf16", 1e6, 1e9, 1e-6, 1, 1e-5, PEAKS, None)
    assert r["bound"] == "tensor" and r["unit"] == "TFLOP/s"
    assert r["achieved"] == pytest.approx(1000.0)
    assert r["frac"] == pytest.approx(1000.0 / 1500.0)
    # fp32 never takes the bf16 tensor peak.
    r = b.kernel_roofline("k", "f32", 1e6, 1e9, 1e-6, 1, 1e-5, PEAKS, None)
    assert r["bound"] == "hbm"


def test_peaks_fall_back_when_unmeasured():
    b = _bench()
    r = b.kernel_roofline("k", "bf16", 1e6, 1e6, 1e-6, 1, 1e-5, {}, None)
    assert r["peak"] == 6800.0 and r["peak_source"].startswith("fallback")


def test_dominant_kernel_is_the_larger_share_of_the_step():
    b = _bench()
    w = inputs.WORKLOADS["2b-bf16-chain16"]
    batch = inputs.make_batch(w, 0)
    # 28 layers x 7 us = 196 us of attention against 88 us of LM head.
    dom, other = b.step_rooflines(w, batch, 1.97e6, 7e-6, 4.67e8, 88e-6, 290e-6, PEAKS)
    assert dom["kernel"] == "pf_verify_attention" and other["kernel"] == "pf_lmhead_accept"
    assert dom["share_of_step"] == pytest.approx(196 / 290)
    assert dom["launches_per_step"] == 28
    # 28 x 2 us = 56 us of attention: the LM head dominates.
    dom, other = b.step_rooflines(w, batch, 1.97e6, 2e-6, 4.67e8, 88e-6, 150e-6, PEAKS)
    assert dom["kernel"] == "pf_lmhead_accept"


def test_traffic_only_for_matching_sources_and_workload(tmp_path):
    b = _bench()
    files = ("lmhead.cu", "pf_ptx.cuh")
    path = os.path.join(tmp_path, "t.txt")

    def write(fp, wl):
        with open(path, "w") as f:
            f.write("# comment: ignored\nworkload: %s\nsource_fingerprint: %s\n"
                    "dram_bytes_per_launch: 1234\n" % (wl, fp))

    write(b.source_fingerprint(files), "2b-bf16-chain16")
    assert b.profiled_traffic((path, files), "2b-bf16-chain16") == 1234.0
    assert b.profiled_traffic((path, files), "7b-bf16-tree64") is None
    write("0000000000000000", "2b-bf16-chain16")
    assert b.profiled_traffic((path, files), "2b-bf16-chain16") is None
    assert b.profiled_traffic((os.path.join(tmp_path, "missing.txt"), files),
                              "2b-bf16-chain16") is None


def test_reference_steps_stop_at_the_wall_budget():
    b = _bench()
    spec = dict(workload="tiny-f32-chain8", seed=0, mode="whole", steps=50, warmup=0)
    assert b.cpu_worker(dict(spec, wall_budget_s=0.0))["steps"] == 1
    r = b.cpu_worker(dict(spec, steps=3, wall_budget_s=60.0))
    assert r["steps"] == 3
    # whole steps: nothing is projected
    assert r["layers_timed"] == 1 and r["step_s"] == pytest.approx(r["measured_s"])


def test_combined_step_roofline_takes_each_part_at_its_own_bound():
    b = _bench()
    w = inputs.WORKLOADS["7b-bf16-32k-tree128"]
    batch = inputs.make_batch(w, 0)
    attn_b, lm_b, commit_b = 69.2e6, 1.09e9, 2.0e6
    r = b.combined_step_roofline(w, batch, attn_b, lm_b, commit_b, 2e-3, PEAKS)
    flops = b.attention_flops(w, batch)
    # the 32K tree's attention is tensor-bound (about 870 FLOP/B, ridge 250)
    attn = max(attn_b / 6000e9, flops / 1500e12) * w.layers
    assert attn == pytest.approx(flops / 1500e12 * w.layers)
    lm = max(lm_b / 6000e9, b.lmhead_flops(w, batch) / 1500e12)
    ideal = attn + lm + commit_b / 6000e9
    assert r["ideal_us"] == pytest.approx(ideal * 1e6)
    assert r["frac"] == pytest.approx(ideal / 2e-3)
    hbm = (attn_b * w.layers + lm_b + commit_b) / 6000e9
    assert r["hbm_only_frac"] == pytest.approx(hbm / 2e-3)
    assert r["ideal_us"] > r["hbm_only_ideal_us"]


def test_cpu_baseline_mode_is_whole_steps_only_where_they_are_cheap():
    b = _bench()
    W = inputs.WORKLOADS
    assert b.cpu_mode(W["tiny-f32-chain8"]) == "whole"
    assert b.cpu_mode(W["2b-bf16-chain16"]) == "whole"
    for name in ("7b-bf16-tree64", "7b-bf16-batch8-paged", "7b-bf16-32k-tree128"):
        assert b.cpu_mode(W[name]) == "layer"


def test_e2e_copy_pieces_follow_the_layers():
    b = _bench()
    assert b.e2e_cuts(28) == [1, 4, 10, 18]
    assert b.e2e_cuts(1) == []
    assert b.e2e_cuts(2) == [1]
    for L in range(2, 40):
        cuts = b.e2e_cuts(L)
        assert cuts == sorted(set(cuts)) and all(0 < c < L for c in cuts)


def test_input_arena_is_blocked_by_layer():
    """The step's input arena on the host side (torch on the CPU): q and the
    proposal K/V of layer l are one block, the views carry the original
    values, the commit's layer stride is the block, and the copy pieces
    tile the arena in order with the hidden states in the last one."""
    import numpy as np
    import torch
    from paper_2609_32166_gb300.step import VerifyStep
    w = inputs.scaled(inputs.WORKLOADS["7b-bf16-batch8-paged"], layers=3, prefix=(40, 100),
                      vocab=300, hidden=64, batch=2)
    batch = inputs.make_batch(w, 0)
    vs = VerifyStep(w, batch, np.zeros(batch.total_nodes, np.int32), device="cpu")
    bits = lambda t: t.contiguous().view(torch.int16).numpy().view(np.uint16)
    for l in range(w.layers):
        assert np.array_equal(bits(vs.q[l]), inputs.layer_q(w, batch, l))
        tk, tv = inputs.layer_tree_kv(w, batch, l)
        assert np.array_equal(bits(vs.tree_k[l]), tk) and np.array_equal(bits(vs.tree_v[l]), tv)
        assert vs.q[l].is_contiguous() and vs.tree_k[l].is_contiguous()
    blk = vs.tree_k.stride(0) * vs.tree_k.element_size()
    assert vs.q.stride(0) == vs.tree_k.stride(0) == vs.tree_v.stride(0)
    assert vs.tree_k[1].data_ptr() - vs.tree_k[0].data_ptr() == blk
    assert vs.commit_desc.tree_layer_stride == vs.tree_k.stride(0)
    assert np.array_equal(bits(vs.hidden), inputs.hidden_states(w, batch))
    segs = vs.input_segments([1, 2])
    assert [s[2:] for s in segs] == [(0, 1), (1, 2), (2, w.layers + 1)]
    off = 0
    for o, nb, _, _ in segs:
        assert o == off and nb > 0
        off += nb
    assert off == vs.in_arena.numel()
    base = vs.in_arena.data_ptr()
    assert vs.q[1].data_ptr() - base == segs[1][0]  # a piece starts at its first layer's block
    assert vs.hidden.data_ptr() - base >= segs[-1][0]
    assert vs.tokens.data_ptr() - base < segs[0][1]


def test_attention_descriptors_carry_host_copies_of_the_lengths():
    """Every layer's attention descriptor points at the step's own host
    copies of cu_nodes and prefix_len (the two-block kernel's team plan is
    made from them): equal to the batch's lengths, and copies, so that
    changing them leaves the batch -- and the oracle that reads it -- alone."""
    import ctypes as C
    import numpy as np
    from paper_2609_32166_gb300.step import VerifyStep
    w = inputs.scaled(inputs.WORKLOADS["7b-bf16-batch8-paged"], layers=2, prefix=(40, 100),
                      vocab=300, hidden=64, batch=3)
    batch = inputs.make_batch(w, 0)
    vs = VerifyStep(w, batch, np.zeros(batch.total_nodes, np.int32), device="cpu")
    B = w.batch
    for d in vs.attn_descs:
        cu = np.ctypeslib.as_array(C.cast(d.host_cu_nodes, C.POINTER(C.c_int32)), (B + 1,))
        pl = np.ctypeslib.as_array(C.cast(d.host_prefix_len, C.POINTER(C.c_int32)), (B,))
        assert np.array_equal(cu, batch.cu_nodes) and np.array_equal(pl, batch.prefix_lens)
    before = batch.prefix_lens.copy()
    vs.h_prefix_len[:] = vs.h_prefix_len[::-1].copy()
    assert np.array_equal(batch.prefix_lens, before)
