"""Benchmark of the verify step (tree attention x L layers, LM head with
greedy acceptance, KV commit) on seeded synthetic inputs.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME]
    python bench.py --impl reference ...      # the fp64 CPU oracle, timed
    python bench.py --ell-sweep               # verify latency vs proposal length

Prints one JSON line.  The metric is accepted tokens/s of whole verify steps
(sum over sequences of accepted drafts + 1 bonus token, divided by the step
time), with the attention time per layer and the step's achieved HBM
bandwidth alongside.  The headline workload is the largest single-GPU one
(the 8-sequence paged 7B batch); `per_workload` times the other bf16
workloads in the same run.  Steps run as CUDA graphs of L attention calls,
one LM-head call and one commit call; a 256 MB memset between steps (outside
the per-step events) evicts L2.  Multi-GPU runs are independent replicas
(one process per GPU under torchrun); the value is the sum of tokens over
ranks divided by the slowest rank's time.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "verify-step µs/layer & accepted tokens/s; achieved HBM GB/s vs ~8 TB/s peak"
DEFAULT_WORKLOAD = "7b-bf16-batch8-paged"
# the other bf16 workloads, timed in the same run (`per_workload`)
PER_WORKLOAD = ("7b-bf16-tree64", "7b-bf16-32k-tree128", "2b-bf16-chain16")
L2_FLUSH_BYTES = 256 << 20
# per-part (attention / LM head / commit) breakdown: at least this much
# replay time, whatever --steps is
PARTS_MIN_SECONDS = 0.5
# the reference arm (the fp64 oracle on the host cores) times the requested
# steps, or as many as fit this much wall time
REFERENCE_WALL_BUDGET_S = 150.0
CSRC = os.path.join(ROOT, "paper_2609_32166_gb300", "csrc")
# Committed ncu DRAM-traffic summaries, each valid only for the kernel sources
# it was captured on (a fingerprint of the files that define the kernel and
# its launch shape) and for the workload it names.
LMHEAD_TRAFFIC = (os.path.join(ROOT, "profiles", "lmhead_traffic.txt"),
                  ("lmhead.cu", "pf_ptx.cuh"))
ATTENTION_TRAFFIC = (os.path.join(ROOT, "profiles", "attention_traffic.txt"),
                     ("api.cu", "attention.cu", "attention_tc.cu", "attention_tc2.cu",
                      "attention_2blk.cu", "attention_pair.cu", "attn_common.cuh",
                      "pf_internal.h", "pf_ptx.cuh"))


def parse(argv=None):
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=400)
    p.add_argument("--warmup", type=int, default=10)
    p.add_argument("--workload", default=DEFAULT_WORKLOAD)
    p.add_argument("--layers", type=int, default=None,
                   help="profiling aid: the step over the workload's first N layers only "
                        "(recorded in the line's config; default: every layer)")
    p.add_argument("--seed", type=int, default=0)
    p.add_argument("--impl", default="ours", choices=["ours", "reference"])
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--no-next-rows", action="store_true",
                   help="skip the re-rotation, retrieval, prefix and ell-sweep measurements")
    p.add_argument("--no-per-workload", action="store_true",
                   help="time the headline workload only")
    p.add_argument("--ell-sweep", action="store_true",
                   help="only the verify-step latency vs proposal length curve")
    p.add_argument("--cpu-worker", default=None, help=argparse.SUPPRESS)
    return p.parse_args(argv)


# ---------------------------------------------------------------------------
# algorithmic bytes and FLOPs
# ---------------------------------------------------------------------------
def step_bytes(w, batch, accept_lens):
    """(attention bytes per layer, LM-head bytes, commit bytes) of one step:
    every prefix K/V row, the proposal's K/V, q and out read or written once;
    the LM weight and hidden states once; the committed rows read and written
    in every layer."""
    es = 2 if w.dtype == "bf16" else 4
    T = batch.total_nodes
    prefix = int(np.sum(batch.prefix_lens))
    attn = (2 * prefix * w.hkv * w.d + 2 * T * w.hkv * w.d + 2 * T * w.hq * w.d) * es + T * 16
    lm = (w.vocab * w.hidden + T * w.hidden) * es + T * 4 * 4
    rows = int(np.sum(np.asarray(accept_lens) + 1))
    commit = 2 * rows * w.hkv * w.d * es * 2 * w.layers
    return attn, lm, commit


def attention_flops(w, batch):
    """FLOPs of one layer's tree attention: QK^T and PV over every prefix row
    and every proposal row (the masked tree part counted dense), i.e.
    4 * N * Hq * (P + N) * D summed over the sequences."""
    return float(sum(4 * len(par) * w.hq * (int(p) + len(par)) * w.d
                     for par, p in zip(batch.parents, batch.prefix_lens)))


def lmhead_flops(w, batch):
    return 2.0 * batch.total_nodes * w.vocab * w.hidden


def source_fingerprint(files):
    h = hashlib.sha256()
    for f in files:
        h.update(open(os.path.join(CSRC, f), "rb").read())
    return h.hexdigest()[:16]


def profiled_traffic(spec, workload):
    """dram bytes per launch from a committed ncu summary, if it was taken on
    the current kernel sources for this workload; else None."""
    path, files = spec
    if not os.path.exists(path):
        return None
    kv = {}
    for line in open(path):
        if ":" in line and not line.startswith("#"):
            k, v = line.split(":", 1)
            kv[k.strip()] = v.strip()
    if kv.get("source_fingerprint") != source_fingerprint(files):
        return None
    if kv.get("workload") != workload:
        return None
    try:
        return float(kv["dram_bytes_per_launch"])
    except (KeyError, ValueError):
        return None


def peak_values(peaks):
    hbm = peaks.get("hbm_gbs")
    tc = peaks.get("bf16_tflops_sustained")
    return (hbm or 6800.0, tc or 1700.0,
            "measured copy bandwidth" if hbm else "fallback copy bandwidth",
            "measured bf16 sustained" if tc else "fallback bf16 sustained")


def kernel_roofline(kernel, dtype, bytes_per_launch, flops_per_launch, seconds_per_launch,
                    launches_per_step, step_seconds, peaks, traffic):
    """Roofline of one kernel from its algorithmic bytes and FLOPs per launch
    and its mean in-step launch time.  The bound is the tensor pipe when the
    arithmetic intensity of a bf16 kernel lies above the ridge of the two
    measured peaks (bf16 sustained, since every kernel here is timed inside a
    long run, over copy bandwidth), else HBM."""
    hbm, tc, hbm_src, tc_src = peak_values(peaks)
    ridge = tc * 1e12 / (hbm * 1e9)
    intensity = flops_per_launch / bytes_per_launch if bytes_per_launch else 0.0
    if dtype == "bf16" and intensity > ridge:
        achieved = flops_per_launch / seconds_per_launch / 1e12
        out = {"bound": "tensor", "achieved": achieved, "peak": tc, "unit": "TFLOP/s",
               "frac": achieved / tc, "peak_source": tc_src}
    else:
        achieved = bytes_per_launch / seconds_per_launch / 1e9
        out = {"bound": "hbm", "achieved": achieved, "peak": hbm, "unit": "GB/s",
               "frac": achieved / hbm, "peak_source": hbm_src}
    out.update({"kernel": kernel, "traffic": traffic,
                "algorithmic_bytes": bytes_per_launch, "algorithmic_flops": flops_per_launch,
                "intensity_flop_per_byte": intensity, "ridge_flop_per_byte": ridge,
                "us_per_launch": seconds_per_launch * 1e6,
                "launches_per_step": launches_per_step,
                "share_of_step": seconds_per_launch * launches_per_step / step_seconds})
    return out


def step_rooflines(w, batch, attn_bytes, attn_s_per_layer, lm_bytes, lm_s, step_s, peaks):
    """(dominant, other): the roofline of the kernel with the larger share of
    the step's time, and that of the other one."""
    attn = kernel_roofline("pf_verify_attention", w.dtype, attn_bytes,
                           attention_flops(w, batch), attn_s_per_layer, w.layers, step_s, peaks,
                           profiled_traffic(ATTENTION_TRAFFIC, w.name))
    lm = kernel_roofline("pf_lmhead_accept", w.dtype, lm_bytes, lmhead_flops(w, batch), lm_s, 1,
                         step_s, peaks, profiled_traffic(LMHEAD_TRAFFIC, w.name))
    return (attn, lm) if attn["share_of_step"] >= lm["share_of_step"] else (lm, attn)


def combined_step_roofline(w, batch, attn_bytes, lm_bytes, commit_bytes, step_s, peaks):
    """The step's ideal time with each part at its own bound -- attention per
    layer and the LM head each at max(bytes / HBM, FLOPs / bf16 tensor peak),
    the commit at bytes / HBM -- against the measured step; and the HBM-only
    ideal (all algorithmic bytes at the copy bandwidth)."""
    hbm, tc, _, _ = peak_values(peaks)
    B, F = hbm * 1e9, tc * 1e12
    attn_ideal = max(attn_bytes / B, attention_flops(w, batch) / F) * w.layers
    lm_ideal = max(lm_bytes / B, lmhead_flops(w, batch) / F)
    commit_ideal = commit_bytes / B
    ideal = attn_ideal + lm_ideal + commit_ideal
    hbm_ideal = (attn_bytes * w.layers + lm_bytes + commit_bytes) / B
    return {"ideal_us": ideal * 1e6, "frac": ideal / step_s,
            "attention_ideal_us": attn_ideal * 1e6, "lmhead_ideal_us": lm_ideal * 1e6,
            "commit_ideal_us": commit_ideal * 1e6,
            "hbm_only_ideal_us": hbm_ideal * 1e6, "hbm_only_frac": hbm_ideal / step_s,
            "rule": "sum over parts of max(bytes / measured copy bandwidth, FLOPs / measured "
                    "bf16 sustained peak), divided by the measured step time"}


def load_peaks():
    pk = os.path.join(ROOT, "MEASURED_PEAKS.json")
    return json.load(open(pk)) if os.path.exists(pk) else {}


# ---------------------------------------------------------------------------
# clocks
# ---------------------------------------------------------------------------
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def start(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "50"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        rows = []
        for line in open(self.path):
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                rows.append(dict(sm=float(parts[1]), max=float(parts[2]),
                                 power=float(parts[3]) if parts[3] not in ("[N/A]", "N/A") else 0.0,
                                 hw=parts[5], hwt=parts[6], swt=parts[7], pcap=parts[8]))
            except ValueError:
                continue
        os.unlink(self.path)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        pmax = max(r["power"] for r in rows)
        load = [r for r in rows if r["power"] >= 0.5 * pmax] or rows
        reasons = set()
        for r in rows:
            for key, name in (("hw", "hw_slowdown"), ("hwt", "hw_thermal_slowdown"),
                              ("swt", "sw_thermal_slowdown"), ("pcap", "sw_power_cap")):
                if r[key].lower().startswith("active"):
                    reasons.add(name)
        return {"sm_mhz": statistics.median(r["sm"] for r in load),
                "sm_max_mhz": max(r["max"] for r in rows), "reasons": sorted(reasons),
                "samples": len(rows), "samples_under_load": len(load),
                "power_w_max": pmax}


# ---------------------------------------------------------------------------
# CPU oracle timing (cpu_baseline and --impl reference); runs in a fresh
# interpreter so its BLAS thread count is set before numpy loads
# ---------------------------------------------------------------------------
def cpu_worker(spec: dict) -> dict:
    """Times the fp64 oracle on one workload.  mode "whole": whole verify
    steps, every layer and sequence.  mode "layer": one sampled step =
    attention and commit of layer 0 for every sequence, the full LM head and
    the acceptance walks; the whole-step time is projected as
    L * (attention + commit of one layer) + LM head + walks."""
    from oracle import accept as OAcc
    from oracle import attention as OA
    from oracle import commit as OC
    from oracle import lmhead as OL
    from paper_2609_32166_gb300 import inputs as I

    w = I.WORKLOADS[spec["workload"]]
    if spec.get("layers"):
        w = I.scaled(w, layers=spec["layers"])
    batch = I.make_batch(w, spec["seed"])
    f = (lambda x: I.bf16_bits_to_f32(x)) if w.dtype == "bf16" else (lambda x: x)
    hidden = f(I.hidden_states(w, batch))
    weight = f(I.lm_weight(w, batch.seed))
    nl = w.layers if spec["mode"] == "whole" else 1
    layers = []
    for l in range(nl):
        q = f(I.layer_q(w, batch, l))
        tk, tv = (f(x) for x in I.layer_tree_kv(w, batch, l))
        pre = [tuple(f(x) for x in I.layer_prefix_kv(w, batch, l, s)) for s in range(w.batch)]
        layers.append((q, tk, tv, pre))
    cu = batch.cu_nodes
    ends = I.step_forced_ends(batch, 50)
    counter = [0]

    def one_step():
        g = counter[0] % len(ends)
        counter[0] += 1
        t0 = time.perf_counter()
        for (q, tk, tv, pre) in layers:
            for s in range(w.batch):
                c0, c1 = int(cu[s]), int(cu[s + 1])
                OA.tree_attention(q[c0:c1], pre[s][0], pre[s][1], tk[c0:c1], tv[c0:c1],
                                  batch.parents[s])
        t_attn = time.perf_counter() - t0
        t1 = time.perf_counter()
        am, _, _ = OL.greedy(OL.logits(hidden, weight))
        tokens = I.plant_tokens(batch, am, ends[g], salt=g)   # this step's proposal
        acc = []
        for s in range(w.batch):
            c0, c1 = int(cu[s]), int(cu[s + 1])
            acc.append(OAcc.accept_walk(batch.parents[s], tokens[c0:c1], am[c0:c1]))
        t_lm = time.perf_counter() - t1
        t2 = time.perf_counter()
        for (q, tk, tv, pre) in layers:
            for s in range(w.batch):
                c0, c1 = int(cu[s]), int(cu[s + 1])
                P = int(batch.prefix_lens[s])
                rows = np.zeros((w.hkv, P + w.nodes, w.d), dtype=np.float32)
                OC.commit_rows(rows, P, acc[s][1], tk[c0:c1])
                OC.commit_rows(rows, P, acc[s][1], tv[c0:c1])
        t_commit = time.perf_counter() - t2
        measured = t_attn + t_lm + t_commit
        whole = (t_attn + t_commit) * (w.layers / nl) + t_lm
        return measured, whole, sum(a[0] + 1 for a in acc)

    meas, whole, toks = [], [], []
    n = spec.get("steps")
    budget = spec.get("wall_budget_s")
    for _ in range(spec.get("warmup", 0)):
        one_step()
    counter[0] = 0
    t_start = time.perf_counter()
    # the requested steps, or as many as fit the wall budget (at least one)
    while len(meas) < (n if n is not None else 1 << 30):
        if meas and budget is not None and time.perf_counter() - t_start > budget:
            break
        m, wh, tok = one_step()
        meas.append(m)
        whole.append(wh)
        toks.append(tok)
    return dict(measured_s=float(np.mean(meas)), step_s=float(np.mean(whole)), steps=len(meas),
                tokens_per_step=float(np.mean(toks)), layers_timed=nl)


def run_cpu_worker(spec: dict, threads: int = None) -> dict:
    cores = os.cpu_count() or 1
    threads = threads or cores
    env = dict(os.environ)
    for k in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS"):
        env[k] = str(threads)
    env["CUDA_VISIBLE_DEVICES"] = ""
    r = subprocess.run([sys.executable, os.path.abspath(__file__), "--cpu-worker", json.dumps(spec)],
                       capture_output=True, text=True, env=env, cwd=ROOT)
    if r.returncode != 0:
        raise RuntimeError("CPU oracle worker failed:\n" + r.stderr[-2000:])
    out = json.loads(r.stdout.strip().splitlines()[-1])
    out["cores"] = threads
    out["host_cores"] = cores
    return out


def cpu_mode(w):
    """Whole steps where one fits a few seconds of fp64 numpy (the 2B chain
    and smaller), else a one-layer sample."""
    return "whole" if (w.hq * w.nodes * w.batch <= 256 and w.prefix[1] <= 4096) else "layer"


def cpu_sample_text(w, r):
    if r["layers_timed"] == w.layers:
        what = (f"whole verify steps of {w.name} in fp64 numpy: attention of all {w.layers} "
                f"layers, full LM head ({w.vocab}x{w.hidden}), acceptance, commit")
    else:
        what = (f"one sampled step of {w.name} in fp64 numpy: attention and commit of layer 0 "
                f"for all {w.batch} sequence(s), full LM head ({w.vocab}x{w.hidden}), acceptance; "
                f"whole-step time projected as {w.layers} x (attention + commit of one layer) "
                f"+ LM head + acceptance")
    return what + f"; {r['steps']} step(s) timed, {r['cores']} thread(s)"


def cpu_baseline_entry(w, spec_base):
    """The oracle on all host cores and on one core; value = accepted
    tokens per (projected) whole-step second."""
    out = {}
    for label, threads in (("all_cores", None), ("single_thread", 1)):
        r = run_cpu_worker(dict(spec_base, mode=cpu_mode(w)), threads=threads)
        out[label] = {"value": r["tokens_per_step"] / r["step_s"], "unit": "tokens/s",
                      "cores": r["cores"], "kind": "oracle", "ms_per_step": r["step_s"] * 1e3,
                      "measured_ms_per_sample": r["measured_s"] * 1e3,
                      "sample": cpu_sample_text(w, r)}
    base = dict(out["all_cores"])
    base["single_thread"] = out["single_thread"]
    return base


# ---------------------------------------------------------------------------
# multi-rank aggregation (replicas: one process per GPU, no data exchange)
# ---------------------------------------------------------------------------
def max_over_ranks(x: float, world: int, device: str = "cpu") -> float:
    """The largest x over all ranks (the slowest replica's time); x itself
    when there is one rank.  `device` is where the reduction tensor lives
    (cuda for nccl, cpu for gloo)."""
    if world <= 1:
        return float(x)
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(units_per_rank: float, slowest_seconds: float, world: int) -> float:
    """Units all ranks processed (every replica runs the same work) per
    second of the slowest rank."""
    return world * float(units_per_rank) / float(slowest_seconds)


# ---------------------------------------------------------------------------
# reference arm: the oracle as it stands, on the host cores
# ---------------------------------------------------------------------------
def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    from paper_2609_32166_gb300 import inputs as I
    w = I.WORKLOADS[args.workload]
    mode = cpu_mode(w)
    spec = dict(workload=args.workload, seed=args.seed, mode=mode, steps=args.steps,
                warmup=min(args.warmup, 1), wall_budget_s=REFERENCE_WALL_BUDGET_S)
    t0 = time.perf_counter()
    r = run_cpu_worker(spec)
    wall = time.perf_counter() - t0
    value = r["tokens_per_step"] / r["step_s"]
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s",
        "n_gpus": args.gpus, "steps": r["steps"], "steps_requested": args.steps,
        "warmup": args.warmup,
        # the measured time of the steps this run executed (for a one-layer
        # sample: the sample, not the projected whole step)
        "ms_per_step": r["measured_s"] * 1e3,
        "projected_ms_per_whole_step": r["step_s"] * 1e3,
        "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic (seeded generator)",
        "config": config_dict(w, args),
        "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": r["cores"],
                         "kind": "oracle",
                         "sample": cpu_sample_text(w, r) +
                         f"; {r['steps']} of {args.steps} steps timed (the steps that fit "
                         f"{REFERENCE_WALL_BUDGET_S:.0f} s of wall time)"},
        "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
        "wall_s": wall,
    }
    print(json.dumps(line))


def config_dict(w, args):
    return {"workload": w.name, "layers": w.layers, "batch": w.batch, "q_heads": w.hq,
            "kv_heads": w.hkv, "head_dim": w.d, "hidden": w.hidden, "vocab": w.vocab,
            "prefix": list(w.prefix), "nodes": w.nodes, "tree": w.tree, "kv_layout": w.layout,
            "seed": args.seed,
            "l2": "256 MB memset between steps (outside the per-step events); "
                  "step inputs also exceed the 129 MB L2"}


# ---------------------------------------------------------------------------
# our arm: one workload, device-timed
# ---------------------------------------------------------------------------
def _graph_events_supported():
    import torch
    try:
        torch.cuda.Event(enable_timing=True, external=True)
        return True
    except TypeError:
        return False


def prepare_workload(w, seed, weight_dev=None):
    """Device state of a workload (bulk tensors drawn on the device), draft
    tokens planted from the GPU's own greedy predictions for a seeded
    sequence of per-step accepted paths."""
    import torch
    from paper_2609_32166_gb300 import inputs as I
    from paper_2609_32166_gb300.step import VerifyStep
    batch = I.make_batch(w, seed)
    vs = VerifyStep(w, batch, np.zeros(batch.total_nodes, np.int32), fill="device",
                    weight_dev=weight_dev)
    vs.lmhead()
    torch.cuda.synchronize()
    greedy = vs.argmax.cpu().numpy()
    G = 50
    ends = I.step_forced_ends(batch, G)
    depth = [I.node_depths(p) for p in batch.parents]
    planned = [int(sum(depth[b][e[b]] + 1 for b in range(w.batch))) for e in ends]
    tok_table = torch.from_numpy(np.stack([I.plant_tokens(batch, greedy, e, salt=g)
                                           for g, e in enumerate(ends)])).cuda()
    return vs, batch, tok_table, planned


def time_steps(vs, tok_table, planned, K, warmup, stream, flush, parts, world=1, dist=None):
    """K verify steps in CUDA graphs of up to 50 steps, events at every step
    boundary (parts=False) or also around the attention / LM head / commit
    of every step (parts=True; those events split the programmatic-launch
    chain between the parts).  Returns (per-step ms, per-part ms lists,
    accepted tokens per step)."""
    import torch
    G_tab = tok_table.shape[0]
    with torch.cuda.stream(stream):
        for k in range(max(warmup, 3)):
            flush.zero_()
            vs.tokens.copy_(tok_table[k % G_tab])
            vs.step()
            stream.synchronize()
            got = int((vs.accept_len + 1).sum().item())
            assert got == planned[k % G_tab], (k, got, planned[k % G_tab])
    per_step, attn_t, lm_t, commit_t, toks = [], [], [], [], []
    done = 0
    graph_events = _graph_events_supported()
    while done < K:
        n = min(50, K - done)
        if graph_events:
            ev = [[torch.cuda.Event(enable_timing=True, external=True) for _ in range(4)]
                  for _ in range(n)]
            graph = torch.cuda.CUDAGraph()
            with torch.cuda.graph(graph, stream=stream):
                s = torch.cuda.current_stream()
                for g in range(n):
                    flush.zero_()
                    vs.tokens.copy_(tok_table[(done + g) % G_tab])
                    ev[g][0].record(s)
                    for l in range(vs.L):
                        vs.attention(l, s.cuda_stream)
                    if parts:
                        ev[g][1].record(s)
                    vs.lmhead(s.cuda_stream)
                    if parts:
                        ev[g][2].record(s)
                    vs.commit(s.cuda_stream)
                    ev[g][3].record(s)
            with torch.cuda.stream(stream):
                graph.replay()   # untimed: uploads the graph
            stream.synchronize()
            if dist is not None and world > 1:
                dist.barrier()
            torch.cuda.synchronize()
            with torch.cuda.stream(stream):
                graph.replay()
            stream.synchronize()
            del graph
        else:
            ev = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(n)]
            with torch.cuda.stream(stream):
                for g in range(n):
                    flush.zero_()
                    vs.tokens.copy_(tok_table[(done + g) % G_tab])
                    ev[g][0].record(stream)
                    for l in range(vs.L):
                        vs.attention(l, stream.cuda_stream)
                    ev[g][1].record(stream)
                    vs.lmhead(stream.cuda_stream)
                    ev[g][2].record(stream)
                    vs.commit(stream.cuda_stream)
                    ev[g][3].record(stream)
            stream.synchronize()
        for g in range(n):
            per_step.append(ev[g][0].elapsed_time(ev[g][3]))
            if parts or not graph_events:
                attn_t.append(ev[g][0].elapsed_time(ev[g][1]))
                lm_t.append(ev[g][1].elapsed_time(ev[g][2]))
                commit_t.append(ev[g][2].elapsed_time(ev[g][3]))
            toks.append(planned[(done + g) % G_tab])
        done += n
    res = vs.results()
    assert res["err"] == 0, f"device error flag {res['err']}"
    assert int(np.sum(res["accept_len"] + 1)) == toks[-1]
    return per_step, (attn_t, lm_t, commit_t), toks


def measure_workload(w, args, K, stream, flush, peaks, weight_dev=None, world=1, dist=None,
                     clocks=None):
    """Device-timed steps of one workload: the step time over exactly K
    steps (step-boundary events only), then a per-part pass of at least
    PARTS_MIN_SECONDS of replays with events around every step's parts."""
    import torch
    vs, batch, tok_table, planned = prepare_workload(w, args.seed, weight_dev)
    if clocks is not None:
        clocks.start()
        time.sleep(0.3)
    per_step, _, toks = time_steps(vs, tok_table, planned, K, args.warmup, stream, flush,
                                   parts=False, world=world, dist=dist)
    clk = clocks.stop() if clocks is not None else None
    t_total_ms = max_over_ranks(float(np.sum(per_step)), world, "cuda")
    ms_step = t_total_ms / K
    k_parts = max(20, int(np.ceil(PARTS_MIN_SECONDS / (ms_step * 1e-3))))
    _, (attn_t, lm_t, commit_t), _ = time_steps(vs, tok_table, planned, k_parts, 0, stream,
                                                flush, parts=True)
    res = vs.results()
    attn_b, lm_b, commit_b = step_bytes(w, batch, res["accept_len"])
    step_b = attn_b * w.layers + lm_b + commit_b
    attn_ms = float(np.mean(attn_t))
    lm_ms = float(np.mean(lm_t))
    hbm = peak_values(peaks)[0]
    roof, other = step_rooflines(w, batch, attn_b, attn_ms * 1e-3 / w.layers, lm_b, lm_ms * 1e-3,
                                 ms_step * 1e-3, peaks)
    out = {
        "workload": w.name, "steps": K, "ms_per_step": ms_step,
        "value": whole_job_rate(float(np.sum(toks)), t_total_ms / 1e3, world),
        "unit": "tokens/s", "accepted_tokens_per_step": float(np.mean(toks)),
        "us_per_layer_attention": attn_ms * 1e3 / w.layers,
        "us_lmhead": lm_ms * 1e3, "us_commit": float(np.mean(commit_t)) * 1e3,
        "parts": {"steps": len(attn_t), "seconds": float(np.sum(attn_t) + np.sum(lm_t) +
                                                         np.sum(commit_t)) * 1e-3,
                  "ms_per_step_with_part_events": float(np.mean(attn_t) + np.mean(lm_t) +
                                                        np.mean(commit_t)),
                  "attention_us_per_layer_sd": float(np.std(attn_t)) * 1e3 / w.layers,
                  "lmhead_us_sd": float(np.std(lm_t)) * 1e3},
        "step_hbm_gbs": step_b / (ms_step * 1e-3) / 1e9,
        "step_hbm_frac": step_b / (ms_step * 1e-3) / 1e9 / hbm,
        "step_bytes": step_b,
        "step_roofline": combined_step_roofline(w, batch, attn_b, lm_b, commit_b, ms_step * 1e-3,
                                                peaks),
        "roofline": roof,
        "other_roofline": other,
        "gpu_launches_per_step": vs.launches_per_step(),
    }
    if clk is not None:
        out["clocks"] = clk
    return out, vs, batch, tok_table, planned


# ---------------------------------------------------------------------------
# end to end through the library's calls
# ---------------------------------------------------------------------------
def e2e_cuts(L: int) -> list:
    """Layer boundaries of the end-to-end leg's host copies: a first copy of
    the per-step arrays and layer 0, then growing groups of layers (for 28
    layers: 1-3, 4-9, 10-17, 18-27 with the hidden states), so each copy
    lands before the layers that read it while the earlier layers run."""
    return sorted({max(1, min(L - 1, int(round(L * f)))) for f in (1 / 28, 4 / 28, 10 / 28, 18 / 28)}
                  ) if L > 1 else []


def run_e2e(vs, w, K, stream, flush, world, tok_table, planned):
    """The same metric end to end, as a caller of the library sees it, timed
    on the host wall clock: every step copies its inputs (queries, proposal
    K/V of every layer, hidden states, tokens, tree and lengths) from pinned
    host memory, issues the C-ABI calls eagerly -- the device tree bitmaps
    (pf_tree_prepare_device), L attention calls, the LM head, the commit --
    reads its outputs (accepted lengths, tokens, new lengths: one arena)
    back and synchronises.  The input copy goes in a few pieces on a copy
    stream (the per-step arrays and layer 0 first, then groups of layers,
    the hidden states last), each layer's attention waiting only for the
    piece that holds its inputs, so the copy overlaps the earlier layers.
    The L2 flush between steps is outside the timed region.  A second
    figure replays the same step -- copies, calls and the read-back -- as
    one CUDA graph (device events around it)."""
    import torch
    host_in = vs.in_arena.detach().cpu().pin_memory()
    host_out = torch.empty(vs.out_arena.numel(), dtype=torch.uint8).pin_memory()
    tok_off = vs.tokens.data_ptr() - vs.in_arena.data_ptr()
    tok_bytes = vs.tokens.numel() * vs.tokens.element_size()
    host_tokens = [t.cpu().contiguous().view(torch.uint8) for t in tok_table]
    acc_off = vs.accept_len.data_ptr() - vs.out_arena.data_ptr()
    h2d, d2h = host_in.numel(), host_out.numel()
    n = min(K, 200)
    segs = vs.input_segments(e2e_cuts(vs.L))
    copy_stream = torch.cuda.Stream()
    landed = [torch.cuda.Event() for _ in segs]

    def issue():
        """One step's copies and calls on `stream` (and the copy stream)."""
        sp = torch.cuda.current_stream().cuda_stream
        cur = torch.cuda.current_stream()
        copy_stream.wait_stream(cur)  # the arena is free: the previous step is done
        with torch.cuda.stream(copy_stream):
            for (o, nb, _, _), ev in zip(segs, landed):
                vs.in_arena[o:o + nb].copy_(host_in[o:o + nb], non_blocking=True)
                ev.record(copy_stream)
        cur.wait_event(landed[0])
        vs.tree_prepare(sp)
        si = 0
        for l in range(vs.L):
            while segs[si][3] <= l:
                si += 1
                cur.wait_event(landed[si])
            vs.attention(l, sp)
        for ev in landed[si + 1:]:
            cur.wait_event(ev)  # the hidden states' piece
        vs.lmhead(sp)
        vs.commit(sp)
        host_out.copy_(vs.out_arena, non_blocking=True)

    def one(k, graph=None, events=None):
        host_in[tok_off:tok_off + tok_bytes].copy_(host_tokens[k % len(host_tokens)])
        with torch.cuda.stream(stream):
            flush.zero_()
        stream.synchronize()
        t0 = time.perf_counter()
        with torch.cuda.stream(stream):
            if events:
                events[0].record(stream)
            if graph is None:
                issue()
            else:
                graph.replay()
            if events:
                events[1].record(stream)
        stream.synchronize()
        t = time.perf_counter() - t0
        got = int((host_out[acc_off:acc_off + 4 * w.batch].view(torch.int32) + 1).sum())
        assert got == planned[k % len(planned)]
        return t, got

    for k in range(3):
        one(k)
    wall, tok = [], 0
    for k in range(n):
        t, got = one(k)
        wall.append(t)
        tok += got
    t_wall = max_over_ranks(float(np.sum(wall)), world, "cuda")
    # graph variant: the copies, the calls and the read-back in one graph
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        issue()
    with torch.cuda.stream(stream):
        g.replay()
    stream.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    gt, gtok = [], 0
    for k in range(n):
        _, got = one(k, graph=g, events=(e0, e1))
        gt.append(e0.elapsed_time(e1))
        gtok += got
    t_graph = max_over_ranks(float(np.sum(gt)), world, "cuda")
    res = vs.results()
    assert res["err"] == 0
    return {"value": whole_job_rate(tok, t_wall, world), "unit": "tokens/s",
            "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "steps": n,
            "ms_per_step": t_wall * 1e3 / n,
            "timing": "host wall clock (time.perf_counter) around the H2D copies, eager C-ABI "
                      "calls (pf_tree_prepare_device, %d x pf_verify_attention, "
                      "pf_lmhead_accept, pf_kv_commit), D2H and a stream synchronise, per step"
                      % vs.L,
            "copies_per_step": {"h2d": len(segs), "d2h": 1},
            "h2d_pieces_first_layers": [s[2] for s in segs],
            "graph": {"value": whole_job_rate(gtok, t_graph * 1e-3, world),
                      "ms_per_step": t_graph / n,
                      "timing": "the same step (copies, calls, read-back) as one CUDA-graph "
                                "replay, device events around it"}}


# ---------------------------------------------------------------------------
# widened rows and the verify latency curve
# ---------------------------------------------------------------------------
def _time_events(stream, flush, fn, iters, warmup=3):
    """Mean device time (ms) of fn(i) over iters calls, L2 flushed before each
    call outside the events.  The calls are captured in one CUDA graph with
    event nodes (so host launch overhead stays out of the numbers) when this
    torch supports graph events, else launched eagerly."""
    import torch
    with torch.cuda.stream(stream):
        for i in range(warmup):
            flush.zero_()
            fn(i)
    stream.synchronize()
    if _graph_events_supported():
        ev = [(torch.cuda.Event(enable_timing=True, external=True),
               torch.cuda.Event(enable_timing=True, external=True)) for _ in range(iters)]
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            s = torch.cuda.current_stream()
            for i in range(iters):
                flush.zero_()
                ev[i][0].record(s)
                fn(warmup + i)
                ev[i][1].record(s)
        with torch.cuda.stream(stream):
            g.replay()   # untimed: uploads the graph
            stream.synchronize()
            g.replay()
        stream.synchronize()
    else:
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in range(iters)]
        with torch.cuda.stream(stream):
            for i in range(iters):
                flush.zero_()
                ev[i][0].record(stream)
                fn(warmup + i)
                ev[i][1].record(stream)
        stream.synchronize()
    return float(np.mean([a.elapsed_time(b) for a, b in ev]))


def measure_next_rows(stream, flush, hbm_peak, reps=4):
    """Rolling-image key re-rotation, decoding-memory retrieval and prompt-
    prefix carryover, each on a workload of the paper's shape, timed with
    CUDA events on the launching stream.  Each timed iteration makes `reps`
    calls on `reps` disjoint buffers (every call cold in L2; L2 flushed
    between iterations), so the fixed cost of the event pair is spread over
    several calls."""
    import torch
    from paper_2609_32166_gb300 import binding as pb
    from paper_2609_32166_gb300 import inputs as I
    out = {}
    sp = stream.cuda_stream
    # --- pf_kv_shift: two retained 1300-token screenshots move down by one
    # screenshot in every layer of a 7B-VLM-shaped cache (and back again on
    # the next iteration); `reps` independent 4096-position sequences
    L, Hkv, D, S = 28, 4, 128, 4096
    src, dst, count = 1400, 100, 2600
    k = torch.empty((L, reps, Hkv, S, D), dtype=torch.bfloat16, device="cuda").normal_()
    v = torch.empty_like(k).normal_()
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    descs = [[], []]
    for way, (a, b) in enumerate(((src, dst), (dst, src))):
        for seq in range(reps):
            d = pb.pf_shift_desc()
            d.dtype, d.n_layers, d.n_kv_heads, d.head_dim = pb.PF_BF16, L, Hkv, D
            d.seq, d.batch, d.src, d.dst, d.count, d.rope_base = seq, reps, a, b, count, 1e6
            d.cache.layout, d.cache.k, d.cache.v, d.cache.max_seq = (
                pb.PF_KV_CONTIGUOUS, k.data_ptr(), v.data_ptr(), S)
            d.cache_layer_stride = reps * Hkv * S * D
            d.error_flag = err.data_ptr()
            descs[way].append(d)

    def shift_all(i):
        for d in descs[i % 2]:
            pb.pf_kv_shift(d, sp)

    ms = _time_events(stream, flush, shift_all, 20) / reps
    assert int(err.item()) == 0
    shift_bytes = count * L * Hkv * D * 2 * 2 * 2   # K and V rows, read once and written once
    gbs = shift_bytes / (ms * 1e-3) / 1e9
    out["kv_shift"] = {
        "workload": "28 layers x 4 KV heads x D=128 bf16; 2600 rows shifted by 1300 "
                    "(two 1300-token screenshots), rope base 1e6",
        "us": ms * 1e3, "algorithmic_bytes": shift_bytes, "achieved_gbs": gbs,
        "peak_gbs": hbm_peak, "frac": gbs / hbm_peak, "launches_per_call": 2,
        "timing": f"{reps} calls on {reps} sequences per event pair, L2 flushed between pairs"}
    del k, v
    # --- pf_retrieval_key + pf_retrieve over a 290K-entry memory (74 MiB at
    # 256 + 12 bytes per entry); `reps` copies at different addresses
    M, H = 290000, 3584
    mem = I.decoding_memory(M, seed=11)
    mems = []
    for r in range(reps):
        mems.append(dict(keys=torch.from_numpy(mem.keys).cuda(),
                         token=torch.from_numpy(mem.token).cuda(),
                         pos=torch.from_numpy(mem.pos).cuda(),
                         bound=torch.from_numpy(mem.bound).cuda()))
    h = torch.empty(H, dtype=torch.bfloat16, device="cuda").normal_()
    P = torch.empty((I.KEY_DIM, H), dtype=torch.bfloat16, device="cuda").normal_()
    qkey = torch.zeros(I.KEY_DIM, dtype=torch.int8, device="cuda")
    best = torch.zeros(1, dtype=torch.int32, device="cuda")
    sim = torch.zeros(1, dtype=torch.float32, device="cuda")
    nws = pb.pf_retrieval_workspace_size()
    ws = torch.zeros(nws, dtype=torch.uint8, device="cuda")
    kd = pb.pf_key_desc()
    kd.dtype, kd.hidden, kd.hidden_state, kd.projection = pb.PF_BF16, H, h.data_ptr(), P.data_ptr()
    kd.key_out, kd.error_flag = qkey.data_ptr(), err.data_ptr()
    tokens, counts = np.unique(mem.token, return_counts=True)
    elig = (mem.pos < mem.bound)
    res = {}
    for label, tok in (("most frequent token", int(tokens[np.argmax(counts)])),
                       ("token of a random entry", int(mem.token[M // 3]))):
        rds = []
        for m in mems:
            rd = pb.pf_retrieval_desc()
            rd.n_entries, rd.lo, rd.hi, rd.token = M, 0, M, tok
            rd.query_key, rd.keys = qkey.data_ptr(), m["keys"].data_ptr()
            rd.entry_token, rd.entry_pos, rd.entry_bound = (
                m["token"].data_ptr(), m["pos"].data_ptr(), m["bound"].data_ptr())
            rd.best, rd.similarity, rd.error_flag = best.data_ptr(), sim.data_ptr(), err.data_ptr()
            rds.append(rd)

        def lookups(i, rds=rds):
            for rd in rds:
                pb.pf_retrieval_key(kd, ws.data_ptr(), nws, sp)
                pb.pf_retrieve(rd, ws.data_ptr(), nws, sp)

        def scans(i, rds=rds):
            for rd in rds:
                pb.pf_retrieve(rd, ws.data_ptr(), nws, sp)

        ms_l = _time_events(stream, flush, lookups, 30) / reps
        ms_s = _time_events(stream, flush, scans, 30) / reps
        n_elig = int(np.sum((mem.token == tok) & elig))
        # token, position and boundary of every entry, the key of every eligible one
        scan_bytes = 12 * M + I.KEY_DIM * n_elig
        res[label] = {"eligible": n_elig, "us_lookup": ms_l * 1e3, "us_scan": ms_s * 1e3,
                      "scan_algorithmic_bytes": scan_bytes,
                      "scan_gbs": scan_bytes / (ms_s * 1e-3) / 1e9}
    assert int(err.item()) == 0
    # --- pf_prefix_match: consecutive action-step prompts of 3.9K keys that
    # share a 2.1K-key system prompt and history, then differ (new screenshot)
    rng = np.random.default_rng(3)
    shared = rng.integers(0, 151936, size=2100)
    pairs = []
    for r in range(reps):
        a = np.concatenate([shared, rng.integers(1 << 30, (1 << 30) + (1 << 20), size=1800)])
        b = np.concatenate([shared, rng.integers(1 << 30, (1 << 30) + (1 << 20), size=1800)])
        pairs.append((torch.from_numpy(a.astype(np.int32)).cuda(),
                      torch.from_numpy(b.astype(np.int32)).cuda()))
    lcp = torch.zeros(2 * reps, dtype=torch.int32, device="cuda")
    pds = []
    for r, (a, b) in enumerate(pairs):
        d = pb.pf_prefix_desc()
        d.prev, d.n_prev, d.next, d.n_next = a.data_ptr(), a.numel(), b.data_ptr(), b.numel()
        d.lcp, d.cache_len = lcp.data_ptr() + 8 * r, lcp.data_ptr() + 8 * r + 4
        pds.append(d)

    def matches(i):
        for d in pds:
            pb.pf_prefix_match(d, sp)

    ms_p = _time_events(stream, flush, matches, 30) / reps
    assert int(lcp[0].item()) >= 2100
    out["prefix_match"] = {
        "workload": "two 3900-key prompts sharing a 2100-key prefix",
        "us": ms_p * 1e3, "bytes": 8 * 2101,
        "timing": f"{reps} calls on {reps} prompt pairs per event pair, L2 flushed between pairs"}
    out["retrieval"] = {
        "workload": f"{M} entries (int8 256-d keys, Zipf(1.2) tokens), H={H} bf16 query state",
        "lookup": "pf_retrieval_key + pf_retrieve",
        "timing": f"{reps} lookups on {reps} copies of the memory per event pair, "
                  "L2 flushed between pairs",
        "queries": res}
    return out


ELL_POINTS = (0, 1, 2, 3, 4, 6, 8, 12, 16, 24, 32, 48, 64, 96, 127)
ELL_RATES = (0.3, 0.6, 0.8, 0.9, 0.95, 0.99)


def ell_sweep(base, seed, stream, flush, steps=50, weight_dev=None):
    """Verify-step latency T(l) for chain proposals of l drafts (N = l + 1
    nodes) on the workload's model shape with one sequence and its largest
    prefix: L attention launches, the LM head with acceptance, the commit;
    CUDA-graph steps with events at every step boundary, L2 flushed between
    steps (outside the events), accepted length drawn per step as in the
    main benchmark.  Returns the curve, a log-quadratic least-squares fit
    log T = c0 + c1 l + c2 l^2 (the latency model of eq. 1's controller) and
    the library controller's choices on it at fixed per-token acceptance."""
    import torch
    from paper_2609_32166_gb300 import binding as pb
    from paper_2609_32166_gb300 import inputs as I
    points = []
    for ell in ELL_POINTS:
        w = I.scaled(base, nodes=ell + 1, max_depth=ell, tree="chain", accept="chain", batch=1,
                     layout="contiguous", prefix=(base.prefix[1], base.prefix[1]))
        vs, batch, tok_table, planned = prepare_workload(w, seed, weight_dev)
        if weight_dev is None:
            weight_dev = vs.weight
        per_step, _, _ = time_steps(vs, tok_table, planned, steps, 3, stream, flush, parts=False)
        points.append({"ell": ell, "nodes": ell + 1, "us_step": float(np.mean(per_step)) * 1e3})
        del vs
        torch.cuda.empty_cache()
    ell = np.array([p["ell"] for p in points], dtype=np.float64)
    logt = np.log(np.array([p["us_step"] for p in points]))
    A = np.stack([np.ones_like(ell), ell, ell * ell], axis=1)
    coef, *_ = np.linalg.lstsq(A, logt, rcond=None)
    l_max = ELL_POINTS[-1]
    ctl = pb.pf_controller_init(l_max, 0.05, 0.0)
    for p in points:
        pb.pf_controller_observe(ctl, p["ell"], 0.0, -1, p["us_step"])
    u = np.arange(l_max + 1) / l_max
    t_hat = np.exp(ctl.c[0] + ctl.c[1] * u + ctl.c[2] * u * u)
    choices = []
    for q in ELL_RATES:
        best, obj = pb.pf_length_select(t_hat, np.full(l_max + 1, q), np.full(l_max + 1, q))
        choices.append({"per_token_acceptance": q, "chosen_length": best,
                        "us_per_token": obj, "tokens_per_s": 1e6 / obj})
    return {"workload": f"{base.name} shape, one sequence, prefix {base.prefix[1]}, chain of l "
                        f"drafts", "unit": "us per verify step", "steps_per_point": steps,
            "points": points, "log_quadratic_fit": [float(c) for c in coef],
            "controller": {"l_max": l_max, "latency_model": list(ctl.c), "choices": choices},
            "timing": "CUDA graphs, events around every step; L2 flushed before every step, "
                      "outside the events"}


def run_ell_sweep(args):
    import torch
    import __graft_entry__
    __graft_entry__.build()
    from paper_2609_32166_gb300 import inputs as I
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device="cuda")
    stream = torch.cuda.Stream()
    r = ell_sweep(I.WORKLOADS[args.workload], args.seed, stream, flush, max(10, args.steps))
    print(json.dumps(dict(mode="ell_sweep", **r)))


# ---------------------------------------------------------------------------
# main
# ---------------------------------------------------------------------------
def main():
    args = parse()
    if args.cpu_worker is not None:
        print(json.dumps(cpu_worker(json.loads(args.cpu_worker))))
        return
    if args.impl == "reference":
        run_reference(args)
        return
    if args.ell_sweep:
        run_ell_sweep(args)
        return

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))

    from paper_2609_32166_gb300 import inputs as I
    w = I.WORKLOADS[args.workload]
    if args.layers is not None:
        w = I.scaled(w, layers=max(1, min(args.layers, w.layers)))

    import torch
    import torch.distributed as dist
    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl")

    import __graft_entry__
    # one process per GPU: local rank 0 builds (or finds the library up to
    # date) before the others look, so no two ranks write it at once
    if world > 1 and local != 0:
        dist.barrier()
    __graft_entry__.build()
    if world > 1 and local == 0:
        dist.barrier()

    peaks = load_peaks()
    hbm_peak = peak_values(peaks)[0]
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device="cuda")
    stream = torch.cuda.Stream()
    K = args.steps
    clocks = ClockSampler(torch.cuda.current_device())
    head, vs, batch, tok_table, planned = measure_workload(
        w, args, K, stream, flush, peaks, world=world, dist=dist, clocks=clocks)
    e2e = None if args.no_e2e else run_e2e(vs, w, K, stream, flush, world, tok_table, planned)
    weight_7b = vs.weight if (w.vocab, w.hidden) == (152064, 3584) else None
    if world > 1:
        dist.barrier()
    if rank != 0:
        if world > 1:
            dist.destroy_process_group()
        return
    launches = head["gpu_launches_per_step"]
    del vs
    torch.cuda.empty_cache()

    per_workload = {}
    if not args.no_per_workload and args.layers is None:
        for name in PER_WORKLOAD:
            if name == w.name:
                continue
            wo = I.WORKLOADS[name]
            share = weight_7b if (wo.vocab, wo.hidden) == (152064, 3584) else None
            k_w = max(20, min(K, 200))
            r, vso, *_ = measure_workload(wo, args, k_w, stream, flush, peaks, weight_dev=share)
            del vso
            torch.cuda.empty_cache()
            per_workload[name] = r
    next_rows = None
    if not args.no_next_rows:
        next_rows = measure_next_rows(stream, flush, hbm_peak)
        next_rows["ell_sweep"] = ell_sweep(w, args.seed, stream, flush, 50, weight_dev=weight_7b)
    del weight_7b
    torch.cuda.empty_cache()

    line = {
        "metric": METRIC, "value": head["value"], "unit": "tokens/s", "n_gpus": world, "steps": K,
        "warmup": args.warmup, "ms_per_step": head["ms_per_step"], "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": w.dtype,
        "data": "synthetic (seeded device generator; shapes and distributions of the named "
                "workload)",
        "config": config_dict(w, args),
    }
    for k in ("accepted_tokens_per_step", "us_per_layer_attention", "us_lmhead", "us_commit",
              "parts", "step_hbm_gbs", "step_hbm_frac", "step_bytes", "step_roofline",
              "roofline", "other_roofline", "clocks"):
        line[k] = head[k]
    line["gpu_launches"] = K * launches
    line["timing"] = ("step time: CUDA graphs of up to 50 steps with events at every step "
                      "boundary, exactly %d steps; per-part times: a second pass of %d steps with "
                      "events around every step's parts" % (K, head["parts"]["steps"]))
    line["e2e"] = e2e
    line["per_workload"] = per_workload
    line["next_rows"] = next_rows
    if not args.no_cpu_baseline and world == 1:
        spec = dict(workload=w.name, seed=args.seed, layers=args.layers, warmup=0, steps=1)
        line["cpu_baseline"] = cpu_baseline_entry(w, spec)
        for name, r in per_workload.items():
            wo = I.WORKLOADS[name]
            if cpu_mode(wo) == "whole":
                r["cpu_baseline"] = cpu_baseline_entry(
                    wo, dict(workload=name, seed=args.seed, warmup=0, steps=1))
    print(json.dumps(line))
    if world > 1:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
