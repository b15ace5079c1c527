"""Benchmark of the verify step (tree attention x L layers, LM head with
greedy acceptance, KV commit) on seeded synthetic inputs.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME]
    python bench.py --impl reference ...      # the fp64 CPU oracle, timed

Prints one JSON line.  The metric is accepted tokens/s of whole verify steps
(sum over sequences of accepted drafts + 1 bonus token, divided by the step
time), with the attention time per layer and the step's achieved HBM
bandwidth alongside.  Every step is one CUDA-graph segment: L attention
launches, one LM-head launch, one commit launch.  Between steps a 256 MB
memset evicts L2; each step is bracketed by its own CUDA events, so the
flush is outside the measured time.  Multi-GPU runs are independent
replicas (one process per GPU under torchrun); the value is the sum of
tokens over ranks divided by the slowest rank's time.
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
DEFAULT_WORKLOAD = "2b-bf16-chain16"
L2_FLUSH_BYTES = 256 << 20
# the reference arm (the fp64 oracle on the host cores) times the requested
# steps, or as many as fit this much wall time
REFERENCE_WALL_BUDGET_S = 150.0
CSRC = os.path.join(ROOT, "paper_2609_32166_gb300", "csrc")
# Committed ncu DRAM-traffic summaries, each valid only for the kernel sources
# it was captured on (a fingerprint of the files that define the kernel and
# its launch shape).
LMHEAD_TRAFFIC = (os.path.join(ROOT, "profiles", "lmhead_traffic.txt"),
                  ("lmhead.cu", "pf_ptx.cuh"))
ATTENTION_TRAFFIC = (os.path.join(ROOT, "profiles", "attention_traffic.txt"),
                     ("api.cu", "attention.cu", "attention_tc.cu", "attention_tc2.cu",
                      "attn_common.cuh", "pf_internal.h", "pf_ptx.cuh"))


def parse():
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
                   help="skip the key re-rotation and retrieval measurements")
    p.add_argument("--ell-sweep", action="store_true",
                   help="verify-step latency vs proposal length on the workload's chain shape")
    p.add_argument("--cpu-worker", default=None, help=argparse.SUPPRESS)
    return p.parse_args()


# ---------------------------------------------------------------------------
# algorithmic bytes
# ---------------------------------------------------------------------------
def step_bytes(w, batch, accept_lens):
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


def kernel_roofline(kernel, dtype, bytes_per_launch, flops_per_launch, seconds_per_launch,
                    launches_per_step, step_seconds, peaks, traffic):
    """Roofline of one kernel from its algorithmic bytes and FLOPs per launch
    and its mean in-step launch time.  The bound is the tensor pipe when the
    arithmetic intensity of a bf16 kernel lies above the ridge of the two
    measured peaks (bf16 sustained, since every kernel here is timed inside a
    long run, over copy bandwidth), else HBM."""
    hbm = peaks.get("hbm_gbs")
    tc = peaks.get("bf16_tflops_sustained")
    hbm_src = "measured copy bandwidth" if hbm else "fallback copy bandwidth"
    tc_src = "measured bf16 sustained" if tc else "fallback bf16 sustained"
    hbm = hbm or 6800.0
    tc = tc or 1700.0
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
    nl = spec["layers_sample"]
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
        scale = w.layers / nl
        est = (t_attn + t_commit) * scale + t_lm
        return est, sum(a[0] + 1 for a in acc)

    times, toks = [], []
    n = spec.get("steps")
    if n is None:   # time-bounded sample for cpu_baseline
        t_start = time.perf_counter()
        while (time.perf_counter() - t_start < spec["budget_s"] or not times) and len(times) < 50:
            est, tok = one_step()
            times.append(est)
            toks.append(tok)
    else:
        for _ in range(spec["warmup"]):
            one_step()
        counter[0] = 0
        # the requested steps, or as many as fit the wall budget (at least one)
        t_start = time.perf_counter()
        budget = spec.get("wall_budget_s")
        for _ in range(n):
            if times and budget is not None and time.perf_counter() - t_start > budget:
                break
            est, tok = one_step()
            times.append(est)
            toks.append(tok)
    return dict(step_s=float(np.mean(times)), steps=len(times),
                tokens_per_step=float(np.mean(toks)))


def run_cpu_worker(spec: dict) -> dict:
    cores = os.cpu_count() or 1
    env = dict(os.environ)
    for k in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS"):
        env[k] = str(cores)
    env["CUDA_VISIBLE_DEVICES"] = ""
    r = subprocess.run([sys.executable, os.path.abspath(__file__), "--cpu-worker", json.dumps(spec)],
                       capture_output=True, text=True, env=env, cwd=ROOT)
    if r.returncode != 0:
        raise RuntimeError("CPU oracle worker failed:\n" + r.stderr[-2000:])
    out = json.loads(r.stdout.strip().splitlines()[-1])
    out["cores"] = cores
    return out


def cpu_sample_text(w, nl):
    return (f"whole verify steps of {w.name} in fp64 numpy: attention of {nl} of {w.layers} "
            f"layers (time scaled by {w.layers}/{nl}), full LM head ({w.vocab}x{w.hidden}), "
            f"acceptance, commit")


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
    nl = 1
    spec = dict(workload=args.workload, seed=args.seed, layers_sample=nl, steps=args.steps,
                warmup=args.warmup, wall_budget_s=REFERENCE_WALL_BUDGET_S)
    t0 = time.perf_counter()
    r = run_cpu_worker(spec)
    wall = time.perf_counter() - t0
    value = r["tokens_per_step"] / r["step_s"]
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s",
        "n_gpus": args.gpus, "steps": r["steps"], "steps_requested": args.steps,
        "warmup": args.warmup,
        "ms_per_step": r["step_s"] * 1e3, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic (seeded generator)",
        "config": config_dict(w, args),
        "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": r["cores"],
                         "kind": "oracle",
                         "sample": cpu_sample_text(w, nl) +
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
# our arm
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

    cpu_base = None
    from paper_2609_32166_gb300 import inputs as I
    w = I.WORKLOADS[args.workload]
    if args.layers is not None:
        w = I.scaled(w, layers=max(1, min(args.layers, w.layers)))
    nl_cpu = 1
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        # before any CUDA call in this process
        cpu_base = run_cpu_worker(dict(workload=args.workload, seed=args.seed,
                                       layers_sample=nl_cpu, budget_s=12.0, layers=w.layers))

    import torch
    import torch.distributed as dist
    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl")

    import __graft_entry__
    __graft_entry__.build()
    from paper_2609_32166_gb300.step import VerifyStep

    batch = I.make_batch(w, args.seed)
    vs = VerifyStep(w, batch, np.zeros(batch.total_nodes, np.int32))
    # plant the draft tokens from the model's own greedy predictions so the
    # accepted length is the planted one
    vs.lmhead()
    torch.cuda.synchronize()
    greedy = vs.argmax.cpu().numpy()
    # every step verifies a new proposal: the planted accepted path of step k
    # follows the workload's rule, drawn from a seeded per-step stream
    K = args.steps
    G = max(d for d in range(1, min(K, 50) + 1) if K % d == 0)
    ends = I.step_forced_ends(batch, G)
    depth = [I.node_depths(p) for p in batch.parents]
    planned = [int(sum(depth[b][e[b]] + 1 for b in range(w.batch))) for e in ends]
    tok_table = torch.from_numpy(np.stack([I.plant_tokens(batch, greedy, e, salt=g)
                                           for g, e in enumerate(ends)])).cuda()
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device="cuda")

    stream = torch.cuda.Stream()
    torch.cuda.synchronize()
    with torch.cuda.stream(stream):
        for k in range(max(args.warmup, 3)):
            flush.zero_()
            vs.tokens.copy_(tok_table[k % G])
            vs.step()
            stream.synchronize()
            got = int((vs.accept_len + 1).sum().item())
            assert got == planned[k % G], (k, got, planned[k % G])
    accepted_steps = [planned[k % G] for k in range(K)]

    # one graph = G steps; each step: flush, tokens | e0 attention e1 lmhead e2 commit e3
    per_step, attn_t, lm_t, commit_t = [], [], [], []

    def collect(e, parts=True):
        per_step.append(e[0].elapsed_time(e[3]))
        if parts:
            attn_t.append(e[0].elapsed_time(e[1]))
            lm_t.append(e[1].elapsed_time(e[2]))
            commit_t.append(e[2].elapsed_time(e[3]))

    try:
        torch.cuda.Event(enable_timing=True, external=True)
        graph_events = True
    except TypeError:
        graph_events = False
    clocks = ClockSampler(torch.cuda.current_device())
    if graph_events:
        R = K // G
        # step boundaries carry events in every step; the part boundaries
        # (which break the programmatic-dependent-launch chain between the
        # last layer, the LM head and the commit) only in the first step of
        # each graph, which provides the per-kernel breakdown
        ev = [[torch.cuda.Event(enable_timing=True, external=True) for _ in range(4)]
              for _ in range(G)]
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=stream):
            s = torch.cuda.current_stream()
            for g in range(G):
                flush.zero_()
                vs.tokens.copy_(tok_table[g])
                ev[g][0].record(s)
                for l in range(vs.L):
                    vs.attention(l, s.cuda_stream)
                if g == 0:
                    ev[g][1].record(s)
                vs.lmhead(s.cuda_stream)
                if g == 0:
                    ev[g][2].record(s)
                vs.commit(s.cuda_stream)
                ev[g][3].record(s)
        with torch.cuda.stream(stream):
            graph.replay()   # untimed: uploads the graph
        stream.synchronize()
        clocks.start()
        time.sleep(0.3)
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize()
        with torch.cuda.stream(stream):
            for r in range(R):
                graph.replay()
                # the event nodes hold this replay's timestamps: read them
                # before the next replay overwrites them
                stream.synchronize()
                for g in range(G):
                    collect(ev[g], parts=(g == 0))
    else:
        # torch without external graph events: one graph per part, events
        # recorded between graph launches
        parts = []
        for fn in (lambda st: [vs.attention(l, st) for l in range(vs.L)],
                   lambda st: vs.lmhead(st), lambda st: vs.commit(st)):
            gr = torch.cuda.CUDAGraph()
            with torch.cuda.graph(gr, stream=stream):
                fn(torch.cuda.current_stream().cuda_stream)
            parts.append(gr)
        with torch.cuda.stream(stream):
            for gr in parts:
                gr.replay()
        stream.synchronize()
        ev = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(K)]
        clocks.start()
        time.sleep(0.3)
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize()
        with torch.cuda.stream(stream):
            for k in range(K):
                flush.zero_()
                vs.tokens.copy_(tok_table[k % G])
                ev[k][0].record(stream)
                parts[0].replay()
                ev[k][1].record(stream)
                parts[1].replay()
                ev[k][2].record(stream)
                parts[2].replay()
                ev[k][3].record(stream)
        stream.synchronize()
        for k in range(K):
            collect(ev[k])
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    clk = clocks.stop()
    assert len(per_step) == K
    t_total_ms = max_over_ranks(float(np.sum(per_step)), world, "cuda")
    res = vs.results()
    assert res["err"] == 0, f"device error flag {res['err']}"
    assert int(np.sum(res["accept_len"] + 1)) == accepted_steps[-1]

    ms_step = t_total_ms / K
    accepted = float(np.mean(accepted_steps))
    value = whole_job_rate(float(np.sum(accepted_steps)), t_total_ms / 1e3, world)
    attn_b, lm_b, commit_b = step_bytes(w, batch, res["accept_len"])
    attn_b_layer = attn_b
    step_b = attn_b * w.layers + lm_b + commit_b
    lm_ms = float(np.mean(lm_t))
    attn_ms = float(np.mean(attn_t))
    peaks = {}
    pk = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(pk):
        peaks = json.load(open(pk))
    hbm_peak = peaks.get("hbm_gbs", 6800.0)
    roofline, other_roofline = step_rooflines(w, batch, attn_b_layer,
                                              attn_ms * 1e-3 / w.layers, lm_b, lm_ms * 1e-3,
                                              ms_step * 1e-3, peaks)

    e2e = None if args.no_e2e else run_e2e(vs, w, batch, K, stream, flush, world, tok_table,
                                           planned)
    if rank != 0:
        if world > 1:
            dist.destroy_process_group()
        return
    next_rows = None if args.no_next_rows else measure_next_rows(stream, flush, hbm_peak)
    line = {
        "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": K,
        "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": w.dtype,
        "data": "synthetic (seeded generator, shapes of the named workload)",
        "config": config_dict(w, args),
        "accepted_tokens_per_step": accepted,
        "us_per_layer_attention": attn_ms * 1e3 / w.layers,
        "us_lmhead": lm_ms * 1e3, "us_commit": float(np.mean(commit_t)) * 1e3,
        "step_hbm_gbs": step_b / (ms_step * 1e-3) / 1e9,
        "step_hbm_frac": step_b / (ms_step * 1e-3) / 1e9 / hbm_peak,
        "step_bytes": step_b,
        "roofline": roofline,
        "other_roofline": other_roofline,
        "gpu_launches": K * vs.launches_per_step(),
        "timing": ("CUDA graphs of %d steps; event nodes at every step boundary, and around "
                   "the attention / LM-head / commit parts of the first step of each graph "
                   "(those give the per-part times)" % G
                   if graph_events else "one CUDA graph per part, events between graph launches"),
        "clocks": clk,
        "e2e": e2e,
        "next_rows": next_rows,
    }
    if cpu_base is not None:
        line["cpu_baseline"] = {"value": cpu_base["tokens_per_step"] / cpu_base["step_s"],
                                "unit": "tokens/s", "cores": cpu_base["cores"], "kind": "oracle",
                                "sample": cpu_sample_text(w, nl_cpu) +
                                f"; {cpu_base['steps']} step(s) timed"}
    print(json.dumps(line))
    if world > 1:
        dist.destroy_process_group()


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
    try:
        ev = [(torch.cuda.Event(enable_timing=True, external=True),
               torch.cuda.Event(enable_timing=True, external=True)) for _ in range(iters)]
    except TypeError:
        ev = None
    if ev is not None:
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
    """Rolling-image key re-rotation and decoding-memory retrieval, each on a
    workload of the paper's shape, timed with CUDA events on the launching
    stream.  Each timed iteration makes `reps` calls on `reps` disjoint
    buffers (every call cold in L2; L2 flushed between iterations), so the
    fixed cost of the event pair is spread over several calls."""
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


def run_ell_sweep(args):
    """Verify-step latency T(l) for chain proposals of l drafts (N = l + 1
    nodes) on the workload's model shape and prefix: L attention launches,
    the LM head with acceptance, the commit; CUDA-graph steps with events
    at every step boundary, L2 flushed between steps (outside the events),
    accepted length drawn per step as in the main benchmark.  Prints one
    JSON line with the curve and a log-quadratic least-squares fit
    log T = c0 + c1 l + c2 l^2 (the latency model of eq. 1's controller)."""
    import torch
    import __graft_entry__
    __graft_entry__.build()
    from paper_2609_32166_gb300 import inputs as I
    from paper_2609_32166_gb300.step import VerifyStep
    base = I.WORKLOADS[args.workload]
    weight = I.lm_weight(base, args.seed)
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device="cuda")
    stream = torch.cuda.Stream()
    K = max(10, args.steps)
    G = max(d for d in range(1, min(K, 50) + 1) if K % d == 0)
    points = []
    for ell in ELL_POINTS:
        w = I.scaled(base, nodes=ell + 1, max_depth=ell, tree="chain", accept="chain", batch=1,
                     layout="contiguous")
        batch = I.make_batch(w, args.seed)
        vs = VerifyStep(w, batch, np.zeros(batch.total_nodes, np.int32), weight=weight)
        vs.lmhead()
        torch.cuda.synchronize()
        greedy = vs.argmax.cpu().numpy()
        ends = I.step_forced_ends(batch, G)
        toks = torch.from_numpy(np.stack([I.plant_tokens(batch, greedy, e, salt=g)
                                          for g, e in enumerate(ends)])).cuda()
        with torch.cuda.stream(stream):
            for k in range(max(args.warmup, 3)):
                flush.zero_()
                vs.tokens.copy_(toks[k % G])
                vs.step(stream.cuda_stream)
        stream.synchronize()
        ev = [(torch.cuda.Event(enable_timing=True, external=True),
               torch.cuda.Event(enable_timing=True, external=True)) for _ in range(G)]
        gr = torch.cuda.CUDAGraph()
        with torch.cuda.graph(gr, stream=stream):
            st = torch.cuda.current_stream()
            for g in range(G):
                flush.zero_()
                vs.tokens.copy_(toks[g])
                ev[g][0].record(st)
                vs.step(st.cuda_stream)
                ev[g][1].record(st)
        times = []
        with torch.cuda.stream(stream):
            gr.replay()   # untimed: uploads the graph
            stream.synchronize()
            for r in range(K // G):
                gr.replay()
                stream.synchronize()
                times.extend(a.elapsed_time(b) for a, b in ev)
        res = vs.results()
        assert res["err"] == 0
        del vs, gr
        torch.cuda.empty_cache()
        points.append({"ell": ell, "nodes": ell + 1, "us_step": float(np.mean(times)) * 1e3})
    ell = np.array([p["ell"] for p in points], dtype=np.float64)
    logt = np.log(np.array([p["us_step"] for p in points]))
    A = np.stack([np.ones_like(ell), ell, ell * ell], axis=1)
    coef, *_ = np.linalg.lstsq(A, logt, rcond=None)
    # eq. 1 driven by the measured curve: the library's controller fits its
    # latency model to the points; for a per-token acceptance rate q (p1 =
    # pc = q) the chosen length and the resulting tokens per second
    from paper_2609_32166_gb300 import binding as pb
    l_max = ELL_POINTS[-1]
    ctl = pb.pf_controller_init(l_max, 0.05, 0.0)
    for p in points:
        pb.pf_controller_observe(ctl, p["ell"], 0.0, -1, p["us_step"])
    u = np.arange(l_max + 1) / l_max
    t_hat = np.exp(ctl.c[0] + ctl.c[1] * u + ctl.c[2] * u * u)
    choices = []
    for q in (0.3, 0.6, 0.8, 0.9, 0.95, 0.99):
        best, obj = pb.pf_length_select(t_hat, np.full(l_max + 1, q), np.full(l_max + 1, q))
        choices.append({"per_token_acceptance": q, "chosen_length": best,
                        "us_per_token": obj, "tokens_per_s": 1e6 / obj})
    print(json.dumps({"mode": "ell_sweep", "workload": base.name, "unit": "us per verify step",
                      "steps_per_point": K, "points": points,
                      "log_quadratic_fit": [float(c) for c in coef],
                      "controller": {"l_max": l_max, "latency_model": list(ctl.c),
                                     "choices": choices},
                      "timing": "CUDA graphs of %d steps, events around every step; L2 "
                                "flushed before every step, outside the events" % G}))


def run_e2e(vs, w, batch, K, stream, flush, world, tok_table, planned):
    """Same metric through host buffers: every step copies its inputs (the
    queries, proposal K/V of every layer, hidden states, tokens, tree and
    lengths: one packed arena) from pinned host memory, runs the step and
    reads its outputs (accepted lengths, tokens, new lengths: one arena)
    back."""
    import torch
    host_in = vs.in_arena.detach().cpu().pin_memory()
    host_out = torch.empty(vs.out_arena.numel(), dtype=torch.uint8).pin_memory()
    tok_off = vs.tokens.data_ptr() - vs.in_arena.data_ptr()
    tok_bytes = vs.tokens.numel() * vs.tokens.element_size()
    host_tokens = [t.cpu().contiguous().view(torch.uint8) for t in tok_table]
    acc_off = vs.accept_len.data_ptr() - vs.out_arena.data_ptr()
    h2d = host_in.numel()
    d2h = host_out.numel()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        vs.step(torch.cuda.current_stream().cuda_stream)
    with torch.cuda.stream(stream):
        g.replay()
    stream.synchronize()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    times = []
    tok = 0
    n = min(K, 200)
    with torch.cuda.stream(stream):
        for k in range(n):
            flush.zero_()
            host_in[tok_off:tok_off + tok_bytes].copy_(host_tokens[k % len(host_tokens)])
            e0.record(stream)
            vs.in_arena.copy_(host_in, non_blocking=True)
            g.replay()
            host_out.copy_(vs.out_arena, non_blocking=True)
            e1.record(stream)
            stream.synchronize()
            times.append(e0.elapsed_time(e1))
            acc = host_out[acc_off:acc_off + 4 * w.batch].view(torch.int32)
            got = int((acc + 1).sum())
            assert got == planned[k % len(planned)]
            tok += got
    t = max_over_ranks(float(np.sum(times)), world, "cuda")
    return {"value": whole_job_rate(tok, t * 1e-3, world), "unit": "tokens/s",
            "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "steps": n, "ms_per_step": t / n,
            "copies_per_step": {"h2d": 1, "d2h": 1}}


if __name__ == "__main__":
    main()
