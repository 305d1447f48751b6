#!/usr/bin/env python3
"""Benchmark of the gradient-coding hot path on one GB300 (or N replicas).

Default workload (the headline): the decode-dominated batch -- m = N = 256
workers/chunks, cyclic assignment with delta = 16 chunks per worker, given
chunk gradients of length d = 2^20 (fp32 ~ N(0,1), 1.07 GB), 4096 straggler
patterns per step (per pattern a completion fraction f ~ U[0.2, 1], psi_j ~
Binomial(16, f)), communication factor l = 2.

One step (every row of the PS's decode path once, on a fresh pattern batch):
  1. Algorithm 1 for all 4096 patterns -> decode plan,
     coefficient error and estimate                      (gc_decode_plan)
  2. the batched decode: 4096 decoded gradients (17.2 GB)
     written, with each pattern's gradient MSE            (gc_decode_apply)
Both are captured once in a CUDA graph per double buffer; event-record nodes
in instrumented copies time each call inside the timed region.  Step inputs
(the pattern batch) and results (the decoded gradients and per-pattern errors)
are double-buffered so that copies overlap the next step.

Metric: decoded gradients per second (whole job).  `e2e` repeats the timed
loop through the same C-ABI calls with each step's pattern batch copied from
pinned host memory and its 4096 decoded gradients (16 GiB) and per-pattern
errors copied back to pinned host memory.  `--workload` selects the other
configurations (one JSON line each); `--impl reference` times the fp64 CPU
oracle on the host cores instead.
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

def metric_decode(ell: int) -> str:
    return ("decoded gradients/sec (decode-dominated batch: m=N=256, delta=16, d=2^20, "
            f"4096 straggler patterns per step, l={ell})")


def metric_logistic(ell: int) -> str:
    return f"decoded gradients/sec (logistic m=N=20, delta=4, d=4096, 10^4 realizations, l={ell})"


UNIT = "decoded gradients/s"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=None,
                    help="timed steps (default 60 for the decode batch, 200 for logistic)")
    ap.add_argument("--warmup", type=int, default=None,
                    help="untimed warm-up steps (default 10 for the decode batch, 20 for logistic)")
    ap.add_argument("--impl", choices=["gc", "reference"], default="gc")
    ap.add_argument("--ell", type=int, default=2)
    ap.add_argument("--workload", default="decode",
                    choices=["decode", "logistic", "sweep", "sgd", "trigger", "batched", "chunkgrad",
                             "encode"],
                    help="decode: the headline step (default); logistic: the logistic-regression "
                         "step (N replicas like the headline).  The others measure the remaining "
                         "configurations, one JSON line each (1 GPU)")
    ap.add_argument("--small", action="store_true",
                    help="with --workload batched: a 134 MB case (N=64, n_c=1024, d=1024: the "
                         "same tile counts, short K for GEMM 1) for profiler captures instead of "
                         "the 8.6 GB one; with --workload sweep: given chunk gradients instead of "
                         "X (the decode-combine alone, for profiler captures); with --workload "
                         "decode: 256 patterns per step (profiler captures)")
    ap.add_argument("--decode-policy", default="auto", choices=["auto", "dense", "residual"],
                    help="with --workload sweep: the batched decode's path (gc_set_decode_policy); "
                         "dense forces the tensor-core GEMM for profiler captures of it")
    ap.add_argument("--shape", default=None,
                    help="with --workload chunkgrad: one case 'dtype,N,n_c,d' (dtype f32 or bf16) "
                         "timed over --steps calls after --warmup calls, instead of the table of "
                         "8.6 GB cases")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-extras", action="store_true",
                    help="decode: skip the tensor-GEMM and chunk-gradient side measurements")
    ap.add_argument("--min-warm-seconds", type=float, default=1.5,
                    help="keep warming up at least this long (steady clocks, clock samples)")
    a = ap.parse_args()
    dflt = {"decode": (60, 10), "logistic": (200, 20)}.get(a.workload, (10, 3))
    if a.steps is None:
        a.steps = dflt[0]
    if a.warmup is None:
        a.warmup = dflt[1]
    return a


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return d, "measured"
    return FALLBACK_PEAKS, "fallback"


# ------------------------------------------------------------------ clocks
class Clocks:
    """nvidia-smi samples every 200 ms while the GPU is under load."""
    Q = ("index,uuid,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, uuid: str | None):
        self.uuid = uuid
        self.proc = None
        self.path = None

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            cmd = ["nvidia-smi", f"--query-gpu={self.Q}", "--format=csv,noheader,nounits", "-lms", "200"]
            if self.uuid:
                cmd += ["-i", self.uuid]
            self.proc = subprocess.Popen(cmd, stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self) -> dict:
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        sm, mx, reasons, power = [], [], set(), []
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        with open(self.path) as f:
            for line in f:
                parts = [x.strip() for x in line.split(",")]
                if len(parts) < 10:
                    continue
                try:
                    sm.append(float(parts[2]))
                    mx.append(float(parts[3]))
                    power.append(float(parts[4]))
                except ValueError:
                    continue
                for n, v in zip(names, parts[6:10]):
                    if v.lower().startswith("active"):
                        reasons.add(n)
        os.unlink(self.path)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "samples": len(sm),
                "power_w_max": max(power) if power else None, "reasons": sorted(reasons)}


# ------------------------------------------------------------------ multi-rank bookkeeping
def max_over_ranks(values, world, device="cpu"):
    """Element-wise max of per-rank timings (the slowest rank decides)."""
    import torch

    t = torch.tensor([float(v) for v in values], dtype=torch.float64, device=device)
    if world > 1:
        import torch.distributed as tdist
        tdist.all_reduce(t, op=tdist.ReduceOp.MAX)
    return t.tolist()


def job_rate(units_per_rank, world, ms):
    """Whole-job throughput: units all ranks processed / slowest rank's time."""
    return world * units_per_rank / (ms / 1e3)


# ------------------------------------------------------------------ oracle timing
def oracle_step_rate(cfg, data_cpu, ell, n_sample, seed_stream):
    """Time the fp64 oracle on this host: one full chunk-gradient pass plus
    `n_sample` realizations through Algorithm 1, encode and decode; returns
    (decoded gradients/s extrapolated to the full batch, seconds used)."""
    import oracle as O
    from workloads import make_patterns, make_R

    N, m, delta = cfg.N, cfg.m, cfg.delta
    order = O.cyclic_order(N, m, delta)
    R = make_R(cfg, ell)
    X, y, w = data_cpu["X"].numpy(), data_cpu["y"].numpy(), data_cpu["w"].numpy()
    t0 = time.perf_counter()
    G = O.chunk_gradients(X, y, w, N, cfg.n_c, O.LOGISTIC)
    t_cg = time.perf_counter() - t0
    psi = make_patterns(cfg, npat=n_sample, stream=seed_stream)
    t1 = time.perf_counter()
    for b in range(n_sample):
        O.run_pattern(R, order, psi[b], N, G, want_transmit=True)
    t_pat = (time.perf_counter() - t1) / n_sample
    step = t_cg + cfg.npat * t_pat
    return cfg.npat / step, time.perf_counter() - t0, t_cg, t_pat


def reference_arm(args, rank, world):
    from workloads import get, make_data

    if rank != 0:
        return
    if args.workload == "decode":
        reference_decode(args, world)
        return
    if args.workload != "logistic":
        print(json.dumps({"impl": "reference", "unavailable": "the reference arm times the decode "
                          "and logistic workloads; the other workload lines carry the oracle as "
                          "cpu_baseline"}), flush=True)
        return
    cfg = get("logistic")
    data = make_data(cfg, "cpu")
    n_sample = 64
    for t in range(args.warmup):
        oracle_step_rate(cfg, data, args.ell, 8, 10_000 + t)
    rates, t_all = [], time.perf_counter()
    for t in range(args.steps):
        r, _, _, _ = oracle_step_rate(cfg, data, args.ell, n_sample, 20_000 + t)
        rates.append(r)
    wall = time.perf_counter() - t_all
    value = statistics.median(rates)
    cores = os.cpu_count()
    line = {
        "impl": "reference", "metric": metric_logistic(args.ell), "value": value, "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * cfg.npat / value,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic",
        "config": {"workload": "logistic m=N=20 delta=4 d=4096 n_c=512 npat=10000 ell=%d" % args.ell,
                   "l2": "inputs larger than L2 (X 168 MB)"},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                         "sample": f"each step: full fp64 chunk-gradient pass + {n_sample} realizations "
                                   "(Algorithm 1 per worker, eq. 2 encode, decode), extrapolated to 10^4; "
                                   "pattern loop single-threaded NumPy"},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
        "wall_s": wall,
    }
    print(json.dumps(line), flush=True)


# ------------------------------------------------------------------ GPU arm
def _src_hash(names):
    h = hashlib.sha256()
    for n in names:
        with open(os.path.join(ROOT, "paper_2405_19509_gb300", "csrc", n), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def _traffic(kernel, src_files):
    """dram bytes per launch from a committed ncu summary, if it was taken
    on the current kernel source (else None)."""
    p = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(p):
        return None
    with open(p) as f:
        d = json.load(f)
    e = d.get(kernel)
    if not e or e.get("src_hash") != _src_hash(src_files):
        return None
    return e.get("dram_bytes_per_launch")


def oracle_decode_sample(cfg, ell, G32, psi, cols, min_patterns, max_seconds):
    """Time the fp64 oracle on a bounded sample of the decode workload.

    For each pattern (at least `min_patterns`, more while under `max_seconds`):
    Algorithm 1 in full (every worker's least-squares problem), then the
    eq. (2) encode and the Sec. II-B decode on the first `cols` columns of
    every block (the same block structure on a d' = l * cols problem), the
    latter scaled to the full block length.  Returns seconds per decoded
    gradient and the split."""
    import oracle as O
    from workloads import make_R

    N, m, delta, d = cfg.N, cfg.m, cfg.delta, cfg.d
    L = -(-d // ell)
    S = min(cols, L)
    idx = np.concatenate([k * L + np.arange(S) for k in range(ell)])
    idx = idx[idx < d]
    Gs = G32[:, idx].astype(np.float64)
    order = O.cyclic_order(N, m, delta)
    R = make_R(cfg, ell)
    t_alg = t_cod = 0.0
    n = 0
    t0 = time.perf_counter()
    for b in range(psi.shape[0]):
        if n >= min_patterns and time.perf_counter() - t0 > max_seconds:
            break
        ta = time.perf_counter()
        B = O.encoding_matrix(R, order, psi[b], N)
        tb = time.perf_counter()
        T = O.encode(B, Gs, order, psi[b], ell)
        O.decode(R, T, Gs.shape[1])
        tc = time.perf_counter()
        t_alg += tb - ta
        t_cod += tc - tb
        n += 1
    per = (t_alg + t_cod * (L / S)) / n
    return {"s_per_gradient": per, "patterns": n, "seconds": time.perf_counter() - t0,
            "alg1_s": t_alg / n, "codec_s_sample": t_cod / n, "cols": S}


def reference_decode(args, world):
    """--impl reference for the decode batch: the fp64 oracle on the host
    cores, each step one pattern (Algorithm 1 in full, encode + decode on a
    2^14-column sample of each block, scaled to d = 2^20)."""
    from workloads import get, make_chunk_grads, make_patterns

    cfg = get("decode")
    ell = args.ell
    G32 = make_chunk_grads(cfg, "cpu").numpy()
    psi = make_patterns(cfg, stream=900_000)
    for t in range(args.warmup):
        oracle_decode_sample(cfg, ell, G32, psi[t:t + 1], 1 << 14, 1, 0.0)
    per, t_all = [], time.perf_counter()
    for t in range(args.steps):
        r = oracle_decode_sample(cfg, ell, G32, psi[args.warmup + t:args.warmup + t + 1], 1 << 14, 1, 0.0)
        per.append(r["s_per_gradient"])
    wall = time.perf_counter() - t_all
    value = 1.0 / statistics.median(per)
    line = {
        "impl": "reference", "metric": metric_decode(ell), "value": value, "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * cfg.npat / value,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic",
        "config": {"workload": f"decode m=N=256 delta=16 d=2^20 npat=4096 ell={ell}",
                   "l2": "host run"},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": os.cpu_count(), "kind": "oracle",
                         "sample": "each step one pattern: Algorithm 1 in full (per-worker "
                                   "least squares), eq. (2) encode + Sec. II-B decode on 2^14 "
                                   "columns of each block, scaled to d = 2^20; median over steps"},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
        "wall_s": wall,
    }
    print(json.dumps(line), flush=True)


def decode_arm(args, rank, world, local_rank):
    """The headline: Algorithm 1 + the batched decode of 4096 patterns per step."""
    import dataclasses

    import torch

    import paper_2405_19509_gb300 as gc
    from workloads import get, make_chunk_grads, make_patterns, make_R

    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    cfg = get("decode")
    if args.small:
        cfg = dataclasses.replace(cfg, npat=256)
    N, m, delta, d, npat, ell = cfg.N, cfg.m, cfg.delta, cfg.d, cfg.npat, args.ell
    G = make_chunk_grads(cfg, dev)
    _, order, _ = gc.gc_make_assignment(N, m, delta, gc.GC_CYCLIC)
    Rd = torch.from_numpy(make_R(cfg, ell)).to(dev)
    od = torch.from_numpy(order).to(dev)
    S = args.warmup + args.steps
    nbatch = min(S, 16)   # distinct pattern batches, cycled
    base = 1_000_000 * rank
    psi_host = np.stack([make_patterns(cfg, stream=base + t) for t in range(nbatch)])
    psi_all = torch.from_numpy(psi_host).to(dev)
    # step inputs and results double-buffered (index k % 2)
    psi_b = [torch.empty(npat, m, dtype=torch.int32, device=dev) for _ in range(2)]
    Gh_b = [torch.empty(npat, d, dtype=torch.float32, device=dev) for _ in range(2)]
    ce_b = [torch.empty(npat, dtype=torch.float64, device=dev) for _ in range(2)]
    est_b = [torch.empty(npat, dtype=torch.float64, device=dev) for _ in range(2)]
    mse_b = [torch.empty(npat, dtype=torch.float64, device=dev) for _ in range(2)]
    plan_s = torch.empty(int(gc.lib.gc_decode_plan_bytes(N, ell, npat)), dtype=torch.uint8, device=dev)
    wsP, wsA = gc.Workspace(dev), gc.Workspace(dev)
    bi = [0]

    def stage_plan():   # psi -> Algorithm 1 -> decode plan, coefficient error, estimate
        gc.gc_decode_plan(Rd, ell, od, N, m, delta, psi_b[bi[0]], plan=plan_s, coef_err=ce_b[bi[0]],
                          est=est_b[bi[0]], ws=wsP)

    def stage_apply():  # the batched decode: decoded gradients and their MSE
        gc.gc_decode_apply(plan_s, ell, N, npat, G, Ghat=Gh_b[bi[0]], grad_mse=mse_b[bi[0]], ws=wsA)

    for b in range(2):
        bi[0] = b
        psi_b[b].copy_(psi_all[b % nbatch])
        stage_plan()
        stage_apply()
    gc.gc_status(wsP)
    gc.gc_status(wsA)
    torch.cuda.synchronize()
    ser_ev = [torch.cuda.Event(enable_timing=True) for _ in range(4)]
    for rep in range(3):
        bi[0] = rep % 2
        ser_ev[0].record()
        stage_plan()
        ser_ev[1].record()
        ser_ev[2].record()
        stage_apply()
        ser_ev[3].record()
    torch.cuda.synchronize()
    serial_ms = [ser_ev[0].elapsed_time(ser_ev[1]), ser_ev[2].elapsed_time(ser_ev[3])]

    n0 = gc.gc_kernel_launches()
    cap_stream = torch.cuda.Stream(dev)
    graphs = []
    for b in range(2):
        bi[0] = b
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=cap_stream):
            stage_plan()
            stage_apply()
        graphs.append(g)
        if b == 0:
            launches_per_step = gc.gc_kernel_launches() - n0
    # instrumented copies (buffer 0): event-record nodes around each call
    EVERY, NE = 4, 6
    kev = [[[torch.cuda.Event(enable_timing=True, external=True) for _ in range(2)] for _ in range(2)]
           for _ in range(NE)]
    gi = []
    bi[0] = 0
    for j in range(NE):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=cap_stream):
            kev[j][0][0].record(cap_stream)
            stage_plan()
            kev[j][0][1].record(cap_stream)
            kev[j][1][0].record(cap_stream)
            stage_apply()
            kev[j][1][1].record(cap_stream)
        gi.append(g)
    torch.cuda.synchronize()

    stream = torch.cuda.current_stream(dev)
    copy_stream = torch.cuda.Stream(dev)
    NCOPY = 4
    d2h_streams = [torch.cuda.Stream(dev) for _ in range(NCOPY)]
    ev_d2h = [torch.cuda.Event() for _ in range(NCOPY)]
    ev_ready = [torch.cuda.Event() for _ in range(2)]
    ev_done = [torch.cuda.Event() for _ in range(2)]
    ev_out = [torch.cuda.Event() for _ in range(2)]

    def put_inputs(t, b, src):
        with torch.cuda.stream(copy_stream):
            copy_stream.wait_event(ev_done[b])
            psi_b[b].copy_(src[t % nbatch], non_blocking=True)
            ev_ready[b].record(copy_stream)

    def run_step(k, t_next, src, instrumented=False, outs=None):
        b = k % 2
        g = graphs[b]
        if instrumented:
            assert b == 0
            g = gi[(k // EVERY) % NE]
        if t_next is not None:
            put_inputs(t_next, 1 - b, src)
        stream.wait_event(ev_ready[b])
        stream.wait_event(ev_out[b])  # results of step k - 2 have been read out
        g.replay()
        ev_done[b].record(stream)
        if outs is not None:
            # the decoded gradients leave in NCOPY row blocks on their own
            # streams (one copy engine each), the errors on the copy stream
            for q, cs in enumerate(d2h_streams):
                rows = slice(q * npat // NCOPY, (q + 1) * npat // NCOPY)
                with torch.cuda.stream(cs):
                    cs.wait_event(ev_done[b])
                    outs["Ghat"][rows].copy_(Gh_b[b][rows], non_blocking=True)
                    ev_d2h[q].record(cs)
            with torch.cuda.stream(copy_stream):
                copy_stream.wait_event(ev_done[b])
                outs["ce"][k].copy_(ce_b[b], non_blocking=True)
                outs["est"][k].copy_(est_b[b], non_blocking=True)
                outs["mse"][k].copy_(mse_b[b], non_blocking=True)
                for q in range(NCOPY):
                    copy_stream.wait_event(ev_d2h[q])
                ev_out[b].record(copy_stream)

    import torch.distributed as tdist

    def barrier():
        if world > 1:
            tdist.barrier()

    props = torch.cuda.get_device_properties(dev)
    uuid = getattr(props, "uuid", None)
    clocks = Clocks(f"GPU-{uuid}" if uuid is not None else None)
    clocks.start()
    t_w = time.perf_counter()
    put_inputs(0, 0, psi_all)
    k = 0
    while k < args.warmup or time.perf_counter() - t_w < args.min_warm_seconds:
        run_step(k, k + 1, psi_all)
        k += 1
        if k % 32 == 0:
            torch.cuda.synchronize()
    torch.cuda.synchronize()
    K = args.steps
    barrier()
    torch.cuda.synchronize()
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    wall0 = time.perf_counter()
    t_start.record(stream)
    copy_stream.wait_stream(stream)
    put_inputs(args.warmup, 0, psi_all)
    n_inst = 0
    for k in range(K):
        inst = k % EVERY == 0 and k % 2 == 0
        n_inst += inst
        run_step(k, args.warmup + k + 1 if k + 1 < K else None, psi_all, instrumented=inst)
    t_end.record(stream)
    torch.cuda.synchronize()
    barrier()
    wall = time.perf_counter() - wall0
    clk = clocks.stop()
    total_ms = t_start.elapsed_time(t_end)
    n_used = min(NE, n_inst)
    call_ms = np.array([[kev[j][si][0].elapsed_time(kev[j][si][1]) for si in range(2)]
                        for j in range(n_used)]).mean(axis=0)
    gc.gc_status(wsP)
    gc.gc_status(wsA)
    mse_dev = mse_b[(K - 1) % 2].clone()

    # ---- end to end: pattern batches from pinned host memory, decoded
    # gradients and errors back to pinned host memory, every step
    pin_psi = torch.from_numpy(psi_host).pin_memory()
    outs = {"Ghat": torch.empty(npat, d, dtype=torch.float32).pin_memory(),
            "ce": torch.empty(K, npat, dtype=torch.float64).pin_memory(),
            "est": torch.empty(K, npat, dtype=torch.float64).pin_memory(),
            "mse": torch.empty(K, npat, dtype=torch.float64).pin_memory()}
    barrier()
    torch.cuda.synchronize()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    copy_stream.wait_stream(stream)
    put_inputs(args.warmup, 0, pin_psi)
    for k in range(K):
        run_step(k, args.warmup + k + 1 if k + 1 < K else None, pin_psi, outs=outs)
    stream.wait_stream(copy_stream)
    e1.record(stream)
    torch.cuda.synchronize()
    barrier()
    e2e_ms = e0.elapsed_time(e1)
    assert np.all(np.isfinite(outs["mse"].numpy())) and np.all(outs["est"].numpy() >= 0)
    assert torch.isfinite(outs["Ghat"][:4]).all()
    total_ms, e2e_ms = max_over_ranks([total_ms, e2e_ms], world, dev)
    value = job_rate(npat * K, world, total_ms)
    e2e_value = job_rate(npat * K, world, e2e_ms)

    # ---- roofline of the dominant call (the decode; Algorithm 1 is the other)
    pk, pk_src = peaks()
    hbm = float(pk["hbm_gbs"])
    Kp = -(-N * ell // 64) * 64
    plan_b = 2 * npat * ell * Kp * 2
    apply_bytes = npat * d * 4 + N * d * 4 + plan_b + npat * 8          # Ghat written; G, plan read
    plan_bytes_alg = npat * m * 4 + plan_b + 2 * npat * 8                 # psi read; plan, errors written
    achieved = apply_bytes / (call_ms[1] / 1e3) / 1e9
    roofline = {"kernel": "gc_decode_apply (k_decode_resid + helpers)", "bound": "hbm",
                "achieved": achieved, "peak": hbm, "unit": "GB/s", "frac": achieved / hbm,
                "peak_source": f"{pk_src} hbm_gbs",
                "traffic": _traffic("k_decode_resid", ["k_decode_resid.cu"]),
                "algorithmic_bytes_per_call": apply_bytes,
                "timing": "CUDA events recorded by event nodes inside the step's graph around the "
                          f"gc_decode_apply call (every {EVERY}th timed step, the last {n_used} "
                          "averaged); the call is the plan scan, the residual decode (which also "
                          "forms sum_i g), the operand split and GEMM when a tile needs them, and "
                          "the MSE reduction",
                "call_ms": {"gc_decode_plan (Algorithm 1)": float(call_ms[0]),
                            "gc_decode_apply": float(call_ms[1])},
                "call_GBps": {"gc_decode_plan": plan_bytes_alg / (call_ms[0] / 1e3) / 1e9,
                              "gc_decode_apply": achieved},
                "serial_ms": {"gc_decode_plan": serial_ms[0], "gc_decode_apply": serial_ms[1]}}
    line = {
        "metric": metric_decode(ell), "value": value, "unit": UNIT, "n_gpus": world, "steps": K,
        "warmup": args.warmup, "ms_per_step": total_ms / K, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f32 (Algorithm 1 in f64)",
        "data": "synthetic",
        "config": {"workload": f"decode m=N=256 delta=16 d=2^20 npat={npat} ell={ell}",
                   "l2": "inputs larger than L2 (G 1.07 GB read, Ghat 17.2 GB written per step)",
                   "parallelism": f"replicas x{world} (independent pattern batches)"},
        "roofline": roofline,
        "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": int(npat * m * 4),
                "d2h_bytes_per_step": int(npat * d * 4 + 3 * npat * 8),
                "returns": "the step's decoded gradients (npat x d fp32) and per-pattern "
                           "coefficient error, estimate and gradient MSE"},
        "gpu_launches": int(launches_per_step * K),
        "clocks": clk,
        "wall_s_timed": wall,
        "exact_patterns_frac": float((mse_dev == 0).double().mean()),
    }
    if rank == 0 and world == 1 and not args.no_extras:
        line["extras"] = decode_extras(gc, torch, dev, cfg, ell, G, Rd, od, psi_all[0], plan_s,
                                       wsP, wsA, Gh_b[0], mse_b[0], call_ms, pk, pk_src)
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        G32 = G.cpu().numpy()
        r = oracle_decode_sample(cfg, ell, G32, psi_host[0], 1 << 14, 16, 20.0)
        line["cpu_baseline"] = {
            "value": 1.0 / r["s_per_gradient"], "unit": UNIT, "cores": os.cpu_count(), "kind": "oracle",
            "sample": f"{r['patterns']} patterns of the first batch: Algorithm 1 in full "
                      f"({r['alg1_s']:.2f} s per pattern), eq. (2) encode + Sec. II-B decode on "
                      f"{r['cols']} columns of each block ({r['codec_s_sample']:.2f} s) scaled to "
                      f"d = 2^20; {r['seconds']:.1f} s of CPU work, NumPy with its BLAS threads"}
    if rank == 0:
        print(json.dumps(line), flush=True)


def decode_extras(gc, torch, dev, cfg, ell, G, Rd, od, pd, plan, wsP, wsA, Gh, mse, call_ms, pk, pk_src):
    """Side measurements on the headline workload (not part of the step):
    the same decode forced onto the tensor-core GEMM, and the chunk-gradient
    pass of the coded-SGD workload (8.6 GB fp32 X)."""
    from workloads import make_data
    from workloads import get as get_cfg

    N, m, delta, d, npat = cfg.N, cfg.m, cfg.delta, cfg.d, cfg.npat
    out = {}
    bf16s = float(pk.get("bf16_tflops_sustained", pk["bf16_tflops"]))
    gc.gc_decode_plan(Rd, ell, od, N, m, delta, pd, plan=plan, coef_err=False, est=False, ws=wsP)
    gc.gc_set_decode_policy(gc.GC_DECODE_DENSE)
    try:
        t_dense = _time_ms(torch, lambda: gc.gc_decode_apply(plan, ell, N, npat, G, Ghat=Gh,
                                                             grad_mse=mse, ws=wsA), 3)
    finally:
        gc.gc_set_decode_policy(gc.GC_DECODE_AUTO)
    gc.gc_status(wsA)
    L = -(-d // ell)
    Kp = -(-N * ell // 64) * 64
    useful = 2.0 * npat * ell * (N * ell) * L
    issued = 3 * 2.0 * npat * ell * Kp * L
    out["decode_on_tensor_cores"] = {
        "ms_apply": t_dense, "decoded_gradients_per_s_apply_only": npat / (t_dense / 1e3),
        "useful_tflops": useful / (t_dense / 1e3) / 1e12, "issued_tflops": issued / (t_dense / 1e3) / 1e12,
        "frac_useful_of_bf16_sustained": useful / (t_dense / 1e3) / 1e12 / bf16s,
        "frac_issued_of_bf16_sustained": issued / (t_dense / 1e3) / 1e12 / bf16s,
        "note": "gc_decode_apply with every tile on the bf16x3 tcgen05 GEMM (gc_set_decode_policy "
                "DENSE), operand split included; useful = 2 npat N l^2 L, issued = 3 MMAs per K "
                "step over the padded K; peak = measured bf16 sustained",
        "residual_path_speedup": t_dense / float(call_ms[1])}
    sg = get_cfg("sgd")
    data = make_data(sg, dev)
    Gc = torch.empty(sg.N, sg.d, device=dev)
    lo = torch.zeros(1, dtype=torch.float64, device=dev)
    ws = gc.Workspace(dev)
    t_cg = _time_ms(torch, lambda: gc.gc_chunk_grads(data["X"], data["y"], data["w"], sg.N, sg.n_c,
                                                     gc.GC_LOGISTIC, G=Gc, loss_out=lo, ws=ws), 5)
    gc.gc_status(ws)
    nbytes = sg.Ntil * sg.d * 4 + sg.Ntil * 4 + sg.N * sg.d * 4
    out["chunk_grads"] = {
        "workload": "sgd m=N=128 n_c=2048 d=8192 fp32 X (8.6 GB), logistic, with the loss",
        "ms": t_cg, "GB/s": nbytes / (t_cg / 1e3) / 1e9,
        "frac_of_hbm": nbytes / (t_cg / 1e3) / 1e9 / float(pk["hbm_gbs"]),
        "TFLOP/s": 4.0 * sg.Ntil * sg.d / (t_cg / 1e3) / 1e12,
        "note": "two matrix-vector products per chunk (HBM-bound); TFLOP/s = 4 N~ d / t"}
    del data, Gc
    torch.cuda.empty_cache()
    return out


def logistic_arm(args, rank, world, local_rank):
    import torch

    import paper_2405_19509_gb300 as gc
    from workloads import get, make_data, make_patterns, make_R

    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    cfg = get("logistic")
    N, m, delta, d, n_c, ell, npat = cfg.N, cfg.m, cfg.delta, cfg.d, cfg.n_c, args.ell, cfg.npat
    L = -(-d // ell)
    data_cpu = make_data(cfg, "cpu")
    X = data_cpu["X"].to(dev)
    y = data_cpu["y"].to(dev)
    w = data_cpu["w"].to(dev).clone()
    _, order, _ = gc.gc_make_assignment(N, m, delta, gc.GC_CYCLIC)
    Rd = torch.from_numpy(make_R(cfg, ell)).to(dev)
    od = torch.from_numpy(order).to(dev)
    S = args.warmup + args.steps
    # realizations: each rank draws its own batches (replicas over independent patterns)
    base = 1_000_000 * rank
    psi_host = np.stack([make_patterns(cfg, stream=base + t) for t in range(S)])
    live_host = np.stack([make_patterns(cfg, npat=1, stream=base + 500_000 + t) for t in range(S)])
    psi_all = torch.from_numpy(psi_host).to(dev)
    live_all = torch.from_numpy(live_host).to(dev)
    # static buffers
    # step inputs and per-step results are triple-buffered (index t % NB) so
    # that step t + 1's inputs are copied in, and earlier steps' results out,
    # on a copy stream while step t runs
    NB = 3
    psi_b = [torch.empty(npat, m, dtype=torch.int32, device=dev) for _ in range(NB)]
    live_b = [torch.empty(1, m, dtype=torch.int32, device=dev) for _ in range(NB)]
    loss_b = [torch.zeros(1, dtype=torch.float64, device=dev) for _ in range(NB)]
    ce_b = [torch.empty(npat, dtype=torch.float64, device=dev) for _ in range(NB)]
    est_b = [torch.empty(npat, dtype=torch.float64, device=dev) for _ in range(NB)]
    mse_b = [torch.empty(npat, dtype=torch.float64, device=dev) for _ in range(NB)]
    # the chunk gradients and the decode plan are triple-buffered too: the
    # batched decode of step t reads them while step t + 1 computes its own
    G_b = [torch.empty(N, d, dtype=torch.float32, device=dev) for _ in range(NB)]
    plan_b = [torch.empty(int(gc.lib.gc_decode_plan_bytes(N, ell, npat)), dtype=torch.uint8, device=dev)
              for _ in range(NB)]
    Gh_s = torch.empty(npat, d, dtype=torch.float32, device=dev)
    T_s = torch.empty(1, m, L, dtype=torch.float32, device=dev)
    E_s = torch.empty(1, m, delta, ell, dtype=torch.float64, device=dev)
    gh_s = torch.empty(1, d, dtype=torch.float32, device=dev)
    wsA, wsB, wsC, wsD = (gc.Workspace(dev) for _ in range(4))

    bi = [0]  # buffer the stage functions use (set before each capture / eager call)

    def stage_a():
        gc.gc_chunk_grads(X, y, w, N, n_c, gc.GC_LOGISTIC, G=G_b[bi[0]], loss_out=loss_b[bi[0]], ws=wsA)

    # set-up, once per (R, assignment) like the assignment itself: the holder
    # table and Algorithm 1's solution for every (chunk, holder subset)
    prep = gc.gc_decode_prepare(Rd, ell, od, N, m, delta)

    def stage_b():  # Algorithm 1 for the batch -> decode plan (psi side, no G needed)
        gc.gc_decode_plan_prepared(prep, Rd, ell, N, m, delta, psi_b[bi[0]], plan=plan_b[bi[0]],
                                   coef_err=ce_b[bi[0]], est=est_b[bi[0]], ws=wsB)

    def stage_c():  # batched decode-combine from the plan and G
        gc.gc_decode_apply(plan_b[bi[0]], ell, N, npat, G_b[bi[0]], Ghat=Gh_s, grad_mse=mse_b[bi[0]],
                           ws=wsC)

    def stage_d1():  # Algorithm 1 for the live realization (independent of G)
        gc.gc_find_encoding_coeff(Rd, ell, od, N, m, delta, live_b[bi[0]], E=E_s, C=False,
                                  delta_out=False, support=False, coef_err=False, est=False, ws=wsD)

    def stage_d2():  # eq. (2) encode, PS decode, update: one launch
        gc.gc_live_step(E_s, Rd, ell, od, N, m, delta, live_b[bi[0]], G_b[bi[0]], w, cfg.lr,
                        cfg.Ntil, T=T_s, ghat=gh_s)

    stages = [stage_a, stage_b, stage_c, stage_d1, stage_d2]
    # eager run: allocates workspaces, checks the device status words
    psi_b[0].copy_(psi_all[0])
    live_b[0].copy_(live_all[0])
    for f in stages:
        f()
    for ws in (wsA, wsB, wsC, wsD):
        gc.gc_status(ws)
    torch.cuda.synchronize()
    # each stage alone (informational, before the timed loop): its own graph
    # replayed back to back, events on the replay stream; w is restored after
    # the repeated updates
    w_saved = w.clone()
    alone_stream = torch.cuda.Stream(dev)
    bi[0] = 0
    alone_ms = []
    for f in stages:
        ga_ = torch.cuda.CUDAGraph()
        with torch.cuda.graph(ga_, stream=alone_stream):
            f()
        with torch.cuda.stream(alone_stream):
            ga_.replay()
            ea0 = torch.cuda.Event(enable_timing=True)
            ea1 = torch.cuda.Event(enable_timing=True)
            ea0.record(alone_stream)
            for _ in range(10):
                ga_.replay()
            ea1.record(alone_stream)
        torch.cuda.synchronize()
        alone_ms.append(ea0.elapsed_time(ea1) / 10)
        del ga_
    w.copy_(w_saved)
    torch.cuda.synchronize()

    # two graphs per step on two streams.  g1 runs the chunk gradients (A)
    # with Algorithm 1 for the live realization (D1) and for the batch (B) on
    # high-priority side streams beside it, then the live encode / decode /
    # update (D2), which gives the next step's w.  g2 is the batched decode
    # (C); it needs A and B of its step but nothing of the next one, so it
    # runs on its own stream while g1 of the next step streams X (the chunk
    # gradients and the plan are triple-buffered; a step's g1 waits for the
    # decode of three steps before, which read its buffers).
    n0 = gc.gc_kernel_launches()
    cap_stream = torch.cuda.Stream(dev)
    cap_hi = [torch.cuda.Stream(dev, priority=-1) for _ in range(2)]

    def fork_join(main_fns, *side_lists):
        fork = torch.cuda.Event()
        fork.record(cap_stream)
        for f in main_fns:
            f()
        joins = []
        for side, fns in zip(cap_hi, side_lists):
            side.wait_event(fork)
            with torch.cuda.stream(side):
                for f in fns:
                    f()
                joins.append(torch.cuda.Event())
                joins[-1].record(side)
        for j in joins:
            cap_stream.wait_event(j)

    def timed(f, ev):
        # event-record nodes around f on the capture stream (the kernel's stream)
        def g():
            ev[0].record(cap_stream)
            f()
            ev[1].record(cap_stream)
        return g

    g1, g2 = [], []
    for b in range(NB):
        bi[0] = b
        g1.append(torch.cuda.CUDAGraph())
        g2.append(torch.cuda.CUDAGraph())
        with torch.cuda.graph(g1[b], stream=cap_stream):
            fork_join([stage_a], [stage_d1], [stage_b])
            stage_d2()
        with torch.cuda.graph(g2[b], stream=cap_stream):
            stage_c()
        if b == 0:
            launches_per_step = gc.gc_kernel_launches() - n0
    # instrumented copies of buffer 0's graphs for every EVERY-th timed step:
    # event-record nodes bracket the chunk-gradient call (A) and the
    # decode-combine call (C) on their own stream inside the graph; NE copies
    # with their own events, cycled, so the last NE instrumented steps each
    # leave a sample
    EVERY, NE = 8 * NB, 8
    kev = [[[torch.cuda.Event(enable_timing=True, external=True) for _ in range(2)] for _ in range(2)]
           for _ in range(NE)]
    g1i, g2i = [], []
    bi[0] = 0
    for j in range(NE):
        g1i.append(torch.cuda.CUDAGraph())
        g2i.append(torch.cuda.CUDAGraph())
        with torch.cuda.graph(g1i[j], stream=cap_stream):
            fork_join([timed(stage_a, kev[j][0])], [stage_d1], [stage_b])
            stage_d2()
        with torch.cuda.graph(g2i[j], stream=cap_stream):
            timed(stage_c, kev[j][1])()
    torch.cuda.synchronize()

    # g1 (the chunk gradients and the update: the step's critical path) on a
    # high-priority stream, g2 (the batched decode) on a low-priority one:
    # when SMs free up the block scheduler takes g1's blocks first, so the
    # decode's many small blocks do not hold the chunk-gradient kernel (one
    # block per SM) back
    stream = torch.cuda.Stream(dev, priority=-1)
    dec_stream = torch.cuda.Stream(dev, priority=0)  # the batched decode (g2)

    copy_stream = torch.cuda.Stream(dev)
    ev_ready = [torch.cuda.Event() for _ in range(NB)]  # inputs of the buffer's next step are in
    ev_g1 = [torch.cuda.Event() for _ in range(NB)]     # the buffer's g1 has finished
    ev_done = [torch.cuda.Event() for _ in range(NB)]   # the buffer's step (g1 and g2) has finished
    ev_out = [torch.cuda.Event() for _ in range(NB)]    # the buffer's results have been read out

    def put_inputs(t, b, src):
        """Copy step t's realizations into buffer b on the copy stream, once
        the step that last used buffer b has finished."""
        with torch.cuda.stream(copy_stream):
            copy_stream.wait_event(ev_done[b])
            psi_b[b].copy_(src[0][t], non_blocking=True)
            live_b[b].copy_(src[1][t], non_blocking=True)
            ev_ready[b].record(copy_stream)

    def run_step(k, t, t_next, src, evs=None, outs=None):
        """Step k on realization batch t (buffer k % NB, whose inputs are
        already being copied in); queues the copy of batch t_next into the
        other buffer, runs g1 and g2 and, with `outs`, copies the step's
        results to host memory on the copy stream.  With evs (instrumented
        steps, buffer 0) evs[0..3] bracket g1 and g2 and the graphs are the
        instrumented copy (k // EVERY) % NE."""
        b = k % NB
        ga, gb = g1[b], g2[b]
        if evs is not None:
            assert b == 0
            ga, gb = g1i[(k // EVERY) % NE], g2i[(k // EVERY) % NE]

        def rec(i, st):
            if evs is not None:
                evs[i].record(st)
        if t_next is not None:
            put_inputs(t_next, (k + 1) % NB, src)
        stream.wait_event(ev_ready[b])
        stream.wait_event(ev_done[b])  # the decode of step k - NB has read this buffer's G and plan
        stream.wait_event(ev_out[b])   # results of step k - NB have been read out
        with torch.cuda.stream(stream):  # replay() launches on the current stream
            rec(0, stream)
            ga.replay()
            rec(1, stream)
        ev_g1[b].record(stream)
        dec_stream.wait_event(ev_g1[b])
        with torch.cuda.stream(dec_stream):
            rec(2, dec_stream)
            gb.replay()
            rec(3, dec_stream)
        ev_done[b].record(dec_stream)
        if outs is not None:
            with torch.cuda.stream(copy_stream):
                copy_stream.wait_event(ev_done[b])
                outs[0][k].copy_(ce_b[b], non_blocking=True)
                outs[1][k].copy_(est_b[b], non_blocking=True)
                outs[2][k].copy_(mse_b[b], non_blocking=True)
                outs[3][k].copy_(loss_b[b], non_blocking=True)
                ev_out[b].record(copy_stream)

    import torch.distributed as tdist

    def barrier():
        if world > 1:
            tdist.barrier()

    props = torch.cuda.get_device_properties(dev)
    uuid = getattr(props, "uuid", None)
    clocks = Clocks(f"GPU-{uuid}" if uuid is not None else None)
    clocks.start()
    # warm-up: at least W steps and at least --min-warm-seconds
    src_dev = (psi_all, live_all)
    t_w = time.perf_counter()
    put_inputs(0, 0, src_dev)
    k = 0
    while k < args.warmup or time.perf_counter() - t_w < args.min_warm_seconds:
        run_step(k, k % S, (k + 1) % S, src_dev)
        k += 1
        if k % 64 == 0:
            torch.cuda.synchronize()
    torch.cuda.synchronize()

    K = args.steps
    # the stage events bracket g1 and g2 of every EVERY-th timed step
    evs = {k: [torch.cuda.Event(enable_timing=True) for _ in range(4)] for k in range(0, K, EVERY)}
    batch = [(args.warmup + k) % S for k in range(K)]
    barrier()
    torch.cuda.synchronize()
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    wall0 = time.perf_counter()
    t_start.record(stream)
    copy_stream.wait_stream(stream)
    put_inputs(batch[0], 0, src_dev)
    for k in range(K):
        run_step(k, batch[k], batch[k + 1] if k + 1 < K else None, src_dev, evs.get(k))
    stream.wait_stream(dec_stream)
    t_end.record(stream)
    torch.cuda.synchronize()
    barrier()
    wall = time.perf_counter() - wall0
    clk = clocks.stop()
    total_ms = t_start.elapsed_time(t_end)
    stage_ms = np.zeros(2)
    for k, ev in evs.items():
        for si in range(2):
            stage_ms[si] += ev[2 * si].elapsed_time(ev[2 * si + 1])
    stage_ms /= len(evs)
    # kernel-call times from the event nodes: the copies replayed in the timed
    # loop (each holds its last replay's timestamps)
    n_used = min(NE, len(evs))
    call_ms = np.array([[kev[j][si][0].elapsed_time(kev[j][si][1]) for si in range(2)]
                        for j in range(n_used)]).mean(axis=0)
    for ws in (wsA, wsB, wsC, wsD):
        gc.gc_status(ws)

    # ---- end to end through the C-ABI with host buffers
    pin_psi = torch.from_numpy(psi_host).pin_memory()
    pin_live = torch.from_numpy(live_host).pin_memory()
    out_ce = torch.empty(K, npat, dtype=torch.float64).pin_memory()
    out_est = torch.empty(K, npat, dtype=torch.float64).pin_memory()
    out_mse = torch.empty(K, npat, dtype=torch.float64).pin_memory()
    out_loss = torch.empty(K, 1, dtype=torch.float64).pin_memory()
    barrier()
    torch.cuda.synchronize()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    src_host = (pin_psi, pin_live)
    outs = (out_ce, out_est, out_mse, out_loss)
    e0.record(stream)
    copy_stream.wait_stream(stream)
    put_inputs(batch[0], 0, src_host)
    for k in range(K):
        run_step(k, batch[k], batch[k + 1] if k + 1 < K else None, src_host, None, outs)
    stream.wait_stream(copy_stream)  # the last step's results are in host memory
    e1.record(stream)
    torch.cuda.synchronize()
    barrier()
    e2e_ms = e0.elapsed_time(e1)
    assert np.all(np.isfinite(out_mse.numpy())) and np.all(out_est.numpy() >= 0)

    # ---- max over ranks
    total_ms, e2e_ms = max_over_ranks([total_ms, e2e_ms], world, dev)
    value = job_rate(npat * K, world, total_ms)
    e2e_value = job_rate(npat * K, world, e2e_ms)

    # ---- roofline of the dominant stage
    pk, pk_src = peaks()
    hbm = float(pk["hbm_gbs"])
    names = ["k_chunkgrad", "k_patterns", "gc_decode_apply", "k_patterns(live)",
             "encode+decode_tx+sgd"]
    alg_bytes = [
        cfg.Ntil * d * 4 + cfg.Ntil * 4 + N * d * 4,                          # X, y read; G written
        npat * m * 4 + npat * ell * N * ell * 4 + 2 * npat * 8,               # psi read; C (hi+lo), errors written
        npat * d * 4 + npat * ell * N * ell * 4 + N * d * 4 + npat * 8,       # Ghat written; C (hi+lo), G read
        m * 4 + m * delta * ell * 8,                                          # psi read; E written
        N * d * 4 + m * L * 4 * 2 + d * 4 * 3,                                # G read; T; ghat; w
    ]
    srcs = [["k_chunkgrad.cu"], ["k_solve.cu"], ["k_decode_resid.cu"], ["k_solve.cu"],
            ["k_encode.cu"]]
    # the dominant kernel: the longer of the two HBM-bound calls on the
    # critical path (chunk gradients in g1, decode-combine in g2)
    di = 0 if call_ms[0] >= call_ms[1] else 1
    dom = (0, 2)[di]
    achieved = alg_bytes[dom] / (call_ms[di] / 1e3) / 1e9
    roofline = {"kernel": names[dom], "bound": "hbm", "achieved": achieved, "peak": hbm,
                "unit": "GB/s", "frac": achieved / hbm, "peak_source": f"{pk_src} hbm_gbs",
                "traffic": _traffic(names[dom], srcs[dom]),
                "timing": "CUDA events recorded by event nodes inside the step's graphs, on the "
                          "call's stream, around the call (the chunk-gradient kernel with its "
                          "reduction; the batched decode with its scan, s and MSE reduction), "
                          f"in every {EVERY}th timed step (the last {n_used} averaged); the "
                          "decode of step t runs beside the chunk gradients of step t + 1",
                "call_ms": {"k_chunkgrad (+ reduction)": float(call_ms[0]),
                            "gc_decode_apply": float(call_ms[1])},
                "call_frac_of_hbm": {"k_chunkgrad": float(alg_bytes[0] / (call_ms[0] / 1e3) / 1e9 / hbm),
                                     "gc_decode_apply": float(alg_bytes[2] / (call_ms[1] / 1e3) / 1e9 / hbm)},
                "graph_ms": {"g1: k_chunkgrad || Algorithm 1, then live encode/decode/update": float(stage_ms[0]),
                             "g2: batched decode": float(stage_ms[1])},
                "alone_graph_ms": {n: float(v) for n, v in zip(names, alone_ms)},
                "alone_frac_of_hbm": {names[i]: float(alg_bytes[i] / (alone_ms[i] / 1e3) / 1e9 / hbm)
                                      for i in (0, 2)}}

    line = {
        "metric": metric_logistic(ell), "value": value, "unit": UNIT, "n_gpus": world, "steps": K,
        "warmup": args.warmup, "ms_per_step": total_ms / K, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": {"workload": "logistic m=N=20 delta=4 d=4096 n_c=512 npat=10000 ell=%d" % ell,
                   "l2": "inputs larger than L2 (X 168 MB, Ghat 164 MB per step)",
                   "parallelism": f"replicas x{world} (independent realization batches)"},
        "roofline": roofline,
        "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": int(npat * m * 4 + m * 4),
                "d2h_bytes_per_step": int(3 * npat * 8 + 8)},
        "gpu_launches": int(launches_per_step * K),
        "clocks": clk,
        "wall_s_timed": wall,
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        rate, used, t_cg, t_pat = oracle_step_rate(cfg, data_cpu, ell, 256, 7_777)
        line["cpu_baseline"] = {
            "value": rate, "unit": UNIT, "cores": os.cpu_count(), "kind": "oracle",
            "sample": f"full fp64 chunk-gradient pass ({t_cg:.3f} s, BLAS threads) + 256 realizations "
                      f"({1e3 * t_pat:.2f} ms each, single-threaded NumPy), extrapolated to 10^4; "
                      f"{used:.1f} s of CPU work"}
    if rank == 0:
        print(json.dumps(line), flush=True)


# ------------------------------------------------------------------ other workloads
def _time_ms(torch, f, reps, warm=2, flush=None):
    """Mean CUDA-event time of f() (ms); the L2 is flushed before each rep."""
    for _ in range(warm):
        f()
    torch.cuda.synchronize()
    tot = 0.0
    for _ in range(reps):
        if flush is not None:
            flush.zero_()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        f()
        e1.record()
        torch.cuda.synchronize()
        tot += e0.elapsed_time(e1)
    return tot / reps


def _graph_time_ms(torch, f, reps, flush, warm=2):
    """Mean CUDA-event time (ms) of f() captured once in a CUDA graph and
    replayed: the per-call host work of the binding is out of the timed
    region, and the L2 is flushed before each replay.  f must size its
    workspace and take preallocated outputs (it runs once before capture)."""
    f()
    torch.cuda.synchronize()
    side = torch.cuda.Stream()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=side):
        f()
    for _ in range(warm):
        g.replay()
    torch.cuda.synchronize()
    tot = 0.0
    for _ in range(reps):
        flush.zero_()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        g.replay()
        e1.record()
        torch.cuda.synchronize()
        tot += e0.elapsed_time(e1)
    del g
    return tot / reps


def extra_workload(args):
    """One JSON line for a non-headline configuration (single GPU)."""
    import torch

    import paper_2405_19509_gb300 as gc
    from workloads import (get, make_R, make_chunk_grads, make_data, make_patterns,
                           make_worker_times, random_regular_graph)

    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    pk, pk_src = peaks()
    hbm, bf16 = float(pk["hbm_gbs"]), float(pk["bf16_tflops"])
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    n0 = gc.gc_kernel_launches()
    ell = args.ell
    line = {"workload": args.workload, "n_gpus": 1, "data": "synthetic", "dtype": "f32"}
    if args.workload == "encode":
        # eq. (2) on the decode workload's chunk gradients (A4 alone, from
        # Algorithm 1's worker coefficients): per pattern G is read and T written
        cfg = get("decode")
        N, m, delta, d = cfg.N, cfg.m, cfg.delta, cfg.d
        G = make_chunk_grads(cfg, dev)
        _, order, _ = gc.gc_make_assignment(N, m, delta)
        Rd = torch.from_numpy(make_R(cfg, ell)).to(dev)
        od = torch.from_numpy(order).to(dev)
        psi_all = make_patterns(cfg)
        L = -(-d // ell)
        rows = {}
        for ne in (1, 8):
            pe = torch.from_numpy(psi_all[:ne]).to(dev)
            E = gc.gc_find_encoding_coeff(Rd, ell, od, N, m, delta, pe, E=True, C=False, delta_out=False,
                                          coef_err=False, est=False)["E"]
            T = torch.empty(ne, m, L, device=dev)
            t = _time_ms(torch, lambda: gc.gc_encode_with_coeffs(E, ell, od, N, m, delta, pe, G, T=T),
                         max(3, args.steps), warm=max(2, args.warmup), flush=flush)
            alg = ne * (N * d * 4 + m * L * 4)
            dram = N * d * 4 + ne * m * L * 4
            rows[ne] = {"patterns": ne, "ms": t, "GB/s": alg / (t / 1e3) / 1e9,
                        "frac_of_hbm": alg / (t / 1e3) / 1e9 / hbm,
                        "GB/s_G_once": dram / (t / 1e3) / 1e9}
            del T, E
        line.update({
            "metric": f"encode GB/s (eq. 2; m=N=256, delta=16, d=2^20, l={ell}, 1 pattern)",
            "value": rows[1]["GB/s"], "unit": "GB/s", "per_patterns": rows,
            "roofline": {"kernel": "k_encode", "bound": "hbm", "unit": "GB/s",
                         "achieved": rows[1]["GB/s"], "peak": hbm, "frac": rows[1]["frac_of_hbm"],
                         "traffic": _traffic("k_encode", ["k_encode.cu"]),
                         "note": "algorithmic bytes per pattern: G read once (N d 4) + T written "
                                 "(m L 4); GB/s_G_once counts G once for the whole call",
                         "peak_source": f"{pk_src} hbm_gbs"},
            "config": {"workload": f"encode m=N=256 delta=16 d=2^20 ell={ell}, 1 and 8 patterns",
                       "l2": "L2 flushed before each timed call (G 1.07 GB)"}})
    elif args.workload == "sweep":
        cfg = get("mse_sweep")
        N, m, delta, d, npat = cfg.N, cfg.m, cfg.delta, cfg.d, cfg.npat
        if args.small:
            # profiler captures of the decode-combine: given chunk gradients, no X
            G = make_chunk_grads(cfg, dev)
            t_cg = float("nan")
        else:
            data = make_data(cfg, dev)
            G = torch.empty(N, d, device=dev)
            wsA = gc.Workspace(dev)
            t_cg = _time_ms(torch, lambda: gc.gc_chunk_grads(data["X"], data["y"], data["w"], N, cfg.n_c,
                                                             gc.GC_LSQ, G=G, ws=wsA), 5)
            del data
            torch.cuda.empty_cache()
        _, order, _ = gc.gc_make_assignment(N, m, delta)
        Rd = torch.from_numpy(make_R(cfg, ell)).to(dev)
        od = torch.from_numpy(order).to(dev)
        wsM = gc.Workspace(dev)
        wsP, wsA2 = gc.Workspace(dev), gc.Workspace(dev)
        gc.gc_set_decode_policy({"auto": gc.GC_DECODE_AUTO, "dense": gc.GC_DECODE_DENSE,
                                 "residual": gc.GC_DECODE_RESIDUAL}[args.decode_policy])
        res = {}
        t_mse_tot = 0.0
        L = -(-d // ell)
        K = N * ell
        Kp = -(-K // 64) * 64
        # FP32 multiply-add peak from the unit counts: 128 lanes an SM, 2 flops each
        sm_count = torch.cuda.get_device_properties(dev).multi_processor_count
        fp32_peak = sm_count * 128 * 2 * 2.07e9 / 1e12
        ntile = -(-K // 64)
        gram_flops = 2.0 * (ntile * (ntile + 1) // 2) * 64 * 64 * L  # upper-triangle 64 x 64 tiles
        outs = {k: torch.empty(npat, dtype=torch.float64, device=dev) for k in ("ce", "est", "mse")}
        for p in (0.3, 0.5, 0.7):
            psi_h = make_patterns(cfg, p=p)
            pd = torch.from_numpy(psi_h).to(dev)
            # each call captured in a CUDA graph, the L2 flushed before each replay
            t = _graph_time_ms(torch, lambda: gc.gc_mse(Rd, ell, od, N, m, delta, pd, G,
                                                        coef_err=outs["ce"], est=outs["est"],
                                                        grad_mse=outs["mse"], ws=wsM), 5, flush)
            out = gc.gc_mse(Rd, ell, od, N, m, delta, pd, G, ws=wsM)
            gc.gc_status(wsM)
            # the same work as two calls: Algorithm 1 into a plan, then the errors
            pl = gc.gc_decode_plan(Rd, ell, od, N, m, delta, pd, ws=wsP)
            mse_a = torch.empty(npat, dtype=torch.float64, device=dev)
            t_plan = _graph_time_ms(torch, lambda: gc.gc_decode_plan(Rd, ell, od, N, m, delta, pd,
                                                                     plan=pl["plan"],
                                                                     coef_err=pl["coef_err"],
                                                                     est=pl["est"], ws=wsP), 5, flush)
            t_apply = _graph_time_ms(torch, lambda: gc.gc_decode_apply(pl["plan"], ell, N, npat, G,
                                                                       Ghat=False, grad_mse=mse_a,
                                                                       ws=wsA2), 5, flush)
            gc.gc_status(wsP)
            gc.gc_status(wsA2)
            # useful flops of the quadratic forms: 2 nz^2 a row, nz = its non-zero entries
            cs = pl["plan"][:2 * npat * ell * Kp * 2].view(torch.bfloat16).view(2, npat * ell, Kp)
            v = (cs[0, :, :K].float() + cs[1, :, :K].float())
            eye = (torch.arange(K, device=dev) % ell)[None, :] == (torch.arange(npat * ell, device=dev) % ell)[:, None]
            nz = ((v - eye.float()) != 0).sum(dim=1).double()
            form_flops = float(2.0 * (nz * nz).sum())
            del cs, v, eye, nz
            res[str(p)] = {"ms": t, "patterns/s": npat / (t / 1e3),
                           "plan_ms": t_plan, "apply_ms": t_apply,
                           "apply_tflops": (gram_flops + form_flops) / (t_apply / 1e3) / 1e12,
                           "mean_grad_mse": float(out["grad_mse"].mean()),
                           "mean_coef_err": float(out["coef_err"].mean()),
                           "mean_est": float(out["est"].mean())}
            t_mse_tot += t
        t_mse = t_mse_tot / 3
        r3 = res["0.3"]
        roof = {"kernel": "gc_decode_apply errors only (k_gram_partial, k_gram_reduce, "
                          "k_mse_gram) at p = 0.3, the densest decode matrices",
                "bound": "alu", "unit": "TFLOP/s",
                "achieved": r3["apply_tflops"], "peak": fp32_peak,
                "frac": r3["apply_tflops"] / fp32_peak,
                "note": "each pattern's MSE is a quadratic form in the Gram matrix of the "
                        "N*l chunk blocks; flops = the Gram matrix's upper-triangle tiles "
                        "(2 * 64 * 64 * L each) + 2 nz^2 for every decode row with nz "
                        "non-zero entries of C - I; the sums read H from shared memory "
                        "(one load a multiply-add), which caps them near a quarter of the "
                        "FP32 rate; the timed gc_mse also runs Algorithm 1 (plan_ms)",
                "peak_source": f"derived: {sm_count} SMs x 128 FP32 lanes x 2 flops x 2.07 GHz"}
        if args.decode_policy == "dense":
            # every row tile on the bf16x3 tensor-core GEMM: three MMAs per K step
            issued = 3 * 2.0 * npat * ell * Kp * L
            bf16s = float(pk.get("bf16_tflops_sustained", bf16))
            roof = {"kernel": "gc_decode_apply errors only on the GEMM (k_split_gt, k_combine_tc) "
                              "at p = 0.3", "bound": "tensor", "unit": "TFLOP/s",
                    "achieved": issued / (r3["apply_ms"] / 1e3) / 1e12, "peak": bf16s,
                    "frac": issued / (r3["apply_ms"] / 1e3) / 1e12 / bf16s,
                    "useful_tflops": 2.0 * npat * ell * K * L / (r3["apply_ms"] / 1e3) / 1e12,
                    "note": "issued = three bf16 MMAs per K step over the padded K "
                            "(gc_set_decode_policy(DENSE)); apply_tflops per p assumes the "
                            "Gram path and does not apply",
                    "peak_source": f"{pk_src} bf16_tflops_sustained"}
        line.update({
            "metric": f"patterns/sec (MSE only, m=N=64, delta=8, d=65536, 10^5 patterns, l={ell})",
            "value": npat / (t_mse / 1e3), "unit": "patterns/s",
            "chunk_grads": {"ms": t_cg, "GB/s": cfg.Ntil * d * 2 / (t_cg / 1e3) / 1e9,
                            "frac_of_hbm": cfg.Ntil * d * 2 / (t_cg / 1e3) / 1e9 / hbm,
                            "TFLOP/s": 4.0 * cfg.Ntil * d / (t_cg / 1e3) / 1e12},
            "per_p": res,
            "roofline": roof,
            "dtype": "bf16 X, f32 otherwise",
            "config": {"workload": f"sweep m=N=64 delta=8 d=65536 n_c=1024 bf16 npat=10^5 ell={ell}",
                       "decode_policy": args.decode_policy,
                       "l2": "chunk gradients: inputs larger than L2 (X 8.6 GB); error calls: "
                             "L2 flushed before each replay of the call's CUDA graph"}})
        gc.gc_set_decode_policy(gc.GC_DECODE_AUTO)
    elif args.workload == "sgd":
        cfg = get("sgd")
        N, m, delta, d = cfg.N, cfg.m, cfg.delta, cfg.d
        data = make_data(cfg, dev, w_which="zero")
        X, y, w = data["X"], data["y"], data["w"].clone()
        _, order, _ = gc.gc_make_assignment(N, m, delta)
        Rd = torch.from_numpy(make_R(cfg, ell)).to(dev)
        od = torch.from_numpy(order).to(dev)
        psi = torch.from_numpy(np.stack([make_patterns(cfg, npat=1, stream=t)[0]
                                         for t in range(cfg.iters)])).to(dev)
        G = torch.empty(N, d, device=dev)
        loss = torch.zeros(cfg.iters, dtype=torch.float64, device=dev)
        ws = gc.Workspace(dev)
        L = -(-d // ell)
        T = torch.empty(1, m, L, device=dev)
        gh = torch.empty(1, d, device=dev)

        def run():
            for it in range(cfg.iters):
                gc.gc_chunk_grads(X, y, w, N, cfg.n_c, gc.GC_LOGISTIC, G=G, loss_out=loss[it:it + 1], ws=ws)
                gc.gc_encode(Rd, ell, od, N, m, delta, psi[it:it + 1], G, T=T, ws=ws)
                gc.gc_decode_tx(Rd, ell, m, T, d, ghat=gh)
                gc.gc_sgd_step(w, gh[0], cfg.lr, cfg.Ntil)
        w0 = w.clone()
        run()  # sizes the workspace; then the 64 iterations are one CUDA graph
        torch.cuda.synchronize()
        w.copy_(w0)
        g64 = torch.cuda.CUDAGraph()
        cap = torch.cuda.Stream(dev)
        with torch.cuda.graph(g64, stream=cap):
            run()
        torch.cuda.synchronize()
        w.copy_(w0)
        t = _time_ms(torch, g64.replay, 3, warm=1)
        w.copy_(w0)
        t_cg = _time_ms(torch, lambda: gc.gc_chunk_grads(X, y, w, N, cfg.n_c, gc.GC_LOGISTIC, G=G, ws=ws), 5)
        gc.gc_status(ws)
        line.update({
            "metric": f"coded SGD iterations/sec (m=N=128, delta=6, d=8192, n_c=2048, l={ell})",
            "value": cfg.iters / (t / 1e3), "unit": "iterations/s", "ms_64_iterations": t,
            "note": "the 64 iterations (chunk gradients, Algorithm 1 + encode of the live "
                    "realization, PS decode, update) replayed as one CUDA graph",
            "roofline": {"kernel": "k_chunkgrad", "bound": "hbm", "unit": "GB/s",
                         "achieved": cfg.Ntil * d * 4 / (t_cg / 1e3) / 1e9, "peak": hbm,
                         "frac": cfg.Ntil * d * 4 / (t_cg / 1e3) / 1e9 / hbm,
                         "ms_chunk_grads": t_cg, "peak_source": f"{pk_src} hbm_gbs"},
            "config": {"workload": f"sgd m=N=128 delta=6 d=8192 n_c=2048 64 iterations ell={ell}",
                       "l2": "inputs larger than L2 (X 8.6 GB)"}})
    elif args.workload == "batched":
        cfg = get("mse_sweep")
        if args.small:
            import dataclasses
            cfg = dataclasses.replace(cfg, N=64, m=64, n_c=1024, d=1024)
        N, d, n_c = cfg.N, cfg.d, cfg.n_c
        data = make_data(cfg, dev)
        X, y = data["X"], data["y"]
        res = {}
        for n_w in ((256,) if args.small else (128, 256)):
            W = torch.randn(n_w, d, generator=torch.Generator(device=dev).manual_seed(n_w),
                            device=dev) / d ** 0.5
            G = torch.empty(n_w, N, d, device=dev)
            ws = gc.Workspace(dev)
            t = _time_ms(torch, lambda: gc.gc_chunk_grads_batched(X, y, W, N, n_c, gc.GC_LSQ, G=G, ws=ws), 3)
            gc.gc_status(ws)
            useful = 4.0 * cfg.Ntil * d * n_w
            res[n_w] = {"ms": t, "useful_tflops": useful / (t / 1e3) / 1e12,
                        "issued_tflops": 2 * useful / (t / 1e3) / 1e12,
                        "X_read_GBps": 2 * cfg.Ntil * d * 2 / (t / 1e3) / 1e9}
            del G
            torch.cuda.empty_cache()
        r = res[256]
        line.update({
            "metric": f"chunk-gradient TFLOP/s, n_w parameter vectors at once (m=N={N}, d={d}, n_c={n_c}, bf16 X)",
            "value": r["useful_tflops"], "unit": "TFLOP/s (useful)", "per_n_w": res,
            "roofline": {"kernel": "k_gemm_w (two GEMMs)", "bound": "tensor", "unit": "TFLOP/s",
                         "achieved": r["issued_tflops"], "peak": bf16, "frac": r["issued_tflops"] / bf16,
                         "note": "issued = two bf16 MMAs per K step (hi/lo parts of W, R); X is read "
                                 "twice (once per GEMM)",
                         "peak_source": f"{pk_src} bf16_tflops"},
            "dtype": "bf16 X, f32 accumulate",
            "config": {"workload": f"batched chunk gradients N={N} n_c={n_c} d={d} bf16, "
                                   f"n_w={'256' if args.small else '128 and 256'}, lsq",
                       "l2": f"inputs larger than L2 (X {cfg.Ntil * d * 2 / 1e9:.2f} GB)"}})
    elif args.workload == "trigger":
        nsim = 100_000
        rows = {}
        for name, N, nu, alpha_of in (("cyclic N=m=200 delta=8", 200, 8, lambda l: 8 - l),
                                      ("random 8-regular m=200 (Alg. 2 order)", 200, 8, lambda l: 7)):
            if name.startswith("cyclic"):
                _, order, _ = gc.gc_make_assignment(N, N, nu)
                t_alg2 = None
            else:
                A = random_regular_graph(N, nu, 1)
                t0 = time.perf_counter()
                order, _ = gc.gc_chunk_ordering(A)
                t_alg2 = (time.perf_counter() - t0) * 1e3
            od = torch.from_numpy(order).to(dev)
            ws = gc.Workspace(dev)
            for l in (1, 2, 3, 4):
                tau = torch.from_numpy(make_worker_times(N, nsim, 20 + l, alpha=alpha_of(l))).to(dev)
                T = torch.empty(nsim, dtype=torch.float64, device=dev)
                TF = torch.empty_like(T)
                psi = torch.empty(nsim, N, dtype=torch.int32, device=dev)
                t = _time_ms(torch, lambda: gc.gc_trigger_times(od, N, N, nu, tau, l, 0, T=T, psi=psi,
                                                                T_full=TF, ws=ws), 5, flush=flush)
                fin = torch.isfinite(T) & torch.isfinite(TF)
                rows[f"{name}, l={l}"] = {
                    "ms": t, "realizations/s": nsim / (t / 1e3),
                    "mean_T": float(T[fin].mean()), "mean_T_full": float(TF[fin].mean()),
                    "mean_ratio_T_full_over_T": float((TF[fin] / T[fin]).mean()),
                    "alg2_host_ms": t_alg2}
        r0 = rows["cyclic N=m=200 delta=8, l=2"]
        bytes_r = 200 * 8 + 200 * 4 + 16  # tau read, psi written, two times written
        line.update({
            "metric": "simulated realizations/sec (completion time + trigger + psi, N=m=200, delta=8, l=2)",
            "value": r0["realizations/s"], "unit": "realizations/s", "per_case": rows,
            "roofline": {"kernel": "k_trigger", "bound": "hbm", "unit": "GB/s",
                         "achieved": bytes_r * r0["realizations/s"] / 1e9, "peak": hbm,
                         "frac": bytes_r * r0["realizations/s"] / 1e9 / hbm,
                         "note": "latency/ALU-bound selection; bytes = tau read + outputs",
                         "peak_source": f"{pk_src} hbm_gbs"},
            "dtype": "f64",
            "config": {"workload": "trigger cyclic N=m=200 delta=8 alpha=delta-l, 10^5 realizations; "
                                   "and 8-regular m=200 alpha=7",
                       "l2": "L2 flushed before each timed call (tau 160 MB)"}})
    elif args.workload == "chunkgrad":
        # chunk-gradient bandwidth over row lengths: every case reads 8.6 GB of X
        # (one pass), from one CTA per row slice up to clusters of 8
        shapes = [args.shape] if args.shape else [
            "bf16,64,1024,65536", "bf16,128,1024,32768", "bf16,256,1024,16384", "bf16,512,1024,8192",
            "f32,64,512,65536", "f32,128,512,32768", "f32,256,512,16384", "f32,512,512,8192"]
        gen = torch.Generator(device=dev).manual_seed(5)
        rows = {}
        for sh in shapes:
            dt, N, n_c, d = sh.split(",")
            N, n_c, d = int(N), int(n_c), int(d)
            tdt = torch.bfloat16 if dt == "bf16" else torch.float32
            X = torch.empty(N * n_c, d, dtype=tdt, device=dev).normal_(generator=gen).mul_(d ** -0.5)
            y = torch.sign(torch.randn(N * n_c, device=dev, generator=gen))
            w = torch.randn(d, device=dev, generator=gen)
            G = torch.empty(N, d, device=dev)
            lo = torch.zeros(1, dtype=torch.float64, device=dev)
            ws = gc.Workspace(dev)
            t = _time_ms(torch, lambda: gc.gc_chunk_grads(X, y, w, N, n_c, gc.GC_LOGISTIC, G=G,
                                                          loss_out=lo, ws=ws),
                         max(1, args.steps if args.shape else 10), warm=max(1, args.warmup if args.shape else 3),
                         flush=flush if X.numel() * X.element_size() < (256 << 20) else None)
            gc.gc_status(ws)
            nbytes = X.numel() * X.element_size() + N * n_c * 4 + N * d * 4
            rows[sh] = {"ms": t, "GB/s": nbytes / (t / 1e3) / 1e9, "frac_of_hbm": nbytes / (t / 1e3) / 1e9 / hbm}
            del X, y, w, G, ws
            torch.cuda.empty_cache()
        key = shapes[0]
        line.update({
            "metric": f"chunk-gradient bandwidth (logistic, {key})", "value": rows[key]["GB/s"], "unit": "GB/s",
            "per_shape": rows,
            "roofline": {"kernel": "k_chunkgrad", "bound": "hbm", "unit": "GB/s",
                         "achieved": rows[key]["GB/s"], "peak": hbm, "frac": rows[key]["frac_of_hbm"],
                         "note": "bytes = X and y read, G written; k_chunkgrad plus its reduction",
                         "peak_source": f"{pk_src} hbm_gbs"},
            "dtype": "bf16 or f32 X (per shape), f32 accumulate",
            "config": {"workload": "chunk gradients 'dtype,N,n_c,d': " + ", ".join(shapes),
                       "l2": "inputs larger than L2 (8.6 GB per case), else flushed"}})
    line["gpu_launches_total"] = int(gc.gc_kernel_launches() - n0)
    if not args.no_cpu_baseline:
        torch.cuda.synchronize()
        line["cpu_baseline"] = oracle_baseline(args, line)
    print(json.dumps(line), flush=True)


def oracle_baseline(args, line):
    """The fp64 oracle on the host cores, on a bounded sample of the same
    workload (synthetic inputs of the same shapes; the timing does not depend
    on the values), in the unit of the line's metric."""
    import oracle as O
    from workloads import (get, make_patterns, make_R, make_worker_times, random_regular_graph)

    ell = args.ell
    rng = np.random.default_rng(12345)
    cores = os.cpu_count()
    w = args.workload
    t0 = time.perf_counter()

    def chunk_rate(N, n_c, d, dtype, loss, k):
        # k chunks through the oracle's chunk gradient (fp64), seconds per chunk
        X = rng.standard_normal((k * n_c, d), dtype=np.float32)
        if dtype == "bf16":
            import torch
            X = torch.from_numpy(X).to(torch.bfloat16)
        y = np.sign(rng.standard_normal(k * n_c)).astype(np.float32)
        wv = rng.standard_normal(d) / np.sqrt(d)
        ta = time.perf_counter()
        O.chunk_gradients(X, y, wv, k, n_c, loss)
        return (time.perf_counter() - ta) / k

    if w == "encode":
        cfg = get("decode")
        N, m, delta, d = cfg.N, cfg.m, cfg.delta, cfg.d
        L = -(-d // ell)
        S = 1 << 14
        order = O.cyclic_order(N, m, delta)
        psi = make_patterns(cfg, npat=1)[0]
        B = O.encoding_matrix(make_R(cfg, ell), order, psi, N)
        Gs = rng.standard_normal((N, ell * S))
        ta = time.perf_counter()
        O.encode(B, Gs, order, psi, ell)
        t = (time.perf_counter() - ta) * (L / S)
        v = (N * d * 4 + m * L * 4) / t / 1e9
        sample = f"eq. (2) encode of one pattern on {S} columns of each block, scaled to d = 2^20"
    elif w == "sweep":
        cfg = get("mse_sweep")
        N, m, delta, d = cfg.N, cfg.m, cfg.delta, cfg.d
        order = O.cyclic_order(N, m, delta)
        R = make_R(cfg, ell)
        G = rng.standard_normal((N, d))
        psi = make_patterns(cfg, npat=16, p=0.5)
        ta = time.perf_counter()
        for b in range(psi.shape[0]):
            O.run_pattern(R, order, psi[b], N, G, want_transmit=False)
        per = (time.perf_counter() - ta) / psi.shape[0]
        v = 1.0 / per
        cg = chunk_rate(N, cfg.n_c, d, "bf16", O.LSQ, 2)
        sample = (f"16 patterns (p = 0.5): Algorithm 1, decode and errors over all of d "
                  f"({per:.3f} s each); chunk gradients {cg:.2f} s per chunk "
                  f"({N * cg:.1f} s per 8.6 GB pass, from 2 chunks)")
    elif w == "sgd":
        cfg = get("sgd")
        N, m, delta, d = cfg.N, cfg.m, cfg.delta, cfg.d
        cg = chunk_rate(N, cfg.n_c, d, "f32", O.LOGISTIC, 2)
        order = O.cyclic_order(N, m, delta)
        R = make_R(cfg, ell)
        psi = make_patterns(cfg, npat=1)[0]
        G = rng.standard_normal((N, d))
        ta = time.perf_counter()
        B = O.encoding_matrix(R, order, psi, N)
        gh = O.decode(R, O.encode(B, G, order, psi, ell), d)
        O.sgd_step(np.zeros(d), gh, cfg.lr, cfg.Ntil)
        rest = time.perf_counter() - ta
        it = 2 * N * cg + rest   # the loss is a second pass over X in the oracle
        v = 1.0 / it
        sample = (f"chunk gradients of 2 chunks ({cg:.2f} s each), scaled to 128 chunks and counted "
                  f"twice (gradient pass and loss pass); Algorithm 1 + encode + decode + update of "
                  f"one realization ({rest:.2f} s)")
    elif w == "batched":
        cfg = get("mse_sweep")
        cg = chunk_rate(cfg.N, cfg.n_c, cfg.d, "bf16", O.LSQ, 2)
        n_w = 256
        t = cg * cfg.N * n_w
        v = 4.0 * cfg.Ntil * cfg.d * n_w / t / 1e12
        sample = f"one parameter vector, 2 chunks ({cg:.2f} s each), scaled to 64 chunks x 256 vectors"
    elif w == "trigger":
        N, delta = 200, 8
        order = O.cyclic_order(N, N, delta)
        tau = make_worker_times(N, 200, 22, alpha=delta - ell)
        ta = time.perf_counter()
        O.completion_times(order, tau, N, ell)
        v = 200 / (time.perf_counter() - ta)
        sample = "200 realizations, cyclic N=m=200, delta=8, alpha = delta - l"
    elif w == "chunkgrad":
        sh = (args.shape or "bf16,64,1024,65536").split(",")
        dt, N, n_c, d = sh[0], int(sh[1]), int(sh[2]), int(sh[3])
        cg = chunk_rate(N, n_c, d, dt, O.LOGISTIC, 2)
        v = (n_c * d * (2 if dt == "bf16" else 4) + n_c * 4 + d * 4) / cg / 1e9
        sample = f"2 chunks of shape {dt},{n_c}x{d} ({cg:.2f} s each)"
    else:
        return None
    return {"value": v, "unit": line.get("unit"), "cores": cores, "kind": "oracle",
            "sample": sample + f"; {time.perf_counter() - t0:.1f} s of CPU work, NumPy with its BLAS threads"}


def main():
    args = parse()
    if args.workload not in ("decode", "logistic") and args.impl == "gc":
        extra_workload(args)
        return
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        reference_arm(args, rank, world)
        return
    if world > 1:
        import torch
        import torch.distributed as tdist
        torch.cuda.set_device(local_rank)
        tdist.init_process_group("nccl", device_id=torch.device("cuda", local_rank))
    if args.workload == "decode":
        decode_arm(args, rank, world, local_rank)
    else:
        logistic_arm(args, rank, world, local_rank)
    if world > 1:
        import torch.distributed as tdist
        tdist.destroy_process_group()


if __name__ == "__main__":
    main()
