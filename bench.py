"""Benchmark of the stage-boundary codec on GB300.

One step is one pass of the whole boundary for one microbatch of the
large-stream workload (T = 16 x 4096 tokens, d = 8192, k = 82, vocab 128256,
Zipf(1.1) ids, 5% off-subspace energy):

  sn_compress_fwd -> wire (device -> pinned host -> device) -> sn_decompress_fwd
  sn_compress_bwd -> wire -> sn_decompress_bwd
  sn_project_weight of the stage's attention out-projection W_o [8192, 8192]
  (projected every iteration, Sec. 5)

Inputs are resident in HBM when the timed region starts; L2 is flushed (a
512 MiB write, then a read of the same buffer) before every timed step.  `value` is boundary tokens/s over the
whole job; `e2e` is the same metric with the step's activation, ids and
gradient copied in from pinned host memory and the reconstructed activation
and gradient copied back, inside the timed region.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
"""
import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

WORKLOAD = "large"
W_O_SHAPE = (8192, 8192)
# smaller cases with the same step, for profiling (the default is the large stream)
PROFILE_WORKLOADS = {"large": ("large", (8192, 8192)), "8b": ("8b", (4096, 4096)),
                     "1b": ("1b", (2048, 2048))}
METRIC = "boundary tokens/sec (compress+decompress) and achieved HBM GB/s vs GB300 peak"
L2_FLUSH_BYTES = 512 << 20
MIN_TIMED_S = 1.5      # the timed region lasts at least this long (clock samples)


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=300)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--cpu-seconds", type=float, default=12.0,
                    help="target CPU time of the oracle baseline sample")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-graph", action="store_true", help="skip the CUDA-graph replay timing")
    ap.add_argument("--no-next", action="store_true", help="skip the NEXT-row measurements")
    ap.add_argument("--workload", choices=sorted(PROFILE_WORKLOADS), default=WORKLOAD,
                    help="large (default, the benchmark) or a smaller case for profiling")
    ap.add_argument("--passes", type=int, default=0,
                    help="passes per timed step (0: enough for a ~%.1f s timed region)"
                         % MIN_TIMED_S)
    ap.add_argument("--no-configs", action="store_true",
                    help="skip the 8B-class and weight-projection per-call tables")
    return ap.parse_args()


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


# ---- algorithmic bytes (each unique embedding row counted once) --------------

def algorithmic_bytes(T, d, k, n, u, m_cols, s=2):
    """HBM bytes each call must move at minimum."""
    emb = s * u * d + s * min(n, T) * d
    return {
        "sn_compress_fwd": s * T * d + emb + 4 * d * k + s * T * k,
        "sn_decompress_fwd": s * T * d + emb + 4 * d * k + s * T * k,
        "sn_compress_bwd": s * T * d + s * T * k + 4 * d * k,
        "sn_decompress_bwd": s * T * d + s * T * k + 4 * d * k,
        "sn_project_weight": 2 * s * d * m_cols,
    }


def kernel_sources_sha1():
    """Hash of the sources the step's kernels and their launch set-up are
    built from (the tensor-core kernels, their host side and headers)."""
    import glob
    import hashlib
    h = hashlib.sha1()
    for p in sorted(glob.glob(os.path.join(ROOT, "paper_2506_01260_gb300", "csrc", "sn_tc*.cu*"))):
        h.update(os.path.basename(p).encode())
        with open(p, "rb") as f:
            h.update(f.read())
    return h.hexdigest()


def measured_traffic(call):
    """DRAM bytes per launch of `call` from the committed ncu capture, or None
    when the kernel sources changed since the counters were taken."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(path):
        return None
    with open(path) as f:
        t = json.load(f)
    if t.get("sources_sha1") != kernel_sources_sha1():
        return None
    return t.get("per_launch_bytes", {}).get(call)


# ---- clocks ---------------------------------------------------------------------

class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), "--query-gpu=" + self.FIELDS,
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    sm.append(float(parts[1]))
                    mx.append(float(parts[2]))
                except ValueError:
                    continue
                for name, val in zip(names, parts[5:9]):
                    if val.lower() == "active":
                        reasons.add(name)
        os.unlink(self.path)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx),
                "samples": len(sm), "reasons": sorted(reasons)}


# ---- distributed plumbing (independent replicas: no data-path collective) ----

def dist_setup(args):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    pg = None
    if world > 1:
        import torch.distributed as dist
        import torch
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        if backend == "nccl":
            torch.cuda.set_device(local)
        dist.init_process_group(backend)
        pg = dist
    return world, rank, local, pg


def barrier(pg):
    if pg is not None:
        pg.barrier()


def max_over_ranks(pg, value, device=None):
    if pg is None:
        return value
    import torch
    t = torch.tensor([float(value)], dtype=torch.float64,
                     device=device if device is not None else "cpu")
    pg.all_reduce(t, op=pg.ReduceOp.MAX)
    return float(t.item())


# ---- CPU oracle baseline ---------------------------------------------------------

def _oracle_inputs(seed):
    sys.path.insert(0, ROOT)
    import oracle as O
    from paper_2506_01260_gb300 import workloads as W
    wl = W.WORKLOADS[WORKLOAD]
    rng = np.random.default_rng(seed)
    U = W.orthonormal_basis(wl.d, wl.k, rng).astype(np.float32)
    return O.default(), W, rng, U, wl


def _oracle_boundary(orc, W, rng, U, S, d):
    """S tokens through the four boundary calls of the oracle; seconds."""
    tok = W.to_bf16(0.02 * rng.standard_normal((S, d)))
    pe = W.to_bf16(0.02 * rng.standard_normal((S, d)))
    ids = np.arange(S, dtype=np.int32)
    pos = np.arange(S, dtype=np.int32)
    X = W.to_bf16(0.1 * rng.standard_normal((S, d)))
    G = W.to_bf16(rng.standard_normal((S, d)))
    t0 = time.perf_counter()
    C, _, _ = orc.compress_fwd(X, ids, tok, U, S, pos_emb=pe, pos=pos)
    orc.decompress_fwd(C, ids, tok, U, S, pos_emb=pe, pos=pos)
    Cg, _, _ = orc.compress_bwd(G, U)
    orc.decompress_bwd(Cg, U)
    return time.perf_counter() - t0


def _oracle_project(orc, W, rng, U, c, d):
    """c columns of a [d, c] weight through the oracle's projection; seconds."""
    Wc = W.to_bf16(0.02 * rng.standard_normal((d, c)))
    t0 = time.perf_counter()
    orc.project_weight(Wc, U)
    return time.perf_counter() - t0


def _oracle_worker(job):
    """One process of the all-cores baseline: ("boundary", S) or ("project", c)."""
    kind, size, seed = job
    orc, W, rng, U, wl = _oracle_inputs(seed)
    if size == 0:
        return 0.0
    if kind == "boundary":
        return _oracle_boundary(orc, W, rng, U, size, wl.d)
    return _oracle_project(orc, W, rng, U, size, wl.d)


def cpu_oracle_step_time(target_s, seed=7):
    """Time the fp64 oracle on a bounded sample of the large-stream step and
    scale it to a full step: S tokens through the four boundary calls, plus c
    columns of W_o through the projection.  Returns (seconds per full step,
    description of the sample, seconds spent, (S, c))."""
    orc, W, rng, U, wl = _oracle_inputs(seed)
    d = wl.d
    t_probe = _oracle_boundary(orc, W, rng, U, 8, d) / 8
    S = int(max(8, min(wl.T, 0.85 * target_s / max(t_probe, 1e-9))))
    tb = _oracle_boundary(orc, W, rng, U, S, d)
    p_probe = _oracle_project(orc, W, rng, U, 4, d) / 4
    c = int(max(4, min(W_O_SHAPE[1], 0.15 * target_s / max(p_probe, 1e-9))))
    tp = _oracle_project(orc, W, rng, U, c, d)
    step = tb * wl.T / S + tp * W_O_SHAPE[1] / c
    desc = ("fp64 oracle, 1 thread: %d of %d tokens through compress_fwd+decompress_fwd+"
            "compress_bwd+decompress_bwd (%.1f s) and %d of %d W_o columns through "
            "project_weight (%.1f s), scaled to one full step" % (S, wl.T, tb, c, W_O_SHAPE[1], tp))
    return step, desc, tb + tp, (S, c)


def cpu_oracle_step_time_all_cores(S, c, seed=11):
    """The same sample as cpu_oracle_step_time split over every host core: one
    spawned process per core takes an equal share of the S tokens, then of the
    c columns (the oracle itself is single-threaded; the shards are independent
    rows and columns).  A phase takes as long as its slowest process's oracle
    calls (each process builds its inputs first, untimed, like the one-thread
    sample); scaled to one full step."""
    import multiprocessing as mp
    from paper_2506_01260_gb300 import workloads as W
    wl = W.WORKLOADS[WORKLOAD]
    n = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else os.cpu_count()
    n = max(1, int(n))
    ctx = mp.get_context("spawn")
    with ctx.Pool(n) as pool:
        tb = max(pool.map(_oracle_worker,
                          [("boundary", S // n + (i < S % n), seed + i) for i in range(n)]))
        tp = max(pool.map(_oracle_worker,
                          [("project", c // n + (i < c % n), seed + i) for i in range(n)]))
    step = tb * wl.T / S + tp * W_O_SHAPE[1] / c
    desc = ("fp64 oracle in %d processes (one per host core): the same %d tokens (slowest "
            "process %.2f s) and %d W_o columns (slowest %.2f s), scaled to one full step"
            % (n, S, tb, c, tp))
    return step, desc, n


def run_reference(args, world, rank):
    """The oracle on the host cores, on the same workload, metric and unit."""
    if rank != 0:
        return
    steps = []
    desc = None
    for i in range(args.warmup + args.steps):
        st, desc, _, (S, c) = cpu_oracle_step_time(max(1.0, args.cpu_seconds / 4), seed=100 + i)
        if i >= args.warmup:
            steps.append(st)
            sampled = (S, c)
    from paper_2506_01260_gb300 import workloads as W
    T = W.WORKLOADS[WORKLOAD].T
    ms = 1e3 * statistics.mean(steps)
    value = T / (ms / 1e3)
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": config_dict(args.workload),
        "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": 1, "kind": "oracle",
                         "sample": desc},
        "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
        # each of the `steps` runs the oracle on a sample of the step and scales its time
        # to the full step: the steps are extrapolated, not timed over the whole workload
        "extrapolated": True,
        "sampled_tokens_per_step": sampled[0], "sampled_w_o_columns_per_step": sampled[1],
        "tokens_per_step": T,
    }
    print(json.dumps(line), flush=True)


def config_dict(workload=WORKLOAD):
    from paper_2506_01260_gb300 import workloads as W
    wname, wo = PROFILE_WORKLOADS[workload]
    wl = W.WORKLOADS[wname]
    if workload == "large":
        desc = ("large stream: T=16x4096 tokens, d=8192, k=82, vocab 128256, bf16, Zipf(1.1) "
                "ids, 5% off-subspace energy; fwd+bwd boundary round trip through a pinned "
                "host wire, plus project_weight of W_o [8192, 8192]")
    else:
        desc = ("%s-class: T=%dx%d tokens, d=%d, k=%d, vocab %d, bf16; fwd+bwd boundary round "
                "trip through a pinned host wire, plus project_weight of W_o [%d, %d]"
                % (wname.upper(), wl.batch, wl.seq_len, wl.d, wl.k, wl.vocab, wo[0], wo[1]))
    return {"workload": desc, "T": wl.T, "d": wl.d, "k": wl.k, "vocab": wl.vocab,
            "seq_len": wl.seq_len, "w_o": list(wo),
            "l2": "flushed before every timed pass (512 MiB written, then read back so that "
                  "no dirty line is left for the timed kernels to write back)",
            "timing": "each of the --steps timed steps runs passes_per_step back-to-back "
                      "passes of the path (enough for a timed region of >= 1.5 s, so the "
                      "clock sampler sees the load); ms_per_step and every per-call figure "
                      "are per pass",
            "parallelism": "independent replicas (one process per GPU)",
            "wire": "pinned-host D2H + H2D of C on a copy stream, overlapped with the next "
                    "compute call; the receiving call waits on it"}


# ---- lossy comparators at the codec's wire size ---------------------------------------

def lossy_comparison(args, sn, basis, X, Xr, ids, tok, pe, n, flush, stream, hbm, pg, dev):
    """Relative reconstruction error ||X' - X|| / ||X|| of the subspace codec and
    of the lossy comparators on the same activation batch, with the wire bytes of
    each: top-k at the codec's wire size (kk = k / 2: a bf16 value and a 16-bit
    column per kept entry), sign quantization (1 bit per entry, the smallest
    quantizer), row-scaled int8 and fp8 e4m3 quantization (8 bits per entry)
    and the randomized rank-r factorisation of the whole batch at the
    codec's wire size (r = T k / (T + d)).  Top-k, sign and the 8-bit
    quantizers are timed like the step's kernels."""
    import torch
    from paper_2506_01260_gb300 import comparators

    T, d = X.shape
    k = basis.k
    sn.sn_compress_fwd(basis, X, ids, tok, n, pos_emb=pe, out=torch.empty(T, k, dtype=X.dtype,
                                                                           device=dev))
    Xf = X.float()
    xn = float(Xf.norm())

    def rel(Xh):
        return float((Xh.float() - Xf).norm()) / xn

    def timed(fn, reps):
        for _ in range(args.warmup):
            flush_l2(flush)
            fn()
        evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
               for _ in range(reps)]
        for a_, b_ in evs:
            flush_l2(flush)
            a_.record(stream)
            fn()
            b_.record(stream)
        torch.cuda.synchronize()
        return max_over_ranks(pg, statistics.mean(a_.elapsed_time(b_) for a_, b_ in evs), dev)

    out = {"subspace": {"wire_bytes": 2 * T * k, "rel_error": rel(Xr)}}
    kk = k // 2
    vals = torch.empty(T, kk, dtype=X.dtype, device=dev)
    cols = torch.empty(T, kk, dtype=torch.int16, device=dev)
    tms = timed(lambda: sn.sn_topk_compress(X, kk, values=vals, cols=cols), min(args.steps, 20))
    Xh, wb = comparators.topk_roundtrip(X, kk)
    tab = 2 * T * d + 4 * T * kk
    out["topk"] = {"kk": kk, "wire_bytes": wb, "rel_error": rel(Xh), "compress_ms": tms,
                   "compress_gbs": tab / (tms / 1e3) / 1e9,
                   "compress_frac": tab / (tms / 1e3) / 1e9 / hbm}
    del Xh, vals, cols
    words = (d + 31) // 32
    bits = torch.empty(T, words, dtype=torch.int32, device=dev)
    scale = torch.empty(T, dtype=torch.float32, device=dev)
    sms = timed(lambda: sn.sn_sign_compress(X, bits=bits, scale=scale), min(args.steps, 20))
    Xh, wb = comparators.sign_roundtrip(X)
    sab = 2 * T * d + 4 * T * words + 4 * T
    out["sign"] = {"wire_bytes": wb, "rel_error": rel(Xh), "compress_ms": sms,
                   "compress_gbs": sab / (sms / 1e3) / 1e9,
                   "compress_frac": sab / (sms / 1e3) / 1e9 / hbm}
    del Xh, bits, scale
    codes = torch.empty(T, d, dtype=torch.uint8, device=dev)
    qscale = torch.empty(T, dtype=torch.float32, device=dev)
    qab = 2 * T * d + T * d + 4 * T
    for fmt in ("int8", "e4m3"):
        qms = timed(lambda: sn.sn_quant_compress(X, fmt, codes=codes, scale=qscale),
                    min(args.steps, 20))
        Xh, wb = comparators.quant_roundtrip(X, fmt)
        out[fmt] = {"wire_bytes": wb, "rel_error": rel(Xh), "compress_ms": qms,
                    "compress_gbs": qab / (qms / 1e3) / 1e9,
                    "compress_frac": qab / (qms / 1e3) / 1e9 / hbm}
        del Xh
    del codes, qscale
    r = T * k // (T + d)
    Xh, wb = comparators.lowrank_roundtrip(X, r)
    out["lowrank"] = {"r": r, "wire_bytes": wb, "rel_error": rel(Xh)}
    del Xh, Xf
    out["note"] = ("same X as the step (embeddings + in-span signal + off-subspace noise); "
                   "errors relative to ||X||; the codec subtracts the embeddings the "
                   "receiver recomputes, the comparators send X itself")
    return out


def paper_context(T, d, k, codec_ms, link_mbps=80.0):
    """The paper's own figures (other hardware, other setting), reported beside
    the measurement as context, not as its target: the compression ratio of the
    wire against the activation (Sec. 1, Sec. 8.1: up to 99%, ~100x at k = 40,
    d = 4096) and what one step's boundary traffic costs on the consumer links
    of its experiments (80 Mbps, Sec. 8.1) with and without the codec."""
    wire = 2 * (T * k * 2)                   # C forward + Cg backward, bf16
    full = 2 * (T * d * 2)                   # X forward + G backward uncompressed
    bytes_per_ms = link_mbps * 1e6 / 8 / 1e3
    return {
        "paper": "up to 99% compression (~100x, k = 40 at d = 4096) and up to 100x "
                 "communication efficiency; 80 Mbps links matching 100 Gbps convergence "
                 "(A10G / L4 GPUs, Sec. 1, Sec. 8.1)",
        "wire_bytes_per_step": wire, "uncompressed_bytes_per_step": full,
        "compression_ratio": full / wire, "compression_pct": 100.0 * (1 - wire / full),
        "link_mbps": link_mbps,
        "wire_ms_at_link": wire / bytes_per_ms, "uncompressed_ms_at_link": full / bytes_per_ms,
        "codec_ms_per_step": codec_ms,
        "note": "context, not the target: the codec's GPU time per step against the time its "
                "output needs on the paper's slowest links"}


def flush_l2(buf):
    """Evict L2 before a timed region: write a buffer larger than L2, then read
    it back, so that L2 holds only clean lines of the buffer.  The timed kernels
    start with none of their inputs cached and without the flush's dirty lines
    to write back (≈ 129 MB of DRAM writes, 15 µs on the first call after a
    write-only flush)."""
    import torch
    buf.zero_()
    buf.view(torch.int64).sum()


def timed_call(fn, flush, stream, warmup, reps):
    """Mean CUDA-event time (ms) of fn on `stream`, L2 flushed before every call."""
    import torch
    for _ in range(warmup):
        flush_l2(flush)
        fn()
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
           for _ in range(reps)]
    for a_, b_ in evs:
        flush_l2(flush)
        a_.record(stream)
        fn()
        b_.record(stream)
    torch.cuda.synchronize()
    return statistics.mean(a_.elapsed_time(b_) for a_, b_ in evs)


def config_tables(args, sn, dev, flush, stream, hbm, pg):
    """Per-call timings of the other configurations the roofline target names,
    each call alone with L2 flushed before it: the 8B-class boundary step (T =
    4 x 4096, d = 4096, k = 41, uniform ids) and the weight-projection
    configuration (W_o [4096, 4096] and W_down [4096, 14336], U [4096, 41])."""
    import torch
    from paper_2506_01260_gb300 import workloads as W
    reps = 50
    out = {}
    wl = W.WORKLOADS["8b"]
    inp = W.generate_on_device(wl, dev, grad=True)
    T, d, k, n = wl.T, wl.d, wl.k, wl.seq_len
    u = W.unique_ids(inp["ids_host"])
    basis = sn.Basis(inp["U"])
    X, ids, tok, pe, G = inp["X"], inp["ids"], inp["tok_emb"], inp["pos_emb"], inp["G"]
    C = torch.empty(T, k, dtype=torch.bfloat16, device=dev)
    Cg = torch.empty_like(C)
    Xr = torch.empty_like(X)
    Gr = torch.empty_like(G)
    sn.sn_compress_fwd(basis, X, ids, tok, n, pos_emb=pe, out=C)
    sn.sn_compress_bwd(basis, G, out=Cg)
    calls = {
        "sn_compress_fwd": lambda: sn.sn_compress_fwd(basis, X, ids, tok, n, pos_emb=pe, out=C),
        "sn_decompress_fwd": lambda: sn.sn_decompress_fwd(basis, C, ids, tok, n, pos_emb=pe,
                                                          out=Xr),
        "sn_compress_bwd": lambda: sn.sn_compress_bwd(basis, G, out=Cg),
        "sn_decompress_bwd": lambda: sn.sn_decompress_bwd(basis, Cg, out=Gr),
    }
    ab = algorithmic_bytes(T, d, k, n, u, 0)
    kernels = {}
    for name, fn in calls.items():
        ms = max_over_ranks(pg, timed_call(fn, flush, stream, args.warmup, reps), dev)
        gbs = ab[name] / (ms / 1e3) / 1e9
        kernels[name] = {"ms": ms, "algorithmic_bytes": ab[name], "gbs": gbs, "frac": gbs / hbm}
    sn.sn_check_errors(basis)
    out["8b"] = {"workload": "8B-class: T=4x4096 tokens, d=4096, k=41, vocab 128256, bf16, "
                             "uniform ids, 1e-3 off-subspace noise; G ~ N(0,1)",
                 "unique_ids": u, "reps": reps, "kernels": kernels}
    basis.destroy()
    del inp, X, ids, tok, pe, G, C, Cg, Xr, Gr
    torch.cuda.empty_cache()

    win = W.weight_inputs()
    U = torch.from_numpy(win["U"]).to(dev)
    basis = sn.Basis(U)
    proj = {}
    for name in ("W_o", "W_down"):
        Wd = torch.from_numpy(win[name].view(np.int16)).to(dev).view(torch.bfloat16)
        Wp = torch.empty_like(Wd)
        ws = torch.empty(max(16, sn.sn_project_weight_workspace(basis, torch.bfloat16,
                                                                Wd.shape[1])),
                         dtype=torch.uint8, device=dev)
        ms = max_over_ranks(pg, timed_call(lambda: sn.sn_project_weight(basis, Wd, out=Wp,
                                                                         workspace=ws),
                                           flush, stream, args.warmup, reps), dev)
        b = 2 * 2 * Wd.shape[0] * Wd.shape[1]
        gbs = b / (ms / 1e3) / 1e9
        proj[name] = {"shape": list(Wd.shape), "ms": ms, "algorithmic_bytes": b, "gbs": gbs,
                      "frac": gbs / hbm}
        del Wd, Wp, ws
    sn.sn_check_errors(basis)
    basis.destroy()
    out["weight_projection"] = {"workload": "W_o [4096, 4096] and W_down [4096, 14336] bf16 "
                                            "~N(0, 0.02^2), U [4096, 41]; W' = U (U^T W)",
                                "reps": reps, "sn_project_weight": proj}
    return out


# ---- our arm -------------------------------------------------------------------------

def run_ours(args, world, rank, local, pg):
    import torch
    from paper_2506_01260_gb300 import sn
    from paper_2506_01260_gb300 import workloads as W

    assert torch.cuda.is_available(), "bench needs a CUDA device"
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    wname, wo_shape = PROFILE_WORKLOADS[args.workload]
    wl = W.WORKLOADS[wname]
    T, d, k, n = wl.T, wl.d, wl.k, wl.seq_len
    inp = W.generate_on_device(wl, dev, seed=wl.seed + rank, grad=True)
    u = W.unique_ids(inp["ids_host"])
    g = torch.Generator(device=dev)
    g.manual_seed(wl.seed + 1000 + rank)
    Wo = (0.02 * torch.randn(*wo_shape, generator=g, device=dev)).to(torch.bfloat16)
    basis = sn.Basis(inp["U"])
    X, ids, tok, pe, G = inp["X"], inp["ids"], inp["tok_emb"], inp["pos_emb"], inp["G"]
    C = torch.empty(T, k, dtype=torch.bfloat16, device=dev)
    C_rx = torch.empty_like(C)
    Cg = torch.empty_like(C)
    Cg_rx = torch.empty_like(C)
    Xr = torch.empty_like(X)
    Gr = torch.empty_like(G)
    Wp = torch.empty_like(Wo)
    ws = torch.empty(max(16, sn.sn_project_weight_workspace(basis, torch.bfloat16, wo_shape[1])),
                     dtype=torch.uint8, device=dev)
    wire_f = torch.empty(C.numel() * 2, dtype=torch.uint8, pin_memory=True)
    wire_b = torch.empty(C.numel() * 2, dtype=torch.uint8, pin_memory=True)
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream()

    names = ["sn_compress_fwd", "sn_decompress_fwd", "sn_compress_bwd", "sn_decompress_bwd",
             "sn_project_weight"]

    # The forward and backward boundary transfers are independent of each
    # other, so each crosses the wire on its own copy stream while the compute
    # stream runs the next call (as a pipeline overlaps the activation send of
    # one microbatch with the gradient work of another); the receiving call
    # waits on the copy's event.
    wire_stream = torch.cuda.Stream()
    sync_ev = [torch.cuda.Event() for _ in range(4)]

    def step(ev=None, wev=None):
        # ev: 8 events on the compute stream, wev: 4 on the wire stream
        def mark(i):
            if ev is not None:
                ev[i].record(stream)

        def wmark(i):
            if wev is not None:
                wev[i].record(wire_stream)
        stream = torch.cuda.current_stream()     # the capturing stream under a graph
        mark(0)
        sn.sn_compress_fwd(basis, X, ids, tok, n, pos_emb=pe, out=C)
        sync_ev[0].record(stream)
        mark(1)
        wire_stream.wait_event(sync_ev[0])
        wmark(0)
        sn.sn_wire_send(C, wire_f, stream=wire_stream)
        sn.sn_wire_recv(wire_f, C_rx, stream=wire_stream)
        wmark(1)
        sync_ev[1].record(wire_stream)
        sn.sn_compress_bwd(basis, G, out=Cg)
        sync_ev[2].record(stream)
        mark(2)
        wire_stream.wait_event(sync_ev[2])
        wmark(2)
        sn.sn_wire_send(Cg, wire_b, stream=wire_stream)
        sn.sn_wire_recv(wire_b, Cg_rx, stream=wire_stream)
        wmark(3)
        sync_ev[3].record(wire_stream)
        sn.sn_project_weight(basis, Wo, out=Wp, workspace=ws)
        mark(3)
        stream.wait_event(sync_ev[1])
        mark(4)
        sn.sn_decompress_fwd(basis, C_rx, ids, tok, n, pos_emb=pe, out=Xr)
        mark(5)
        stream.wait_event(sync_ev[3])
        mark(6)
        sn.sn_decompress_bwd(basis, Cg_rx, out=Gr)
        mark(7)

    for _ in range(args.warmup):
        flush_l2(flush)
        step()
    sn.sn_check_errors(basis)
    torch.cuda.synchronize()

    # Each timed step runs `passes` back-to-back passes of the path (L2 flushed
    # before each), enough for the timed region to last about MIN_TIMED_S so that
    # the clock sampler sees the GPU under load; ms_per_step is per pass.
    pe0 = torch.cuda.Event(enable_timing=True)
    pe1 = torch.cuda.Event(enable_timing=True)
    pe0.record(stream)
    flush_l2(flush)
    step()
    pe1.record(stream)
    torch.cuda.synchronize()
    est_ms = max(1e-3, pe0.elapsed_time(pe1))
    passes = args.passes if args.passes > 0 else max(
        1, min(500, int(np.ceil(1e3 * MIN_TIMED_S / (args.steps * est_ms)))))
    npass = args.steps * passes
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(8)] for _ in range(npass)]
    wevs = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(npass)]
    clocks = ClockSampler(local)
    clocks.start()
    barrier(pg)
    torch.cuda.synchronize()
    launches0 = sn.sn_launch_count()
    wall0 = time.perf_counter()
    for i in range(npass):
        flush_l2(flush)
        step(evs[i], wevs[i])
    torch.cuda.synchronize()
    wall = time.perf_counter() - wall0
    launches = sn.sn_launch_count() - launches0
    barrier(pg)
    clk = clocks.stop()
    sn.sn_check_errors(basis)

    per_step = [e[0].elapsed_time(e[7]) for e in evs]          # ms
    seg = {  # ms per launch, averaged over the timed steps
        "sn_compress_fwd": statistics.mean(e[0].elapsed_time(e[1]) for e in evs),
        "sn_compress_bwd": statistics.mean(e[1].elapsed_time(e[2]) for e in evs),
        "sn_project_weight": statistics.mean(e[2].elapsed_time(e[3]) for e in evs),
        "wire_wait": statistics.mean(e[3].elapsed_time(e[4]) + e[5].elapsed_time(e[6])
                                     for e in evs),
        "sn_decompress_fwd": statistics.mean(e[4].elapsed_time(e[5]) for e in evs),
        "sn_decompress_bwd": statistics.mean(e[6].elapsed_time(e[7]) for e in evs),
        "wire_fwd": statistics.mean(w[0].elapsed_time(w[1]) for w in wevs),
        "wire_bwd": statistics.mean(w[2].elapsed_time(w[3]) for w in wevs),
    }
    ms = statistics.mean(per_step)
    ms = max_over_ranks(pg, ms, dev)
    value = world * T / (ms / 1e3)

    hbm, peak_kind = peaks()
    ab = algorithmic_bytes(T, d, k, n, u, wo_shape[1])
    kernels = {}
    for name in names:
        gbs = ab[name] / (seg[name] / 1e3) / 1e9
        kernels[name] = {"ms": seg[name], "algorithmic_bytes": ab[name], "gbs": gbs,
                         "frac": gbs / hbm}
    dom = max(names, key=lambda nm: seg[nm])
    traffic = measured_traffic(dom) if args.workload == WORKLOAD else None

    # ---- the same step captured once into a CUDA graph and replayed ----
    graph_line = None
    if not args.no_graph:
        graph = torch.cuda.CUDAGraph()
        side = torch.cuda.Stream()
        side.wait_stream(stream)
        l0 = sn.sn_launch_count()
        with torch.cuda.stream(side):
            with torch.cuda.graph(graph, stream=side, capture_error_mode="thread_local"):
                step()
        per_graph = sn.sn_launch_count() - l0
        stream.wait_stream(side)
        for _ in range(args.warmup):
            flush_l2(flush)
            graph.replay()
        torch.cuda.synchronize()
        gev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
               for _ in range(args.steps)]
        barrier(pg)
        torch.cuda.synchronize()
        for a_, b_ in gev:
            flush_l2(flush)
            a_.record(stream)
            graph.replay()
            b_.record(stream)
        torch.cuda.synchronize()
        barrier(pg)
        sn.sn_check_errors(basis)
        gms = max_over_ranks(pg, statistics.mean(a_.elapsed_time(b_) for a_, b_ in gev), dev)
        graph_line = {"ms_per_step": gms, "value": world * T / (gms / 1e3), "unit": "tokens/s",
                      "launches_per_step": per_graph,
                      "note": "the step above captured once (wire stream joined by events, "
                              "chained launches as programmatic edges) and replayed; L2 "
                              "flushed before every replay"}
        del graph

    # ---- NEXT f3, reported apart from the step: compress with projected tables
    nxt = None
    if not args.no_next:
        TU, PU = sn.sn_project_tables(basis, tok, pos_emb=pe)        # warm-up
        bev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
               for _ in range(3)]
        for a_, b_ in bev:
            flush_l2(flush)
            a_.record(stream)
            sn.sn_project_tables(basis, tok, pos_emb=pe, TU=TU, PU=PU)
            b_.record(stream)
        torch.cuda.synchronize()
        build_ms = statistics.mean(a_.elapsed_time(b_) for a_, b_ in bev)
        Cp = torch.empty_like(C)
        for _ in range(args.warmup):
            flush_l2(flush)
            sn.sn_compress_fwd_projected(basis, X, ids, TU, n, PU=PU, out=Cp)
        pev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
               for _ in range(min(args.steps, 50))]
        for a_, b_ in pev:
            flush_l2(flush)
            a_.record(stream)
            sn.sn_compress_fwd_projected(basis, X, ids, TU, n, PU=PU, out=Cp)
            b_.record(stream)
        torch.cuda.synchronize()
        sn.sn_check_errors(basis)
        pms = max_over_ranks(pg, statistics.mean(a_.elapsed_time(b_) for a_, b_ in pev), dev)
        pab = 2 * T * d + 4 * u * k + 4 * min(n, T) * k + 4 * d * k + 2 * T * k
        nxt = {"f3_projected_compress": {
            "ms": pms, "algorithmic_bytes": pab, "gbs": pab / (pms / 1e3) / 1e9,
            "frac": pab / (pms / 1e3) / 1e9 / hbm,
            "table_build_ms": build_ms,
            "speedup_vs_sn_compress_fwd": seg["sn_compress_fwd"] / pms,
            "note": "C = X U - (T_fixed U)[ids] - (P U)[pos] with the tables projected once "
                    "(sn_project_tables); same C as sn_compress_fwd"}}
        del TU, PU, Cp
        # NEXT f1: the Grassmann accumulation M += G^T Cg (every iteration) and the
        # step (every K iterations), at the workload's G and U
        Mg = torch.zeros(d, k, dtype=torch.float32, device=dev)
        wsa, wss = sn.sn_grassmann_workspace(basis, T)
        wsa = torch.empty(max(256, wsa), dtype=torch.uint8, device=dev)
        wss = torch.empty(max(256, wss), dtype=torch.uint8, device=dev)
        sn.sn_compress_bwd(basis, G, out=Cg)
        for _ in range(args.warmup):
            flush_l2(flush)
            sn.sn_grassmann_accumulate(basis, G, Cg, Mg, workspace=wsa)
        gev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
               for _ in range(min(args.steps, 30))]
        for a_, b_ in gev:
            flush_l2(flush)
            a_.record(stream)
            sn.sn_grassmann_accumulate(basis, G, Cg, Mg, workspace=wsa)
            b_.record(stream)
        torch.cuda.synchronize()
        gms = max_over_ranks(pg, statistics.mean(a_.elapsed_time(b_) for a_, b_ in gev), dev)
        Unew = torch.empty(d, k, dtype=torch.float32, device=dev)
        from paper_2506_01260_gb300.shard import allreduce_grassmann
        allreduce_grassmann(Mg)        # data-parallel replicas sum M before the step
        Mg.div_(len(gev) + args.warmup)
        sn.sn_grassmann_step(basis, Mg, 1, 1e-3, out=Unew, workspace=wss)
        sev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
               for _ in range(5)]
        for a_, b_ in sev:
            a_.record(stream)
            sn.sn_grassmann_step(basis, Mg, 1, 1e-3, out=Unew, workspace=wss)
            b_.record(stream)
        torch.cuda.synchronize()
        sn.sn_check_errors(basis)
        sms_ = statistics.mean(a_.elapsed_time(b_) for a_, b_ in sev)
        orth = float((Unew.double().t() @ Unew.double() - torch.eye(k, dtype=torch.float64,
                                                                      device=dev)).abs().max())
        gab = 2 * T * d + 2 * T * k + 2 * 4 * d * k
        nxt["f1_grassmann"] = {
            "accumulate_ms": gms, "accumulate_algorithmic_bytes": gab,
            "accumulate_gbs": gab / (gms / 1e3) / 1e9,
            "accumulate_frac": gab / (gms / 1e3) / 1e9 / hbm,
            "step_ms": sms_, "step_orthonormality_error": orth,
            "note": "M += G^T (G U) per iteration on the tensor cores (the [d, d] S is never "
                    "formed); every K iterations: tangent step + CholeskyQR2 retraction"}
        del Mg, wsa, wss, Unew
        # NEXT f2: one row-constant AdamW step on an fp32 master copy of W_o
        # (bf16 gradient), the weight whose columns the paper keeps in S
        Wm = Wo.float()
        gW = (0.01 * torch.randn(wo_shape, generator=g, device=dev)).to(torch.bfloat16)
        Mm = torch.zeros_like(Wm)
        Vm = torch.zeros_like(Wm)
        aws = torch.empty(wo_shape[1], dtype=torch.float32, device=dev)
        for t_ in range(1, args.warmup + 1):
            flush_l2(flush)
            sn.sn_adamw_rowconst(Wm, gW, Mm, Vm, t_, 1e-4, workspace=aws)
        aev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
               for _ in range(min(args.steps, 30))]
        for i_, (a_, b_) in enumerate(aev):
            flush_l2(flush)
            a_.record(stream)
            sn.sn_adamw_rowconst(Wm, gW, Mm, Vm, args.warmup + 1 + i_, 1e-4, workspace=aws)
            b_.record(stream)
        torch.cuda.synchronize()
        ams = max_over_ranks(pg, statistics.mean(a_.elapsed_time(b_) for a_, b_ in aev), dev)
        nel = wo_shape[0] * wo_shape[1]
        aab = nel * (2 + 8 + 8 + 8)
        nxt["f2_adamw_rowconst"] = {
            "ms": ams, "algorithmic_bytes": aab, "gbs": aab / (ams / 1e3) / 1e9,
            "frac": aab / (ams / 1e3) / 1e9 / hbm, "shape": list(wo_shape),
            "note": "fp32 W, M, V, bf16 gradient; V + column sums of V^ (pass 1), M and W "
                    "with one rate per column (pass 2, reads g again): 28 B moved per element"}
        del Wm, gW, Mm, Vm, aws
        nxt["f4_lossy"] = lossy_comparison(args, sn, basis, X, Xr, ids, tok, pe, n, flush,
                                           stream, hbm, pg, dev)

    # ---- the other configurations of the roofline target, per call ----
    tables = None
    if not args.no_configs and args.workload == WORKLOAD:
        tables = config_tables(args, sn, dev, flush, stream, hbm, pg)

    # ---- end to end through the C ABI with host buffers ----
    e2e_line = None
    if not args.no_e2e:
        Xh = torch.empty(X.shape, dtype=X.dtype, pin_memory=True)
        Gh = torch.empty(G.shape, dtype=G.dtype, pin_memory=True)
        idsh = torch.empty(ids.shape, dtype=ids.dtype, pin_memory=True)
        Xoh = torch.empty_like(Xh, pin_memory=True)
        Goh = torch.empty_like(Gh, pin_memory=True)
        Xh.copy_(X)
        Gh.copy_(G)
        idsh.copy_(ids)
        h2d = Xh.numel() * 2 + Gh.numel() * 2 + idsh.numel() * 4
        d2h = Xoh.numel() * 2 + Goh.numel() * 2

        # Host copies ride their own streams and the device side of every host
        # buffer is doubled, so the link never waits for compute: step i + 1's
        # uploads start as soon as step i's are done (X, ids and G of the step
        # before last have been read by then), and each step's X' and G' leave
        # while the next step's inputs arrive (the link runs both directions at
        # once).  Every step still copies its own inputs in and its results
        # out; events keep each buffer from being overwritten while it is read
        # or sent.
        h2d_stream = torch.cuda.Stream()
        d2h_stream = torch.cuda.Stream()
        # the eager step's outputs on the same inputs: what every e2e step must download
        torch.cuda.synchronize()
        Xr_ref, Gr_ref = Xr.clone(), Gr.clone()
        Xd, Gd, idsd = [X, torch.empty_like(X)], [G, torch.empty_like(G)], [ids, torch.empty_like(ids)]
        Xrd, Grd = [Xr, torch.empty_like(Xr)], [Gr, torch.empty_like(Gr)]
        ev = {name: [torch.cuda.Event() for _ in range(2)]
              for name in ("x_free", "g_free", "x_in", "g_in", "xr_done", "gr_done", "xr_free",
                           "gr_free")}
        for b_ in range(2):
            for name in ("x_free", "g_free"):
                ev[name][b_].record(stream)
            for name in ("xr_free", "gr_free"):
                ev[name][b_].record(d2h_stream)
        step_no = [0]

        def e2e_step():
            b_ = step_no[0] % 2
            step_no[0] += 1
            h2d_stream.wait_event(ev["x_free"][b_])     # X, ids of two steps ago are read
            sn.sn_wire_recv(Xh, Xd[b_], stream=h2d_stream)
            sn.sn_wire_recv(idsh, idsd[b_], stream=h2d_stream)
            ev["x_in"][b_].record(h2d_stream)
            h2d_stream.wait_event(ev["g_free"][b_])
            sn.sn_wire_recv(Gh, Gd[b_], stream=h2d_stream)
            ev["g_in"][b_].record(h2d_stream)
            stream.wait_event(ev["x_in"][b_])
            sn.sn_compress_fwd(basis, Xd[b_], idsd[b_], tok, n, pos_emb=pe, out=C)
            sync_ev[0].record(stream)
            wire_stream.wait_event(sync_ev[0])
            sn.sn_wire_send(C, wire_f, stream=wire_stream)
            sn.sn_wire_recv(wire_f, C_rx, stream=wire_stream)
            sync_ev[1].record(wire_stream)
            stream.wait_event(ev["g_in"][b_])
            sn.sn_compress_bwd(basis, Gd[b_], out=Cg)
            ev["g_free"][b_].record(stream)
            sync_ev[2].record(stream)
            wire_stream.wait_event(sync_ev[2])
            sn.sn_wire_send(Cg, wire_b, stream=wire_stream)
            sn.sn_wire_recv(wire_b, Cg_rx, stream=wire_stream)
            sync_ev[3].record(wire_stream)
            sn.sn_project_weight(basis, Wo, out=Wp, workspace=ws)
            stream.wait_event(sync_ev[1])
            stream.wait_event(ev["xr_free"][b_])         # X' of two steps ago has left
            sn.sn_decompress_fwd(basis, C_rx, idsd[b_], tok, n, pos_emb=pe, out=Xrd[b_])
            ev["x_free"][b_].record(stream)
            ev["xr_done"][b_].record(stream)
            d2h_stream.wait_event(ev["xr_done"][b_])
            sn.sn_wire_send(Xrd[b_], Xoh, stream=d2h_stream)
            ev["xr_free"][b_].record(d2h_stream)
            stream.wait_event(sync_ev[3])
            stream.wait_event(ev["gr_free"][b_])
            sn.sn_decompress_bwd(basis, Cg_rx, out=Grd[b_])
            ev["gr_done"][b_].record(stream)
            d2h_stream.wait_event(ev["gr_done"][b_])
            sn.sn_wire_send(Grd[b_], Goh, stream=d2h_stream)
            ev["gr_free"][b_].record(d2h_stream)

        for _ in range(min(args.warmup, 3)):
            e2e_step()
        torch.cuda.synchronize()
        e2e_ms = []
        nrep = max(3, min(args.steps, 40) // 2)
        for _ in range(3):                        # three timed runs of nrep steps each
            a = torch.cuda.Event(enable_timing=True)
            b = torch.cuda.Event(enable_timing=True)
            torch.cuda.synchronize()
            a.record(stream)
            for _ in range(nrep):
                e2e_step()
            stream.wait_stream(d2h_stream)          # the run ends when the last X', G' are on the host
            b.record(stream)
            b.synchronize()
            e2e_ms.append(a.elapsed_time(b) / nrep)
        sn.sn_check_errors(basis)
        e2e = max_over_ranks(pg, statistics.mean(e2e_ms), dev)
        torch.cuda.synchronize()
        verified = bool(torch.equal(Xoh.to(dev).view(torch.int16), Xr_ref.view(torch.int16)) and
                        torch.equal(Goh.to(dev).view(torch.int16), Gr_ref.view(torch.int16)))
        del Xr_ref, Gr_ref
        e2e_line = {"value": world * T / (e2e / 1e3), "unit": "tokens/s",
                    "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "ms_per_step": e2e,
                    "outputs_match_eager_step": verified,
                    "pipelining": "up to two steps in flight: uploads, compute and downloads on "
                                  "their own streams, device-side host buffers doubled"}

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline and args.workload == WORKLOAD:
        st, desc, _, (S, c) = cpu_oracle_step_time(args.cpu_seconds)
        cpu = {"value": T / st, "unit": "tokens/s", "cores": 1, "kind": "oracle",
               "sample": desc}
        try:
            st_all, desc_all, n_all = cpu_oracle_step_time_all_cores(S, c)
            cpu["all_cores"] = {"value": T / st_all, "unit": "tokens/s", "cores": n_all,
                                "sample": desc_all}
        except Exception as exc:          # a host without spawnable workers
            cpu["all_cores"] = {"unavailable": repr(exc)[:200]}

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic", "config": config_dict(args.workload),
            "roofline": {"bound": "hbm", "kernel": dom,
                         "achieved": kernels[dom]["gbs"], "peak": hbm,
                         "peak_kind": peak_kind, "unit": "GB/s",
                         "frac": kernels[dom]["gbs"] / hbm, "traffic": traffic,
                         "algorithmic_bytes_per_launch": ab[dom]},
            "kernels": kernels,
            "passes_per_step": passes, "timed_passes": npass,
            "configs": tables,
            "wire_ms": {"fwd": seg["wire_fwd"], "bwd": seg["wire_bwd"],
                        "compute_stream_wait": seg["wire_wait"]},
            "boundary_hbm_gbs": sum(ab[nm] for nm in names) / (
                sum(seg[nm] for nm in names) / 1e3) / 1e9,
            # tokens/s of each round trip alone (compress + decompress), beside the
            # whole step's `value`
            "round_trip_tokens_per_s": {
                "fwd": world * T / ((seg["sn_compress_fwd"] + seg["sn_decompress_fwd"]) / 1e3),
                "bwd": world * T / ((seg["sn_compress_bwd"] + seg["sn_decompress_bwd"]) / 1e3)},
            "next": nxt,
            "e2e": e2e_line,
            "graph": graph_line,
            "paper_context": paper_context(T, d, k, ms),
            "gpu_launches": launches,
            "unique_ids": u,
            "wall_s_timed_region": wall,
            "clocks": clk,
            "cpu_baseline": cpu,
        }
        print(json.dumps(line), flush=True)
    basis.destroy()


def main():
    args = parse()
    world, rank, local, pg = dist_setup(args)
    if args.impl == "reference":
        run_reference(args, world, rank)
    else:
        run_ours(args, world, rank, local, pg)
    if pg is not None:
        pg.destroy_process_group()


if __name__ == "__main__":
    main()
