"""Benchmark of the pvMVMD hot path on GB300.

A step is one pass of the whole online path over one batch of synthetic
inputs (the 4096 x 4096 single-projection workload, batch 1):
    pvmvmd_encode        (100 vectors)
    pvmvmd_server_mvm    100 times at batch 1 (one grouped call)
    pvmvmd_decode_verify (100 vectors)
By default (--step-schedule overlap) the next batch's encode runs on a second
stream beside this batch's decode; every step still encodes, multiplies and
decodes 100 vectors.  Preprocessing (P^T and Q) happens once, before timing.
The 100 GEMVs rotate
over 64 copies of the weights (1 GiB in all), so every timed GEMV streams its
matrix from HBM rather than from the 126 MB L2.

Prints one JSON line (rank 0).  `--impl reference` times the CPU oracle on the
same workload instead (a bounded sample of vectors per step).
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "field MAC/s and achieved HBM GB/s (batch-1) / int8 tensor-pipe % (batched)"
UNIT = "field MAC/s"
M = K = 4096
VECTORS = 100
REPLICAS = 64
SEED_W, SEED_X = 2, 3


# --------------------------------------------------------------------------- host CPU and the oracle on all cores

def host_cpu() -> dict:
    """The host's logical CPU count and model (from /proc/cpuinfo)."""
    import platform
    model = ""
    try:
        with open("/proc/cpuinfo") as f:
            for line in f:
                key, _, val = line.partition(":")
                key, val = key.strip().lower(), val.strip()
                if key == "model name" and val:
                    model = val
                    break
                if key == "cpu part" and val and not model:
                    model = "CPU part " + val
    except OSError:
        pass
    return {"cpu_count": os.cpu_count(), "model": model or platform.machine()}


_ORACLE_W = None


def _oracle_rows_init(W):
    global _ORACLE_W
    _ORACLE_W = W


def _oracle_rows(job):
    import oracle
    x, r0, r1 = job
    return oracle.server_mvm(_ORACLE_W[r0:r1], x)


def oracle_rows_parallel(W, X, procs: int):
    """The oracle's server MVM (unchanged) of every vector of X with the rows
    of W split over `procs` spawned processes.  Returns (field MACs, seconds,
    the product of the last vector)."""
    import multiprocessing as mp
    m = W.shape[0]
    bounds = [(m * i // procs, m * (i + 1) // procs) for i in range(procs)]
    with mp.get_context("spawn").Pool(procs, initializer=_oracle_rows_init, initargs=(W,)) as pool:
        pool.map(_oracle_rows, [(X[0], r0, r1) for r0, r1 in bounds])  # every worker has loaded the oracle
        t0 = time.perf_counter()
        for x in X:
            parts = pool.map(_oracle_rows, [(x, r0, r1) for r0, r1 in bounds])
        dt = time.perf_counter() - t0
    return len(X) * W.size, dt, np.concatenate(parts)


# --------------------------------------------------------------------------- distributed helpers

def dist_env():
    return int(os.environ.get("RANK", 0)), int(os.environ.get("WORLD_SIZE", 1)), \
        int(os.environ.get("LOCAL_RANK", 0))


def max_over_ranks(value: float, device=None) -> float:
    """Max of a float over all ranks (identity without torch.distributed)."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()):
        return value
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def barrier(device=None):
    import torch.distributed as dist
    if dist.is_available() and dist.is_initialized():
        if device is not None and dist.get_backend() == "nccl":
            dist.barrier(device_ids=[device.index])
        else:
            dist.barrier()


# --------------------------------------------------------------------------- clocks

class ClockSampler:
    """Samples nvidia-smi SM clocks and throttle reasons while running.

    start() returns once the first sample has arrived, so the sampler is live
    before the timed region begins; region_started() marks the start of the
    region, and stop() summarises the samples taken from that mark on (the
    timed region and the load queued after it, see clock_tail)."""
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.lines = []
        self.t_mark = None

    def start(self, wait_s: float = 3.0):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except (OSError, ValueError):
            self.proc = None
            return
        t_end = time.monotonic() + wait_s
        while not self.lines and time.monotonic() < t_end and self.proc.poll() is None:
            time.sleep(0.01)

    def region_started(self):
        self.t_mark = time.monotonic()

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append((time.monotonic(), line.strip()))

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"], "samples": 0}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.thread.join(timeout=2)
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        lines = [ln for ts, ln in self.lines if self.t_mark is None or ts >= self.t_mark]
        for line in lines:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 7:
                continue
            try:
                sm.append(float(parts[0]))
                smax.append(float(parts[1]))
            except ValueError:
                continue
            for n, v in zip(names, parts[3:7]):
                if v.lower() == "active":
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(smax), "reasons": sorted(reasons),
                "samples": len(sm), "window": "from the start of the timed region to the end of the "
                                              "same steps queued after it (clock tail)"}


CLOCK_TAIL_S = 0.5


def clock_tail(replay, ms_per_call: float, seconds: float | None = None) -> int:
    """Queue untimed calls of `replay` after the timed region's stop event, so
    that the clock sampler (100 ms period) sees the GPU under the same load
    for `seconds` even when the timed region itself is only milliseconds
    long.  Returns the number of calls queued."""
    seconds = CLOCK_TAIL_S if seconds is None else seconds
    if seconds <= 0:
        return 0
    n = max(1, int(seconds * 1e3 / max(ms_per_call, 1e-3)))
    for i in range(n):
        replay(i)
    return n


# --------------------------------------------------------------------------- roofline inputs

def measured_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return json.load(f), "measured"
    except OSError:
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0}, "fallback"


def gemv_traffic_per_launch():
    """DRAM bytes per GEMV launch from the committed ncu summary, or None when
    the kernel source changed since the counters were taken."""
    path = os.path.join(ROOT, "profiles", "gemv_4096x4096_traffic.json")
    try:
        with open(path) as f:
            rec = json.load(f)
    except OSError:
        return None
    src = os.path.join(ROOT, "paper_2609_10264_gb300", "csrc", "gemv.cu")
    sha = hashlib.sha256(open(src, "rb").read()).hexdigest()
    if rec.get("gemv_cu_sha256") != sha:
        return None
    return rec.get("dram_bytes_per_launch")


# --------------------------------------------------------------------------- CPU oracle (baseline)

class OracleWorkload:
    """The oracle, as it stands, on this workload (preprocessing done once)."""

    def __init__(self):
        import oracle
        from paper_2609_10264_gb300 import workloads as wl
        self.o = oracle
        self.W = wl.weights_gaussian(M, K, SEED_W)
        self.x = oracle.lift(wl.int8_vectors(VECTORS, K, SEED_X))
        self.pp = oracle.PublicParams(self.W, oracle.key_from_seed(20))

    def client(self, b: int):
        """Encrypt, server MVM, verify and decrypt of vector b (full vector)."""
        o, pp = self.o, self.pp
        xh, s, v = pp.encrypt(self.x[b], o.key_from_seed(21), b)
        yh = o.server_mvm(self.W, xh)
        assert pp.verify(xh, yh, o.key_from_seed(22))
        pp.decrypt(s, v, yh)
        return xh

    def full_vectors(self, n: int):
        """Time n full vectors.  Returns (field MACs, seconds)."""
        t0 = time.perf_counter()
        for b in range(n):
            self.client(b % VECTORS)
        return n * M * K, time.perf_counter() - t0


def run_reference(args):
    """Each step: the server MVM of one vector restricted to R rows, plus that
    vector's client work (encrypt, verify, decrypt) once every 4096/R steps,
    so that server and client work keep the proportions of a full vector."""
    rank, world, _ = dist_env()
    if rank != 0:
        return 0
    ow = OracleWorkload()
    o = ow.o
    xh0 = ow.client(0)
    t0 = time.perf_counter()
    o.server_mvm_rows(ow.W, xh0, np.arange(256))
    t_row = (time.perf_counter() - t0) / 256
    budget_s = float(os.environ.get("PVMVMD_REF_BUDGET_S", "90"))
    R = int(max(8, min(M, budget_s / ((args.steps + args.warmup) * t_row))))
    every = -(-M // R)
    rng = np.random.default_rng(0)

    def one_step(s):
        b = s % VECTORS
        t = time.perf_counter()
        if s % every == 0:
            xh = ow.client(b)            # includes the full-vector server MVM: count it
            macs = M * K
        else:
            rows = rng.choice(M, size=R, replace=False)
            o.server_mvm_rows(ow.W, xh0, rows)
            macs = R * K
        return macs, time.perf_counter() - t

    for w in range(args.warmup):
        one_step(w + 1)
    total_macs, total_s = 0, 0.0
    for s in range(args.steps):
        mac, dt = one_step(s)
        total_macs += mac
        total_s += dt
    value = total_macs / total_s
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * total_s / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "u32 (F_q, exact)",
        "data": "synthetic", "config": arm_config(args),
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": 1, "kind": "oracle",
                         "sample": f"per step: server MVM of one vector on {R} sampled rows; every "
                                   f"{every} steps one full vector (encrypt, MVM, verify, decrypt); "
                                   "single-threaded C oracle"},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


def workload_config():
    return {"workload": "pvMVMD batch-1 round trip: W 4096x4096 int8 (Gaussian sigma 32, clipped), "
                        "100 int8 vectors per step: encode -> 100 batch-1 GEMVs -> decode+verify",
            "m": M, "K": K, "vectors_per_step": VECTORS, "w_replicas": REPLICAS,
            "params": "lambda 128, kappa 40, rate 8, delta 1/2, t_x 157, t_y 31, ell 2",
            "l2": "inputs larger than L2: 64 weight copies (1 GiB) rotate over the GEMVs; "
                  "P^T and Q are 0.5 GiB each",
            "parallelism": "replicas (one independent workload per GPU)",
            "server": "100 independent batch-1 products (one weight copy each) in one "
                      "pvmvmd_server_mvm_multi call"}


def arm_config(args) -> dict:
    """The `config` of the default workload's line, identical for both arms."""
    overlap = args.mode == "standard" and args.step_schedule == "overlap"
    cfg = dict(workload_config(), mode=args.mode,
               step_schedule=("overlap: each step's server call, then its decode beside the next batch's "
                              "encode on a second stream" if overlap else "serial: encode, server, decode"))
    if args.mode == "boost":
        cfg["masks"] = "prepared ahead and reused across the timed steps (the same work as fresh masks)"
    return cfg


# --------------------------------------------------------------------------- our arm

def run_ours(args):
    import torch
    rank, world, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    device = torch.device("cuda", local)
    torch.cuda.set_device(device)
    import paper_2609_10264_gb300 as pv
    from paper_2609_10264_gb300 import workloads as wl

    W = wl.weights_gaussian(M, K, SEED_W)
    x = wl.int8_vectors(VECTORS, K, SEED_X)
    X = np.mod(x, pv.PVMVMD_Q).astype(np.uint32)
    Wd = torch.from_numpy(W).to(device)
    Wrep = Wd.repeat(REPLICAS, 1).contiguous()           # 64 distinct copies, 1 GiB
    Xd = torch.from_numpy(X.view(np.int32)).to(device)
    params = pv.pvmvmd_params()
    params.scratch_batch = VECTORS                        # one encode chunk per step
    ctx = pv.pvmvmd_preprocess(Wd, key=20, params=params)
    torch.cuda.synchronize(device)   # the inputs, made on torch's stream, are ready for `stream`
    stream = torch.cuda.Stream(device)
    # "overlap" (standard mode): the next batch's encode runs on enc_stream
    # beside this batch's decode (an encode and a decode of one context share
    # no scratch), so x_hat and st alternate between two sets
    overlap = args.mode == "standard" and args.step_schedule == "overlap"
    enc_stream = torch.cuda.Stream(device)
    Xh_sets = [torch.empty_like(Xd) for _ in range(2 if overlap else 1)]
    st_sets = [torch.empty((VECTORS, 2 * ctx.t_x), dtype=torch.int32, device=device)
               for _ in range(2 if overlap else 1)]
    Xh, st = Xh_sets[0], st_sets[0]
    Yh = torch.empty((VECTORS, M), dtype=torch.int32, device=device)
    Y = torch.empty_like(Yh)
    acc = torch.empty(VECTORS, dtype=torch.int32, device=device)
    Wv = [Wrep[(b % REPLICAS) * M:(b % REPLICAS + 1) * M] for b in range(VECTORS)]

    # Boost mode (Sec. 7.2): masks prepared ahead.  "boost" prepares them
    # before the timed region; "pipelined" (standard mode with pipelining)
    # prepares step j+1's masks on a second stream while step j runs, inside
    # the timed region.  Two mask sets alternate between steps.
    boost = args.mode != "standard"
    nsets = 2 if args.mode == "pipelined" else 1
    if boost:
        mi = [torch.empty((VECTORS, K), dtype=torch.int32, device=device) for _ in range(nsets)]
        mo = [torch.empty((VECTORS, M), dtype=torch.int32, device=device) for _ in range(nsets)]
        mst = [torch.empty((VECTORS, 2 * ctx.t_x), dtype=torch.int32, device=device) for _ in range(nsets)]
    prep_stream = torch.cuda.Stream(device)

    def prepare(k, on):
        pv.pvmvmd_boost_prepare(ctx, VECTORS, 41 + rank + k, mask_in=mi[k], mask_out=mo[k], st=mst[k],
                                stream=on)

    cur = [0]

    def encode():
        if boost:
            pv.pvmvmd_boost_encode(Xd, mi[cur[0]], Xhat=Xh, stream=stream)
            return
        pv.pvmvmd_encode(ctx, Xd, 21 + rank, Xhat=Xh, st=st, stream=stream)

    side = [torch.cuda.Stream(device) for _ in range(args.server_streams)]
    jobs_sets = [pv.mvm_jobs([(Wv[b], xs[b], Yh[b]) for b in range(VECTORS)]) for xs in Xh_sets]
    jobs = jobs_sets[0]

    def server():
        if args.server_mode == "multi":
            # the 100 independent batch-1 requests in one grouped call
            pv.pvmvmd_server_mvm_multi(jobs, stream=stream)
            return
        # one call per request, spread over a few streams
        fork = torch.cuda.Event()
        fork.record(stream)
        for ss in side:
            ss.wait_event(fork)
        for b in range(VECTORS):
            pv.pvmvmd_server_mvm(Wv[b], Xh[b], Yhat=Yh[b], stream=side[b % len(side)])
        for ss in side:
            join = torch.cuda.Event()
            join.record(ss)
            stream.wait_event(join)

    def decode():
        if boost:
            pv.pvmvmd_boost_decode_verify(ctx, mo[cur[0]], Xh, Yh, 22 + rank, Y=Y, accept=acc, stream=stream)
            return
        pv.pvmvmd_decode_verify(ctx, st, Xh, Yh, 22 + rank, Y=Y, accept=acc, stream=stream)

    # eager run once (sets kernel attributes, checks the result), then capture
    if boost:
        for k in range(nsets):
            with torch.cuda.stream(prep_stream):
                prepare(k, prep_stream)
        prep_stream.synchronize()
    with torch.cuda.stream(stream):
        encode(); server(); decode()
    stream.synchronize()
    pv.pvmvmd_device_status(stream)
    assert int(acc.sum()) == VECTORS, "honest outputs must be accepted"
    Yc = pv.as_u32(Y)
    rows = [0, 1, 2047, 4095]
    exact = x.astype(np.float64) @ W[rows].astype(np.float64).T
    assert np.array_equal(np.where(Yc[:, rows] > (pv.PVMVMD_Q - 1) // 2,
                                   Yc[:, rows].astype(np.int64) - pv.PVMVMD_Q,
                                   Yc[:, rows].astype(np.int64)), exact.astype(np.int64))

    def capture(fn, on):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=on):
            fn()
        return g

    g_encs, g_decs, g_preps = [], [], []
    for k in range(nsets):
        cur[0] = k
        g_encs.append(capture(encode, stream))
        g_decs.append(capture(decode, stream))
        if args.mode == "pipelined":
            g_preps.append(capture(lambda k=k: prepare(k, prep_stream), prep_stream))
    cur[0] = 0
    g_srv = capture(server, stream)

    # the whole step (for pipelined mode with the other set's preparation
    # forked onto prep_stream and joined back) as one graph per mask set:
    # what `value` times; the per-phase graphs above give the phase split
    def whole_step(k):
        cur[0] = k
        if args.mode == "pipelined":
            fork = torch.cuda.Event()
            fork.record(stream)
            prep_stream.wait_event(fork)
            with torch.cuda.stream(prep_stream):
                prepare(1 - k, prep_stream)
        encode(); server(); decode()
        if args.mode == "pipelined":
            join = torch.cuda.Event()
            join.record(prep_stream)
            stream.wait_event(join)

    def overlapped_step(k, x_in=None, host_in=None, host_out=None):
        # this batch (set k): server, then decode on `stream`; the next batch
        # (set 1 - k): encode on enc_stream, forked after the server call.
        # (Forked at the start of the step instead, beside the server call,
        # it saved nothing: 338 against 330 us per step; enqueueing the
        # decode before the encode changed nothing either.)
        pv.pvmvmd_server_mvm_multi(jobs_sets[k], stream=stream)
        fork = torch.cuda.Event()
        fork.record(stream)
        enc_stream.wait_event(fork)
        with torch.cuda.stream(enc_stream):
            src = Xd
            if host_in is not None:
                x_in[1 - k].copy_(host_in, non_blocking=True)
                src = x_in[1 - k]
            pv.pvmvmd_encode(ctx, src, 21 + rank, Xhat=Xh_sets[1 - k], st=st_sets[1 - k], stream=enc_stream)
        pv.pvmvmd_decode_verify(ctx, st_sets[k], Xh_sets[k], Yh, 22 + rank, Y=Y, accept=acc, stream=stream)
        if host_out is not None:
            host_out[0].copy_(Y, non_blocking=True)
            host_out[1].copy_(acc, non_blocking=True)
        join = torch.cuda.Event()
        join.record(enc_stream)
        stream.wait_event(join)

    if overlap:
        # set 0 holds an encoded batch before the first step
        with torch.cuda.stream(stream):
            pv.pvmvmd_encode(ctx, Xd, 21 + rank, Xhat=Xh_sets[0], st=st_sets[0], stream=stream)
        stream.synchronize()
        n_launch0 = pv.pvmvmd_kernel_launches()
        g_steps = [capture(lambda k=k: overlapped_step(k), stream) for k in range(2)]
    else:
        n_launch0 = pv.pvmvmd_kernel_launches()
        g_steps = [capture(lambda k=k: whole_step(k), stream) for k in range(nsets)]
    # kernels the library enqueued into the step graphs (each replay launches them again)
    counted_per_step = (pv.pvmvmd_kernel_launches() - n_launch0) / len(g_steps)
    cur[0] = 0
    # encode: the fused syndrome kernel (standard), or k_field_add with masks
    # prepared ahead (boost; pipelined adds the preparation: fused syndrome +
    # k_output_mask); decode: challenge syndrome, k_verify_u, k_decrypt, k_check
    enc_launches = {"standard": 1, "boost": 1, "pipelined": 1 + 2}[args.mode]
    expected_per_step = enc_launches + (1 if args.server_mode == "multi" else VECTORS) + 4
    # the library's own count is what the line reports; the expected count is
    # a consistency check of the path the calls took
    launches_per_step = int(round(counted_per_step))
    if launches_per_step != expected_per_step:
        print(f"note: {launches_per_step} library launches per step, {expected_per_step} expected",
              file=sys.stderr, flush=True)
    step_no = [0]

    def step(record=None):
        k = step_no[0] % nsets
        step_no[0] += 1
        if args.mode == "pipelined":
            # the other set was used by the previous step, which is complete on
            # `stream` when this step starts: refill it for the next step
            fork = torch.cuda.Event()
            fork.record(stream)
            prep_stream.wait_event(fork)
            with torch.cuda.stream(prep_stream):
                g_preps[1 - k].replay()
        if record is not None:
            record[0].record(stream)
        g_encs[k].replay()
        if record is not None:
            record[1].record(stream)
        g_srv.replay()
        if record is not None:
            record[2].record(stream)
        g_decs[k].replay()
        if record is not None:
            record[3].record(stream)
        if args.mode == "pipelined":
            join = torch.cuda.Event()
            join.record(prep_stream)
            stream.wait_event(join)

    with torch.cuda.stream(stream):
        for _ in range(args.warmup):
            step()
    stream.synchronize()

    # ---- timed region: whole steps, one graph per step
    nsteps_sets = len(g_steps)
    w0, w1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        w0.record(stream)
        for w in range(args.warmup):
            g_steps[w % nsteps_sets].replay()
        w1.record(stream)
    stream.synchronize()
    ms_est = w0.elapsed_time(w1) / args.warmup
    clocks = ClockSampler(device.index)
    clocks.start()
    barrier(device)
    torch.cuda.synchronize(device)
    t_start = torch.cuda.Event(enable_timing=True)
    t_stop = torch.cuda.Event(enable_timing=True)
    clocks.region_started()
    with torch.cuda.stream(stream):
        t_start.record(stream)
        for s in range(args.steps):
            g_steps[s % nsteps_sets].replay()
        t_stop.record(stream)
        # untimed: the same steps, so that the clock samples see this load
        clock_tail(lambda i: g_steps[(args.steps + i) % nsteps_sets].replay(), ms_est)
    stream.synchronize()
    torch.cuda.synchronize(device)
    clk = clocks.stop()
    barrier(device)
    ms_local = t_start.elapsed_time(t_stop)
    ms = max_over_ranks(ms_local, device)

    # ---- the same steps as one graph per phase, with per-phase events on the
    # launching stream (the split reported in phases_ms and the GEMV launch
    # the roofline uses)
    phase_events = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(args.steps)]
    step_no[0] = 0
    with torch.cuda.stream(stream):
        for s in range(args.steps):
            step(phase_events[s])
    stream.synchronize()
    enc_ms = sum(e[0].elapsed_time(e[1]) for e in phase_events) / args.steps
    srv_ms = sum(e[1].elapsed_time(e[2]) for e in phase_events) / args.steps
    dec_ms = sum(e[2].elapsed_time(e[3]) for e in phase_events) / args.steps

    macs_per_step = VECTORS * M * K
    value = world * macs_per_step * args.steps / (ms / 1e3)
    gemv_s = srv_ms / 1e3 / VECTORS                     # per request
    gemv_bytes = M * K + 4 * K + 4 * M                  # W int8 + x_hat + y_hat per request
    peaks, peak_kind = measured_peaks()
    achieved = gemv_bytes / gemv_s / 1e9
    traffic = gemv_traffic_per_launch()

    # ---- end to end through the public API with pinned host buffers
    Xhost = torch.from_numpy(X.view(np.int32)).pin_memory()
    Yhost = torch.empty((VECTORS, M), dtype=torch.int32).pin_memory()
    Ahost = torch.empty(VECTORS, dtype=torch.int32).pin_memory()
    Xin = torch.empty_like(Xd)

    def e2e_step():
        Xin.copy_(Xhost, non_blocking=True)
        if boost:
            pv.pvmvmd_boost_encode(Xin, mi[0], Xhat=Xh, stream=stream)
        else:
            pv.pvmvmd_encode(ctx, Xin, 31 + rank, Xhat=Xh, st=st, stream=stream)
        server()
        if boost:
            pv.pvmvmd_boost_decode_verify(ctx, mo[0], Xh, Yh, 32 + rank, Y=Y, accept=acc, stream=stream)
        else:
            pv.pvmvmd_decode_verify(ctx, st, Xh, Yh, 32 + rank, Y=Y, accept=acc, stream=stream)
        Yhost.copy_(Y, non_blocking=True)
        Ahost.copy_(acc, non_blocking=True)

    if overlap:
        # the same pipeline through the public calls: the next batch's host
        # copy and encode beside this batch's decode and copy back
        Xins = [torch.empty_like(Xd) for _ in range(2)]
        with torch.cuda.stream(stream):
            Xins[0].copy_(Xhost, non_blocking=True)
            pv.pvmvmd_encode(ctx, Xins[0], 21 + rank, Xhat=Xh_sets[0], st=st_sets[0], stream=stream)
        stream.synchronize()
        ges = [capture(lambda k=k: overlapped_step(k, Xins, Xhost, (Yhost, Ahost)), stream) for k in range(2)]
    else:
        with torch.cuda.stream(stream):
            e2e_step()
        stream.synchronize()
        ges = [capture(e2e_step, stream)]
    e2e_steps = max(2, args.steps // 2)
    with torch.cuda.stream(stream):
        for w in range(args.warmup):
            ges[w % len(ges)].replay()
    stream.synchronize()
    barrier(device)
    t0 = time.perf_counter()
    with torch.cuda.stream(stream):
        for s_ in range(e2e_steps):
            ges[s_ % len(ges)].replay()
    stream.synchronize()
    e2e_s = max_over_ranks(time.perf_counter() - t0, device)
    assert int(Ahost.sum()) == VECTORS
    e2e_value = world * macs_per_step * e2e_steps / e2e_s

    cpu = cpu_all = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        n = args.cpu_vectors
        ow = OracleWorkload()
        macs, dt = ow.full_vectors(n)
        host = host_cpu()
        cpu = {"value": macs / dt, "unit": UNIT, "cores": 1, "kind": "oracle",
               "sample": f"{n} vector round trips (encrypt, server MVM, verify, decrypt) cycling over "
                         f"the workload's {VECTORS} vectors; single-threaded C oracle on the host; "
                         "its preprocessing untimed", "host": host}
        # the oracle's server MVM on every core: rows of W split over processes
        procs = max(1, host["cpu_count"] or 1)
        Xo = np.stack([ow.x[b % VECTORS] for b in range(8 * procs)])
        macs_p, dt_p, y_last = oracle_rows_parallel(ow.W, Xo, procs)
        assert np.array_equal(y_last, ow.o.server_mvm(ow.W, Xo[-1]))
        cpu_all = {"value": macs_p / dt_p, "unit": UNIT, "cores": procs, "kind": "oracle",
                   "sample": f"server MVM only (the bulk of a round trip) of {len(Xo)} vectors, the rows "
                             f"of W split over {procs} spawned processes running the unchanged C oracle",
                   "host": host}

    line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms / args.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "u32 (F_q exact; int8 weights, dp4a digits)",
            "data": "synthetic", "config": arm_config(args),
            "hbm_gbs_gemv": achieved,
            "phases_ms": {"encode": enc_ms, "server_100_gemv": srv_ms, "decode_verify": dec_ms},
            "roofline": {"bound": "hbm", "kernel": "k_gemv_multi (batch-1 field GEMV, 100 requests per launch)",
                         "achieved": achieved,
                         "peak": peaks["hbm_gbs"], "unit": "GB/s", "frac": achieved / peaks["hbm_gbs"],
                         "peak_kind": f"{peak_kind} hbm_gbs", "traffic": traffic,
                         "algorithmic_bytes_per_launch": gemv_bytes * (VECTORS if args.server_mode == "multi" else 1),
                         "launch_ms": srv_ms if args.server_mode == "multi" else srv_ms / VECTORS},
            "cpu_baseline": cpu,
            "cpu_baseline_all_cores": cpu_all,
            "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": int(Xhost.numel() * 4),
                    "d2h_bytes_per_step": int(Yhost.numel() * 4 + Ahost.numel() * 4),
                    "how": "CUDA graph of the public calls with pinned host copies inside, replayed"
                           + ("; the next batch's copy-in and encode beside this batch's decode" if overlap else "")
                           + ("" if args.mode == "standard" else "; masks prepared ahead (boost encode and decode)")},
            "gpu_launches": launches_per_step * args.steps,
            "clocks": clk,
        }
    ctx.destroy()
    del Wrep, Wd, jobs_sets, jobs, g_steps, ges, g_encs, g_decs, g_preps, g_srv
    torch.cuda.synchronize(device)
    torch.cuda.empty_cache()
    if world == 1 and not args.no_extra_configs:
        # the other configurations the metric is quoted on, as sub-records of
        # this line: the 8B- and 70B-class batched pipelines (the tensor-core
        # half of the metric) and one 8B-class token at batch 1, the server's
        # chain alone and with the client's encodes and decodes of every call
        line["configs"] = {
            "layer8b-b64": measure_batched(args, "layer8b-b64", device, rank, world,
                                           with_cpu=not args.no_cpu_baseline),
            "layer70b-b256": measure_batched(args, "layer70b-b256", device, rank, world,
                                             with_cpu=not args.no_cpu_baseline),
            "token8b-b1": measure_token(args, device, rank),
            "token8b-b1-client": measure_token_client(args, device, rank),
        }
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()
    return 0


# --------------------------------------------------------------------------- batched workloads

BATCHED = {
    # one 8B-class decoder layer, 64 vectors per projection
    "layer8b-b64": {"B": 64, "shapes": [("q", 4096, 4096), ("k", 1024, 4096), ("v", 1024, 4096),
                                        ("o", 4096, 4096), ("gate", 14336, 4096), ("up", 14336, 4096),
                                        ("down", 4096, 14336)]},
    # one Qwen3-4B block (the paper's evaluation model) with an eight-token prompt
    "layerqwen4b-b8": {"B": 8, "shapes": [("q", 4096, 2560), ("k", 1024, 2560), ("v", 1024, 2560),
                                          ("o", 2560, 4096), ("gate", 9728, 2560), ("up", 9728, 2560),
                                          ("down", 2560, 9728)]},
    # 70B-class projections, 256 vectors each
    "layer70b-b256": {"B": 256, "shapes": [("q", 8192, 8192), ("kv", 1024, 8192), ("gate_up", 28672, 8192),
                                           ("down", 8192, 28672)]},
}


def measure_batched(args, workload, device, rank=0, world=1, with_cpu=True, with_e2e=True):
    """Step = for every projection of the layer: encode B vectors, the
    batched server product, decode+verify.  The server phase (tcgen05 digit
    GEMM) is reported against the 16-bit tensor peak: it executes
    2 * m * K * 4 * B fp16 flops (four digit planes per field MAC).  Returns
    the record (a dict); run_batched prints it as the bench line."""
    import torch
    import paper_2609_10264_gb300 as pv
    from paper_2609_10264_gb300 import workloads as wl
    spec = BATCHED[workload]
    B = spec["B"]
    torch.cuda.synchronize(device)
    stream = torch.cuda.Stream(device)
    projs = []
    for j, (name, m, K) in enumerate(spec["shapes"]):
        W = wl.weights_gaussian(m, K, (7, j))
        x = wl.int8_vectors(B, K, (8, j))
        X = np.mod(x, pv.PVMVMD_Q).astype(np.uint32)
        Wd = torch.from_numpy(W).to(device)
        Xd = torch.from_numpy(X.view(np.int32)).to(device)
        params = pv.pvmvmd_params()
        params.scratch_batch = B
        ctx = pv.pvmvmd_preprocess(Wd, key=100 + j, params=params)
        projs.append(dict(name=name, m=m, K=K, W=Wd, X=Xd, ctx=ctx, x=x, Wh=W,
                          Xh=torch.empty_like(Xd), st=torch.empty((B, 2 * ctx.t_x), dtype=torch.int32, device=device),
                          Yh=torch.empty((B, m), dtype=torch.int32, device=device),
                          Y=torch.empty((B, m), dtype=torch.int32, device=device),
                          acc=torch.empty(B, dtype=torch.int32, device=device)))
    torch.cuda.synchronize(device)   # the inputs, made on torch's stream, are ready for the others

    def enc():
        for p in projs:
            pv.pvmvmd_encode(p["ctx"], p["X"], 21, Xhat=p["Xh"], st=p["st"], stream=stream)
    # the layer's independent server products, spread over a few streams so
    # that a small projection's product can use the SMs a larger one leaves
    srv_streams = [torch.cuda.Stream(device) for _ in range(max(1, args.server_streams))]

    grouped_jobs = pv.batch_jobs([(p["W"], p["Xh"], p["Yh"]) for p in projs])

    def srv():
        if args.server_call == "grouped":
            # the layer's products in one call: one persistent launch
            pv.pvmvmd_server_mvm_grouped(grouped_jobs, stream=stream)
            return
        fork = torch.cuda.Event()
        fork.record(stream)
        for ss in srv_streams:
            ss.wait_event(fork)
        for j, p in enumerate(projs):
            ss = srv_streams[j % len(srv_streams)]
            pv.pvmvmd_server_mvm(p["W"], p["Xh"], Yhat=p["Yh"], stream=ss)
        for ss in srv_streams:
            join = torch.cuda.Event()
            join.record(ss)
            stream.wait_event(join)

    def dec():
        for p in projs:
            pv.pvmvmd_decode_verify(p["ctx"], p["st"], p["Xh"], p["Yh"], 22, Y=p["Y"], accept=p["acc"], stream=stream)

    # --schedule projections: each projection's encode -> product -> decode
    # runs in order on one of a few streams, so one projection's client work
    # overlaps another's server product (the same calls, reordered across
    # independent projections)
    proj_streams = [torch.cuda.Stream(device) for _ in range(max(1, args.server_streams))]

    def pipelined(host=None):
        fork = torch.cuda.Event()
        fork.record(stream)
        for ss in proj_streams:
            ss.wait_event(fork)
        for j, p in enumerate(projs):
            ss = proj_streams[j % len(proj_streams)]
            with torch.cuda.stream(ss):
                src = p["X"]
                if host is not None:      # end to end: the inputs arrive from pinned host memory
                    p["Xin"].copy_(p["Xhost"], non_blocking=True)
                    src = p["Xin"]
                pv.pvmvmd_encode(p["ctx"], src, 21, Xhat=p["Xh"], st=p["st"], stream=ss)
                pv.pvmvmd_server_mvm(p["W"], p["Xh"], Yhat=p["Yh"], stream=ss)
                pv.pvmvmd_decode_verify(p["ctx"], p["st"], p["Xh"], p["Yh"], 22, Y=p["Y"], accept=p["acc"],
                                        stream=ss)
                if host is not None:
                    p["Yhost"].copy_(p["Y"], non_blocking=True)
                    p["Ahost"].copy_(p["acc"], non_blocking=True)
        for ss in proj_streams:
            join = torch.cuda.Event()
            join.record(ss)
            stream.wait_event(join)

    def phases():
        enc(); srv(); dec()

    def forked(per_proj):
        # per_proj(p, on) for every projection on one of the side streams
        fork = torch.cuda.Event()
        fork.record(stream)
        for ss in proj_streams:
            ss.wait_event(fork)
        for j, p in enumerate(projs):
            ss = proj_streams[j % len(proj_streams)]
            with torch.cuda.stream(ss):
                per_proj(p, ss)
        for ss in proj_streams:
            join = torch.cuda.Event()
            join.record(ss)
            stream.wait_event(join)

    def grouped(host=None):
        # --schedule grouped: the encodes side by side on the side streams,
        # the layer's products in one grouped call, the decodes side by side
        def e(p, on):
            src = p["X"]
            if host is not None:
                p["Xin"].copy_(p["Xhost"], non_blocking=True)
                src = p["Xin"]
            pv.pvmvmd_encode(p["ctx"], src, 21, Xhat=p["Xh"], st=p["st"], stream=on)

        def d(p, on):
            pv.pvmvmd_decode_verify(p["ctx"], p["st"], p["Xh"], p["Yh"], 22, Y=p["Y"], accept=p["acc"], stream=on)
            if host is not None:
                p["Yhost"].copy_(p["Y"], non_blocking=True)
                p["Ahost"].copy_(p["acc"], non_blocking=True)
        forked(e)
        pv.pvmvmd_server_mvm_grouped(grouped_jobs, stream=stream)
        forked(d)

    # --schedule pipeline: three batches in flight.  Step k encodes batch
    # k + 1, runs the server products of batch k (one grouped call) and
    # decodes batch k - 1, the three branches side by side on their own
    # streams; every step still encodes, multiplies and decodes one batch of
    # every projection.  Three sets of buffers rotate (an encode and a decode
    # of one context may overlap; two of either never do).
    nsets = 3
    # zero-filled: the first two eager steps decode sets that hold no batch
    # yet, and a zero mask state indexes row 0 of P^T, which exists
    for p in projs:
        p["sets"] = [dict(Xh=torch.zeros_like(p["X"]), st=torch.zeros_like(p["st"]), Yh=torch.zeros_like(p["Yh"]),
                          Y=torch.zeros_like(p["Y"]), acc=torch.zeros_like(p["acc"])) for _ in range(nsets)]
    set_jobs = [pv.batch_jobs([(p["W"], p["sets"][i]["Xh"], p["sets"][i]["Yh"]) for p in projs])
                for i in range(nsets)]
    srv_stream = torch.cuda.Stream(device)
    dec_streams = [torch.cuda.Stream(device) for _ in range(max(1, args.server_streams))]

    def pipeline_step(k, host=None):
        se, sv, sd = (k + 1) % nsets, k % nsets, (k - 1) % nsets
        fork = torch.cuda.Event()
        fork.record(stream)
        branches = proj_streams + dec_streams + [srv_stream]
        for ss in branches:
            ss.wait_event(fork)
        for j, p in enumerate(projs):
            ss = proj_streams[j % len(proj_streams)]
            with torch.cuda.stream(ss):
                src, b = p["X"], p["sets"][se]
                if host is not None:
                    b["Xin"].copy_(p["Xhost"], non_blocking=True)
                    src = b["Xin"]
                pv.pvmvmd_encode(p["ctx"], src, 21, Xhat=b["Xh"], st=b["st"], stream=ss)
        pv.pvmvmd_server_mvm_grouped(set_jobs[sv], stream=srv_stream)
        for j, p in enumerate(projs):
            ss = dec_streams[j % len(dec_streams)]
            with torch.cuda.stream(ss):
                b = p["sets"][sd]
                pv.pvmvmd_decode_verify(p["ctx"], b["st"], b["Xh"], b["Yh"], 22, Y=b["Y"], accept=b["acc"],
                                        stream=ss)
                if host is not None:
                    b["Yhost"].copy_(b["Y"], non_blocking=True)
                    b["Ahost"].copy_(b["acc"], non_blocking=True)
        for ss in branches:
            join = torch.cuda.Event()
            join.record(ss)
            stream.wait_event(join)

    if args.schedule == "pipeline":
        # fill the pipeline eagerly: after steps -1, 0, 1 batch 0 is decoded
        with torch.cuda.stream(stream):
            for k in (-1, 0, 1):
                pipeline_step(k)
        stream.synchronize()
        for p in projs:
            b = p["sets"][0]
            p["Y"].copy_(b["Y"])
            p["acc"].copy_(b["acc"])
        torch.cuda.synchronize(device)

    step_fn = {"projections": pipelined, "phases": phases, "grouped": grouped, "pipeline": None}[args.schedule]
    # eager runs of every schedule that is captured below (the first call on
    # a stream sizes its scratch, which a capture may not do)
    with torch.cuda.stream(stream):
        if step_fn is not None:
            enc(); srv(); dec()
            step_fn()
        else:   # the pipeline's output was checked out above; the phases still run eagerly once
            Ysave = [(p["Y"].clone(), p["acc"].clone()) for p in projs]
            enc(); srv(); dec()
    stream.synchronize()
    if step_fn is None:
        for p, (yv, av) in zip(projs, Ysave):
            assert torch.equal(yv, p["Y"]) and torch.equal(av, p["acc"]), "pipelined batch differs from the phases"
    assert pv.pvmvmd_device_status(stream) == 0
    for p in projs:
        assert int(p["acc"].sum()) == B
        rows = [0, p["m"] // 2, p["m"] - 1]
        got = pv.as_u32(p["Y"])[:, rows].astype(np.int64)
        got = np.where(got > (pv.PVMVMD_Q - 1) // 2, got - pv.PVMVMD_Q, got)
        assert np.array_equal(got, p["x"] @ p["Wh"][rows].astype(np.int64).T), p["name"]
    graphs = []
    # the phases as the step runs them: with the grouped and pipeline
    # schedules the encodes and the decodes run side by side on the side
    # streams (one after the other on `stream` for --schedule phases)
    if args.schedule in ("grouped", "pipeline"):
        def enc_side(p, on):
            pv.pvmvmd_encode(p["ctx"], p["X"], 21, Xhat=p["Xh"], st=p["st"], stream=on)

        def dec_side(p, on):
            pv.pvmvmd_decode_verify(p["ctx"], p["st"], p["Xh"], p["Yh"], 22, Y=p["Y"], accept=p["acc"], stream=on)
        phase_fns = (lambda: forked(enc_side), srv, lambda: forked(dec_side))
        with torch.cuda.stream(stream):   # eager once before the captures
            for fn in phase_fns:
                fn()
        stream.synchronize()
    else:
        phase_fns = (enc, srv, dec)
    for fn in phase_fns:
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            fn()
        graphs.append(g)
    # the whole step as one graph (what `value` times); the per-phase graphs
    # give the phase split.  The library counts the kernels it enqueues, also
    # while a stream is captured: the count around the step captures is the
    # kernels every replay of those graphs launches.
    n_launch0 = pv.pvmvmd_kernel_launches()
    if step_fn is not None:
        g_step = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g_step, stream=stream):
            step_fn()
        step_graphs = [g_step]
    else:
        step_graphs = []
        for k in range(nsets):
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                pipeline_step(k)
            step_graphs.append(g)
    nsg = len(step_graphs)
    launches_per_graph = (pv.pvmvmd_kernel_launches() - n_launch0) / nsg
    w0, w1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        for g in graphs:
            g.replay()
        w0.record(stream)
        for w in range(args.warmup * nsg):
            step_graphs[w % nsg].replay()
        w1.record(stream)
    stream.synchronize()
    ms_est = w0.elapsed_time(w1) / (args.warmup * nsg)
    clocks = ClockSampler(device.index)
    clocks.start()
    barrier(device)
    torch.cuda.synchronize(device)
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    clocks.region_started()
    with torch.cuda.stream(stream):
        t0.record(stream)
        for s_ in range(args.steps):
            step_graphs[s_ % nsg].replay()
        t1.record(stream)
        clock_tail(lambda i: step_graphs[(args.steps + i) % nsg].replay(), ms_est)
    stream.synchronize()
    if step_fn is None:
        # the batch decoded by the last timed step completed its three steps
        last = (args.steps - 2) % nsets
        for p in projs:
            assert int(p["sets"][last]["acc"].sum()) == B, "pipelined batch rejected"
    torch.cuda.synchronize(device)
    clk = clocks.stop()
    barrier(device)
    ms = max_over_ranks(t0.elapsed_time(t1), device)
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(args.steps)]
    with torch.cuda.stream(stream):
        for s in range(args.steps):
            for k, g in enumerate(graphs):
                ev[s][k].record(stream)
                g.replay()
            ev[s][3].record(stream)
    stream.synchronize()
    ph = [sum(e[k].elapsed_time(e[k + 1]) for e in ev) / args.steps for k in range(3)]
    macs = sum(p["m"] * p["K"] for p in projs) * B
    flops = 2 * 4 * macs
    peaks, kind = measured_peaks()

    # the dominant kernel as the step launches it, alone, by CUDA events on
    # its stream: the layer's products in one grouped call (one launch of
    # k_batched_grouped), or the largest projection's product when the
    # products are separate calls
    big = max(projs, key=lambda p: p["m"] * p["K"])
    grouped_call = args.server_call == "grouped"

    def one_product():
        if grouped_call:
            pv.pvmvmd_server_mvm_grouped(grouped_jobs, stream=stream)
        else:
            pv.pvmvmd_server_mvm(big["W"], big["Xh"], Yhat=big["Yh"], stream=stream)
    with torch.cuda.stream(stream):   # sizes this stream's scratch before the capture
        one_product()
    stream.synchronize()
    g_big = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g_big, stream=stream):
        one_product()
    k0, k1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    reps = max(args.steps, 5)
    with torch.cuda.stream(stream):
        for _ in range(args.warmup):
            g_big.replay()
        k0.record(stream)
        for _ in range(reps):
            g_big.replay()
        k1.record(stream)
    stream.synchronize()
    big_ms = k0.elapsed_time(k1) / reps

    if B <= 16 and args.server_call == "grouped":
        # a few vectors in 16-vector tensor-core tiles: one pass over M per
        # call, so the product is bound by HBM, not by the tensor pipe
        nbytes = sum(p["m"] * p["K"] + 4 * B * (p["K"] + p["m"]) for p in projs)
        roof = {"bound": "hbm", "kernel": "k_batched_grouped<16> (tcgen05, 16-vector tiles), server phase",
                "achieved": nbytes / (ph[1] / 1e3) / 1e9, "peak": peaks.get("hbm_gbs", 0.0), "unit": "GB/s",
                "peak_kind": f"{kind} hbm_gbs", "bytes_per_step": nbytes, "traffic": None}
        dtype = "u32 (F_q exact; fp16 digit MMAs, fp32 TMEM accumulation)"
    elif B <= 16 and all(p["K"] % 16 == 0 for p in projs):
        # a few vectors run the dp4a GEMV over four vectors' digit planes: one
        # pass over M per four vectors, x_hat read and y_hat written once
        nbytes = sum(p["m"] * p["K"] * ((B + 3) // 4) + 4 * B * (p["K"] + p["m"]) for p in projs)
        roof = {"bound": "hbm", "kernel": "k_gemv_nb (dp4a, four vectors per pass over M), server phase",
                "achieved": nbytes / (ph[1] / 1e3) / 1e9, "peak": peaks.get("hbm_gbs", 0.0), "unit": "GB/s",
                "peak_kind": f"{kind} hbm_gbs", "bytes_per_step": nbytes, "traffic": None}
        dtype = "u32 (F_q exact; int8 weights, dp4a digits)"
    else:
        peak = peaks.get("bf16_tflops_sustained", peaks["bf16_tflops"])
        big_flops = 2 * 4 * (macs if grouped_call else big["m"] * big["K"] * B)
        roof = {"bound": "tensor",
                "kernel": ("k_batched_grouped (tcgen05 kind::f16 digit GEMM) over the layer's products, one "
                           "pvmvmd_server_mvm_grouped call as the step makes it" if grouped_call else
                           f"k_batched_grouped (tcgen05 kind::f16 digit GEMM) on {big['name']} "
                           f"{big['m']}x{big['K']}x{B}, one pvmvmd_server_mvm call") +
                          " (k_digit_tiles_grouped + k_batched_grouped, + k_split_finish when K is split), "
                          "timed alone by CUDA events",
                "achieved": big_flops / (big_ms / 1e3) / 1e12, "peak": peaks["bf16_tflops"], "unit": "TFLOP/s",
                "peak_kind": f"{kind} bf16_tflops (burst; the kernel timed alone)", "traffic": None,
                "flops_per_launch": big_flops, "launch_ms": big_ms,
                "server_phase": {"achieved": flops / (ph[1] / 1e3) / 1e12, "peak": peak, "unit": "TFLOP/s",
                                 "frac": flops / (ph[1] / 1e3) / 1e12 / peak,
                                 "peak_kind": f"{kind} bf16_tflops_sustained (inside the step)",
                                 "flops_per_step": flops}}
        dtype = "u32 (F_q exact; fp16 digit MMAs, fp32 TMEM accumulation)"
    roof["frac"] = roof["achieved"] / roof["peak"] if roof["peak"] else None
    roof["field_macs_per_step"] = macs
    roof["field_mac_per_s_server"] = macs / (ph[1] / 1e3)

    e2e = None
    if with_e2e:
        for p in projs:
            p["Xhost"] = pv_host_copy(p["X"])
            p["Xin"] = torch.empty_like(p["X"])
            p["Yhost"] = torch.empty((B, p["m"]), dtype=torch.int32).pin_memory()
            p["Ahost"] = torch.empty(B, dtype=torch.int32).pin_memory()
        if args.schedule == "pipeline":
            for p in projs:
                for b in p["sets"]:
                    b["Xin"] = torch.empty_like(p["X"])
                    b["Yhost"] = torch.empty((B, p["m"]), dtype=torch.int32).pin_memory()
                    b["Ahost"] = torch.empty(B, dtype=torch.int32).pin_memory()
            with torch.cuda.stream(stream):
                for k in (-1, 0, 1):
                    pipeline_step(k, host=True)
            stream.synchronize()
            e2e_graphs = []
            for k in range(nsets):
                g = torch.cuda.CUDAGraph()
                with torch.cuda.graph(g, stream=stream):
                    pipeline_step(k, host=True)
                e2e_graphs.append(g)
        else:
            e2e_fn = grouped if args.schedule == "grouped" else pipelined
            with torch.cuda.stream(stream):
                e2e_fn(host=True)
            stream.synchronize()
            g_e2e = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g_e2e, stream=stream):
                e2e_fn(host=True)
            e2e_graphs = [g_e2e]
        ne = len(e2e_graphs)
        with torch.cuda.stream(stream):
            for w in range(args.warmup * ne):
                e2e_graphs[w % ne].replay()
        stream.synchronize()
        barrier(device)
        n_e2e = max(3, args.steps)
        te = time.perf_counter()
        with torch.cuda.stream(stream):
            for i in range(n_e2e):
                e2e_graphs[i % ne].replay()
        stream.synchronize()
        e2e_s = max_over_ranks(time.perf_counter() - te, device)
        for p in projs:
            hosts = [b["Ahost"] for b in p["sets"]] if args.schedule == "pipeline" else [p["Ahost"]]
            assert any(int(h.sum()) == B for h in hosts)
        e2e = {"value": world * macs * n_e2e / e2e_s, "unit": UNIT,
               "h2d_bytes_per_step": int(sum(p["Xhost"].numel() * 4 for p in projs)),
               "d2h_bytes_per_step": int(sum(p["Yhost"].numel() * 4 + p["Ahost"].numel() * 4 for p in projs)),
               "how": ("CUDA graphs of the public calls, three batches in flight (batch k + 1's encodes, "
                       "batch k's grouped product call and batch k - 1's decodes side by side)"
                       if args.schedule == "pipeline" else
                       "CUDA graph of the public calls (the encodes side by side on "
                       f"{len(proj_streams)} streams, one grouped product call, the decodes side by side)"
                       if args.schedule == "grouped" else
                       "CUDA graph of the public calls (each projection's encode, product, decode on one of "
                       f"{len(proj_streams)} streams)") + " with pinned host copies of X in and Y, accept out, "
                      "replayed; wall clock"}

    cpu = None
    if with_cpu and rank == 0:
        # the oracle's server MVM (the per-MAC C loop, unchanged) on every host
        # core, on a row sample of the dominant projection
        host = host_cpu()
        procs = max(1, host["cpu_count"] or 1)
        rows = min(big["m"], 2048)
        Xo = pv.as_u32(big["Xh"])[: min(B, 4 * procs)]
        macs_p, dt_p, y_last = oracle_rows_parallel(np.ascontiguousarray(big["Wh"][:rows]), Xo, procs)
        assert np.array_equal(y_last, pv.as_u32(big["Yh"])[len(Xo) - 1, :rows]), "oracle and GPU products differ"
        cpu = {"value": macs_p / dt_p, "unit": UNIT, "cores": procs, "kind": "oracle",
               "sample": f"server MVM only, {len(Xo)} masked vectors of the {big['name']} projection on its first "
                         f"{rows} rows (K = {big['K']}), the rows split over {procs} spawned processes running "
                         "the unchanged C oracle; its last product equals the GPU's",
               "host": host}
    rec = {
        "metric": METRIC, "value": world * macs * args.steps / (ms / 1e3), "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": dtype, "data": "synthetic",
        "config": {"workload": workload, "B": B, "projections": [[p["name"], p["m"], p["K"]] for p in projs],
                   "schedule": args.schedule, "server_call": args.server_call, "streams": args.server_streams,
                   "l2": "weights, P^T and Q of the layer exceed L2"},
        "phases_ms": {"encode": ph[0], "server_batched": ph[1], "decode_verify": ph[2]},
        "roofline": roof, "e2e": e2e, "cpu_baseline": cpu,
        "gpu_launches": int(round(launches_per_graph * args.steps)), "clocks": clk}
    for p in projs:
        p["ctx"].destroy()
    projs.clear()
    torch.cuda.synchronize(device)
    torch.cuda.empty_cache()
    return rec


def pv_host_copy(t):
    """A pinned host copy of a device tensor."""
    return t.cpu().pin_memory()


def run_batched(args):
    import torch
    rank, world, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    device = torch.device("cuda", local)
    torch.cuda.set_device(device)
    rec = measure_batched(args, args.workload, device, rank, world, with_cpu=not args.no_cpu_baseline)
    if rank == 0:
        print(json.dumps(rec), flush=True)
    return 0


TOKEN_GROUPS = (("q", "k", "v"), ("o",), ("gate", "up"), ("down",))


def measure_token(args, device, rank=0):
    """One token of 32 independent 8B-class layers at batch 1 (the server's
    side).  Within a layer the products depend on one another as in a
    decoder: q, k and v read the layer input; o reads the attention output;
    gate and up read the attention block's output; down reads the MLP's
    hidden state.  So a token is 4 dependent grouped calls per layer,
    {q,k,v} -> o -> {gate,up} -> down, 128 calls in order on one stream (one
    CUDA graph).  Weights are seeded int8 (Gaussian, sigma 32, rounded and
    clipped), 6.98 GB per token, so every token streams them from HBM; x_hat
    is uniform in F_q.  The relaxed schedules (one grouped call per layer,
    one per token) are reported beside it as context."""
    import torch
    import paper_2609_10264_gb300 as pv
    from paper_2609_10264_gb300 import workloads as wl
    Q = pv.PVMVMD_Q
    nlayers = 32
    gen = torch.Generator(device=device)
    layers = []
    for l in range(nlayers):
        trip = {}
        for j, (name, (m, K)) in enumerate(wl.LAYER_8B.items()):
            gen.manual_seed(1000 + 7 * l + j)
            W = (torch.randn((m, K), generator=gen, device=device) * 32.0).round_().clamp_(-127, 127).to(torch.int8)
            xh = torch.randint(0, Q, (K,), generator=gen, device=device, dtype=torch.int64).to(torch.int32)
            trip[name] = (W, xh, torch.empty(m, dtype=torch.int32, device=device))
        layers.append(trip)
    torch.cuda.synchronize(device)   # the inputs, made on torch's stream, are ready for `stream`
    dep_jobs = [[pv.mvm_jobs([t[n] for n in grp]) for grp in TOKEN_GROUPS] for t in layers]
    layer_jobs = [pv.mvm_jobs(list(t.values())) for t in layers]
    all_jobs = pv.mvm_jobs([v for t in layers for v in t.values()])
    torch.cuda.synchronize(device)
    stream = torch.cuda.Stream(device)

    def token_dep():
        for l in range(nlayers):
            for jobs in dep_jobs[l]:
                pv.pvmvmd_server_mvm_multi(jobs, stream=stream)

    def token_layer():
        for l in range(nlayers):
            pv.pvmvmd_server_mvm_multi(layer_jobs[l], stream=stream)

    def token_one():
        pv.pvmvmd_server_mvm_multi(all_jobs, stream=stream)

    with torch.cuda.stream(stream):
        token_dep()
    stream.synchronize()
    assert pv.pvmvmd_device_status(stream) == 0
    # exact check of sampled rows of every projection of two layers (int64 numpy)
    for l in (0, nlayers - 1):
        for name, (W, xh, yh) in layers[l].items():
            rows = [0, 1, W.shape[0] // 2, W.shape[0] - 1]
            Wr = W[rows].cpu().numpy().astype(np.int64)
            x = pv.as_u32(xh).astype(np.int64)
            assert np.array_equal(pv.as_u32(yh)[rows].astype(np.int64), (Wr @ x) % Q), f"layer {l} {name}"
    graphs = {}
    for key, fn in (("dep", token_dep), ("layer", token_layer), ("one", token_one)):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            fn()
        graphs[key] = g
    w0, w1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        w0.record(stream)
        for _ in range(args.warmup):
            graphs["dep"].replay()
        w1.record(stream)
    stream.synchronize()
    ms_est = w0.elapsed_time(w1) / args.warmup
    clocks = ClockSampler(device.index)
    clocks.start()
    torch.cuda.synchronize(device)
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    clocks.region_started()
    with torch.cuda.stream(stream):
        t0.record(stream)
        for _ in range(args.steps):
            graphs["dep"].replay()
        t1.record(stream)
        clock_tail(lambda i: graphs["dep"].replay(), ms_est)
    stream.synchronize()
    clk = clocks.stop()
    assert pv.pvmvmd_device_status(stream) == 0
    ms = t0.elapsed_time(t1) / args.steps
    relaxed = {}
    for key in ("layer", "one"):
        with torch.cuda.stream(stream):
            for _ in range(args.warmup):
                graphs[key].replay()
            t0.record(stream)
            for _ in range(args.steps):
                graphs[key].replay()
            t1.record(stream)
        stream.synchronize()
        relaxed[key] = t0.elapsed_time(t1) / args.steps
    macs = nlayers * sum(m * K for (m, K) in wl.LAYER_8B.values())
    nbytes = nlayers * sum(m * K + 4 * K + 4 * m for (m, K) in wl.LAYER_8B.values())
    peaks, kind = measured_peaks()
    achieved = nbytes / (ms / 1e3) / 1e9
    del graphs, layers
    torch.cuda.synchronize(device)
    torch.cuda.empty_cache()
    return {
        "metric": METRIC, "value": macs / (ms / 1e3), "unit": UNIT, "n_gpus": 1, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms, "ms_per_token": ms, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "u32 (F_q exact; int8 weights, dp4a digits)",
        "data": "synthetic",
        "config": {"workload": "token8b-b1", "layers": nlayers, "projections": list(wl.LAYER_8B),
                   "schedule": "per layer {q,k,v} -> o -> {gate,up} -> down: 4 dependent grouped "
                               "pvmvmd_server_mvm_multi calls, 128 per token, in order on one stream",
                   "weight_bytes_per_token": nbytes,
                   "l2": "6.98 GB of distinct weights per token (larger than L2)"},
        "relaxed_schedules": {
            "one_call_per_layer": {"ms": relaxed["layer"], "hbm_gbs": nbytes / (relaxed["layer"] / 1e3) / 1e9,
                                   "note": "the 7 products of a layer in one call, ignoring o's and "
                                           "down's dependence on q/k/v and gate/up"},
            "one_call_per_token": {"ms": relaxed["one"], "hbm_gbs": nbytes / (relaxed["one"] / 1e3) / 1e9,
                                   "note": "all 224 products in one call (a replay of a finished token)"}},
        "roofline": {"bound": "hbm", "kernel": "k_gemv_multi (1-3 requests per launch, 128 dependent launches)",
                     "achieved": achieved, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                     "frac": achieved / peaks["hbm_gbs"], "peak_kind": f"{kind} hbm_gbs", "traffic": None,
                     "algorithmic_bytes_per_token": nbytes},
        "gpu_launches": 4 * nlayers * args.steps, "clocks": clk}


def measure_token_client(args, device, rank=0):
    """One token through 32 8B-class layers at batch 1 with the client's work
    of every call in the chain: per layer, {q,k,v} -> o -> {gate,up} -> down,
    each group as the encodes of its inputs, one grouped server call and the
    decodes (verify + decrypt) of its outputs, the group's projections side by
    side, so every server call waits for its encodes and the next group for
    the decodes (224 encodes, 128 server calls and 224 decodes per token, one
    CUDA graph).  The client needs P^T and Q per matrix (13.8 GB for one
    layer), so the 32 layers share one layer's weights and contexts; part of
    each layer's 218 MB of weights then stays in the 126 MB L2, which the
    same chain without the client work (reported beside it) shows."""
    import torch
    import paper_2609_10264_gb300 as pv
    from paper_2609_10264_gb300 import workloads as wl
    Q = pv.PVMVMD_Q
    nlayers = 32
    projs = {}
    for j, (name, (m, K)) in enumerate(wl.LAYER_8B.items()):
        W = wl.weights_gaussian(m, K, (11, j))
        x = wl.int8_vectors(1, K, (12, j))
        Wd = torch.from_numpy(W).to(device)
        Xd = torch.from_numpy(np.mod(x, Q).astype(np.uint32).view(np.int32)).to(device)
        ctx = pv.pvmvmd_preprocess(Wd, key=300 + j)
        projs[name] = dict(W=Wd, Wh=W, x=x, X=Xd, ctx=ctx, Xh=torch.empty_like(Xd),
                           st=torch.empty((1, 2 * ctx.t_x), dtype=torch.int32, device=device),
                           Yh=torch.empty((1, m), dtype=torch.int32, device=device),
                           Y=torch.empty((1, m), dtype=torch.int32, device=device),
                           acc=torch.empty(1, dtype=torch.int32, device=device))
    torch.cuda.synchronize(device)
    jobs = [pv.mvm_jobs([(projs[n]["W"], projs[n]["Xh"][0], projs[n]["Yh"][0]) for n in grp])
            for grp in TOKEN_GROUPS]
    stream = torch.cuda.Stream(device)
    # a group's projections are independent: their encodes (and decodes) run
    # side by side, one side stream each, joined before the next step
    side = [torch.cuda.Stream(device) for _ in range(3)]

    def side_by_side(grp, call):
        if len(grp) == 1:
            call(projs[grp[0]], stream)
            return
        fork = torch.cuda.Event()
        fork.record(stream)
        for i, n in enumerate(grp):
            side[i].wait_event(fork)
            with torch.cuda.stream(side[i]):
                call(projs[n], side[i])
            join = torch.cuda.Event()
            join.record(side[i])
            stream.wait_event(join)

    def token(client=True):
        for l in range(nlayers):
            for g, grp in enumerate(TOKEN_GROUPS):
                if client:
                    side_by_side(grp, lambda p, on: pv.pvmvmd_encode(p["ctx"], p["X"], 4 * l + g + 1, Xhat=p["Xh"],
                                                                     st=p["st"], stream=on))
                pv.pvmvmd_server_mvm_multi(jobs[g], stream=stream)
                if client:
                    side_by_side(grp, lambda p, on: pv.pvmvmd_decode_verify(p["ctx"], p["st"], p["Xh"], p["Yh"],
                                                                            1000 + 4 * l + g, Y=p["Y"],
                                                                            accept=p["acc"], stream=on))

    with torch.cuda.stream(stream):
        token()
    stream.synchronize()
    assert pv.pvmvmd_device_status(stream) == 0
    for n, p in projs.items():   # every decoded output equals W x over the integers
        assert int(p["acc"].sum()) == 1, n
        y = pv.as_u32(p["Y"])[0].astype(np.int64)
        y = np.where(y > (Q - 1) // 2, y - Q, y)
        assert np.array_equal(y, p["Wh"].astype(np.int64) @ p["x"][0].astype(np.int64)), n
    graphs, launches = {}, {}
    for key, client in (("client", True), ("server", False)):
        n0 = pv.pvmvmd_kernel_launches()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            token(client)
        launches[key] = pv.pvmvmd_kernel_launches() - n0
        graphs[key] = g
    steps = max(3, min(args.steps, 20))
    ms = {}
    clk = None
    for key in ("client", "server"):
        with torch.cuda.stream(stream):
            for _ in range(args.warmup):
                graphs[key].replay()
        stream.synchronize()
        clocks = ClockSampler(device.index) if key == "client" else None
        if clocks:
            clocks.start()
        t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        if clocks:
            clocks.region_started()
        with torch.cuda.stream(stream):
            t0.record(stream)
            for _ in range(steps):
                graphs[key].replay()
            t1.record(stream)
        stream.synchronize()
        if clocks:
            clk = clocks.stop()
        ms[key] = t0.elapsed_time(t1) / steps
    assert pv.pvmvmd_device_status(stream) == 0 and all(int(p["acc"].sum()) == 1 for p in projs.values())
    macs = nlayers * sum(m * K for (m, K) in wl.LAYER_8B.values())
    for p in projs.values():
        p["ctx"].destroy()
    projs.clear()
    del graphs
    torch.cuda.synchronize(device)
    torch.cuda.empty_cache()
    return {
        "metric": METRIC, "value": macs / (ms["client"] / 1e3), "unit": UNIT, "n_gpus": 1, "steps": steps,
        "warmup": args.warmup, "ms_per_step": ms["client"], "ms_per_token": ms["client"], "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "u32 (F_q exact; int8 weights, dp4a digits)",
        "data": "synthetic",
        "config": {"workload": "token8b-b1-client", "layers": nlayers, "projections": list(wl.LAYER_8B),
                   "schedule": "per layer {q,k,v} -> o -> {gate,up} -> down; each group: the encodes of its "
                               "inputs side by side, one pvmvmd_server_mvm_multi call, the decodes of its outputs "
                               "side by side; the groups in order (224 encodes, 128 server calls, 224 decodes per "
                               "token)",
                   "weights": "one 8B-class layer's weights and client contexts shared by the 32 layers"},
        "server_only_ms_per_token": ms["server"],
        "client_ms_per_token": ms["client"] - ms["server"],
        "gpu_launches": launches["client"] * steps,
        "launches_per_token": launches, "clocks": clk}

def run_token(args):
    import torch
    rank, world, local = dist_env()
    device = torch.device("cuda", local)
    torch.cuda.set_device(device)
    rec = measure_token(args, device, rank)
    if rank == 0:
        print(json.dumps(rec), flush=True)
    return 0


def run_bv(args):
    """Batch verification (Protocol 2) of B = 8 claims y_b = M_b x_b with
    1024 x 1024 matrices: one round = the client's primary challenges, the
    server's projection u = Qt e and the client's checks (z_b = G^T y_b,
    secondary challenges and G' e', all checks).  Preprocessing (Qs and
    Qaux, 2.1 GB) runs before timing."""
    import torch
    rank, world, local = dist_env()
    device = torch.device("cuda", local)
    torch.cuda.set_device(device)
    import paper_2609_10264_gb300 as pv
    Q = pv.PVMVMD_Q
    B, m, n = 8, 1024, 1024
    gen = torch.Generator(device=device)
    gen.manual_seed(77)
    Ws = (torch.randn((B, m, n), generator=gen, device=device) * 32.0).round_().clamp_(-127, 127).to(torch.int8)
    X = torch.randint(0, Q, (B, n), generator=gen, device=device, dtype=torch.int64).to(torch.int32)
    # honest claims y_b = M_b x_b from the library's product (parity-tested)
    Y = torch.stack([pv.pvmvmd_server_mvm(Ws[b], X[b]) for b in range(B)])
    t0 = time.perf_counter()
    ctx = pv.pvmvmd_bv_preprocess(Ws, key=61)
    torch.cuda.synchronize(device)
    prep_s = time.perf_counter() - t0
    torch.cuda.synchronize(device)
    stream = torch.cuda.Stream(device)
    chal = torch.empty((ctx.ell, 2 * ctx.t), dtype=torch.int32, device=device)
    u = torch.empty((ctx.ell, B * n), dtype=torch.int32, device=device)
    acc = torch.empty(1, dtype=torch.int32, device=device)

    def rnd():
        pv.pvmvmd_bv_challenge(ctx, 62, chal=chal, stream=stream)
        pv.pvmvmd_bv_server_project(ctx, chal, u=u, stream=stream)
        pv.pvmvmd_bv_check(ctx, X, Y, chal, u, 63, accept=acc, stream=stream)

    with torch.cuda.stream(stream):
        rnd()
    stream.synchronize()
    pv.pvmvmd_device_status(stream)
    assert int(acc.item()) == 1, "honest claims must be accepted"
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        rnd()
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(4)]
    with torch.cuda.stream(stream):
        for _ in range(args.warmup):
            g.replay()
        ev[0].record(stream)
        for _ in range(args.steps):
            g.replay()
        ev[1].record(stream)
        # the server's projection alone
        for _ in range(args.warmup):
            pv.pvmvmd_bv_server_project(ctx, chal, u=u, stream=stream)
        ev[2].record(stream)
        for _ in range(args.steps):
            pv.pvmvmd_bv_server_project(ctx, chal, u=u, stream=stream)
        ev[3].record(stream)
    stream.synchronize()
    ms = ev[0].elapsed_time(ev[1]) / args.steps
    ms_srv = ev[2].elapsed_time(ev[3]) / args.steps
    macs = B * m * n
    if rank == 0:
        print(json.dumps({
            "metric": "batch-verified field MAC/s (Protocol 2)", "value": macs / (ms / 1e3), "unit": "field MAC/s",
            "n_gpus": 1, "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "u32 (F_q exact)", "data": "synthetic",
            "config": {"workload": "bv-b8-1024", "B": B, "m": m, "n": n, "N": ctx.N, "N2": ctx.N2,
                       "t": ctx.t, "ell": ctx.ell, "t2": ctx.t2, "ell2": ctx.ell2},
            "server_project_ms": ms_srv, "preprocess_s": prep_s,
            "gpu_launches": None}), flush=True)
    ctx.destroy()
    return 0


def run_encode_shape(args):
    """Encrypt alone for B vectors of length K (``--shape KxB``): x_hat =
    x + G_x e_x with fresh sparse masks, timed over --steps calls.  The
    matrix has 256 rows, so preprocessing and its tables stay small."""
    import torch
    rank, world, local = dist_env()
    device = torch.device("cuda", local)
    torch.cuda.set_device(device)
    import paper_2609_10264_gb300 as pv
    Q = pv.PVMVMD_Q
    K, B = (int(v) for v in args.shape.lower().split("x"))
    gen = torch.Generator(device=device)
    gen.manual_seed(81)
    W = torch.randint(-127, 128, (256, K), generator=gen, device=device, dtype=torch.int8)
    X = torch.randint(0, Q, (B, K), generator=gen, device=device, dtype=torch.int64).to(torch.int32)
    params = pv.pvmvmd_params()
    params.scratch_batch = max(B, 1)
    ctx = pv.pvmvmd_preprocess(W, key=82, params=params)
    torch.cuda.synchronize(device)
    stream = torch.cuda.Stream(device)
    Xh = torch.empty_like(X)
    st = torch.empty((B, 2 * ctx.t_x), dtype=torch.int32, device=device)
    with torch.cuda.stream(stream):
        for s in range(args.warmup):
            pv.pvmvmd_encode(ctx, X, 83 + s, Xhat=Xh, st=st, stream=stream)
    stream.synchronize()
    pv.pvmvmd_device_status(stream)
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        t0.record(stream)
        for s in range(args.steps):
            pv.pvmvmd_encode(ctx, X, 1000 + s, Xhat=Xh, st=st, stream=stream)
        t1.record(stream)
    stream.synchronize()
    pv.pvmvmd_device_status(stream)
    ms = t0.elapsed_time(t1) / args.steps
    N = ctx.N_x
    if rank == 0:
        print(json.dumps({
            "metric": "encrypted vectors/s", "value": B / (ms / 1e3), "unit": "vectors/s", "n_gpus": 1,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "u32 (F_q exact)", "data": "synthetic",
            "config": {"workload": "encode-shape", "K": K, "B": B, "N_x": N, "t_x": ctx.t_x},
            "gpu_launches": None}), flush=True)
    ctx.destroy()
    return 0


def run_encoder_shape(args):
    """The RAA encoder G^T alone (App. B; the operation preprocessing runs):
    ``--shape mxK`` encodes the m rows of an m x K matrix with G_x, i.e. L = m
    lanes of length n = K into N_x = 8K positions, as pvmvmd_preprocess does
    for P^T.  Each call is two gather / scale / decoupled-look-back
    prefix-scan launches over the N_x x m array.  Inputs are uniform in F_q;
    the arrays (a 4096 x 4096 shape moves 1.7 GB per call) exceed L2."""
    import torch
    rank, world, local = dist_env()
    device = torch.device("cuda", local)
    torch.cuda.set_device(device)
    import paper_2609_10264_gb300 as pv
    Q = pv.PVMVMD_Q
    m, K = (int(v) for v in args.shape.lower().split("x")[:2])
    gen = torch.Generator(device=device)
    gen.manual_seed(85)
    W = torch.randint(-127, 128, (16, K), generator=gen, device=device, dtype=torch.int8)
    ctx = pv.pvmvmd_preprocess(W, key=86)
    X = torch.randint(0, Q, (K, m), generator=gen, device=device, dtype=torch.int64).to(torch.int32)
    N = ctx.N_x
    Y = torch.empty((N, m), dtype=torch.int32, device=device)
    scratch = torch.empty(pv.pvmvmd_code_encode_scratch(ctx, 0, m), dtype=torch.uint8, device=device)
    torch.cuda.synchronize(device)
    stream = torch.cuda.Stream(device)
    with torch.cuda.stream(stream):
        for _ in range(args.warmup):
            pv.pvmvmd_code_encode_lanes(ctx, 0, X, Y=Y, scratch=scratch, stream=stream)
    stream.synchronize()
    assert pv.pvmvmd_device_status(stream) == 0
    clocks = ClockSampler(device.index)
    clocks.start()
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        t0.record(stream)
        for _ in range(args.steps):
            pv.pvmvmd_code_encode_lanes(ctx, 0, X, Y=Y, scratch=scratch, stream=stream)
        t1.record(stream)
    stream.synchronize()
    clk = clocks.stop()
    assert pv.pvmvmd_device_status(stream) == 0
    ms = t0.elapsed_time(t1) / args.steps
    # one read of X, the intermediate written and read once, Y written once
    nbytes = 4 * m * (K + 3 * N)
    peaks, kind = measured_peaks()
    achieved = nbytes / (ms / 1e3) / 1e9
    if rank == 0:
        print(json.dumps({
            "metric": "encoded field elements/s", "value": N * m / (ms / 1e3), "unit": "elements/s",
            "n_gpus": 1, "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "u32 (F_q exact)",
            "data": "synthetic",
            "config": {"workload": "encoder-shape", "lanes": m, "n": K, "N": N,
                       "l2": "arrays larger than L2"},
            "roofline": {"bound": "hbm", "kernel": "k_encode_scan (two launches per call)",
                         "achieved": achieved, "peak": peaks.get("hbm_gbs", 0.0), "unit": "GB/s",
                         "frac": achieved / peaks["hbm_gbs"] if peaks.get("hbm_gbs") else None,
                         "peak_kind": f"{kind} hbm_gbs", "algorithmic_bytes_per_call": nbytes},
            "gpu_launches": 2 * args.steps, "clocks": clk}), flush=True)
    ctx.destroy()
    return 0


def run_preprocess_shape(args):
    """pvmvmd_preprocess alone for an m x K int8 matrix (``--shape mxK``):
    both codes sampled on the host, P^T = G_x^T M^T and Q = G_y^T M encoded
    on the device, wall-clock per call (allocation included).  The paper's
    single-threaded CPU figures for the same step are 6.03 s at n = 2^12 and
    135.8 s at n = 2^14 (context, another machine)."""
    import torch
    rank, world, local = dist_env()
    device = torch.device("cuda", local)
    torch.cuda.set_device(device)
    import paper_2609_10264_gb300 as pv
    m, K = (int(v) for v in args.shape.lower().split("x")[:2])
    gen = torch.Generator(device=device)
    gen.manual_seed(87)
    W = torch.randint(-127, 128, (m, K), generator=gen, device=device, dtype=torch.int8)
    torch.cuda.synchronize(device)
    stream = torch.cuda.Stream(device)
    for w in range(args.warmup):
        pv.pvmvmd_preprocess(W, key=88 + w, stream=stream).destroy()
    torch.cuda.synchronize(device)
    times = []
    for s_ in range(args.steps):
        t0 = time.perf_counter()
        ctx = pv.pvmvmd_preprocess(W, key=200 + s_, stream=stream)
        stream.synchronize()
        times.append(time.perf_counter() - t0)
        assert pv.pvmvmd_device_status(stream) == 0
        ctx.destroy()
    sec = statistics.median(times)
    if rank == 0:
        print(json.dumps({
            "metric": "preprocessing time", "value": sec, "unit": "s", "n_gpus": 1, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": sec * 1e3, "higher_is_better": False, "scaling": "weak",
            "vs_baseline": None, "dtype": "u32 (F_q exact)", "data": "synthetic",
            "config": {"workload": "preprocess-shape", "m": m, "K": K, "N_x": 8 * K, "N_y": 8 * m,
                       "tables_bytes": 4 * 8 * 2 * m * K, "timing": "wall clock per call, median"},
            "gpu_launches": None}), flush=True)
    return 0


def run_server_shape(args):
    """The batched server product Y_hat = M X_hat alone on one m x K x B
    shape (``--shape MxKxB``), timed over --steps launches after --warmup.
    Each step rotates over enough independent weight copies that the weights
    read per step exceed the L2 cache."""
    import torch
    rank, world, local = dist_env()
    device = torch.device("cuda", local)
    torch.cuda.set_device(device)
    import paper_2609_10264_gb300 as pv
    from paper_2609_10264_gb300 import workloads as wl
    m, K, B = (int(v) for v in args.shape.lower().split("x"))
    copies = max(1, -(-256 * 2**20 // (m * K)))  # > 2x the 129 MB L2 in rotation
    Wh = wl.weights_gaussian(m, K, (9, 0))
    W0 = torch.from_numpy(Wh).to(device)
    W = [W0] + [W0.clone() for _ in range(copies - 1)]
    x = wl.int8_vectors(B, K, (10, 0))
    Xd = torch.from_numpy(np.mod(x, pv.PVMVMD_Q).astype(np.uint32).view(np.int32)).to(device)
    Y = torch.empty((B, m), dtype=torch.int32, device=device)
    torch.cuda.synchronize(device)
    stream = torch.cuda.Stream(device)
    with torch.cuda.stream(stream):
        pv.pvmvmd_server_mvm(W0, Xd, Yhat=Y, stream=stream)
    stream.synchronize()
    pv.pvmvmd_device_status(stream)
    rows = [0, m // 2, m - 1]
    got = pv.as_u32(Y)[:, rows].astype(np.int64)
    got = np.where(got > (pv.PVMVMD_Q - 1) // 2, got - pv.PVMVMD_Q, got)
    assert np.array_equal(got, x @ Wh[rows].astype(np.int64).T), "server product mismatch"
    # one CUDA graph of one call per weight copy, so that host-side call
    # overhead is not timed
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        for c in range(copies):
            pv.pvmvmd_server_mvm(W[c], Xd, Yhat=Y, stream=stream)
    reps = max(1, -(-args.steps // copies))
    with torch.cuda.stream(stream):
        for s in range(args.warmup):
            g.replay()
    stream.synchronize()
    clocks = ClockSampler(device.index)
    clocks.start()
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    clocks.region_started()
    with torch.cuda.stream(stream):
        t0.record(stream)
        for s in range(reps):
            g.replay()
        t1.record(stream)
        clock_tail(lambda i: g.replay(), 0.03 * copies)
    stream.synchronize()
    clk = clocks.stop()
    pv.pvmvmd_device_status(stream)
    ms = t0.elapsed_time(t1) / (reps * copies)
    macs = m * K * B
    peaks, kind = measured_peaks()
    if B <= 16 and K % 16 == 0:
        # small batches run the dp4a GEMV over four vectors' digit planes:
        # one pass over M per four vectors, x_hat read and y_hat written once
        nbytes = m * K * ((B + 3) // 4) + 4 * B * (K + m)
        roof = {"bound": "hbm", "kernel": "k_gemv_nb (dp4a, four vectors per pass over M)",
                "achieved": nbytes / (ms / 1e3) / 1e9, "peak": peaks.get("hbm_gbs", 0.0), "unit": "GB/s",
                "bytes_per_call": nbytes, "peak_kind": f"{kind} hbm_gbs"}
        launches = 2 * args.steps  # k_nb_planes + k_gemv_nb
    else:
        flops = 2 * 4 * macs
        roof = {"bound": "tensor", "kernel": "k_batched (tcgen05 kind::f16 digit GEMM) + k_digit_tiles",
                "achieved": flops / (ms / 1e3) / 1e12, "peak": peaks.get("bf16_tflops", 0.0), "unit": "TFLOP/s",
                "peak_kind": f"{kind} bf16_tflops (burst)"}
        launches = None  # k_digit_tiles_grouped + k_batched_grouped (+ k_split_finish when K is split)
    roof["frac"] = roof["achieved"] / roof["peak"] if roof["peak"] else None
    if rank == 0:
        print(json.dumps({
            "metric": "server_field_mac_per_s", "value": macs / (ms / 1e3), "unit": "field-MAC/s",
            "n_gpus": 1, "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": ("u32 (F_q exact; int8 weights, dp4a digits)" if roof["bound"] == "hbm"
                      else "u32 (F_q exact; fp16 digit MMAs, fp32 TMEM accumulation)"), "data": "synthetic",
            "config": {"workload": "server-shape", "m": m, "K": K, "B": B, "weight_copies": copies,
                       "calls_timed": reps * copies, "timing": "CUDA graph of one call per weight copy",
                       "l2": "weights rotated over copies larger than L2"},
            "roofline": roof, "gpu_launches": launches, "clocks": clk}), flush=True)
    return 0


def run_server_layer(args):
    """The server's products of one layer alone (``--shape`` = a batched
    workload name: layer8b-b64, layer70b-b256, layerqwen4b-b8), as one
    pvmvmd_server_mvm_grouped call, timed inside a CUDA graph.  Only the
    weights and the masked vectors are on the device (no client context), so
    the launch also serves as a small case for a profiler."""
    import torch
    rank, world, local = dist_env()
    device = torch.device("cuda", local)
    torch.cuda.set_device(device)
    import paper_2609_10264_gb300 as pv
    Q = pv.PVMVMD_Q
    spec = BATCHED[args.shape]
    B = spec["B"]
    gen = torch.Generator(device=device)
    gen.manual_seed(91)
    ins = []
    for name, m, K in spec["shapes"]:
        W = (torch.randn((m, K), generator=gen, device=device) * 32.0).round_().clamp_(-127, 127).to(torch.int8)
        X = torch.randint(0, Q, (B, K), generator=gen, device=device, dtype=torch.int64).to(torch.int32)
        ins.append((W, X, torch.empty((B, m), dtype=torch.int32, device=device)))
    torch.cuda.synchronize(device)
    stream = torch.cuda.Stream(device)
    jobs = pv.batch_jobs(ins)
    with torch.cuda.stream(stream):
        pv.pvmvmd_server_mvm_grouped(jobs, stream=stream)
    stream.synchronize()
    assert pv.pvmvmd_device_status(stream) == 0
    for W, X, Y in ins:   # sampled rows against an exact int64 product
        rows = [0, W.shape[0] // 2, W.shape[0] - 1]
        exp = (W[rows].cpu().numpy().astype(np.int64) @ pv.as_u32(X).astype(np.int64).T) % Q
        assert np.array_equal(pv.as_u32(Y)[:, rows].T.astype(np.int64), exp)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        pv.pvmvmd_server_mvm_grouped(jobs, stream=stream)
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        for _ in range(args.warmup):
            g.replay()
        t0.record(stream)
        for _ in range(args.steps):
            g.replay()
        t1.record(stream)
    stream.synchronize()
    ms = t0.elapsed_time(t1) / args.steps
    macs = sum(m * K for _, m, K in spec["shapes"]) * B
    peaks, kind = measured_peaks()
    if rank == 0:
        tf = 8 * macs / (ms / 1e3) / 1e12
        print(json.dumps({
            "metric": "server_field_mac_per_s", "value": macs / (ms / 1e3), "unit": "field-MAC/s", "n_gpus": 1,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "u32 (F_q exact; fp16 digit MMAs)", "data": "synthetic",
            "config": {"workload": "server-layer", "layer": args.shape, "B": B,
                       "projections": [list(x) for x in spec["shapes"]],
                       "timing": "CUDA graph of one pvmvmd_server_mvm_grouped call per step"},
            "roofline": {"bound": "tensor", "kernel": "k_digit_tiles_grouped + k_batched_grouped (+ k_split_finish)",
                         "achieved": tf, "peak": peaks["bf16_tflops"], "unit": "TFLOP/s",
                         "frac": tf / peaks["bf16_tflops"], "peak_kind": f"{kind} bf16_tflops (burst)"},
            "gpu_launches": None}), flush=True)
    return 0


def run_decode_shape(args):
    """pvmvmd_decode_verify alone (``--shape mxKxB``): preprocessing, one
    encode and one server product first, then --steps decode calls with fresh
    challenge keys.  4096x8192x256 holds 2 GiB of P^T and Q, a small case of
    the 70B-class decode for a profiler."""
    import torch
    rank, world, local = dist_env()
    device = torch.device("cuda", local)
    torch.cuda.set_device(device)
    import paper_2609_10264_gb300 as pv
    from paper_2609_10264_gb300 import workloads as wl
    m, K, B = (int(v) for v in args.shape.lower().split("x"))
    W = torch.from_numpy(wl.weights_gaussian(m, K, (13, 0))).to(device)
    x = wl.int8_vectors(B, K, (13, 1))
    X = torch.from_numpy(np.mod(x, pv.PVMVMD_Q).astype(np.uint32).view(np.int32)).to(device)
    params = pv.pvmvmd_params()
    params.scratch_batch = B
    ctx = pv.pvmvmd_preprocess(W, key=131, params=params)
    torch.cuda.synchronize(device)
    stream = torch.cuda.Stream(device)
    with torch.cuda.stream(stream):
        Xh, st = pv.pvmvmd_encode(ctx, X, key=132, stream=stream)
        Yh = pv.pvmvmd_server_mvm(W, Xh, stream=stream)
        Y, acc = pv.pvmvmd_decode_verify(ctx, st, Xh, Yh, 133, stream=stream)
    stream.synchronize()
    assert int(acc.sum()) == B
    supp = pv.as_u32(st)[:, :ctx.t_x]
    distinct = len(np.unique(supp))
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        for s_ in range(args.warmup):
            pv.pvmvmd_decode_verify(ctx, st, Xh, Yh, 200 + s_, Y=Y, accept=acc, stream=stream)
        t0.record(stream)
        for s_ in range(args.steps):
            pv.pvmvmd_decode_verify(ctx, st, Xh, Yh, 300 + s_, Y=Y, accept=acc, stream=stream)
        t1.record(stream)
    stream.synchronize()
    assert pv.pvmvmd_device_status(stream) == 0 and int(acc.sum()) == B
    ms = t0.elapsed_time(t1) / args.steps
    peaks, kind = measured_peaks()
    # the decrypt's bytes when every needed row of P^T is read once (the
    # distinct rows of the batch's supports), plus y_hat read and y written
    nbytes = distinct * 4 * m + 8 * B * m
    if rank == 0:
        print(json.dumps({
            "metric": "decoded vectors/s", "value": B / (ms / 1e3), "unit": "vectors/s", "n_gpus": 1,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "u32 (F_q exact)", "data": "synthetic",
            "config": {"workload": "decode-shape", "m": m, "K": K, "B": B, "t_x": ctx.t_x,
                       "support_draws": int(supp.size), "distinct_rows": distinct,
                       "bytes_distinct_rows": nbytes, "bytes_per_vector_rows": int(supp.size) * 4 * m + 8 * B * m},
            "roofline": {"bound": "hbm", "kernel": "pvmvmd_decode_verify call (k_decrypt dominant)",
                         "achieved": nbytes / (ms / 1e3) / 1e9, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                         "frac": nbytes / (ms / 1e3) / 1e9 / peaks["hbm_gbs"], "peak_kind": f"{kind} hbm_gbs"},
            "gpu_launches": None}), flush=True)
    ctx.destroy()
    return 0


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--clock-tail-s", type=float, default=0.5,
                    help="seconds of untimed steps queued after each timed region so that the clock "
                         "sampler sees the load (0 under a profiler)")
    ap.add_argument("--no-extra-configs", action="store_true",
                    help="default workload: skip the 70B-class batched and 8B-class token sub-records")
    ap.add_argument("--cpu-vectors", type=int, default=150)
    ap.add_argument("--server-mode", choices=["multi", "calls"], default="multi")
    ap.add_argument("--workload", choices=["batch1-4096", "server-shape", "server-layer", "decode-shape",
                                           "encode-shape", "encoder-shape",
                                           "preprocess-shape", "token8b-b1", "token8b-b1-client", "bv-b8-1024"]
                    + sorted(BATCHED),
                    default="batch1-4096")
    ap.add_argument("--shape", default="4096x4096x64",
                    help="m x K x B for --workload server-shape and decode-shape, K x B for --workload "
                         "encode-shape, a batched workload name for --workload server-layer")
    ap.add_argument("--server-streams", type=int, default=4)
    ap.add_argument("--schedule", choices=["phases", "projections", "grouped", "pipeline"], default="grouped",
                    help="batched workloads: all encodes, then all products, then all decodes "
                         "(phases); each projection's three calls in order on one of "
                         "--server-streams streams (projections); or the encodes side by side on those "
                         "streams, one grouped product call, the decodes side by side (grouped); or three "
                         "batches in flight, batch k+1's encodes beside batch k's products and batch k-1's "
                         "decodes (pipeline)")
    ap.add_argument("--server-call", choices=["grouped", "per-projection"], default="grouped",
                    help="batched workloads, server phase: one pvmvmd_server_mvm_grouped call for the layer, "
                         "or one pvmvmd_server_mvm call per projection spread over --server-streams streams")
    ap.add_argument("--step-schedule", choices=["overlap", "serial"], default="overlap",
                    help="batch1-4096 standard mode: overlap the next batch's encode with this batch's "
                         "decode on a second stream, or run encode, server and decode in order")
    ap.add_argument("--mode", choices=["standard", "boost", "pipelined"], default="standard",
                    help="client mode of the batch-1 workload (Sec. 7.2): standard (masks drawn during "
                         "the step), boost (masks prepared ahead, untimed) or pipelined (standard mode "
                         "with the next step's masks prepared on a second stream, timed)")
    args = ap.parse_args(argv)
    global CLOCK_TAIL_S
    CLOCK_TAIL_S = args.clock_tail_s
    if args.warmup < 3:
        ap.error("--warmup must be at least 3")
    if args.impl == "reference":
        return run_reference(args)
    if args.workload in BATCHED:
        return run_batched(args)
    if args.workload == "server-shape":
        return run_server_shape(args)
    if args.workload == "server-layer":
        return run_server_layer(args)
    if args.workload == "decode-shape":
        return run_decode_shape(args)
    if args.workload == "token8b-b1-client":
        import torch
        rank, world, local = dist_env()
        device = torch.device("cuda", local)
        torch.cuda.set_device(device)
        rec = measure_token_client(args, device, rank)
        if rank == 0:
            print(json.dumps(rec), flush=True)
        return 0
    if args.workload == "token8b-b1":
        return run_token(args)
    if args.workload == "bv-b8-1024":
        return run_bv(args)
    if args.workload == "encoder-shape":
        return run_encoder_shape(args)
    if args.workload == "preprocess-shape":
        return run_preprocess_shape(args)
    if args.workload == "encode-shape":
        return run_encode_shape(args)
    return run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
