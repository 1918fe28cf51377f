"""Benchmark of the quantized-matmul hot path on GB300.

Workload (default): one Llama-7B-shaped decoder layer (q, k, v, o 4096x4096;
gate, up 11008x4096; down 4096x11008), Student-t(4) weights with sigma 0.01
(q, k), 0.02 (v, o), 0.04 (MLP), quantized to 3-bit non-uniform codes with a
per-group 8-entry fp16 LUT (Lloyd-Max, group 128 along k).  One step = one
decode token through all seven matrices: the decode dependency chain
q,k,v | o | gate,up | down at batch 1 as the four phases of one persistent
qx_gemv_fused launch (each phase reads its x once every CTA has written the
previous phase's y; one CUDA graph).  Metric: HBM GB/s of the packed weights
(+ x, y) per step.  The same step as four qx_gemv_multi launches (PDL) is
reported beside it.

Also reported on the same line: the prefill GEMM (M = 2048 tokens against the
11008x4096 and 4096x11008 3-bit LUT matrices, tcgen05), the same layer with
4-bit uniform g128 and 3-bit uniform g64 weights at batch 1, 4 and 16, the
mixed-recipe LLaVA-shaped stack (32 language layers decoded, 24 vision layers
prefilled), the roofline of the dominant kernel, the CPU oracle as a
baseline, SM clocks during the timed region and an end-to-end number with
host buffers.

Launch: python bench.py [--gpus N --steps K --warmup W] [--impl reference];
for N > 1 under torch.distributed.run (one rank per GPU, weak scaling: every
rank decodes its own copy of the layer; no collective on the data path).
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "3/4-bit dequant-GEMV HBM GB/s (% of 8 TB/s); prefill dequant-GEMM TFLOP/s"
NOMINAL_HBM_GBS = 8000.0
LAYER = [  # name, n, k, sigma, stream id
    ("q_proj", 4096, 4096, 0.01, 0),
    ("k_proj", 4096, 4096, 0.01, 1),
    ("v_proj", 4096, 4096, 0.02, 2),
    ("o_proj", 4096, 4096, 0.02, 3),
    ("gate_proj", 11008, 4096, 0.04, 4),
    ("up_proj", 11008, 4096, 0.04, 5),
    ("down_proj", 4096, 11008, 0.04, 6),
]
GEMM_M = 2048
GEMM_MATS = [("gate_proj", 11008, 4096, 0.04, 4), ("down_proj", 4096, 11008, 0.04, 6)]
REF_BUDGET_S = float(os.environ.get("QX_REF_BUDGET_S", "150"))  # wall time of the whole reference (oracle) arm


def _peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), float(d["bf16_tflops"]), float(d["bf16_tflops_sustained"]), "measured"
    except Exception:
        return 6800.0, 1900.0, 1700.0, "fallback"


def _src_sha(name: str) -> str:
    with open(os.path.join(ROOT, "paper_2505_07531_gb300", "csrc", name), "rb") as f:
        return hashlib.sha256(f.read()).hexdigest()[:16]


def _traffic(kernel_file: str, key: str):
    """DRAM bytes per launch from a committed ncu summary, if taken on this source."""
    path = os.path.join(ROOT, "profiles", "traffic.txt")
    if not os.path.exists(path):
        return None
    sha = _src_sha(kernel_file)
    with open(path) as f:
        for line in f:
            parts = line.split()
            if len(parts) >= 4 and parts[0] == key and parts[1] == sha:
                return float(parts[2])
    return None


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled every 200 ms."""

    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.Q}", "--format=csv,noheader,nounits",
                 "-lms", "200"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        out, _ = self.proc.communicate(timeout=10)
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in out.strip().splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx.append(float(f[2]))
            except ValueError:
                continue
            for nm, v in zip(names, f[5:9]):
                if v.lower() == "active":
                    reasons.add(nm)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": sorted(reasons), "samples": len(sm)}


def _dist():
    """(dist module or None, rank, world size, local rank) of a torchrun launch:
    one process per GPU over NCCL; gloo where no GPU is visible (the host-side
    tests of the multi-rank path)."""
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    if ws > 1:
        import torch
        import torch.distributed as dist

        dist.init_process_group("nccl" if torch.cuda.is_available() else "gloo")
        return dist, dist.get_rank(), ws, int(os.environ.get("LOCAL_RANK", "0"))
    return None, 0, 1, 0


def _max_over_ranks(dist, v: float, device) -> float:
    """The largest of every rank's v (each rank's timed region is its own; the
    job takes as long as its slowest rank)."""
    if dist is None:
        return v
    import torch

    t = torch.tensor([v], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def _job_rate(units_per_rank: float, world: int, ms: float) -> float:
    """Whole-job throughput (weak scaling: every rank processes units_per_rank)
    in units per second, timed by the slowest rank's ms."""
    return units_per_rank * world / (ms * 1e-3)


# --------------------------------------------------------------- CPU oracle leg
def _oracle_sample(rows_per_matrix: int, seed: int = 0):
    """Oracle-quantized samples of the layer's matrices (first rows of each)."""
    import oracle
    import synth
    from oracle.pack import Recipe as ORecipe

    rec = ORecipe(3, 128, "lut", 25)
    mats = []
    for name, n, k, sigma, sid in LAYER:
        W = synth.student_t_weights(rows_per_matrix, k, sigma, seed=seed, stream=100 + sid)
        p = oracle.quantize(W, rec)
        x = synth.activations(1, k, seed=seed, stream=200 + sid)
        nbytes = p["codes"].nbytes + p["luts"].nbytes + x.nbytes + 2 * rows_per_matrix
        mats.append((p, x, k, nbytes))
    return rec, mats


def _oracle_pass(rec, mats):
    import oracle

    for p, x, k, _ in mats:
        oracle.gemv(p, rec, x, k)


_POOL_SAMPLE = None


def _pool_init(sample):
    global _POOL_SAMPLE
    _POOL_SAMPLE = sample


def _pool_passes(passes: int) -> float:
    rec, mats = _POOL_SAMPLE
    t0 = time.perf_counter()
    for _ in range(passes):
        _oracle_pass(rec, mats)
    return time.perf_counter() - t0


class _OraclePool:
    """The oracle on every host core: one single-threaded process per core,
    each making whole passes over its own copy of the sample (started with
    spawn, in a process that has not touched the GPU)."""

    def __init__(self, rec, mats, workers: int):
        import multiprocessing as mp

        self.workers = workers
        self.pool = mp.get_context("spawn").Pool(workers, initializer=_pool_init, initargs=((rec, mats),))
        self.pool.map(_pool_passes, [1] * workers)  # start-up and first touch

    def run(self, passes: int) -> float:
        """Wall seconds for `passes` passes on every worker."""
        t0 = time.perf_counter()
        self.pool.map(_pool_passes, [passes] * self.workers)
        return time.perf_counter() - t0

    def close(self):
        self.pool.close()
        self.pool.join()


def _single_thread_env():
    return dict(os.environ, OMP_NUM_THREADS="1", OPENBLAS_NUM_THREADS="1", MKL_NUM_THREADS="1",
                CUDA_VISIBLE_DEVICES="")


def cpu_baseline_child(seconds: float):
    """Run in a subprocess with single-threaded numpy: oracle GB/s on a bounded
    sample, on one core and on every core."""
    rec, mats = _oracle_sample(64)
    nbytes = sum(m[3] for m in mats)
    _oracle_pass(rec, mats)
    t0 = time.perf_counter()
    reps = 0
    while True:
        _oracle_pass(rec, mats)
        reps += 1
        if time.perf_counter() - t0 >= seconds:
            break
    dt = time.perf_counter() - t0
    one = nbytes * reps / dt / 1e9
    workers = os.cpu_count() or 1
    pool = _OraclePool(rec, mats, workers)
    chunk = max(1, int(seconds / (dt / reps)) // 16)  # bounded in time whatever the cores' speed
    passes, dtp = 0, 0.0
    while dtp < seconds:
        dtp += pool.run(chunk)
        passes += chunk
    pool.close()
    allc = nbytes * passes * workers / dtp / 1e9
    print(json.dumps({"value": allc, "unit": "GB/s", "cores": workers, "kind": "oracle",
                      "value_1_core": one,
                      "sample": f"the first 64 rows of each of the 7 layer matrices ({nbytes / 1e6:.2f} MB packed "
                                f"per pass), numpy float64: {workers} single-threaded processes x {passes} passes "
                                f"each in {dtp:.1f} s; on 1 core {reps} passes in {dt:.1f} s"}))


def run_cpu_baseline(seconds: float = 12.0):
    r = subprocess.run([sys.executable, os.path.abspath(__file__), "--cpu-baseline-child", str(seconds)],
                       capture_output=True, text=True, env=_single_thread_env(), timeout=900)
    try:
        return json.loads(r.stdout.strip().splitlines()[-1])
    except Exception:
        return {"value": None, "unit": "GB/s", "cores": None, "kind": "oracle", "sample": "failed: " + r.stderr[-200:]}


def run_reference(args):
    """The oracle as the reference arm: same metric and config, on every host
    core, bounded samples per step.

    The oracle quantizes a fixed sample (the first 64 rows of each of the seven
    matrices) once; a step is a whole number of dequantize + float64 matvec passes
    over that sample on each of os.cpu_count() single-threaded processes, sized so
    that warm-up plus timed steps take about QX_REF_BUDGET_S seconds of wall time.
    """
    dist, rank, ws, _ = _dist()
    if rank != 0:
        return
    if os.environ.get("QX_REF_CHILD") != "1":
        # numpy single-threaded in every process: the processes are the cores
        env = dict(_single_thread_env(), QX_REF_CHILD="1")
        env.pop("RANK", None)
        env.pop("WORLD_SIZE", None)
        r = subprocess.run([sys.executable, os.path.abspath(__file__), "--impl", "reference", "--gpus", str(ws),
                            "--steps", str(args.steps), "--warmup", str(args.warmup)], capture_output=True, text=True,
                           env=env, timeout=1800)
        out = [ln for ln in r.stdout.splitlines() if ln.startswith("{")]
        if r.returncode != 0 or not out:
            print(json.dumps({"impl": "reference", "unavailable": "oracle arm failed: " + r.stderr[-200:]}))
            return
        line = json.loads(out[-1])
        line["n_gpus"] = ws
        print(json.dumps(line))
        return
    steps, warmup = args.steps, args.warmup
    workers = os.cpu_count() or 1
    per_step = REF_BUDGET_S / max(1, steps + warmup)
    rows = 64
    rec, mats = _oracle_sample(rows)
    nbytes = sum(m[3] for m in mats)
    _oracle_pass(rec, mats)
    t0 = time.perf_counter()
    _oracle_pass(rec, mats)
    t_pass = max(time.perf_counter() - t0, 1e-6)
    if t_pass > per_step and rows > 1:  # very many steps: shrink the sample instead
        rows = max(1, int(rows * per_step / t_pass))
        rec, mats = _oracle_sample(rows)
        nbytes = sum(m[3] for m in mats)
        _oracle_pass(rec, mats)
        t0 = time.perf_counter()
        _oracle_pass(rec, mats)
        t_pass = max(time.perf_counter() - t0, 1e-6)
    passes = max(1, int(per_step / t_pass))
    pool = _OraclePool(rec, mats, workers)
    for _ in range(warmup):
        pool.run(passes)
    dt = 0.0
    for _ in range(steps):
        dt += pool.run(passes)
    pool.close()
    v = nbytes * passes * workers * steps / dt / 1e9
    sample = (f"{workers} single-threaded processes, each {passes} pass(es) per step over the first {rows} rows of "
              f"each of the 7 layer matrices ({nbytes / 1e6:.2f} MB packed per pass), numpy float64")
    line = {
        "impl": "reference", "metric": METRIC, "value": v, "unit": "GB/s", "n_gpus": ws, "steps": steps,
        "warmup": warmup, "ms_per_step": dt / steps * 1e3, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": "llama7b_layer_decode_L3g128_b1", "sample_rows_per_matrix": rows,
                   "passes_per_step_per_process": passes},
        "cpu_baseline": {"value": v, "unit": "GB/s", "cores": workers, "kind": "oracle", "sample": sample},
        "e2e": {"value": v, "unit": "GB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line))


# --------------------------------------------------------------- GPU arm
def _quantize_layer(qx, torch, dev, mats, recipe, seed=0):
    import synth

    out = []  # [(name, PackedMatrix)]
    for name, n, k, sigma, sid in mats:
        W = synth.student_t_weights_torch(n, k, sigma, seed=seed, stream=sid, device=dev)
        out.append((name, qx.quantize(W, recipe)))
        del W
    if qx.device_status() != 0:
        raise RuntimeError("quantize reported a device error")
    return out


def _clone(qx, P):
    c = lambda t: None if t is None else t.clone()
    return qx.PackedMatrix(P.n, P.k, P.recipe, c(P.codes), c(P.scales), c(P.zeros), c(P.luts))


def _summary(line, hbm, tf_burst):
    """The headline figures in a few keys (the end of the line)."""
    def get(d, *path):
        for p in path:
            if not isinstance(d, dict) or p not in d:
                return None
            d = d[p]
        return d

    out = {"decode_L3g128_b1_GBps": line["value"], "frac_of_measured_hbm": line["value"] / hbm,
           "decode_L3g128_b1_4_launches_GBps": get(line, "chain_4_launches", "GBps"),
           "e2e_GBps": get(line, "e2e", "value"),
           "prefill_TFLOPs": get(line, "gemm", "value"), "prefill_frac_of_bf16_burst": get(line, "gemm", "roofline", "frac")}
    for rec in ("U4g128", "U3g64"):
        for b in (1, 4, 16):
            v = get(line, "config3", f"llama7b_layer_decode_{rec}_b{b}", "GBps")
            if v is not None:
                out[f"decode_{rec}_b{b}_GBps"] = v
    for b in (1, 4, 16):
        v = get(line, "q4x", f"llama7b_layer_decode_Q4X_b{b}", "GBps")
        if v is not None:
            out[f"decode_Q4X_b{b}_GBps"] = v
    return out


def run_ours(args):
    import torch

    import synth
    import paper_2505_07531_gb300.qx as qx

    dist, rank, ws, local = _dist()
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    qx._lib()  # fails loudly when the library is missing
    hbm, tf_burst, tf_sust, peak_src = _peaks()
    props = torch.cuda.get_device_properties(dev)
    l2 = getattr(props, "L2_cache_size", 0) or 126 * 2 ** 20

    recipe = qx.Recipe(3, 128, qx.LUT, 25)
    base = dict(_quantize_layer(qx, torch, dev, LAYER, recipe))
    layer_bytes = sum(P.nbytes() for P in base.values())
    copies = max(2, math.ceil(4 * l2 / layer_bytes))
    layers = [base] + [{nm: _clone(qx, P) for nm, P in base.items()} for _ in range(copies - 1)]
    # decode dependency chain of one token through the layer: q, k, v share the
    # attention input; o reads the attention output; gate, up share the MLP
    # input; down reads act(gate) * up.  Activations are synthetic N(0, 1).
    # the four activations and the seven outputs are views of one input and one
    # output buffer, so that the end-to-end loop moves each with one copy
    x_flat = torch.empty(3 * 4096 + 11008, dtype=torch.float16, device=dev)
    x_attn, x_o, x_mlp = (x_flat[4096 * i:4096 * (i + 1)].view(1, 4096) for i in range(3))
    x_down = x_flat[3 * 4096:].view(1, 11008)
    for i, x in enumerate((x_attn, x_o, x_mlp)):
        x.copy_(synth.activations_torch(1, 4096, seed=0, stream=50 + i, device=dev))
    x_down.copy_(synth.activations_torch(1, 11008, seed=0, stream=53, device=dev))
    y_flat = torch.empty(sum(n for _, n, *_ in LAYER), dtype=torch.float16, device=dev)
    ys, off = {}, 0
    for nm, n, *_ in LAYER:
        ys[nm] = y_flat[off:off + n].view(1, n)
        off += n
    CHAIN = [(["q_proj", "k_proj", "v_proj"], x_attn), (["o_proj"], x_o),
             (["gate_proj", "up_proj"], x_mlp), (["down_proj"], x_down)]
    io_bytes = sum(x.numel() * 2 for x in (x_attn, x_o, x_mlp, x_down)) + sum(y.numel() * 2 for y in ys.values())
    step_bytes = layer_bytes + io_bytes

    stream = torch.cuda.Stream(dev)

    def launch(c, j):
        names, x = CHAIN[j]
        qx.gemv_multi([layers[c][nm] for nm in names], [x] * len(names), outs=[ys[nm] for nm in names], pdl=True)

    def chain_step(c):
        for j in range(len(CHAIN)):
            launch(c, j)

    # the timed step: the four groups as phases of ONE persistent launch
    # (qx_gemv_fused, CTAs balanced slice by slice, a group's x read once every
    # CTA has written the previous group's y), one workspace per weight copy
    fsteps = [qx.GemvChain([([layers[c][nm] for nm in names], [x] * len(names), [ys[nm] for nm in names])
                            for names, x in CHAIN], fused=True) for c in range(copies)]

    def step(c):
        fsteps[c]()

    with torch.cuda.stream(stream):
        for c in range(copies):
            step(c)
    torch.cuda.synchronize(dev)
    graphs = []
    for c in range(copies):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            step(c)
        graphs.append(g)
    # one graph of a step on every copy in turn: programmatic dependent launch
    # links consecutive steps inside it (it does not cross graph boundaries)
    g_all = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g_all, stream=stream):
        for c in range(copies):
            step(c)
    torch.cuda.synchronize(dev)

    uuid = getattr(props, "uuid", None)
    sampler = ClockSampler(f"GPU-{uuid}" if uuid is not None else str(dev.index or 0))
    sampler.start()
    with torch.cuda.stream(stream):
        for i in range(args.warmup):
            graphs[i % copies].replay()
        # soak ~1.5 s so the clocks are sampled under this load, then time exactly K steps
        t_end = time.time() + 1.5
        i = 0
        while time.time() < t_end:
            for _ in range(64):
                graphs[i % copies].replay()
                i += 1
            stream.synchronize()
    if dist is not None:
        dist.barrier()
    torch.cuda.synchronize(dev)
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        ev0.record(stream)
        for _ in range(args.steps // copies):  # exactly K steps: whole rounds, then single steps
            g_all.replay()
        for i in range(args.steps % copies):
            graphs[i].replay()
        ev1.record(stream)
    torch.cuda.synchronize(dev)
    clocks = sampler.stop()
    ms = ev0.elapsed_time(ev1) / args.steps
    ms = _max_over_ranks(dist, ms, dev)
    value = _job_rate(step_bytes, ws, ms) / 1e9

    # The timed region holds only gemv_kernel<3,LUT,-1> launches, one per step,
    # so the launch duration is ms and its algorithmic bytes are step_bytes:
    # achieved = step_bytes / ms.
    launch_us = ms * 1e3
    achieved = step_bytes / (ms * 1e-3) / 1e9
    # steady-state duration of each launch of the chain: one graph per launch
    # kind, `copies` back-to-back launches (PDL) over rotating weight copies
    reps = 20
    per_launch_us = {}
    for j in range(len(CHAIN)):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            for c in range(copies):
                launch(c, j)
        with torch.cuda.stream(stream):
            for _ in range(3):
                g.replay()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            for _ in range(reps):
                g.replay()
            e1.record(stream)
        torch.cuda.synchronize(dev)
        per_launch_us["+".join(CHAIN[j][0])] = 1e3 * e0.elapsed_time(e1) / (reps * copies)
        del g

    # the seven matrices as independent problems in one launch (upper bound of the chain)
    xs7 = {nm: (x_down if nm == "down_proj" else x_attn) for nm, _, _, _, _ in LAYER}
    reps = 200
    with torch.cuda.stream(stream):
        for r in range(3):
            qx.gemv_multi([layers[r % copies][nm] for nm, *_ in LAYER], [xs7[nm] for nm, *_ in LAYER],
                          outs=[ys[nm] for nm, *_ in LAYER], pdl=True)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for r in range(reps):
            qx.gemv_multi([layers[r % copies][nm] for nm, *_ in LAYER], [xs7[nm] for nm, *_ in LAYER],
                          outs=[ys[nm] for nm, *_ in LAYER], pdl=True)
        e1.record(stream)
    torch.cuda.synchronize(dev)
    one_launch_ms = e0.elapsed_time(e1) / reps

    # the same step as four qx_gemv_multi launches (PDL), whole row blocks per
    # CTA, and as four balanced launches (qx_gemv_fused with QX_GEMV_SEPARATE)
    alt_us = {}
    sep = [qx.GemvChain([([layers[c][nm] for nm in names], [x] * len(names), [ys[nm] for nm in names])
                         for names, x in CHAIN], separate=True) for c in range(copies)]
    for nm_, fn in (("chain_4_launches", chain_step), ("balanced_4_launches", lambda c: sep[c]())):
        try:
            with torch.cuda.stream(stream):
                for c in range(copies):
                    fn(c)
            torch.cuda.synchronize(dev)
            ga = torch.cuda.CUDAGraph()
            with torch.cuda.graph(ga, stream=stream):
                for c in range(copies):
                    fn(c)
            us = _time_graph(torch, stream, ga, 20) / copies * 1e3
            alt_us[nm_] = {"us": us, "GBps": step_bytes / (us * 1e-6) / 1e9}
            del ga
        except Exception as e:  # noqa: BLE001
            alt_us[nm_] = f"unavailable: {type(e).__name__}: {e}"[:160]
    del sep

    # end to end through the public API with host buffers: the step's activations
    # in from pinned host memory (one copy), the four decode calls, the outputs
    # back (one copy), then a stream synchronisation, per step
    hx = x_flat.cpu().pin_memory()
    hy = torch.empty(y_flat.shape, dtype=y_flat.dtype).pin_memory()
    # a step is one qx_decode_step_fused call (copy in, the one launch, copy
    # out, synchronize; arguments bound once per weight copy); if it cannot be
    # built or run, the step is the torch copies around the fused call
    e2e_call, e2e_path = None, "torch copies + 1 qx_gemv_fused call + synchronize per step"
    try:
        dsteps = [qx.DecodeStep([([layers[c][nm] for nm in names], [x] * len(names), [ys[nm] for nm in names])
                                 for names, x in CHAIN], h2d=[(x_flat, hx)], d2h=[(hy, y_flat)], fused=True)
                  for c in range(copies)]
        with torch.cuda.stream(stream):
            for ds in dsteps:
                ds()
        if qx.device_status(stream) != 0:
            raise RuntimeError("device status after the decode step")
        e2e_call = lambda c: dsteps[c]()  # noqa: E731
        e2e_path = ("1 qx_decode_step_fused call per step: copy in (copy kernel reading the pinned host x), "
                    "1 launch, copy out (copy kernel writing the pinned host y), synchronize")
    except Exception as e:  # noqa: BLE001
        e2e_path += f" (decode step unavailable: {type(e).__name__}: {e})"[:200]
    e2e_steps = max(3, min(args.steps, 2000))
    if dist is not None:
        dist.barrier()
    torch.cuda.synchronize(dev)
    t0 = time.perf_counter()
    with torch.cuda.stream(stream):
        for i in range(e2e_steps):
            c = i % copies
            if e2e_call is not None:
                e2e_call(c)
                continue
            x_flat.copy_(hx, non_blocking=True)
            step(c)
            hy.copy_(y_flat, non_blocking=True)
            stream.synchronize()
    e2e_ms = _max_over_ranks(dist, (time.perf_counter() - t0) * 1e3 / e2e_steps, dev)
    e2e_value = _job_rate(step_bytes, ws, e2e_ms) / 1e9

    section = lambda fn, *a: _section(torch, fn, *a)  # noqa: E731
    gemm = section(run_gemm_part, qx, torch, dev, stream, tf_burst, peak_src) if not args.skip_gemm else None
    del layers, graphs, g_all, fsteps
    extra = {}
    if not args.skip_configs:
        extra["config3"] = section(run_config3, qx, torch, dev, stream, l2, hbm)
        extra["recipe_select"] = section(run_select, qx, torch, dev, stream)
        extra["config5"] = section(run_config5, qx, torch, dev, stream)
        extra["q4x"] = section(run_q4x, qx, torch, dev, stream, l2, hbm, tf_burst)

    if rank == 0:
        cpu = run_cpu_baseline() if not args.skip_cpu_baseline else None
        line = {
            "metric": METRIC, "value": value, "unit": "GB/s", "n_gpus": ws, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f16", "data": "synthetic",
            "pct_of_8TBs": 100.0 * value / ws / NOMINAL_HBM_GBS,
            "config": {"workload": "llama7b_layer_decode_L3g128_b1",
                       "matrices": {nm: [n, k] for nm, n, k, _, _ in LAYER},
                       "recipe": "3-bit LUT (8 fp16 levels, Lloyd-Max) group 128",
                       "batch": 1, "bytes_per_step": step_bytes,
                       "step": "qkv | o | gate+up | down as the 4 phases of one qx_gemv_fused launch (PDL "
                               "between steps); CUDA graphs of one step on every weight copy in turn",
                       "l2": f"{copies} rotating weight copies ({copies * layer_bytes / 1e6:.0f} MB) > "
                             f"4x L2 ({l2 / 1e6:.0f} MB)"},
            # the long sections first: the record keeps the end of the line
            **extra,
            "chain_per_launch_us": per_launch_us,
            "one_launch_7_matrices": {"us": one_launch_ms * 1e3,
                                      "GBps": step_bytes / (one_launch_ms * 1e-3) / 1e9},
            **alt_us,
            "cpu_baseline": cpu,
            "clocks": clocks,
            "e2e": {"value": e2e_value, "unit": "GB/s", "ms_per_step": e2e_ms,
                    "h2d_bytes_per_step": hx.numel() * hx.element_size(),
                    "d2h_bytes_per_step": hy.numel() * hy.element_size(), "path": e2e_path},
            "gpu_launches": args.steps,
            "roofline": {"bound": "hbm", "achieved": achieved, "peak": hbm, "unit": "GB/s",
                         "frac": achieved / hbm, "peak_source": f"{peak_src} hbm_gbs",
                         "kernel": "gemv_kernel<3,LUT,-1> (4 phases)", "launches_per_step": 1,
                         "launch_us": launch_us, "bytes_per_launch": step_bytes,
                         "traffic": _traffic("qx_gemv.cu", "gemv_L3g128_b1")},
            "gemm": gemm,
        }
        line["summary"] = _summary(line, hbm, tf_burst)
        print(json.dumps(line))
    if dist is not None:
        dist.destroy_process_group()


def _section(torch, fn, *a):
    """fn(*a), or {"error": ...} if it raises: a section that fails reports its
    error in its own key, and the headline figures and the other sections
    stand.  The caching allocator's free blocks are released either way."""
    try:
        return fn(*a)
    except Exception as e:  # noqa: BLE001
        return {"error": f"{type(e).__name__}: {e}"[:300]}
    finally:
        torch.cuda.empty_cache()


def run_gemm_part(qx, torch, dev, stream, tf_burst, peak_src):
    """Prefill GEMM, M = 2048, 3-bit LUT g128 11008x4096 and 4096x11008."""
    import synth

    recipe = qx.Recipe(3, 128, qx.LUT, 25)
    mats = _quantize_layer(qx, torch, dev, GEMM_MATS, recipe, seed=1)
    Xs = [synth.activations_torch(GEMM_M, P.k, seed=1, stream=70 + i, device=dev) for i, (_, P) in enumerate(mats)]
    Ys = [torch.empty((GEMM_M, P.n), dtype=torch.float16, device=dev) for _, P in mats]
    flops = sum(2.0 * GEMM_M * P.n * P.k for _, P in mats)
    with torch.cuda.stream(stream):
        for _ in range(3):
            for (nm, P), X, Y in zip(mats, Xs, Ys):
                qx.gemm(P, X, out=Y)
    torch.cuda.synchronize(dev)
    if qx.device_status(stream) != 0:
        raise RuntimeError("gemm reported a device error")
    reps = 20
    evs = [[(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in mats]
           for _ in range(reps)]
    with torch.cuda.stream(stream):
        for r in range(reps):
            for j, ((nm, P), X, Y) in enumerate(zip(mats, Xs, Ys)):
                evs[r][j][0].record(stream)
                qx.gemm(P, X, out=Y)
                evs[r][j][1].record(stream)
    torch.cuda.synchronize(dev)
    ms = sum(a.elapsed_time(b) for row in evs for a, b in row) / reps
    per = {mats[j][0]: 1e3 * sum(evs[r][j][0].elapsed_time(evs[r][j][1]) for r in range(reps)) / reps
           for j in range(len(mats))}
    tflops = flops / (ms * 1e-3) / 1e12
    try:
        a8 = _a8_prefill(qx, torch, dev, stream, mats, Xs, Ys, flops)
    except Exception as e:  # noqa: BLE001
        a8 = {"error": f"{type(e).__name__}: {e}"[:300]}
    return {"value": tflops, "unit": "TFLOP/s", "ms_per_step": ms, "per_matrix_us": per, "a8_prefill": a8,
            "config": {"workload": "prefill_M2048_L3g128", "m": GEMM_M,
                       "matrices": {nm: [P.n, P.k] for nm, P in mats}, "mma": "tcgen05 kind::f16, fp32 accumulate",
                       "l2": "weights 22.5 MB and X 16-22 MB are L2-resident (compute-bound kernel)"},
            "roofline": {"bound": "tensor", "achieved": tflops, "peak": tf_burst, "unit": "TFLOP/s",
                         "frac": tflops / tf_burst,
                         "peak_source": f"{peak_src} bf16_tflops (burst) x 1.0 nominal fp16/bf16 ratio",
                         "kernel": "gemm_kernel<3,LUT>", "traffic": _traffic("qx_gemm.cu", "gemm_L3g128_m2048")}}


def _a8_prefill(qx, torch, dev, stream, mats, Xs, Ys, flops):
    """The same prefill with 8-bit per-token activations (Tables 1-2, W.A8):
    qx_quantize_act, qx_dequant_act (x_hat = fp16(s_b q)) and qx_gemm per
    matrix, all three timed."""
    bufs = [(torch.empty(X.shape, dtype=torch.int8, device=dev), torch.empty((X.shape[0],), dtype=torch.float32,
                                                                              device=dev), torch.empty_like(X))
            for X in Xs]
    lib = qx._lib()

    def step():
        for (nm, P), X, Y, (q, s, xh) in zip(mats, Xs, Ys, bufs):
            m, k = X.shape
            qx._check(lib.qx_quantize_act(qx._ptr(X), m, k, qx._ptr(q), qx._ptr(s), qx._stream(dev)),
                      "qx_quantize_act")
            qx.dequant_act(q, s, out=xh)
            qx.gemm(P, xh, out=Y)

    with torch.cuda.stream(stream):
        for _ in range(3):
            step()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(10):
            step()
        e1.record(stream)
    torch.cuda.synchronize(dev)
    if qx.device_status(stream) != 0:
        raise RuntimeError("W.A8 prefill reported a device error")
    ms = e0.elapsed_time(e1) / 10
    return {"ms_per_step": ms, "TFLOPs": flops / (ms * 1e-3) / 1e12,
            "path": "qx_quantize_act + qx_dequant_act + qx_gemm per matrix (fp16 tensor cores on x_hat)"}


def _chain_graph(qx, torch, stream, layers, chain, outs, pdl=True):
    """One CUDA graph of the decode chain over every layer copy in `layers`."""
    def body():
        for L in layers:
            for names, x in chain:
                qx.gemv_multi([L[nm] for nm in names], [x] * len(names), outs=[outs[nm] for nm in names], pdl=pdl)

    with torch.cuda.stream(stream):
        body()
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        body()
    return g


def _splitk_graph(qx, torch, stream, layers, xs, outs):
    """One CUDA graph of the seven tensor-core (split-k) matmuls over every layer copy."""
    def body():
        for L in layers:
            for nm, P in L.items():
                qx.gemm_splitk(P, xs[nm], out=outs[nm], pdl=True)

    with torch.cuda.stream(stream):
        body()  # also sizes the stream's workspace before capture
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        body()
    return g


def _time_graph(torch, stream, g, reps):
    with torch.cuda.stream(stream):
        for _ in range(3):
            g.replay()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(reps):
            g.replay()
        e1.record(stream)
    torch.cuda.synchronize()
    return e0.elapsed_time(e1) / reps  # ms per replay


def run_config3(qx, torch, dev, stream, l2, hbm):
    """Llama-7B layer, 4-bit uniform g128 and 3-bit uniform g64, batch 1 / 4 / 16:
    the decode chain (qx_gemv_multi, PDL; products on the CUDA cores at batch
    1, on mma.sync at 4 and 16) and, for batch 4 and 16, the tcgen05 split-k
    matmul (qx_gemm_splitk, one launch per matrix) beside it."""
    import synth

    out = {}
    for bits, g in ((4, 128), (3, 64)):
        recipe = qx.Recipe(bits, g, qx.UNIFORM)
        base = dict(_quantize_layer(qx, torch, dev, LAYER, recipe))
        layer_bytes = sum(P.nbytes() for P in base.values())
        copies = max(2, math.ceil(4 * l2 / layer_bytes))
        layers = [base] + [{nm: _clone(qx, P) for nm, P in base.items()} for _ in range(copies - 1)]
        for batch in (1, 4, 16):
            xs = [synth.activations_torch(batch, k, seed=batch, stream=60 + i, device=dev)
                  for i, k in enumerate((4096, 4096, 4096, 11008))]
            ys = {nm: torch.empty((batch, n), dtype=torch.float16, device=dev) for nm, n, *_ in LAYER}
            chain = [(["q_proj", "k_proj", "v_proj"], xs[0]), (["o_proj"], xs[1]),
                     (["gate_proj", "up_proj"], xs[2]), (["down_proj"], xs[3])]
            gr = _chain_graph(qx, torch, stream, layers, chain, ys)
            ms = _time_graph(torch, stream, gr, 20) / copies
            del gr
            io = sum(x.numel() * 2 for x in xs) + sum(y.numel() * 2 for y in ys.values())
            gbps = (layer_bytes + io) / (ms * 1e-3) / 1e9
            out[f"llama7b_layer_decode_U{bits}g{g}_b{batch}"] = {
                "us_per_layer": ms * 1e3, "GBps": gbps, "frac_of_measured_hbm": gbps / hbm,
                "weight_bytes": layer_bytes,
                "path": "4 qx_gemv_multi launches (PDL): " + ("CUDA-core" if batch <= 2 else "mma.sync") + " products"}
            if batch in (1, 4):
                # W.A8: the four distinct activations quantized per token to int8,
                # then seven integer-dot matmuls (qx_quantize_act + qx_gemv_a8)
                xd = {"attn": xs[0], "o": xs[1], "mlp": xs[2], "down": xs[3]}
                src = {"q_proj": "attn", "k_proj": "attn", "v_proj": "attn", "o_proj": "o", "gate_proj": "mlp",
                       "up_proj": "mlp", "down_proj": "down"}
                qa = {key: (torch.empty(x.shape, dtype=torch.int8, device=dev),
                            torch.empty((batch,), dtype=torch.float32, device=dev)) for key, x in xd.items()}

                def a8_step(L):
                    for key, x in xd.items():
                        qx._check(qx._lib().qx_quantize_act(qx._ptr(x), batch, x.shape[1], qx._ptr(qa[key][0]),
                                                            qx._ptr(qa[key][1]), qx._stream(dev)), "qx_quantize_act")
                    for nm, *_ in LAYER:
                        qx.gemv_a8(L[nm], qa[src[nm]][0], qa[src[nm]][1], out=ys[nm])

                with torch.cuda.stream(stream):
                    for L in layers:
                        a8_step(L)
                torch.cuda.synchronize()
                gr = torch.cuda.CUDAGraph()
                with torch.cuda.graph(gr, stream=stream):
                    for L in layers:
                        a8_step(L)
                ms = _time_graph(torch, stream, gr, 20) / copies
                del gr
                out[f"llama7b_layer_decode_U{bits}g{g}_b{batch}_a8"] = {
                    "us_per_layer": ms * 1e3, "GBps": (layer_bytes + io) / (ms * 1e-3) / 1e9,
                    "weight_bytes": layer_bytes,
                    "path": "qx_quantize_act x4 + qx_gemv_a8 x7 (int8 activations, dp4a)"}
            if batch >= 4:
                xn = {nm: xs[3] if nm == "down_proj" else xs[0] for nm, *_ in LAYER}
                gr = _splitk_graph(qx, torch, stream, layers, xn, ys)
                ms = _time_graph(torch, stream, gr, 20) / copies
                del gr
                out[f"llama7b_layer_decode_U{bits}g{g}_b{batch}_tensorcore"] = {
                    "us_per_layer": ms * 1e3, "GBps": (layer_bytes + io) / (ms * 1e-3) / 1e9,
                    "weight_bytes": layer_bytes, "path": "qx_gemm_splitk per matrix with PDL (tcgen05, k split)"}
        del layers, base
    if qx.device_status(stream) != 0:
        raise RuntimeError("config-3 decode reported a device error")
    return out


def run_q4x(qx, torch, dev, stream, l2, hbm, tf_burst):
    """Q4X shared codebooks (groups of 64 with an fp16 scale and a 2-bit book
    index, 4-bit codes, four 16-level codebooks learned per matrix): the
    learner's device time per Llama-7B layer matrix, and the decode matmul over
    the layer at batch 1, 4 and 16 (q,k,v | o | gate,up | down: four
    qx_q4x_gemv_multi launches per layer copy in one CUDA graph, weights
    rotated over copies larger than 4x L2), and the tensor-core prefill
    (qx_q4x_gemm) at M = 2048 against the two MLP shapes."""
    import synth

    def learn(name, n, k, sigma, sid):
        W = synth.student_t_weights_torch(n, k, sigma, seed=0, stream=sid, device=dev)
        with torch.cuda.stream(stream):
            stream.wait_stream(torch.cuda.default_stream(dev))  # W is drawn on the default stream
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            P = qx.q4x_quantize(W)
            e1.record(stream)
        torch.cuda.synchronize(dev)
        return P, e0.elapsed_time(e1)

    learn(*LAYER[0])  # sizes the caching allocator's workspace block
    base, learn_ms = {}, {}
    for spec in LAYER:
        base[spec[0]], learn_ms[spec[0]] = learn(*spec)
    st_code = qx.device_status(stream)
    if st_code != 0:
        raise RuntimeError(f"q4x_quantize reported device status {st_code}")
    layer_bytes = sum(P.nbytes() for P in base.values())
    copies = max(2, math.ceil(4 * l2 / layer_bytes))
    dup = lambda P: qx.Q4xMatrix(P.n, P.k, P.codes.clone(), P.scales.clone(), P.books.clone(), P.codebooks.clone())
    layers = [base] + [{nm: dup(P) for nm, P in base.items()} for _ in range(copies - 1)]
    out = {"learn_ms": learn_ms, "weight_bytes": layer_bytes,
           "bits_per_weight": 8.0 * layer_bytes / sum(n * k for _, n, k, _, _ in LAYER)}
    for batch in (1, 4, 16):
        xs = {k: synth.activations_torch(batch, k, seed=batch, stream=70 + i, device=dev)
              for i, k in enumerate((4096, 11008))}
        ys = {nm: torch.empty((batch, n), dtype=torch.float16, device=dev) for nm, n, *_ in LAYER}

        chain = (["q_proj", "k_proj", "v_proj"], ["o_proj"], ["gate_proj", "up_proj"], ["down_proj"])

        def body():
            for L in layers:
                for names in chain:
                    qx.q4x_gemv_multi([L[nm] for nm in names], [xs[L[nm].k] for nm in names],
                                      outs=[ys[nm] for nm in names])

        with torch.cuda.stream(stream):
            body()
        torch.cuda.synchronize(dev)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            body()
        ms = _time_graph(torch, stream, g, 20) / copies
        del g
        io = sum(2 * batch * k for _, _, k, _, _ in LAYER) + sum(y.numel() * 2 for y in ys.values())
        gbps = (layer_bytes + io) / (ms * 1e-3) / 1e9
        out[f"llama7b_layer_decode_Q4X_b{batch}"] = {
            "us_per_layer": ms * 1e3, "GBps": gbps, "frac_of_measured_hbm": gbps / hbm,
            "path": "4 qx_q4x_gemv_multi launches: weights dequantized in registers from TMA-staged codes, "
                    "the codebooks as pair tables in shared memory"}
    if qx.device_status(stream) != 0:
        raise RuntimeError("q4x decode reported a device error")
    # prefill on the tensor cores (qx_q4x_gemm): M = 2048 tokens against the two
    # MLP shapes, as the per-group prefill benchmark
    del layers
    pre = {}
    for nm in ("gate_proj", "down_proj"):
        P = base[nm]
        X = synth.activations_torch(GEMM_M, P.k, seed=3, stream=80, device=dev)
        Y = torch.empty((GEMM_M, P.n), dtype=torch.float16, device=dev)
        with torch.cuda.stream(stream):
            for _ in range(3):
                qx.q4x_gemm(P, X, out=Y)
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            for _ in range(10):
                qx.q4x_gemm(P, X, out=Y)
            e1.record(stream)
        torch.cuda.synchronize(dev)
        us = e0.elapsed_time(e1) * 1e3 / 10
        tflops = 2.0 * GEMM_M * P.n * P.k / (us * 1e-6) / 1e12
        pre[f"{P.n}x{P.k}"] = {"us": us, "TFLOPs": tflops, "frac_of_measured_bf16": tflops / tf_burst}
    if qx.device_status(stream) != 0:
        raise RuntimeError("q4x prefill reported a device error")
    out[f"prefill_m{GEMM_M}"] = pre
    return out


def _llava_table():
    """The LLaVA-v1.6-7B-shaped model's per-matrix recipes (a JSON table in the
    package): language matrices as (name, n, k, sigma, stream, (bits, g,
    kind)), vision matrices as (name, n, k, sigma, stream) with their one
    shared recipe."""
    with open(os.path.join(ROOT, "paper_2505_07531_gb300", "recipes", "llava_v1_6_7b.json")) as f:
        t = json.load(f)
    kinds = {"uniform": 0, "lut": 1}
    rec = lambda m: (m["recipe"]["bits"], m["recipe"]["group_size"], kinds[m["recipe"]["kind"]])  # noqa: E731
    lang = [(m["name"], m["n"], m["k"], m["sigma"], m["stream"], rec(m)) for m in t["language"]["matrices"]]
    vis = [(m["name"], m["n"], m["k"], m["sigma"], m["stream"]) for m in t["vision"]["matrices"]]
    vrec = {rec(m) for m in t["vision"]["matrices"]}
    if len(vrec) != 1:
        raise ValueError("the vision matrices share one recipe in this benchmark")
    return t, lang, vis, vrec.pop()


LLAVA, LLAVA_LANG, LLAVA_VISION, LLAVA_VISION_RECIPE = _llava_table()


def run_select(qx, torch, dev, stream):
    """Per-matrix recipe selection (qx_select_recipe) on one 4096x4096
    Student-t matrix among 3-bit uniform g64, 3-bit LUT g128, 4-bit uniform
    g64 and g128: quantize, dequantize and exact error per candidate."""
    import synth

    W = synth.student_t_weights_torch(4096, 4096, 0.02, seed=6, stream=0, device=dev)
    cands = [qx.Recipe(3, 64, qx.UNIFORM), qx.Recipe(3, 128, qx.LUT), qx.Recipe(4, 64, qx.UNIFORM),
             qx.Recipe(4, 128, qx.UNIFORM)]
    with torch.cuda.stream(stream):
        stream.wait_stream(torch.cuda.default_stream(dev))  # W is drawn on the default stream
        qx.select_recipe(W, cands)  # warm-up
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        best, errs, bpws = qx.select_recipe(W, cands)
        e1.record(stream)
    torch.cuda.synchronize()
    names = ["U3g64", "L3g128", "U4g64", "U4g128"]
    norm = float(W.float().norm())
    out = {"matrix": [4096, 4096], "candidates": names, "ms": e0.elapsed_time(e1),
           "chosen": names[best] if best is not None else None,
           "rel_frobenius_error": {nm: math.sqrt(e / float(1 << 48)) / norm for nm, e in zip(names, errs)},
           "bpw": dict(zip(names, bpws))}
    # the same four and a Q4X candidate (shared codebooks, 25 learner steps)
    cands5 = cands + [qx.Recipe(4, 64, qx.Q4X, 25)]
    with torch.cuda.stream(stream):
        qx.select_recipe(W, cands5)  # warm-up
        e0.record(stream)
        best5, errs5, bpws5 = qx.select_recipe(W, cands5)
        e1.record(stream)
    torch.cuda.synchronize()
    st_code = qx.device_status(stream)
    if st_code != 0:
        raise RuntimeError(f"recipe selection reported device status {st_code}")
    names5 = names + ["Q4Xg64"]
    out["with_q4x"] = {"ms": e0.elapsed_time(e1), "chosen": names5[best5] if best5 is not None else None,
                       "rel_frobenius_error": math.sqrt(errs5[4] / float(1 << 48)) / norm, "bpw": bpws5[4]}
    return out


def run_config5(qx, torch, dev, stream):
    """LLaVA-v1.6-7B-shaped stack with the mixed per-layer recipe.

    Decode: one token through the seven GEMVs of each of 32 language layers
    (q,k | v | o | gate,up | down: launches group matrices that share the
    activations and the recipe), PDL, one CUDA graph.  Prefill: 576 image
    tokens through the six GEMMs of each of 24 vision layers.
    """
    import synth

    base = {}
    for nm, n, k, sigma, sid, (bits, g, kind) in LLAVA_LANG:
        W = synth.student_t_weights_torch(n, k, sigma, seed=5, stream=sid, device=dev)
        base[nm] = qx.quantize(W, qx.Recipe(bits, g, kind))
        del W
    n_lang = LLAVA["language"]["layers"]
    lang = [base] + [{nm: _clone(qx, P) for nm, P in base.items()} for _ in range(n_lang - 1)]
    lang_bytes = n_lang * sum(P.nbytes() for P in base.values())
    xs = {k: synth.activations_torch(1, k, seed=5, stream=80 + i, device=dev) for i, k in enumerate((4096, 11008))}
    xa, xo, xm = (synth.activations_torch(1, 4096, seed=5, stream=90 + i, device=dev) for i in range(3))
    ys = {nm: torch.empty((1, n), dtype=torch.float16, device=dev) for nm, n, *_ in LLAVA_LANG}
    chain = [(["q_proj", "k_proj"], xa), (["v_proj"], xa), (["o_proj"], xo),
             (["gate_proj", "up_proj"], xm), (["down_proj"], xs[11008])]
    gr = _chain_graph(qx, torch, stream, lang, chain, ys)
    dec_ms = _time_graph(torch, stream, gr, 10)
    del gr, lang

    vrec = qx.Recipe(*LLAVA_VISION_RECIPE)
    vbase = dict(_quantize_layer(qx, torch, dev, LLAVA_VISION, vrec, seed=5))
    # q, k and v read the same activations and share the recipe: stacked along
    # n they are one 3n x k matrix (a fused QKV projection).  Every group lies
    # within one row, so its codes are those of the three matrices, row for row.
    qkv = [m for m in LLAVA_VISION if m[0] in ("q_proj", "k_proj", "v_proj")]
    Wqkv = torch.cat([synth.student_t_weights_torch(n, k, sig, seed=5, stream=sid, device=dev)
                      for _, n, k, sig, sid in qkv])
    vbase["qkv_proj"] = qx.quantize(Wqkv, vrec)
    del Wqkv
    n_vis = LLAVA["vision"]["layers"]
    vis = [vbase] + [{nm: _clone(qx, P) for nm, P in vbase.items()} for _ in range(n_vis - 1)]
    M = LLAVA["vision"]["tokens"]
    X1 = synth.activations_torch(M, 1024, seed=5, stream=95, device=dev)
    X4 = synth.activations_torch(M, 4096, seed=5, stream=96, device=dev)
    separate = [(nm, n, k) for nm, n, k, *_ in LLAVA_VISION]
    fused = [("qkv_proj", sum(m[1] for m in qkv), qkv[0][2])] + [m for m in separate if m[0] not in
                                                                  ("q_proj", "k_proj", "v_proj")]
    Ys = {nm: torch.empty((M, n), dtype=torch.float16, device=dev) for nm, n, _ in separate + fused}

    def vision_ms(gemm, mats):
        """The vision layers' matrices `mats` through `gemm` (qx.gemm or
        qx.gemm_splitk), one CUDA graph."""
        def vision_pass():
            for L in vis:
                for nm, n, k in mats:
                    gemm(L[nm], X4 if k == 4096 else X1, out=Ys[nm])

        with torch.cuda.stream(stream):
            vision_pass()  # also sizes the stream's split-k workspace before capture
        torch.cuda.synchronize()
        if qx.device_status(stream) != 0:
            raise RuntimeError("vision gemm reported a device error")
        gv = torch.cuda.CUDAGraph()
        with torch.cuda.graph(gv, stream=stream):
            vision_pass()
        ms = _time_graph(torch, stream, gv, 10)
        del gv
        return ms

    splitk = lambda P, X, out: qx.gemm_splitk(P, X, out=out, pdl=True)  # noqa: E731
    pre_ms = vision_ms(splitk, fused)
    pre_ms_sep = vision_ms(splitk, separate)
    pre_ms_tile = vision_ms(qx.gemm, separate)
    flops = n_vis * sum(2.0 * M * n * k for _, n, k, *_ in LLAVA_VISION)
    del vis
    return {"workload": "llava16_7b_mixed_recipe",
            "recipe": {"language": "q,k L3g128; v,o,gate,up,down U4g64", "vision": "all U4g128"},
            "decode_token_us": dec_ms * 1e3, "decode_GBps": lang_bytes / (dec_ms * 1e-3) / 1e9,
            "decode_launches": n_lang * len(chain), "language_weight_bytes": lang_bytes,
            "vision_prefill_us": pre_ms * 1e3, "vision_prefill_TFLOPs": flops / (pre_ms * 1e-3) / 1e12,
            "vision_prefill_path": "qx_gemm_splitk with PDL (64- or 256-token tiles, k split where the tiles "
                                   "leave SMs idle); q, k, v stacked as one 3072x1024 matrix",
            "vision_prefill_us_separate_qkv": pre_ms_sep * 1e3,
            "vision_prefill_us_one_cta_per_tile": pre_ms_tile * 1e3,
            "vision_tokens": M, "vision_gemm_launches": n_vis * len(fused),
            "vision_gemm_launches_separate_qkv": n_vis * len(separate),
            "recipe_table": "paper_2505_07531_gb300/recipes/llava_v1_6_7b.json"}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=50)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--skip-gemm", action="store_true")
    ap.add_argument("--skip-cpu-baseline", action="store_true")
    ap.add_argument("--skip-configs", action="store_true", help="skip the config-3 / config-5 sections")
    ap.add_argument("--cpu-baseline-child", type=float, default=None, help=argparse.SUPPRESS)
    args = ap.parse_args()
    if args.cpu_baseline_child is not None:
        cpu_baseline_child(args.cpu_baseline_child)
        return
    if args.warmup < 3:
        args.warmup = 3
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
