"""Benchmark of the ESPACE projected linear layer on GB300.

Headline workload: the GPT3-22B / Nemotron4-15B-shaped transformer layer at 16,384 tokens,
the largest single-GPU configuration of the benchmark: QKV (K = 6144 -> M = 18432), FC1
(6144 -> 24576) and FC2 (24576 -> 6144), each at rank L = K/2, bf16 inputs, fp32
accumulation, with synthetic activations (power-law spectrum i^-0.8, 1 % outlier channels
x20, log-normal channel scales), W ~ N(0, 1/K) and a seeded random P folded on the device.

A step is one espace_linear_forward per layer over the 16,384-token batch (the rank-L
projection Z = bf16(X P) and the folded product Y = Z W' of Eq. 3, one persistent launch
each). value = algorithmic TFLOP/s, sum over the three layers of 2 N (K L + L M) per step,
over the K timed steps (max over ranks). Every layer's X (>= 201 MB) is larger than the
129 MB L2, so every step reads its inputs from HBM.

Output: the side measurements first, one compact JSON line each ({"row": ...}), then the
headline as the LAST line (a few hundred bytes): value, roofline of the dominant kernel,
e2e through host buffers, cpu_baseline, clocks.

--impl reference times the fp64 CPU oracle (the only reference this method has: the paper
publishes no code) on a bounded sample of the same workload on the host cores.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402

import synth  # noqa: E402

WORKLOAD = "gpt3_22b_layer_prefill"
LAYERS = ("gpt3_22b_qkv", "gpt3_22b_fc1", "gpt3_22b_fc2")
METRIC = "ESPACE linear forward TFLOP/s (GPT3-22B layer: QKV+FC1+FC2 at L=K/2, N=16384)"
UNIT = "TFLOP/s"
SETS = 4

# DRAM bytes (read + write) of the dominant kernel per launch at this workload, averaged
# over the three layers' launches, from one ncu capture of dram__bytes_read.sum and
# dram__bytes_write.sum (the gpt3_22b_layer profile case); None until captured for the
# kernel build that runs.
FUSED_LAYER_TRAFFIC_BYTES = (1562229248 + 678923008 + 1823628032 + 878194944 + 16414597120 + 595352832) / 3
FUSED_LAYER_TRAFFIC_SOURCE = ("ncu dram__bytes_read.sum + dram__bytes_write.sum of launches 4-6 of tc_gemm_pair_kernel "
                              "in bench.py --profile-case gpt3_layer (QKV 2.24, FC1 2.70, FC2 17.01 GB)")


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-rows", action="store_true", help="skip the side measurements")
    ap.add_argument("--profile-case", choices=["gpt3_layer", "fused", "split", "syrk", "syrk24k", "decode", "train", "nl", "epilogue"],
                    help="run a few launches of one kernel on a fixed case (for ncu) and exit")
    return ap.parse_args()


def dist_init(n_gpus):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        torch.distributed.init_process_group(backend=backend)
    return world, rank, local


def barrier(world):
    if world > 1:
        torch.distributed.barrier()


def max_over_ranks(x, world):
    if world == 1:
        return x
    t = torch.tensor([x], dtype=torch.float64, device="cuda" if torch.cuda.is_available() else "cpu")
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return float(t.item())


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            d = json.load(f)
        return d.get("bf16_tflops", 1900.0), d.get("bf16_tflops_sustained", 1700.0), d.get("hbm_gbs", 6800.0), "measured"
    return 1900.0, 1700.0, 6800.0, "fallback"


def emit(obj):
    """One compact JSON line on stdout."""
    print(json.dumps(obj, separators=(",", ":")), flush=True)


def rounded(obj, digits=4):
    """Floats rounded to `digits` significant digits (compact output lines)."""
    if isinstance(obj, float):
        return float(f"{obj:.{digits}g}")
    if isinstance(obj, dict):
        return {k: rounded(v, digits) for k, v in obj.items()}
    if isinstance(obj, (list, tuple)):
        return [rounded(v, digits) for v in obj]
    return obj


class ClockSampler:
    """nvidia-smi clock / throttle samples while the GPU works."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index):
        self.proc = None
        self.device_index = device_index

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.device_index), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except (FileNotFoundError, OSError):
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
            out, _ = self.proc.communicate()
        rows = []
        for line in out.strip().splitlines():
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                rows.append((float(parts[1]), float(parts[2]), parts[5:9]))
            except ValueError:
                continue
        if not rows:
            return None
        maxc = max(r[1] for r in rows)
        loaded = [r for r in rows if r[0] > 0.5 * maxc] or rows
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in loaded for i, v in enumerate(r[2]) if v.lower() == "active"})
        return {"sm_mhz": statistics.median(r[0] for r in loaded), "sm_max_mhz": maxc,
                "reasons": reasons, "samples": len(rows)}


def cuda_events(n):
    return [torch.cuda.Event(enable_timing=True) for _ in range(n)]


def layer_shapes():
    out = []
    for name in LAYERS:
        c = synth.CONFIGS[name]
        out.append((name, c["K"], c["M"], c["L"], c["N"]))
    return out


def step_flops():
    return sum(2.0 * N * (K * L + L * M) for _, K, M, L, N in layer_shapes())


# ----------------------------------------------------------------------------- reference arm

def oracle_sample(tokens, seed):
    """Per layer of the headline workload: `tokens` tokens of X, a random bf16 P and a
    random bf16 W' of the layer's shapes (the fold is offline, Sec. 2.2, and the values do
    not change the oracle's time)."""
    import oracle
    out = []
    for name, K, M, L, N in layer_shapes():
        rng = np.random.default_rng(seed + K + M)
        X = synth.bf16_to_f64(synth.ActivationModel(K, seed=seed).sample(tokens))
        Pb = oracle.bf16_round(rng.standard_normal((K, L)) * K ** -0.5)
        Wf = oracle.bf16_round(rng.standard_normal((L, M)) * L ** -0.5)
        out.append((X, Pb, Wf))
    return out


def oracle_step(sample):
    import oracle
    for X, Pb, Wf in sample:
        oracle.contract(oracle.project(X, Pb), Wf)


def sample_tokens():
    return max(1, min(16, os.cpu_count() or 1))


def run_reference(args, world, rank):
    """fp64 oracle on the host cores, on a bounded sample of the workload."""
    if rank != 0:
        return
    t = sample_tokens()
    sample = oracle_sample(t, synth.BASE_SEED + 900)
    flops = step_flops() / synth.CONFIGS[LAYERS[0]]["N"] * t
    times = []
    for i in range(args.warmup + args.steps):
        t0 = time.perf_counter()
        oracle_step(sample)
        dt = time.perf_counter() - t0
        if i >= args.warmup:
            times.append(dt)
    total = sum(times)
    value = flops * len(times) / total / 1e12
    cores = min(int(os.environ.get("OMP_NUM_THREADS", os.cpu_count() or 1)), t)
    desc = f"{t} of 16384 tokens per step through each of QKV, FC1, FC2 (projection + folded product; fold offline)"
    emit({
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * total / len(times),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": {"workload": WORKLOAD, "layers": "qkv 6144x18432, fc1 6144x24576, fc2 24576x6144",
                                        "L": "K/2", "N": 16384},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle", "sample": desc},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    })


def cpu_baseline_leg():
    t = sample_tokens()
    sample = oracle_sample(t, synth.BASE_SEED + 900)
    flops = step_flops() / synth.CONFIGS[LAYERS[0]]["N"] * t
    oracle_step(sample)                     # first touch of the arrays
    t0 = time.perf_counter()
    reps = 0
    while True:
        oracle_step(sample)
        reps += 1
        if time.perf_counter() - t0 > 10.0 or reps >= 5:
            break
    dt = time.perf_counter() - t0
    return {"value": flops * reps / dt / 1e12, "unit": UNIT, "cores": min(os.cpu_count() or 1, t),
            "kind": "oracle",
            "sample": f"{t} tokens x {reps} repetitions through QKV, FC1 and FC2 of the fp64 oracle forward"}


# ----------------------------------------------------------------------------- our arm

def build_layers(esp, seed):
    layers = []
    for name, K, M, L, N in layer_shapes():
        X = synth.ActivationModel(K, seed=seed).sample_device(N)
        W = synth.weights_device(M, K, seed=seed)
        p = device_projection(esp, K, L, W, seed)
        Lp = (L + 63) // 64 * 64
        layers.append({"name": name, "K": K, "M": M, "L": L, "N": N, "X": X, "W": W, "p": p,
                       "Y": torch.empty((N, M), dtype=torch.bfloat16, device="cuda"),
                       "flops": 2.0 * N * (K * L + L * M), "dense_flops": 2.0 * N * K * M,
                       "bytes": 2.0 * (N * K + K * Lp + Lp * M + N * M)})
    torch.cuda.synchronize()
    return layers


def run_ours(args, world, rank, local):
    import paper_2410_05437_gb300 as esp
    torch.cuda.set_device(local)
    seed = synth.BASE_SEED + 800 + 1000 * rank
    peak_tc, peak_tc_sus, peak_hbm, peak_kind = load_peaks()
    layers = build_layers(esp, seed)
    flops = sum(l["flops"] for l in layers)
    launches = [esp.espace_linear_forward_launches(l["p"], l["N"]) for l in layers]

    sampler = ClockSampler(local)
    sampler.start()
    for i in range(args.warmup):
        for l in layers:
            esp.espace_linear_forward(l["p"], l["X"], l["Y"])
    torch.cuda.synchronize()

    # ---- timed region: exactly K steps; an event before each layer's launch
    ev = [cuda_events(len(layers) + 1) for _ in range(args.steps)]
    for row in ev:
        for e in row:
            e.record()                       # materialize the event handles
    torch.cuda.synchronize()
    barrier(world)
    torch.cuda.synchronize()
    t_begin, t_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t_begin.record()
    for i in range(args.steps):
        for j, l in enumerate(layers):
            ev[i][j].record()
            esp.espace_linear_forward(l["p"], l["X"], l["Y"])
        ev[i][-1].record()
    t_end.record()
    torch.cuda.synchronize()
    barrier(world)
    total_ms = max_over_ranks(t_begin.elapsed_time(t_end), world)
    layer_ms = [[ev[i][j].elapsed_time(ev[i][j + 1]) for i in range(args.steps)] for j in range(len(layers))]
    step_ms = [ev[i][0].elapsed_time(ev[i][-1]) for i in range(args.steps)]
    ms_per_step = total_ms / args.steps
    value = flops * args.steps * world / (total_ms * 1e-3) / 1e12
    esp.espace_check()
    clocks = sampler.stop()

    # ---- end to end through the C ABI with host buffers (pinned), copies inside the timed
    # region: espace_linear_forward_host_many takes the three layers' host X through one
    # pipeline (copies in on one stream, the products in layer order on this stream, copies
    # out on another, so that one layer's copies overlap another's products) and returns
    # with every Y in host memory. Each step is timed on its own: the host link is shared
    # with other work on the machine, and the per-step times show when it was busy.
    Xh = [l["X"].cpu().pin_memory() for l in layers]
    Yh = [torch.empty((l["N"], l["M"]), dtype=torch.bfloat16).pin_memory() for l in layers]
    e2e_steps = max(3, min(3 * args.steps, 30))
    hp = [l["p"] for l in layers]
    esp.espace_linear_forward_host_many(hp, Xh, Yh)
    torch.cuda.synchronize()
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(e2e_steps + 1)]
    ev[0].record()
    for i in range(e2e_steps):
        esp.espace_linear_forward_host_many(hp, Xh, Yh)
        ev[i + 1].record()
    torch.cuda.synchronize()
    e2e_step_ms = [ev[i].elapsed_time(ev[i + 1]) for i in range(e2e_steps)]
    e2e_ms = max_over_ranks(ev[0].elapsed_time(ev[-1]), world) / e2e_steps
    h2d = sum(2 * l["N"] * l["K"] for l in layers)
    d2h = sum(2 * l["N"] * l["M"] for l in layers)
    del Xh, Yh

    # ---- the dense layer on the same kernels (speedup), and the side rows
    dense_ms = []
    for l in layers:
        dense_ms.append(events_ms(lambda i, l=l: esp.espace_dense_forward(l["X"], l["W"], l["Y"]), reps=5, warm=2))
    esp.espace_check()
    per_layer = {}
    for j, l in enumerate(layers):
        k_ms = statistics.mean(layer_ms[j])
        per_layer[l["name"]] = {"K": l["K"], "M": l["M"], "L": l["L"], "N": l["N"], "launches": launches[j],
                                "espace_ms": k_ms, "dense_ms": dense_ms[j], "speedup": dense_ms[j] / k_ms,
                                "espace_tflops": l["flops"] / k_ms / 1e9,
                                "frac_tensor_peak": l["flops"] / k_ms / 1e9 / peak_tc}
    if rank == 0:
        emit({"row": "gpt3_22b_layer_per_layer", **rounded(per_layer)})
    if not args.no_rows:
        for name, row in side_rows(esp, args, peak_tc, peak_hbm):
            if rank == 0:
                emit({"row": name, **rounded(row)})
    for l in layers:
        esp.espace_proj_destroy(l["p"])
    del layers

    # ---- roofline of the dominant kernel: the fused forward (tc_gemm_pair_kernel), one
    # launch per layer; per launch on average = all three launches' flops over their time
    fused = all(n == 1 for n in launches)
    kern_ms = sum(statistics.mean(m) for m in layer_ms)
    achieved = flops / (kern_ms * 1e-3) / 1e12
    n_l = len(LAYERS)
    algo_bytes = sum(2.0 * (N * K + K * L + L * M + N * M) for _, K, M, L, N in layer_shapes()) / n_l
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded power-law activations with outlier channels; random-init W; random P)",
        "config": {"workload": WORKLOAD, "layers": "qkv 6144x18432, fc1 6144x24576, fc2 24576x6144",
                   "L": "K/2", "N": 16384, "parallelism": f"replicas{world}",
                   "l2": "no flush: every layer's X (>= 201 MB) and W' exceed the 129 MB L2"},
        "roofline": {"kernel": "tc_gemm_pair_kernel (fused forward, one launch per layer)" if fused
                     else "tc_gemm_pair_kernel (forward launches)",
                     "bound": "tensor", "achieved": achieved, "peak": peak_tc, "unit": "TFLOP/s",
                     "frac": achieved / peak_tc, "peak_kind": f"{peak_kind} bf16 burst",
                     "frac_of_sustained": achieved / peak_tc_sus,
                     "flops_per_launch": flops / n_l, "ms_per_launch": kern_ms / n_l,
                     "traffic": FUSED_LAYER_TRAFFIC_BYTES if fused else None,
                     "traffic_source": FUSED_LAYER_TRAFFIC_SOURCE if fused else None,
                     "algorithmic_bytes": algo_bytes},
        "step_ms": {"mean": statistics.mean(step_ms), "median": statistics.median(step_ms),
                    "min": min(step_ms), "max": max(step_ms)},
        "speedup_over_dense": sum(dense_ms) / kern_ms,
        "e2e": {"value": flops * world / (e2e_ms * 1e-3) / 1e12, "unit": UNIT, "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h, "ms_per_step": e2e_ms,
                "step_ms": {"median": statistics.median(e2e_step_ms), "min": min(e2e_step_ms),
                            "max": max(e2e_step_ms)},
                "api": "espace_linear_forward_host_many (three layers in one pipeline), pinned host X and Y"},
        "gpu_launches": sum(launches) * args.steps,
        "clocks": clocks,
    }
    if rank == 0 and world == 1:
        try:
            line["cpu_baseline"] = cpu_baseline_leg()
        except Exception as ex:   # the baseline must not sink the GPU line
            line["cpu_baseline"] = {"error": repr(ex)}
    if rank == 0:
        emit(rounded(line, 6))


def side_rows(esp, args, peak_tc, peak_hbm):
    """(name, row) pairs of the other workloads: the Llama2-7B QKV prefill layer (fused,
    two launches, dense, decode sweep), its calibration SYRK, and the rest of the benchmark's
    workloads (config_rows)."""
    rows = []
    K, M, L, N = 4096, 12288, 2048, 4096
    seed = synth.config_seed("llama2_qkv_prefill")
    model = synth.ActivationModel(K, seed=seed)
    # four independent (X, P, W') sets rotate so that no call finds its inputs in L2
    sets = []
    for s in range(SETS):
        W = synth.weights_device(M, K, seed=seed, chunk=s)
        sets.append({"X": model.sample_device(N, chunk=s), "W": W, "p": device_projection(esp, K, L, W, seed + s),
                     "Y": torch.empty((N, M), dtype=torch.bfloat16, device="cuda")})
    try:
        flops, dflops = 2.0 * N * (K * L + L * M), 2.0 * N * K * M
        reps = max(10, args.steps)
        f_ms = events_ms(lambda i: esp.espace_linear_forward(sets[i % SETS]["p"], sets[i % SETS]["X"], sets[i % SETS]["Y"]), reps=reps)
        s_ms = events_ms(lambda i: esp.espace_linear_forward_path(sets[i % SETS]["p"], sets[i % SETS]["X"], sets[i % SETS]["Y"],
                                                                  esp.PATH_TENSOR_SPLIT), reps=reps)
        d_ms = events_ms(lambda i: esp.espace_dense_forward(sets[i % SETS]["X"], sets[i % SETS]["W"], sets[i % SETS]["Y"]), reps=reps)
        esp.espace_check()
        rows.append(("llama2_qkv_prefill", {"K": K, "M": M, "L": L, "N": N, "fused_ms": f_ms, "two_launch_ms": s_ms,
                                            "dense_ms": d_ms, "speedup": d_ms / f_ms,
                                            "fused_frac_tensor_peak": flops / f_ms / 1e9 / peak_tc,
                                            "dense_frac_tensor_peak": dflops / d_ms / 1e9 / peak_tc}))
        rows.append(("decode_sweep_llama2_qkv", decode_sweep(esp, K, M, L, 0, peak_hbm, sets=sets)))
    finally:
        for s in sets:
            esp.espace_proj_destroy(s["p"])
    del sets
    # calibration: S += X^T X over 65,536 tokens (tcgen05 SYRK)
    n_cal = synth.CONFIGS["llama2_qkv_prefill"]["calib_tokens"]
    Xc = model.sample_device(n_cal, stream="calib_tokens")
    h = esp.espace_calib_create(K)
    try:
        cal_ms = events_ms(lambda i: esp.espace_calib_accumulate(h, Xc), reps=3, warm=1)
        esp.espace_check()
    finally:
        esp.espace_calib_destroy(h)
    del Xc
    cflops = float(n_cal) * K * (K + 1)
    rows.append(("calib_accumulate_k4096", {"tokens": n_cal, "ms": cal_ms, "tflops_symmetric": cflops / cal_ms / 1e9,
                                            "frac_tensor_peak": cflops / cal_ms / 1e9 / peak_tc}))
    rows.extend(config_rows(esp, peak_tc, peak_hbm))
    return rows


def events_ms(call, reps=10, warm=3):
    """Mean GPU time of one call, from CUDA events around `reps` calls after `warm` calls."""
    for i in range(warm):
        call(i)
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    for i in range(reps):
        call(i)
    b.record()
    torch.cuda.synchronize()
    return a.elapsed_time(b) / reps


def device_projection(esp, K, L, W, seed):
    """A projection handle for timing only: a seeded random bf16 P^T on the device, folded
    with W on the device (the kernels' time depends on the shapes, not the values)."""
    gen = torch.Generator(device="cuda")
    gen.manual_seed(int(seed) % (1 << 63))
    PT = (torch.randn((L, K), generator=gen, device="cuda") * K ** -0.5).to(torch.bfloat16)
    p = esp.espace_proj_from_device(PT, W)
    del PT
    return p


def tp_projection(esp, kind, tp, K, L, W, seed):
    """A tensor-parallel handle for timing only: tp seeded random projections folded with W."""
    Kr = K // tp if kind == "row" else K
    P = np.random.default_rng(seed).standard_normal((tp, Kr, L)) * Kr ** -0.5
    return esp.espace_proj_tp_from_host(esp.TP_ROW if kind == "row" else esp.TP_COLUMN, P, W)


def table2_rows(esp, peak_tc):
    """Table 2's per-rank configurations folded onto one GPU, each GEMM of a transformer
    block timed alone at batch 1 and the model's sequence length (App. B.4), dense against
    ESPACE. Column-parallel ranks calibrated by Thm. 1 share one projection (they see the
    same inputs), so those layers are the plain projected layer with the rank's L;
    row-parallel ranks each have their own, which makes the first product block-diagonal."""
    out = {}
    seed = synth.BASE_SEED + 700
    for model, cfg in synth.TABLE2.items():
        tp, N = cfg["tp"], cfg["seq"]
        layers = {}
        for name, kind, K, M, L in cfg["layers"]:
            W = synth.weights_device(M, K, seed=seed)
            X = synth.ActivationModel(K, seed=seed).sample_device(N)
            Y = torch.empty((N, M), dtype=torch.bfloat16, device="cuda")
            per_rank = kind == "row" and tp > 1
            p = tp_projection(esp, kind, tp, K, L, W, seed) if per_rank else device_projection(esp, K, L, W, seed)
            try:
                e_ms = events_ms(lambda i: esp.espace_linear_forward(p, X, Y))
                d_ms = events_ms(lambda i: esp.espace_dense_forward(X, W, Y))
                esp.espace_check()
            finally:
                esp.espace_proj_destroy(p)
            width = tp * L if per_rank else L
            flops = 2.0 * N * (K * width // (tp if per_rank else 1) + width * M)
            layers[name] = {"kind": kind, "K": K, "M": M, "L_per_rank": L, "tp": tp, "N": N,
                            "form": "per-rank block-diagonal" if per_rank else "plain", "espace_ms": e_ms,
                            "dense_ms": d_ms, "espace_tflops": flops / e_ms / 1e9,
                            "dense_tflops": 2.0 * N * K * M / d_ms / 1e9}
            del W, X, Y
        e_tot = sum(v["espace_ms"] for v in layers.values())
        d_tot = sum(v["dense_ms"] for v in layers.values())
        out[model] = {"layers": layers, "espace_ms": e_tot, "dense_ms": d_tot,
                      "gemm_latency_reduction": 1.0 - e_tot / d_tot,
                      "paper_reduction_a100": cfg["paper_reduction"]}
    return out


def layer_row(esp, K, M, L, N, seed, peak_tc):
    """One layer at N tokens: the projected forward and the dense one (inputs larger than L2
    are read by every call, so no rotation is needed)."""
    W = synth.weights_device(M, K, seed=seed)
    X = synth.ActivationModel(K, seed=seed).sample_device(N)
    Y = torch.empty((N, M), dtype=torch.bfloat16, device="cuda")
    p = device_projection(esp, K, L, W, seed)
    try:
        e_ms = events_ms(lambda i: esp.espace_linear_forward(p, X, Y))
        d_ms = events_ms(lambda i: esp.espace_dense_forward(X, W, Y))
        esp.espace_check()
    finally:
        esp.espace_proj_destroy(p)
    flops, dflops = 2.0 * N * (K * L + L * M), 2.0 * N * K * M
    return {"K": K, "M": M, "L": L, "N": N, "espace_ms": e_ms, "dense_ms": d_ms, "speedup": d_ms / e_ms,
            "espace_tflops": flops / e_ms / 1e9, "espace_frac_tensor_peak": flops / e_ms / 1e9 / peak_tc,
            "dense_tflops": dflops / d_ms / 1e9}


def decode_sweep(esp, K, M, L, seed, peak_hbm, sets=None):
    """N = 1 .. 512 tokens, projected and dense, each replayed from a CUDA graph of 20 calls
    rotating over four weight sets (so that no call finds its weights in L2)."""
    own = sets is None
    if own:
        sets = []
        for c in range(SETS):
            W = synth.weights_device(M, K, seed=seed, chunk=c)
            sets.append({"W": W, "p": device_projection(esp, K, L, W, seed + c),
                         "X": synth.ActivationModel(K, seed=seed).sample_device(max(synth.DECODE_TOKENS), chunk=c)})
    Lp = (L + 63) // 64 * 64
    sweep = {}
    try:
        for n_tok in synth.DECODE_TOKENS:
            xs = [s["X"][:n_tok].contiguous() for s in sets]
            ys = [torch.empty((n_tok, M), dtype=torch.bfloat16, device="cuda") for _ in sets]

            def espace_call(i, xs=xs, ys=ys):
                esp.espace_linear_forward(sets[i % SETS]["p"], xs[i % SETS], ys[i % SETS])

            def dense_call(i, xs=xs, ys=ys):
                esp.espace_dense_forward(xs[i % SETS], sets[i % SETS]["W"], ys[i % SETS])

            e_us = graph_time_us(espace_call)
            d_us = graph_time_us(dense_call)
            ebytes = 2.0 * (K * Lp + Lp * M + n_tok * (K + M))
            dbytes = 2.0 * (K * M + n_tok * (K + M))
            sweep[str(n_tok)] = {
                "espace_us": e_us, "dense_us": d_us, "speedup": d_us / e_us,
                "espace_gbs": ebytes / e_us / 1e3, "espace_frac_hbm": ebytes / e_us / 1e3 / peak_hbm,
                "espace_tflops": 2.0 * n_tok * (K * L + L * M) / e_us / 1e6,
                "dense_gbs": dbytes / d_us / 1e3,
                "path": ("decode kernel" if esp.espace_linear_forward_launches(sets[0]["p"], n_tok) == 1
                         and n_tok <= 32 else "tcgen05")}
    finally:
        if own:
            for s in sets:
                esp.espace_proj_destroy(s["p"])
    return sweep


def config_rows(esp, peak_tc, peak_hbm):
    """(name, row) pairs of the other workloads of the benchmark: the Llama2-7B MLP over a
    rank sweep, calibration over 1,048,576 tokens at K = 6144 and K = 24576, the decode sweep
    on the other Llama2-7B layers, the whole Llama2-7B layer at batch 1, sequence 4096,
    Table 2's folded tensor-parallel layers (one row per model), the NL-MSE calibration, the
    projection build at K = 4096, 6144 and 11008, and the training step."""
    rows = []
    seed = synth.BASE_SEED + 500
    for name, (K, M) in (("gate_up", (4096, 22016)), ("down", (11008, 4096))):
        sweep = {}
        for frac in (0.8, 0.7, 0.6, 0.5):
            L = int(round(frac * K))
            r = layer_row(esp, K, M, L, 8192, seed, peak_tc)
            sweep[f"L{int(frac * 100)}pct"] = {k: r[k] for k in ("L", "espace_ms", "dense_ms", "speedup",
                                                                 "espace_frac_tensor_peak")}
        rows.append((f"llama2_mlp_{name}_rank_sweep", {"K": K, "M": M, "N": 8192, **sweep}))
    n_total, chunk = 1 << 20, 65536
    for K in (6144, 24576):
        Xc = synth.ActivationModel(K, seed=seed).sample_device(chunk, stream="calib_tokens")
        h = esp.espace_calib_create(K)
        try:
            esp.espace_calib_accumulate(h, Xc)
            esp.espace_calib_reset(h)
            ms = events_ms(lambda i: esp.espace_calib_accumulate(h, Xc), reps=n_total // chunk, warm=0) * (n_total // chunk)
            esp.espace_check()
        finally:
            esp.espace_calib_destroy(h)
        del Xc
        cflops = float(n_total) * K * (K + 1)
        rows.append((f"calibration_1m_tokens_k{K}", {"tokens": n_total, "ms": ms, "tflops_symmetric": cflops / ms / 1e9,
                                                   "frac_tensor_peak": cflops / ms / 1e9 / peak_tc,
                                                   "note": "16 accumulations of one 65,536-token chunk"}))
    for name in ("o", "gate_up", "down"):
        K, M = synth.DECODE_LAYERS[name]
        rows.append((f"decode_sweep_llama2_{name}", decode_sweep(esp, K, M, K // 2, seed, peak_hbm)))
    layer = {}
    for name in ("qkv", "o", "gate_up", "down"):
        K, M = synth.DECODE_LAYERS[name]
        r = layer_row(esp, K, M, K // 2, 4096, seed, peak_tc)
        layer[name] = {"espace_ms": r["espace_ms"], "dense_ms": r["dense_ms"]}
    tot_e = sum(v["espace_ms"] for v in layer.values())
    tot_d = sum(v["dense_ms"] for v in layer.values())
    layer["total"] = {"espace_ms": tot_e, "dense_ms": tot_d, "speedup": tot_d / tot_e}
    rows.append(("llama2_layer_prefill_batch1_seq4096", layer))
    for model, r in table2_rows(esp, peak_tc).items():
        rows.append((f"table2_tp_folded_{model}", r))
    rows.append(("nl_mse_calibration", nl_mse_row(esp, peak_tc, seed)))
    for K, M in ((4096, 12288), (6144, 18432), (11008, 4096)):
        rows.append((f"build_projection_k{K}", build_row(esp, K, M, K // 2, seed)))
    for name, r in training_rows(esp, peak_tc, seed).items():
        rows.append((f"training_step_{name}", r))
    return rows


def build_row(esp, K, M, L, seed, n_cal=65536):
    """espace_build_projection's wall time (synchronous: fp64 eigen-solve of C on the host
    cores, P rounded to bf16 and W' = P^T W folded on the GPU) after a calibration of n_cal
    tokens, at rank L of K inputs and M outputs (Thm. 1, App. B.1)."""
    X = synth.ActivationModel(K, seed=seed).sample_device(n_cal, stream="calib_tokens")
    W = synth.weights_device(M, K, seed=seed)
    h = esp.espace_calib_create(K)
    p = None
    try:
        esp.espace_calib_accumulate(h, X)
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        p = esp.espace_build_projection(h, W, L)
        build_s = time.perf_counter() - t0
        esp.espace_check()
    finally:
        if p:
            esp.espace_proj_destroy(p)
        esp.espace_calib_destroy(h)
    del X, W
    return {"K": K, "M": M, "L": L, "calib_tokens": n_cal, "build_s": build_s, "host_cores": os.cpu_count()}


def nl_mse_row(esp, peak_tc, seed, K=4096, T=4096, reps=4):
    """Thm. 2's NL-MSE calibration at K = 4096, one sequence of 4096 tokens per call with
    synthetic gradients (an independent token model, scaled down): per call two SYRKs of T
    tokens (2 T K (K+1) flop) and six upper-triangle K x K x K products for A B + B A with
    bf16 hi / lo halves (6 K^2 (K+1) flop)."""
    X = synth.ActivationModel(K, seed=seed).sample_device(T, stream="calib_tokens")
    G = (synth.ActivationModel(K, seed=seed + 1, outliers=0, lognormal_sigma=0.0)
         .sample_device(T, stream="calib_tokens", chunk=1).float() * 0.01).to(torch.bfloat16)
    h = esp.espace_calib_create(K)
    try:
        esp.espace_calib_accumulate_nl(h, X, G)          # allocates the handle's scratch
        ms = events_ms(lambda i: esp.espace_calib_accumulate_nl(h, X, G), reps=reps, warm=1)
        esp.espace_check()
    finally:
        esp.espace_calib_destroy(h)
    flops = 2.0 * T * K * (K + 1) + 6.0 * K * K * (K + 1)
    return {"K": K, "tokens_per_sequence": T, "ms_per_sequence": ms, "tflops": flops / ms / 1e9,
            "frac_tensor_peak": flops / ms / 1e9 / peak_tc}


def training_rows(esp, peak_tc, seed, micro=4):
    """The training view of Sec. 2.2 against dense training, one layer's GEMM work per
    optimizer step of `micro` micro-batches: ESPACE refolds W' = P^T W once (after the
    weight update), runs each micro-batch's forward (keeping Z) and backward (dX, and Z^T dY
    accumulated), then forms dW = (sum Z^T dY)^T P^T once; dense runs each micro-batch's
    forward and backward (dX, dW accumulated). Llama2-7B QKV (4096 -> 12288) with 4096-token
    micro-batches, L = K/2 and Table 2's L = 1024; GPT3-22B FC1 (6144 -> 24576) with
    2048-token micro-batches, L = 2048."""
    out = {}
    for name, K, M, L, N in (("llama2_qkv_L2048", 4096, 12288, 2048, 4096), ("llama2_qkv_L1024", 4096, 12288, 1024, 4096),
                             ("gpt3_22b_fc1_L2048", 6144, 24576, 2048, 2048)):
        W = synth.weights_device(M, K, seed=seed)
        X = synth.ActivationModel(K, seed=seed).sample_device(N)
        dY = (torch.randn((N, M), device="cuda") * 0.01).to(torch.bfloat16)
        Y = torch.empty((N, M), dtype=torch.bfloat16, device="cuda")
        dX = torch.empty((N, K), dtype=torch.bfloat16, device="cuda")
        dW = torch.empty((M, K), dtype=torch.float32, device="cuda")
        Lp = (L + 63) // 64 * 64
        Z = torch.empty((N, Lp), dtype=torch.bfloat16, device="cuda")
        p = device_projection(esp, K, L, W, seed)

        def espace_step(i):
            esp.espace_proj_refold(p, W)
            for _ in range(micro):
                esp.espace_train_forward(p, X, Z, Y)
                esp.espace_train_backward(p, dY, Z, dX)
            esp.espace_train_weight_grad(p, dW)

        def dense_step(i):
            for j in range(micro):
                esp.espace_dense_forward(X, W, Y)
                esp.espace_dense_backward(dY, X, W, dX, dW, accumulate=j > 0)

        try:
            e_ms = events_ms(espace_step)
            d_ms = events_ms(dense_step)
            esp.espace_check()
        finally:
            esp.espace_proj_destroy(p)
        T = micro * N
        eflops = 2.0 * M * K * L + 2.0 * T * L * (K + M) + 2.0 * T * L * (2 * M + K) + 2.0 * L * M * K
        dflops = 6.0 * T * K * M
        out[name] = {"K": K, "M": M, "L": L, "tokens_per_micro_batch": N, "micro_batches": micro,
                     "espace_step_ms": e_ms, "dense_step_ms": d_ms, "step_speedup": d_ms / e_ms,
                     "espace_flops_over_dense": eflops / dflops, "espace_tflops": eflops / e_ms / 1e9,
                     "espace_frac_tensor_peak": eflops / e_ms / 1e9 / peak_tc, "dense_tflops": dflops / d_ms / 1e9}
        del W, X, dY, Y, dX, dW, Z
    return out


def graph_time_us(call, per_graph=20, replays=10):
    """Mean GPU time of one call, from CUDA-graph replays (inputs rotate inside the graph)."""
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        # every call of the graph once: scratch and workspaces grow outside the capture
        for i in range(per_graph):
            call(i)
    torch.cuda.current_stream().wait_stream(side)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        for i in range(per_graph):
            call(i)
    g.replay()
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    for _ in range(replays):
        g.replay()
    b.record()
    torch.cuda.synchronize()
    return a.elapsed_time(b) * 1e3 / (per_graph * replays)


def profile_case(which):
    """A few launches of one kernel, with little else on the GPU: the target of the ncu
    captures summarized under profiles/ (gpt3_layer: launches 4-6 of tc_gemm_pair_kernel
    are the three layers' fused forwards, after the three folds; fused: launch 3 of the fused
    forward at the Llama2 QKV prefill shape; split: the same forward as two launches per call
    (launches 2-7 of the kernel); launch 2 of the calibration SYRK; launch 3 of
    the decode kernel; the training view's backward products; the NL-MSE launches; epilogue:
    launches 2-3 of a dense 2048 x 6144 x 512 product, a short reduction)."""
    import paper_2410_05437_gb300 as esp
    torch.cuda.set_device(0)
    if which == "gpt3_layer":
        layers = build_layers(esp, synth.BASE_SEED + 800)
        for l in layers:
            esp.espace_linear_forward(l["p"], l["X"], l["Y"])
        torch.cuda.synchronize()
        for l in layers:
            esp.espace_proj_destroy(l["p"])
    elif which == "epilogue":
        K, M, N = 512, 6144, 2048
        W = synth.weights_device(M, K)
        X = synth.ActivationModel(K).sample_device(N)
        Y = torch.empty(N, M, device="cuda", dtype=torch.bfloat16)
        for _ in range(3):
            esp.espace_dense_forward(X, W, Y)
        torch.cuda.synchronize()
    elif which in ("fused", "split", "decode"):
        K, M, L = 4096, 12288, 2048
        N = 1 if which == "decode" else 4096
        W = synth.weights_device(M, K)
        p = esp.espace_proj_from_host(synth.random_projection(K, L), W)      # launch 1: fold
        X = synth.ActivationModel(K).sample_device(N)
        Y = torch.empty(N, M, device="cuda", dtype=torch.bfloat16)
        path = esp.PATH_TENSOR_SPLIT if which == "split" else esp.PATH_AUTO
        for _ in range(3):
            esp.espace_linear_forward_path(p, X, Y, path)
        torch.cuda.synchronize()
        esp.espace_proj_destroy(p)
    elif which == "train":
        # pair-kernel launches: 1 fold, 2 forward (fused), 3 dZ = dY W', 4 dX = dZ P^T,
        # 5 (dW P)^T += Z^T dY, 6 dW = (dW P) P^T
        K, M, L, N = 4096, 12288, 2048, 4096
        W = synth.weights_device(M, K)
        p = esp.espace_proj_from_host(synth.random_projection(K, L), W)
        X = synth.ActivationModel(K).sample_device(N)
        dY = (torch.randn(N, M, device="cuda") * 0.01).to(torch.bfloat16)
        Z = torch.empty(N, L, device="cuda", dtype=torch.bfloat16)
        Y = torch.empty(N, M, device="cuda", dtype=torch.bfloat16)
        dX = torch.empty(N, K, device="cuda", dtype=torch.bfloat16)
        dW = torch.empty(M, K, device="cuda", dtype=torch.float32)
        esp.espace_train_forward(p, X, Z, Y)
        esp.espace_train_backward(p, dY, Z, dX)
        esp.espace_train_weight_grad(p, dW)
        torch.cuda.synchronize()
        esp.espace_proj_destroy(p)
    elif which == "nl":
        # two NL-MSE sequences of 4096 tokens at K = 4096 (11 launches each)
        K, T = 4096, 4096
        X = synth.ActivationModel(K).sample_device(T, stream="calib_tokens")
        G = (synth.ActivationModel(K, seed=1, outliers=0, lognormal_sigma=0.0)
             .sample_device(T, stream="calib_tokens", chunk=1).float() * 0.01).to(torch.bfloat16)
        h = esp.espace_calib_create(K)
        for _ in range(2):
            esp.espace_calib_accumulate_nl(h, X, G)
        torch.cuda.synchronize()
        esp.espace_calib_destroy(h)
    elif which == "syrk24k":
        # the calibration SYRK at K = 24576 (FC2's input) over one 16,384-token chunk
        K, n = 24576, 16384
        X = synth.ActivationModel(K).sample_device(n, stream="calib_tokens")
        h = esp.espace_calib_create(K)
        for _ in range(2):
            esp.espace_calib_accumulate(h, X)
        torch.cuda.synchronize()
        esp.espace_calib_destroy(h)
    else:
        K, n = 4096, 65536
        X = synth.ActivationModel(K).sample_device(n, stream="calib_tokens")
        h = esp.espace_calib_create(K)
        for _ in range(2):
            esp.espace_calib_accumulate(h, X)
        torch.cuda.synchronize()
        esp.espace_calib_destroy(h)
    esp.espace_check()
    print(json.dumps({"profile_case": which, "ok": True}))


def main():
    args = parse()
    if args.profile_case:
        profile_case(args.profile_case)
        return
    world, rank, local = dist_init(args.gpus)
    if args.impl == "reference":
        run_reference(args, world, rank)
    else:
        run_ours(args, world, rank, local)
    if world > 1:
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
