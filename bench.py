"""Benchmark of the ASP W4A4 + low-rank linear layer on GB300.

One step = one pass of the whole hot path -- kernel (a) (projection, remainder, 4-bit activation
quantization) and kernel (b) (4-bit GEMM with the 16-bit branch in its epilogue) -- over one
batch of the DiT attention-projection workload: X bf16 [M=4096, K=3072], W [3072, 3072],
r = 32, group 64, seeded synthetic data (1% outlier channels x10..30).

Output: one JSON line.  `value` is the effective TOPS (2*M*N*K per step over the device time of
the timed steps of qwam_asp_linear, max over ranks, summed over ranks' work; a step is two
launches, kernel (a) (which for INT4 at 512 or more tokens also writes the float16 weights) and the
GEMM); the per-kernel split comes from a second pass with the two public calls timed apart (there
the GEMM call runs the weight expansion as a launch of its own); `e2e`
repeats the measurement through
the C ABI with the activations copied from pinned host memory and the output copied back inside
the timed region; `roofline` describes the dominant kernel; `cpu_baseline` times the CPU oracle
on a bounded sample of rows.  `--impl reference` times the CPU oracle alone (the reference arm).

Multi-GPU (torchrun): every rank runs the same per-GPU batch (token rows are independent, so
the layer shards by rows with no collective); weak scaling.

The NVFP4 variant (App. B.1: E2M1 with an E4M3 scale per 16 K, block scales applied by the
tensor cores) is timed on the same workload and reported under `variants`; `--format nvfp4` makes
it the headline.  So is the layer with smoothing and the block Hadamard rotation in front (Sec. 3
Eq. (pair)); `--rotate` makes that the headline (one more launch per step with r > 0).  The
denoising-step layer sweep (30 DiT blocks, ASP on a third of them) is reported per format under
`variants.sweep_int4` / `variants.sweep_nvfp4`.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "ASP W4A4+low-rank linear effective TOPS (2*M*N*K per step)"
UNIT = "TOPS"
WORKLOAD = dict(workload="dit_attn_proj_M4096_K3072_N3072_r32_g64", M=4096, K=3072, N=3072, r=32, group=64)
ROTATE_SETS = 6  # distinct input/output/workspace/weight sets cycled through (> L2 in total)
ROTATION = "smoothing alpha 0.5 + block Hadamard B 1024 in front of the layer (Eq. (pair))"


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=2000)
    p.add_argument("--warmup", type=int, default=50)
    p.add_argument("--impl", choices=["ours", "reference"], default="ours")
    p.add_argument("--cpu-rows", type=int, default=0, help="oracle sample rows (0 = sized to ~10 s)")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--rotate", action="store_true",
                   help="headline layer with smoothing (alpha 0.5) and the block Hadamard rotation in front "
                        "(Eq. (pair)); also measured as a variant of the default run")
    p.add_argument("--format", choices=["int4", "nvfp4"], default="int4",
                   help="4-bit format of the headline: INT4 group 64 (the configuration's), or NVFP4 "
                        "(App. B.1's Blackwell format, also measured as a variant of the INT4 run)")
    return p.parse_args()


# ------------------------------------------------------------------ distributed plumbing

def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def init_dist(world, backend):
    import torch.distributed as dist
    if world > 1 and not dist.is_initialized():
        os.environ.setdefault("MASTER_ADDR", "127.0.0.1")
        dist.init_process_group(backend=backend)
    return dist


def max_over_ranks(x: float, world: int, device=None) -> float:
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def aggregate_value(flops_per_step: float, steps: int, world: int, total_ms: float) -> float:
    """Whole-job effective TOPS: every rank's steps over the slowest rank's elapsed time."""
    return flops_per_step * steps * world / (total_ms * 1e-3) / 1e12


def barrier(world: int):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


# ------------------------------------------------------------------ clocks during the timed region

class ClockSampler:
    """nvidia-smi sampling of SM clock and throttle reasons (read-only)."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.samples = []
        self.proc = None
        self.t0 = self.t1 = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu=timestamp,{self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "50"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            threading.Thread(target=self._read, daemon=True).start()
        except Exception:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.samples.append((time.time(), line.strip()))

    def mark(self, which):
        setattr(self, which, time.time())

    def stop(self):
        if self.proc:
            time.sleep(0.12)
            self.proc.terminate()
            try:
                self.proc.wait(timeout=2)
            except Exception:
                self.proc.kill()

    def summary(self):
        rows = []
        for ts, line in self.samples:
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                rows.append((ts, float(parts[1]), float(parts[2]), parts[4:9]))
            except ValueError:
                continue
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        inside = [r for r in rows if self.t0 and self.t1 and self.t0 - 0.05 <= r[0] <= self.t1 + 0.05]
        use = inside or rows
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in use for i, v in enumerate(r[3][1:]) if v.lower().startswith("active")})
        return {"sm_mhz": statistics.median(r[1] for r in use), "sm_max_mhz": max(r[2] for r in use),
                "reasons": reasons, "samples": len(use), "samples_in_timed_region": len(inside)}


# ------------------------------------------------------------------ CPU oracle (baseline / reference arm)

def oracle_sample(rows: int, nvfp4: bool = False, rotate: bool = False):
    """Inputs and packed weights for the oracle timing: the workload's first `rows` tokens; with
    `rotate`, smoothing factors (alpha 0.5, from the batch's channel maxima) for Eq. (pair)."""
    import oracle
    from oracle import subspace
    from paper_2609_33269_gb300 import workloads as wl
    layer = wl.dit_attention().layers[0]
    Xall = layer.x()
    Xb = Xall[:rows].copy()
    U = layer.u()
    s = None
    W = layer.w()
    if rotate:
        xmax = np.abs(oracle.bf16_bits_to_f64(Xall)).max(axis=0)
        s = subspace.smoothing_factors(xmax, oracle.bf16_bits_to_f64(W), 0.5)
    # offline packing: outside the timed sample
    if rotate:
        Wt = oracle.rotate_weights(W, s)
        wts = oracle.pack_nvfp4_f64(Wt, U) if nvfp4 else oracle.pack_f64(Wt, U, layer.G)
    else:
        wts = oracle.pack_nvfp4(W, U) if nvfp4 else oracle.pack(W, U, layer.G)
    layer.s = s
    return Xb, U, wts, layer


def oracle_step(Xb, U, wts, G, nvfp4: bool = False, s=None, rotate: bool = False):
    import oracle
    if rotate:
        Xt = oracle.rotate_acts(Xb, s)
        if nvfp4:
            return oracle.linear_nvfp4(oracle.quantize_act_nvfp4_f64(Xt, U), wts)
        return oracle.linear(oracle.quantize_act_f64(Xt, U, G), wts, G)
    if nvfp4:
        return oracle.linear_nvfp4(oracle.quantize_act_nvfp4(Xb, U), wts)
    act = oracle.quantize_act(Xb, U, G)
    return oracle.linear(act, wts, G)


def cpu_cores() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except Exception:
        return os.cpu_count() or 1


def run_reference(args):
    rank, world, _ = dist_env()
    if rank != 0:
        return 0
    K, N = WORKLOAD["K"], WORKLOAD["N"]
    nv = args.format == "nvfp4"
    rot = args.rotate
    rows = args.cpu_rows
    if not rows:  # size each step so that warm-up + timed steps take about two minutes
        Xb, U, wts, layer = oracle_sample(8, nv, rot)
        t0 = time.perf_counter()
        oracle_step(Xb, U, wts, layer.G, nv, layer.s, rot)
        per_row = (time.perf_counter() - t0) / 8
        rows = int(max(1, min(256, 120.0 / (max(1, args.steps + args.warmup) * per_row))))
    Xb, U, wts, layer = oracle_sample(rows, nv, rot)
    for _ in range(max(0, args.warmup)):
        oracle_step(Xb, U, wts, layer.G, nv, layer.s, rot)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        oracle_step(Xb, U, wts, layer.G, nv, layer.s, rot)
    dt = time.perf_counter() - t0
    value = 2.0 * rows * N * K * args.steps / dt / 1e12
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": dt / args.steps * 1e3,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": dict(WORKLOAD, sample_rows_per_step=rows, parallelism="host cores",
                                            format="nvfp4 (block 16)" if nv else "int4 (group 64)",
                                            **({"rotation": ROTATION} if rot else {})),
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": cpu_cores(), "kind": "oracle",
                         "sample": f"{rows} of 4096 token rows per step (quantize + output); packing offline"},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line))
    return 0


def cpu_baseline(rows_req: int, nvfp4: bool = False, rotate: bool = False, gpu=None):
    """The oracle as it stands on the host cores: whole passes over a sample of the workload's
    rows, repeated until about ten seconds of CPU work (packing excluded, as on the GPU).  With
    `gpu` (the GPU's codes, scales and float32 output for the workload's first rows), the sample's
    oracle result is also compared with them, after the timing (see parity_sample)."""
    K, N = WORKLOAD["K"], WORKLOAD["N"]
    rows = rows_req or WORKLOAD["M"]
    Xb, U, wts, layer = oracle_sample(rows, nvfp4, rotate)
    reps, t0 = 0, time.perf_counter()
    while True:
        oracle_step(Xb, U, wts, layer.G, nvfp4, layer.s, rotate)
        reps += 1
        dt = time.perf_counter() - t0
        if dt >= 10.0 or reps >= 50:
            break
    out = {"value": 2.0 * rows * N * K * reps / dt / 1e12, "unit": UNIT, "cores": cpu_cores(), "kind": "oracle",
           "sample": f"{reps} pass(es) over {rows} of {WORKLOAD['M']} token rows (activation quantization + "
                     f"output, {dt:.1f} s); weight packing offline"}
    if gpu is not None and not rotate:
        n = min(rows, len(gpu["Y"]))
        out["parity_sample"] = parity_sample(Xb[:n], U, wts, layer.G, nvfp4, {k: v[:n] for k, v in gpu.items()})
    return out


def parity_sample(Xb, U, wts, G, nvfp4, gpu):
    """Flip and row-error counts of the timed configuration's GPU result against the oracle on the
    same rows.  At r > 0 the kernel's float32 remainder differs from the oracle's float64 one in
    the last bits, so a code (or an NVFP4 block scale) can round the other way where the float64
    quotient sits next to a rounding midpoint: every such flip is counted and checked to be within
    1e-3 of a midpoint; the output is compared per row (max |dY| / max |Y|), separately for rows
    with and without a flip."""
    import oracle
    oa = oracle.quantize_act(Xb, U, 32 if nvfp4 else G, want_float64=True)
    Xp = oa["Xperp"]
    if nvfp4:
        oa = oracle.quantize_act_nvfp4(Xb, U)
        Yo = oracle.linear_nvfp4(oa, wts)
        tab = np.array([oracle.e4m3_value(b) for b in range(127)])
        mids = (tab[1:] + tab[:-1]) / 2
        M, K = oa["qx"].shape
        t = np.abs(Xp).reshape(M, K // 16, 16).max(axis=2) / 6.0
        sbad = np.argwhere(gpu["sfx"] != oa["sfx"])
        near = [np.abs(mids - t[m, b]).min() <= 1e-3 * t[m, b] for m, b in sbad]
        cbad = np.argwhere((gpu["qx"] != oa["qx"]) & np.repeat(gpu["sfx"] == oa["sfx"], 16, axis=1))
        e2m1_mids = np.array([0.25, 0.75, 1.25, 1.75, 2.5, 3.5, 5.0])
        for m, k in cbad:
            s = tab[int(oa["sfx"][m, k // 16])]
            near.append(s > 0 and np.abs(e2m1_mids - abs(Xp[m, k]) / s).min() <= 1e-3)
        flips, scale_flips = len(sbad) + len(cbad), len(sbad)
        flip_rows = np.any(gpu["qx"] != oa["qx"], axis=1) | np.any(gpu["sfx"] != oa["sfx"], axis=1)
    else:
        Yo = oracle.linear(oa, wts, G)
        bad = np.argwhere(gpu["qx"] != oa["qx"])
        near = []
        for m, k in bad:
            s = float(oa["sx"][m, k // G])
            q = abs(float(Xp[m, k])) / s if s > 0 else 0.0
            near.append(abs(q - np.floor(q) - 0.5) <= 1e-3)
        flips, scale_flips = len(bad), int(np.sum(gpu["sx"].view(np.uint32) != oa["sx"].view(np.uint32)))
        flip_rows = np.any(gpu["qx"] != oa["qx"], axis=1)
    err = np.abs(gpu["Y"] - Yo).max(axis=1) / np.maximum(np.abs(Yo).max(axis=1), 1e-30)
    return {"rows": int(len(Yo)), "codes": int(gpu["qx"].size), "code_or_block_scale_flips": int(flips),
            "all_flips_near_ties": bool(all(near)), "scales_not_bit_equal": int(scale_flips),
            "rows_with_a_flip": int(flip_rows.sum()),
            "max_row_err_rows_without_flip": float(err[~flip_rows].max()) if (~flip_rows).any() else None,
            "max_row_err_rows_with_flip": float(err[flip_rows].max()) if flip_rows.any() else None,
            "note": "bit-exact codes and scales only given the kernel's own float32 remainder at r > 0"}


def kernel_traffic(kernel: str):
    """DRAM bytes per launch of `kernel` from the committed ncu summary, or None when the kernel's
    sources have changed since the counters were taken."""
    import hashlib
    try:
        rec = json.load(open(os.path.join(ROOT, "profiles", "traffic.json")))[kernel]
    except Exception:
        return None
    h = hashlib.sha256()
    for f in rec.get("sources", []):
        with open(os.path.join(ROOT, f), "rb") as fh:
            h.update(fh.read())
    return rec["dram_bytes_per_launch"] if h.hexdigest() == rec.get("sources_sha256") else None


# ------------------------------------------------------------------ GPU arm

def alg_bytes_actquant(M, K, r_pad, G, nvfp4=False):
    """Kernel (a): read X (2MK) and U (hi/lo, twice), write codes (MK/2), scales (INT4: bfloat16
    per group, 2MK/G; NVFP4: one E4M3 byte per 16, MK/16), p_hat."""
    scales = M * K // 16 if nvfp4 else 2 * M * K // G
    return 2 * M * K + M * K // 2 + scales + 2 * M * r_pad + 2 * (2 * K * r_pad) * 2


def small_m_latencies(asp, wl, dev, stream, dev_bf16):
    """The action-expert small-M layers (K = 1024; M 32 and 128; N 1024 and 4096; r 16 and 0), the
    latency-bound regime: the time of one qwam_asp_linear call in each format, from a CUDA graph of
    20 calls replayed 10 times, with the inputs resident on the device."""
    import torch
    out = {}
    side = torch.cuda.Stream(dev)
    for L in wl.action_expert_small_m().layers:
        if L.M not in (32, 128):
            continue
        Xs, Ws = dev_bf16(L.x()), dev_bf16(L.w())
        Us = torch.from_numpy(L.u()).to(dev) if L.r else None
        variants = [(asp.QWAM_FMT_INT4, "int4", False), (asp.QWAM_FMT_NVFP4, "nvfp4", False)]
        if L.r:  # the same layers with smoothing (from the batch's channel maxima) and the rotation
            variants += [(asp.QWAM_FMT_INT4, "int4_rotated", True), (asp.QWAM_FMT_NVFP4, "nvfp4_rotated", True)]
            sm = torch.empty(L.K, dtype=torch.float32, device=dev)
            asp.qwam_asp_smoothing_factors(Xs.float().abs().amax(dim=0).contiguous(), Ws, L.K, L.N, 0.5, sm, stream)
        for fmt, fname, rot in variants:
            lin = asp.AspLinear(Ws, Us, L.G, fmt=fmt, rotate=rot, s=sm if rot else None)
            Ys = torch.empty((L.M, L.N), dtype=torch.bfloat16, device=dev)
            side.wait_stream(stream)
            with torch.cuda.stream(side):
                for _ in range(3):
                    lin(Xs, out=Ys, stream=side)
            side.synchronize()
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=side):
                for _ in range(20):
                    lin(Xs, out=Ys, stream=side)
            g.replay()
            torch.cuda.synchronize()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            for _ in range(10):
                g.replay()
            e1.record()
            torch.cuda.synchronize()
            us = e0.elapsed_time(e1) / 200 * 1e3
            out["%s_%s" % (fname, L.name)] = {"us_per_layer": round(us, 2),
                                              "tops": round(2.0 * L.M * L.N * L.K / us / 1e6, 2)}
            del g
            lin.close()
    return {"what": "one qwam_asp_linear call of an action-expert layer (K=1024), CUDA graph of 20 calls; "
                    "*_rotated: with smoothing and the block Hadamard rotation in front (Eq. (pair))",
            "layers": out}


def denoise_sweep(asp, wl, dev, stream, fmt, steps, hbm_peak, mma_peak, peak_source):
    """The denoising-step layer sweep: 30 DiT blocks x {qkv 3072->9216, o 3072->3072, up
    3072->12288, down 12288->3072} at M = 4096 tokens, ASP (r = 32) on the workload's seeded third of
    the blocks and r = 0 elsewhere, over `steps` denoising steps.  Weights and activations are drawn
    on the device (seeded torch generator) with the recipe's distributions, so that the 120 layers
    pack in seconds (the bases are the workload's own); every layer is packed once.
    Headline (`value`): every step gets fresh activations, drawn in the untimed gap before it,
    and L2 is flushed (a 256 MB write) before it; each step is timed on its own and the steps'
    times are summed.  Within a step two activation sets per input width alternate, so a layer's
    input may still be in L2 from an earlier layer of the step, as the previous layer's output
    would be in a model.  `l2_warm` times the same steps back to back on one activation draw.
    Also: a roofline object (the aggregate against the MMA kind's peak) and the layers' roofline
    fraction (sum over calls of max(algorithmic bytes / HBM, flops / MMA peak) over the measured
    time), and a breakdown by layer kind and rank."""
    import torch
    W = wl.denoise_sweep(steps=steps)
    nv = fmt == asp.QWAM_FMT_NVFP4
    g = torch.Generator(device=dev)
    g.manual_seed(0)
    lins = []
    for L in W.layers:
        Wt = (torch.randn((L.K, L.N), generator=g, device=dev) / np.sqrt(L.K)).to(torch.bfloat16)
        U = torch.from_numpy(L.u()).to(dev) if L.r else None  # the workload's seeded basis (host QR)
        lins.append(asp.AspLinear(Wt, U, L.G, fmt=fmt))
        del Wt
    # activation sets: two per input width, 1 % outlier channels x U(10, 30), and Student-t
    # (nu = 4) for the down projections' input
    def draw(K, student):
        if student:  # t(4) = N(0, 1) / sqrt(chi2(4) / 4)
            z = torch.randn((5, 4096, K), generator=g, device=dev)
            x = z[0] / torch.sqrt((z[1:] ** 2).sum(dim=0) / 4.0)
            del z
        else:
            x = torch.randn((4096, K), generator=g, device=dev)
            ch = torch.randperm(K, generator=g, device=dev)[: K // 100]
            x[:, ch] *= torch.empty(K // 100, device=dev).uniform_(10.0, 30.0, generator=g)
        return x.to(torch.bfloat16).contiguous()

    def draw_all():
        return {(K, st, i): draw(K, st) for K, st in ((3072, False), (12288, True)) for i in range(2)}

    xs = draw_all()
    outs = {N: torch.empty((4096, N), dtype=torch.bfloat16, device=dev) for N in (3072, 9216, 12288)}
    ws = torch.empty(max(asp.qwam_asp_act_workspace_bytes(l.h, 4096) for l in lins), dtype=torch.uint8, device=dev)
    flush = torch.empty(64 * 1024 * 1024, dtype=torch.float32, device=dev)  # 256 MB > L2

    def one_step(i, ev=None):
        for j, (L, lin) in enumerate(zip(W.layers, lins)):
            X = xs[(L.K, L.dist == "student_t", i % 2)]
            if ev is not None:
                ev[2 * j].record(stream)
            asp.qwam_asp_linear(X, 4096, lin.h, outs[L.N], asp.QWAM_Y_BF16, ws, stream)
            if ev is not None:
                ev[2 * j + 1].record(stream)

    one_step(0)
    torch.cuda.synchronize()
    for lin in lins:
        if asp.qwam_asp_get_error(lin.h) != asp.QWAM_OK:
            raise RuntimeError("device error in the sweep warm-up")
    # fresh activations and a cold L2 before every step; each step timed alone
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(2 * len(lins))] for _ in range(steps)]
    step_ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
    for i in range(steps):
        xs = draw_all()
        flush.zero_()
        torch.cuda.synchronize()
        step_ev[i][0].record(stream)
        one_step(i, evs[i])
        step_ev[i][1].record(stream)
    torch.cuda.synchronize()
    total_ms = sum(a.elapsed_time(b) for a, b in step_ev)
    # the same steps back to back on one draw (inputs partly L2-resident across steps)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for i in range(steps):
        one_step(i)
    e1.record(stream)
    torch.cuda.synchronize()
    warm_ms = e0.elapsed_time(e1)
    for lin in lins:
        if asp.qwam_asp_get_error(lin.h) != asp.QWAM_OK:
            raise RuntimeError("device error in the sweep")
    flops = sum(2.0 * L.M * L.N * L.K for L in W.layers) * steps
    # per call: the slower of the algorithmic bytes over HBM (X, packed W and its scales, U, B_hat,
    # the bf16 Y) and the flops over the MMA kind's peak
    t_roof = 0.0
    for L, lin in zip(W.layers, lins):
        w_bytes = L.N * L.K // 2 + (L.N * L.K // 16 if nv else 2 * L.N * L.K // L.G)
        by = 2 * L.M * L.K + w_bytes + 2 * L.K * lin.r_pad + 2 * L.N * lin.r_pad + 2 * L.M * L.N
        t_roof += max(by / (hbm_peak * 1e9), 2.0 * L.M * L.N * L.K / (mma_peak * 1e12))
    t_roof *= steps
    kinds = {}
    for j, L in enumerate(W.layers):
        key = "%s_r%d" % (L.name.split("_", 1)[1], L.r)
        t = sum(evs[i][2 * j].elapsed_time(evs[i][2 * j + 1]) for i in range(steps))
        k = kinds.setdefault(key, [0.0, 0.0, 0])
        k[0] += t
        k[1] += 2.0 * L.M * L.N * L.K * steps
        k[2] += steps
    for lin in lins:
        lin.close()
    value = flops / (total_ms * 1e-3) / 1e12
    return {"value": value, "unit": UNIT, "steps": steps,
            "ms_per_denoising_step": total_ms / steps, "layers_per_step": len(W.layers),
            "inputs": "fresh activations drawn before every step, L2 flushed before every step, steps timed alone",
            "l2_warm": {"value": flops / (warm_ms * 1e-3) / 1e12, "ms_per_denoising_step": warm_ms / steps,
                        "inputs": "one activation draw, steps back to back"},
            "roofline": {"bound": "tensor", "achieved": value, "peak": mma_peak, "unit": "TFLOP/s",
                         "frac": value / mma_peak, "traffic": None, "peak_source": peak_source},
            "layer_roofline_frac": t_roof * 1e3 / total_ms,
            "asp_blocks": W.note, "what": "30 DiT blocks x {qkv, o, up, down} at M = 4096, r = 32 on a third "
            "of the blocks, r = 0 elsewhere; one qwam_asp_linear per layer; device-drawn synthetic data",
            "by_layer": {k: {"us_per_call": round(v[0] / v[2] * 1e3, 1), "tops": round(v[1] / (v[0] * 1e-3) / 1e12, 1)}
                         for k, v in sorted(kinds.items())}}


def run_ours(args):
    import torch
    rank, world, local = dist_env()
    torch.cuda.set_device(local)
    init_dist(world, "nccl")
    dev = torch.device("cuda", local)

    from paper_2609_33269_gb300 import asp, build
    from paper_2609_33269_gb300 import workloads as wl
    build.build()
    asp.load()
    peaks = {}
    try:
        peaks = json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json")))
    except Exception:
        pass
    hbm_peak = peaks.get("hbm_gbs", 6800.0)
    bf16_peak = peaks.get("bf16_tflops", 1900.0)
    f16_peak = bf16_peak        # the INT4 GEMM's MMA kind (kind::f16) runs at the bf16 dense rate
    fp8_peak = 2.0 * bf16_peak  # dense fp8 = 2x dense bf16 (nominal 4.5 / 2.25 PFLOP/s)

    fp4_peak = 6.0 * bf16_peak  # dense fp4 = 6x dense bf16 (nominal 13.5 / 2.25 PFLOP/s)

    layer_def = wl.dit_attention().layers[0]
    M, K, N, r, G = layer_def.M, layer_def.K, layer_def.N, layer_def.r, layer_def.G
    Xb = layer_def.x()
    Wb = layer_def.w()
    U = layer_def.u()

    def dev_bf16(bits):
        return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).to(dev).view(torch.bfloat16)

    W = dev_bf16(Wb)
    Ud = torch.from_numpy(U).to(dev)
    X0 = dev_bf16(Xb)
    stream = torch.cuda.current_stream(dev)
    flops = 2.0 * M * N * K

    def timed(fmt, nsteps, warmup, clocks=None, smooth=None):
        """The layer through qwam_asp_linear (the public call) for `nsteps` timed steps over
        rotating sets (weights packed per set, activations, workspaces, outputs), after `warmup`
        untimed steps; then, outside the timed region, the split of a step into its two calls
        (qwam_asp_quantize_act, qwam_asp_gemm) from CUDA events around each, over up to 200
        steps.  `smooth`: pack rotated layers (Eq. (pair)) with these smoothing factors."""
        sets = []
        for i in range(ROTATE_SETS):
            if smooth is None:
                lin = asp.AspLinear(W, Ud, G, fmt=fmt)
            else:
                lin = asp.AspLinear(W, Ud, G, fmt=fmt, rotate=True, s=smooth)
            X = X0 if i == 0 else X0.clone()
            sets.append((lin, X, lin.workspace(M), torch.empty((M, N), dtype=torch.bfloat16, device=dev)))
        mb = ROTATE_SETS * (2 * M * K + 2 * M * N + lin_ws_bytes(sets[0][0], M) + N * K // 2) / 1e6

        def check(where):
            for lin_, *_ in sets:
                st = asp.qwam_asp_get_error(lin_.h)
                if st != asp.QWAM_OK:
                    raise RuntimeError(f"device error {where}: {asp.status_string(st)}")

        for i in range(warmup):
            lin, X, ws, Y = sets[i % ROTATE_SETS]
            asp.qwam_asp_linear(X, M, lin.h, Y, asp.QWAM_Y_BF16, ws, stream)
        torch.cuda.synchronize()
        check("after warm-up")
        if clocks is not None:
            clocks.start()
            time.sleep(0.3)
        barrier(world)
        torch.cuda.synchronize()
        if clocks is not None:
            clocks.mark("t0")
        start = torch.cuda.Event(enable_timing=True)
        end = torch.cuda.Event(enable_timing=True)
        start.record(stream)
        for i in range(nsteps):
            lin, X, ws, Y = sets[i % ROTATE_SETS]
            asp.qwam_asp_linear(X, M, lin.h, Y, asp.QWAM_Y_BF16, ws, stream)
        end.record(stream)
        torch.cuda.synchronize()
        if clocks is not None:
            clocks.mark("t1")
        barrier(world)
        if clocks is not None:
            clocks.stop()
        total_ms = start.elapsed_time(end)
        check("in the timed region")
        total_ms = max_over_ranks(total_ms, world, dev)
        # the split of a step into its two calls (the GEMM call includes the float16 weight
        # expansion); CUDA events between the calls keep the two from overlapping, so this pass
        # is slightly slower than the timed region
        nsplit = min(nsteps, 200)
        for i in range(3):
            lin, X, ws, Y = sets[i % ROTATE_SETS]
            asp.qwam_asp_quantize_act(X, M, lin.h, ws, stream)
            asp.qwam_asp_gemm(ws, M, lin.h, Y, asp.QWAM_Y_BF16, stream)
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(3 * nsplit)]
        torch.cuda.synchronize()
        for i in range(nsplit):
            lin, X, ws, Y = sets[i % ROTATE_SETS]
            ev[3 * i].record(stream)
            asp.qwam_asp_quantize_act(X, M, lin.h, ws, stream)
            ev[3 * i + 1].record(stream)
            asp.qwam_asp_gemm(ws, M, lin.h, Y, asp.QWAM_Y_BF16, stream)
            ev[3 * i + 2].record(stream)
        torch.cuda.synchronize()
        t_a = sum(ev[3 * i].elapsed_time(ev[3 * i + 1]) for i in range(nsplit)) / nsplit
        t_b = sum(ev[3 * i + 1].elapsed_time(ev[3 * i + 2]) for i in range(nsplit)) / nsplit
        check("in the split pass")
        return dict(sets=sets, total_ms=total_ms, t_a=t_a, t_b=t_b, mb=mb,
                    value=aggregate_value(flops, nsteps, world, total_ms))

    def rooflines(fmt, t_a, t_b, step_ms, r_pad):
        """Per-kernel achieved vs peak, the dominant kernel's roofline object and the layer's
        roofline fraction (slower of the algorithmic bytes over HBM and the MMA kind's peak)."""
        nv = fmt == asp.QWAM_FMT_NVFP4
        a_bytes = alg_bytes_actquant(M, K, r_pad, G, nv)
        peak, pname = (fp4_peak, "fp4") if nv else (f16_peak, "f16")
        gname = "gemm_nvfp4" if nv else "gemm_w4a4_lr"
        kern = {
            "actquant": {"ms": t_a, "bound": "hbm", "alg_bytes": a_bytes,
                         "achieved_gbs": a_bytes / (t_a * 1e-3) / 1e9, "peak_gbs": hbm_peak},
            gname: {"ms": t_b, "bound": "tensor", "alg_flops": flops,
                    "achieved_tflops": flops / (t_b * 1e-3) / 1e12, f"peak_tflops_{pname}": peak},
        }
        kern["actquant"]["frac"] = kern["actquant"]["achieved_gbs"] / hbm_peak
        # what kernel (a) moves: the algorithmic bytes (4-bit codes written packed, as counted),
        # plus, with r > 0, its second pass over X (re-read from L2 after the projection)
        moved = a_bytes + (2 * M * K if r_pad > 0 else 0)
        kern["actquant"].update(moved_bytes=moved, achieved_gbs_of_moved_bytes=moved / (t_a * 1e-3) / 1e9,
                                moved_note="second pass over X served from L2" if r_pad > 0 else "one pass")
        kern[gname]["frac"] = kern[gname]["achieved_tflops"] / peak
        if not nv:  # the same rate against faster MMA kinds, for context
            kern[gname]["frac_of_fp8_peak"] = kern[gname]["achieved_tflops"] / fp8_peak
            kern[gname]["frac_of_fp4_peak"] = kern[gname]["achieved_tflops"] / fp4_peak
        if t_b >= t_a:
            roof = {"kernel": gname, "bound": "tensor", "achieved": kern[gname]["achieved_tflops"],
                    "peak": peak, "unit": "TFLOP/s", "frac": kern[gname]["frac"],
                    "traffic": kernel_traffic("gemm_nvfp4_kernel" if nv else "gemm16_kernel"),
                    "peak_source": ("measured bf16 burst x 6 (nominal fp4/bf16 dense ratio), of measured" if nv else
                                    "measured bf16 burst (the kernel's MMA kind, kind::f16), of measured")}
        else:
            roof = {"kernel": "actquant", "bound": "hbm", "achieved": kern["actquant"]["achieved_gbs"],
                    "peak": hbm_peak, "unit": "GB/s", "frac": kern["actquant"]["frac"],
                    "traffic": kernel_traffic("actquant_kernel_nvfp4" if nv else "actquant_kernel"),
                    "peak_source": "measured HBM copy, of measured"}
        w_bytes = N * K // 2 + (N * K // 16 if nv else 2 * N * K // G)
        t_roof = max((2 * M * K + w_bytes + 2 * K * r_pad + 2 * N * r_pad + 2 * M * N) / (hbm_peak * 1e9),
                     flops / (peak * 1e12))
        return kern, roof, (t_roof * 1e3) / step_ms

    fmt = asp.QWAM_FMT_NVFP4 if args.format == "nvfp4" else asp.QWAM_FMT_INT4
    nsteps = args.steps
    # smoothing factors (alpha = 0.5, from this batch's channel maxima) for the rotated layer
    xmax = X0.float().abs().amax(dim=0).contiguous()
    smooth = torch.empty(K, dtype=torch.float32, device=dev)
    asp.qwam_asp_smoothing_factors(xmax, W, K, N, 0.5, smooth, stream)
    clocks = ClockSampler(local)
    main_run = timed(fmt, nsteps, args.warmup, clocks, smooth=smooth if args.rotate else None)
    sets, total_ms, t_a, t_b = main_run["sets"], main_run["total_ms"], main_run["t_a"], main_run["t_b"]
    value = main_run["value"]
    working_mb = main_run["mb"]
    # the first rows' codes, scales and output, for the oracle comparison in the CPU baseline
    gpu_par = None
    if not args.no_cpu_baseline and world == 1 and not args.rotate:
        gpu_par = gpu_sample(sets[0][0], sets[0][1], M, 512, fmt == asp.QWAM_FMT_NVFP4)

    # End to end through the public API, as a serving loop would run it: every step copies its
    # activations from pinned host memory to the device, runs the layer (qwam_asp_linear) and
    # copies the output back to pinned host memory.  The copies run on their own streams with
    # double-buffered device inputs and outputs, so step i's layer overlaps the input copy of
    # step i + 1 and the output copy of step i - 1; events order each buffer's reuse.
    Xh = torch.from_numpy(np.ascontiguousarray(Xb).view(np.int16)).view(torch.bfloat16).pin_memory()
    Yh = torch.empty((M, N), dtype=torch.bfloat16).pin_memory()
    lin, _, ws, _ = sets[0]
    Xd2 = [torch.empty((M, K), dtype=torch.bfloat16, device=dev) for _ in range(2)]
    Yd2 = [torch.empty((M, N), dtype=torch.bfloat16, device=dev) for _ in range(2)]
    s_in, s_out = torch.cuda.Stream(dev), torch.cuda.Stream(dev)
    e2e_steps = max(3, min(nsteps, 200))

    def e2e_run(n):
        h2d = [torch.cuda.Event() for _ in range(n)]
        comp = [torch.cuda.Event() for _ in range(n)]
        d2h = [torch.cuda.Event() for _ in range(n)]
        for i in range(n):
            b = i % 2
            if i >= 2:
                s_in.wait_event(comp[i - 2])      # X buffer b no longer read by step i - 2
            with torch.cuda.stream(s_in):
                Xd2[b].copy_(Xh, non_blocking=True)
            h2d[i].record(s_in)
            stream.wait_event(h2d[i])
            if i >= 2:
                stream.wait_event(d2h[i - 2])     # Y buffer b already copied out by step i - 2
            lin(Xd2[b], out=Yd2[b], stream=stream)
            comp[i].record(stream)
            s_out.wait_event(comp[i])
            with torch.cuda.stream(s_out):
                Yh.copy_(Yd2[b], non_blocking=True)
            d2h[i].record(s_out)

    e2e_run(3)
    torch.cuda.synchronize()
    barrier(world)
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(s_in)
    e2e_run(e2e_steps)
    s_out.wait_stream(s_in)
    s_out.wait_stream(stream)
    e1.record(s_out)
    torch.cuda.synchronize()
    e2e_ms = max_over_ranks(e0.elapsed_time(e1), world, dev)
    e2e_value = aggregate_value(flops, e2e_steps, world, e2e_ms)

    r_pad = sets[0][0].r_pad
    kern, roof, layer_frac = rooflines(fmt, t_a, t_b, total_ms / nsteps, r_pad)
    variants = {}
    if fmt == asp.QWAM_FMT_INT4 and not args.rotate:
        for lin_, *_ in sets:
            lin_.close()
        sets = []
        vsteps = max(3, min(nsteps, 500))
        vr = timed(asp.QWAM_FMT_NVFP4, vsteps, max(3, min(args.warmup, 20)))
        vk, vroof, vfrac = rooflines(asp.QWAM_FMT_NVFP4, vr["t_a"], vr["t_b"], vr["total_ms"] / vsteps, r_pad)
        variants["nvfp4"] = {"value": vr["value"], "unit": UNIT, "steps": vsteps,
                             "ms_per_step": vr["total_ms"] / vsteps, "dtype": "e2m1",
                             "format": "NVFP4 (App. B.1): E2M1, E4M3 scale per 16 K, float32 per-tensor weight scale",
                             "roofline": vroof, "layer_roofline_frac": vfrac, "kernels": vk}
        for s_ in vr["sets"]:
            s_[0].close()
        variants["small_m"] = small_m_latencies(asp, wl, dev, stream, dev_bf16)
        variants["sweep_int4"] = denoise_sweep(asp, wl, dev, stream, asp.QWAM_FMT_INT4, 10, hbm_peak, f16_peak,
                                               "measured bf16 burst (the GEMM's MMA kind, kind::f16), of measured")
        variants["sweep_nvfp4"] = denoise_sweep(asp, wl, dev, stream, asp.QWAM_FMT_NVFP4, 10, hbm_peak, fp4_peak,
                                                "measured bf16 burst x 6 (nominal fp4/bf16 dense ratio), of measured")
        # Smoothing and the block Hadamard rotation (B = 1024) in front of the same layer: kernel (a)
        # writes the float32 remainder, the rotation kernel rotates and quantizes it (two launches
        # in qwam_asp_quantize_act).
        rr = timed(asp.QWAM_FMT_INT4, vsteps, max(3, min(args.warmup, 20)), smooth=smooth)
        a_fused = alg_bytes_actquant(M, K, r_pad, G)
        a_split = a_fused + 4 * M * K * 2 + 4 * K  # the float32 remainder written and read back, 1/s
        variants["rotated_int4"] = {
            "value": rr["value"], "unit": UNIT, "steps": vsteps, "ms_per_step": rr["total_ms"] / vsteps,
            "what": "smoothing (alpha 0.5) + block Hadamard (B 1024) in front of the INT4 layer (Eq. (pair))",
            "act_path_ms": rr["t_a"], "gemm_ms": rr["t_b"],
            "act_path_gbs_of_fused_bytes": a_fused / (rr["t_a"] * 1e-3) / 1e9,
            "act_path_gbs_of_moved_bytes": a_split / (rr["t_a"] * 1e-3) / 1e9, "peak_gbs": hbm_peak,
            "launches_per_step": 3}
        for s_ in rr["sets"]:
            s_[0].close()

    if rank != 0:
        return 0
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": nsteps, "warmup": args.warmup,
        "ms_per_step": total_ms / nsteps, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "e2m1" if fmt == asp.QWAM_FMT_NVFP4 else "f16", "data": "synthetic",
        "config": dict(WORKLOAD, parallelism=f"replicas by token rows x{world}",
                       format="nvfp4 (block 16)" if fmt == asp.QWAM_FMT_NVFP4 else "int4 (group 64)",
                       l2="rotating buffers: %d sets, %.0f MB > L2" % (ROTATE_SETS, working_mb),
                       **({"rotation": ROTATION} if args.rotate else {})),
        "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": 2 * M * K, "d2h_bytes_per_step": 2 * M * N,
                "steps": e2e_steps,
                "pipeline": "copies on their own streams, overlapping the layer of the neighbouring steps"},
        # per qwam_asp_linear call: kernel (a) and the GEMM, the rotation kernel of a rotated layer
        # with r > 0, and the float16 weight expansion of an INT4 layer of 512 or more tokens as a
        # launch of its own when r = 0 (with r > 0 kernel (a) does it)
        "gpu_launches": (2 + (1 if args.rotate and r > 0 else 0)
                         + (1 if fmt == asp.QWAM_FMT_INT4 and M >= 512 and r == 0 else 0)) * nsteps,
        "roofline": roof,
        "layer_roofline_frac": layer_frac,
        "kernels": kern,
        "variants": variants,
        "clocks": clocks.summary(),
    }
    if not args.no_cpu_baseline and world == 1:
        line["cpu_baseline"] = cpu_baseline(args.cpu_rows, fmt == asp.QWAM_FMT_NVFP4, args.rotate, gpu_par)
    print(json.dumps(line))
    for s_ in sets:
        s_[0].close()
    return 0


def gpu_sample(lin, X, M, rows, nvfp4):
    """The GPU's codes, scales and float32 output for the first `rows` token rows of X (one
    untimed call), decoded to the oracle's layouts: INT4 codes from OB4 words (word j holds
    k = 8j..8j+7 as nibbles c + 8: k = 8j + 2p in bits 4p.., k = 8j + 2p + 1 in bits 16 + 4p..)
    and bfloat16 scales, NVFP4 E2M1 codes two per byte (low nibble first) and block scales from
    the 512-byte atoms."""
    import torch
    Y = lin(X, fp32=True)
    torch.cuda.synchronize()
    out = {"Y": Y[:rows].cpu().numpy().astype(np.float64)}
    if nvfp4:
        codes, atoms, _ = lin.act_views_nvfp4(M)
        p = codes[:rows].cpu().numpy()
        q = np.empty((rows, p.shape[1] * 2), np.uint8)
        q[:, 0::2], q[:, 1::2] = p & 0xF, p >> 4
        a = atoms.cpu().numpy()
        K = q.shape[1]
        rr = np.arange(rows)[:, None]
        b = np.arange(K // 16)[None, :]
        out["qx"] = q
        out["sfx"] = a[((rr // 128) * (K // 64) + b // 4) * 512 + (rr % 32) * 16 + ((rr % 128) // 32) * 4 + b % 4]
    else:
        codes, scales, _ = lin.act_views(M)
        w = np.ascontiguousarray(codes[:rows].cpu().numpy()).view("<u4")
        q = np.empty((rows, w.shape[1], 8), np.int8)
        for p in range(4):
            q[:, :, 2 * p] = ((w >> (4 * p)) & 0xF).astype(np.int16) - 8
            q[:, :, 2 * p + 1] = ((w >> (16 + 4 * p)) & 0xF).astype(np.int16) - 8
        out["qx"] = q.reshape(rows, -1)
        out["sx"] = scales.float().cpu().numpy()[:, :rows].T.copy()
    return out


def lin_ws_bytes(lin, M):
    from paper_2609_33269_gb300 import asp
    return asp.qwam_asp_act_workspace_bytes(lin.h, M)


def main():
    args = parse()
    if args.impl == "reference":
        return run_reference(args)
    return run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
