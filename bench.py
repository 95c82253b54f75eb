"""Throughput benchmark of the Hadamard-domain INT8 convolution stack.

Workload (default): the LIC analysis chain (3->192->192->192->320, 5x5 s2,
WH first layer then DH) and the entropy-model chains (hyperprior
320->640->640->640 plus 8 channel-context slices 32->224->128->32, seeded 30%
WH mask) at batch 8 on 3840x2160 images (latent 240x135), INT8 NHWC
integer-only path, synthetic seeded inputs, random-init weights, scales from
the oracle calibration of the same chains.

One step = one pass of every layer of every chain over one batch of 8 images
(activation transform + quantize where needed, implicit-GEMM conv, fused
requantize/Hadamard epilogue). Prints one JSON line (rank 0).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference]

Under torchrun each rank runs its own batch (replicas, weak scaling); the
ranks meet only at the timing barrier.
"""
from __future__ import annotations

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

from synth import configs as C  # noqa: E402
from synth import inputs as I  # noqa: E402

METRIC = "HaTQ INT8 conv effective TOPS and images/sec (1 GB300); % of INT8 tensor/HBM roofline"
CALIB = os.path.join(ROOT, "tests", "golden", "calibration.json")
PEAKS = os.path.join(ROOT, "MEASURED_PEAKS.json")
FALLBACK_BF16_TFLOPS = 1900.0
FALLBACK_HBM_GBS = 6800.0
# Integer issue capacity of a GB300 for integer-only code: one warp instruction per clock per SM
# sub-partition split between the half-rate ALU and FMA-heavy pipes, 152 SMs x 4 x 32 lanes x 2.07 GHz
INT_OPS_PEAK = 152 * 4 * 32 * 2.07e9


def epilogue_int_ops(L, hb_next):
    """Integer operations per output value of the exact requantize epilogue:
    conversion, bias, 64-bit multiply (3), the ReLU on 64 bits (3), the
    round-half-even shift with clamp (7), packing (1), and two 32-bit
    operations per value for each stage of each int64 Sylvester transform."""
    import math
    hb_out = L.hb_out if L.form == "WH" else 0
    ops = 11 + (3 if L.act == "relu" else 0)
    for hb in (hb_out, hb_next):
        if hb:
            ops += 2 * int(math.log2(hb))
    return ops
CPU_SAMPLE_HW = (1024, 1536)      # bounded oracle sample: one 1536x1024 crop of image 0 (~10-15 s)
CPU_SAMPLE_LATENT = (64, 96)
REF_SAMPLE_HW = (512, 768)        # per step of --impl reference (~3 s), so K steps end within minutes
REF_SAMPLE_LATENT = (32, 48)


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=10)
    p.add_argument("--warmup", type=int, default=3)
    p.add_argument("--impl", default="ours", choices=["ours", "reference"])
    p.add_argument("--workload", default="cfg4",
                   choices=["cfg4", "cfg2", "cfg1", "fwht", "profile", "int8mm", "orders", "decoder", "affine", "gdn"],
                   help="fwht: the INT8 transform+requantize pass alone on the config-4 ga2 input; "
                        "profile: the range-expansion profiling pass on the same tensor; "
                        "int8mm: torch._int_mm 8192^3, the library INT8 GEMM as a reference point; "
                        "orders: the paper's order-192 transform layer and ga2 in that basis at batch 8; "
                        "decoder: a synthesis-side transposed 5x5 s2 layer and a sub-pixel layer at batch 8; "
                        "affine: ga2 with dynamic affine (PTQ) activations at batch 8")
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--no-cpu", action="store_true")
    p.add_argument("--layer", default="", help="time one layer of the config-4 chains (e.g. ga2, h1, s0a)")
    p.add_argument("--batch", type=int, default=8, help="batch for --layer / the FWHT pass")
    p.add_argument("--act", default=None, choices=["none", "relu", "silu", "gelu"],
                   help="--layer: time the layer with this activation instead of its own")
    return p.parse_args()


def workload_chains(name):
    cfg = C.CONFIGS[name]
    calib = json.load(open(CALIB))["configs"]
    scales = {}
    for ch in cfg.chains:
        src = "cfg2" if ch.name == "analysis" else ("cfg3" if name == "cfg4" else name)
        if name in ("cfg1", "cfg2"):
            src = name
        scales[ch.name] = calib[src][ch.name]
    return cfg, scales


def macs_of(chain):
    return chain.macs()


# ------------------------------------------------------------------ clocks

class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.proc = None
        self.path = None

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "50"],
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
        rows = []
        for line in open(self.path):
            parts = [x.strip() for x in line.split(",")]
            if len(parts) >= 9:
                rows.append(parts)
        os.unlink(self.path)
        if not rows:
            return None

        def num(v):
            try:
                return float(v)
            except ValueError:
                return None
        sm = [num(r[1]) for r in rows if num(r[1]) is not None]
        smax = max((num(r[2]) for r in rows if num(r[2]) is not None), default=None)
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i].lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": smax, "reasons": reasons,
                "samples": len(rows), "power_w_max": max((num(r[3]) or 0.0) for r in rows)}


# ------------------------------------------------------------------ oracle (CPU baseline / reference arm)

def oracle_sample(cfg, scales, threads=None, hw=CPU_SAMPLE_HW, latent=CPU_SAMPLE_LATENT):
    """Runs the oracle as it stands on a bounded crop of the same workload and
    returns (seconds, images-equivalent, algorithmic ops, threads)."""
    from oracle import hatq_oracle as O
    if threads:
        O.set_threads(threads)
    threads = O.max_threads()
    t_total, frac_img, ops = 0.0, 0.0, 0
    for ch in cfg.chains:
        if ch.name == "analysis":
            h, w = hw if cfg.name == "cfg4" else (ch.h, ch.w)
        else:
            h, w = latent if cfg.name == "cfg4" else (ch.h, ch.w)
        sub = ch.with_batch(1, h, w, ch.input_seed)
        x = C.chain_input(sub)
        params = C.chain_params(ch)
        preps = O.prepare_chain(ch.layers, params, scales[ch.name], ch.out_f32)
        t0 = time.perf_counter()
        O.chain_forward(ch.layers, preps, x, ch.input_kind, ch.s_in)
        t_total += time.perf_counter() - t0
        ops += 2 * sub.macs()
        if ch.name == "analysis":
            frac_img = (h * w) / (ch.h * ch.w)
    return t_total, frac_img, ops, threads


def run_reference(args, cfg, scales):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    for _ in range(args.warmup):
        oracle_sample(cfg, scales, hw=REF_SAMPLE_HW, latent=REF_SAMPLE_LATENT)
    times = []
    frac = ops = threads = None
    for _ in range(args.steps):
        t, frac, ops, threads = oracle_sample(cfg, scales, hw=REF_SAMPLE_HW, latent=REF_SAMPLE_LATENT)
        times.append(t)
    t = sum(times) / len(times)
    value = frac / t
    sample = (f"oracle (numpy fp64/int64 + C direct conv, OpenMP {threads} threads) on one "
              f"{REF_SAMPLE_HW[1]}x{REF_SAMPLE_HW[0]} crop of image 0 and the matching "
              f"{REF_SAMPLE_LATENT[1]}x{REF_SAMPLE_LATENT[0]} latent crop for every chain, "
              f"scaled to full 3840x2160 images")
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "images/s", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1000 * t, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "int64", "data": "synthetic",
            "effective_tops": ops / t / 1e12,
            "config": {"workload": workload_name(cfg), "global_batch": 8},
            "cpu_baseline": {"value": value, "unit": "images/s", "cores": threads, "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": "images/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def replica_seed(base_seed: int, rank: int) -> int:
    """Input seed of one replica: every rank draws its own batch of images."""
    return base_seed + 7919 * rank


def job_step_time(local_ms: float, dist=None, device=None) -> float:
    """Step time of the whole job: the maximum over ranks (all-reduce MAX)."""
    if dist is None:
        return local_ms
    import torch
    t = torch.tensor([float(local_ms)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(images_per_rank: int, world: int, step_ms: float) -> float:
    """Whole-job images/s: the images all ranks processed over the slowest rank's step."""
    return world * images_per_rank / (step_ms / 1000.0)


def workload_name(cfg):
    if cfg.name == "cfg4":
        return ("cfg4: LIC analysis chain 3->192->192->192->320 (5x5 s2, WH,DH,DH,DH) + hyperprior "
                "320->640->640->640 + 8 context slices 32->224->128->32 (seeded 30% WH mask), batch 8, "
                "3840x2160, INT8 integer-only")
    return f"{cfg.name}: {cfg.description}"


# ------------------------------------------------------------------ single-kernel modes

def time_events(fn, steps, warmup):
    import torch
    for _ in range(max(3, warmup)):
        fn()
    torch.cuda.synchronize()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(steps):
        fn()
    e1.record()
    torch.cuda.synchronize()
    return e0.elapsed_time(e1) / steps


def run_layer_mode(args, cfg, scales):
    """One conv layer of the config-4 chains on a synthetic INT8 operand."""
    import torch
    from paper_2608_01653_gb300 import hatq as H
    H.load()
    for ch in cfg.chains:
        for i, L in enumerate(ch.layers):
            if L.name == args.layer:
                n, h, w = ch.with_batch(args.batch, ch.h, ch.w, 0).shapes()[i]
                params = C.chain_params(ch)[i]
                hb_next = C.plan_chain(ch)[i]
                sc = scales[ch.name][i]
                act = args.act or L.act
                if act in H.GENERAL_ACTS:
                    # same layer through the general transition; the calibrated output scale
                    # stands in for s_z and s_u (timing only: the table's values do not
                    # change the work)
                    if max(L.hb_out if L.form == "WH" else 0, hb_next) > 64:
                        raise SystemExit(f"layer {L.name}: the general transition covers blocks up to 64")
                    P = H.prepare_weights(H.desc_from_spec(L), params[0], params[1], sc["s_x"], sc["s_out"], act,
                                          hb_next, s_z=sc["s_out"], s_u=sc["s_out"])
                else:
                    P = H.prepare_weights(H.desc_from_spec(L), params[0], params[1], sc["s_x"], sc["s_out"], act,
                                          hb_next, False)
                x = torch.from_numpy(I.activations_i8((n, h, w, L.c_in), seed=5, s_in=0.05)).cuda()
                y = torch.empty(P.out_shape(n, h, w), dtype=torch.int8, device="cuda")
                ms = time_events(lambda: H.conv2d_i8(x, P, y=y), args.steps, args.warmup)
                H.sync_status()
                flops = 2 * L.macs(n, h, w)
                peaks = json.load(open(PEAKS)) if os.path.exists(PEAKS) else {}
                peak = peaks.get("bf16_tflops", FALLBACK_BF16_TFLOPS)
                tf = flops / (ms / 1000) / 1e12
                print(json.dumps({"mode": "layer", "layer": L.name, "act": act, "chain": ch.name, "batch": n,
                                  "in_hw": [h, w],
                                  "c_in": L.c_in, "c_out": L.c_out, "k": L.k, "stride": L.stride, "form": L.form,
                                  "hb_next": hb_next, "ms": ms, "tflops": tf, "peak_bf16_burst": peak,
                                  "frac": tf / peak}), flush=True)
                return
    raise SystemExit(f"unknown layer {args.layer}")


def conv_source_sha() -> str:
    """sha256 prefix of the conv kernel's sources (the kernel file and the
    device-helper header it includes), the key of committed counter captures."""
    import hashlib
    h = hashlib.sha256()
    for f in ("hatq_conv.cu", "hatq_conv_pieces.cu", "hatq_tc.h"):
        h.update(open(os.path.join(ROOT, "paper_2608_01653_gb300", "csrc", f), "rb").read())
    return h.hexdigest()[:16]


def fwht_pass(batch, steps, warmup, device="cuda"):
    """The INT8-entry transform + requantize pass (hb 64) on an NHWC tensor
    shaped like the config-4 ga2 input (8 x 1080 x 1920 x 192 at batch 8,
    3.2 GB, larger than L2): 1 byte read + 1 byte written per element. Returns
    (ms per pass, algorithmic bytes per pass, shape)."""
    import torch
    from paper_2608_01653_gb300 import hatq as H
    shape = (batch, 1080, 1920, 192)
    g = torch.Generator(device=device)
    g.manual_seed(9)
    x = torch.randint(-127, 128, shape, dtype=torch.int8, device=device, generator=g)
    y = torch.empty_like(x)
    ms = time_events(lambda: H.quantize_act(x, H.IN_I8, 0.05, 64, 0.07, y=y), steps, warmup)
    H.sync_status()
    return ms, 2 * x.numel(), shape


def run_fwht_mode(args):
    """The transform + quantize pass (hb 64) on the ga2-shaped tensor in its
    three modes: INT8 entry with a static scale (the benchmark's pass), INT8
    entry with the dynamic per-tensor scale (max-abs pass, parameter kernel,
    quantize pass: 3 B/element read + written), FP16 entry with a static scale
    (fp16 read, codes written: 3 B/element)."""
    import torch
    from paper_2608_01653_gb300 import hatq as H
    H.load()
    ms, nbytes, shape = fwht_pass(args.batch, args.steps, args.warmup)
    peaks = json.load(open(PEAKS)) if os.path.exists(PEAKS) else {}
    peak = peaks.get("hbm_gbs", FALLBACK_HBM_GBS)
    gbs = nbytes / (ms / 1000) / 1e9
    g = torch.Generator(device="cuda")
    g.manual_seed(10)
    x = torch.randint(-127, 128, shape, dtype=torch.int8, device="cuda", generator=g)
    y = torch.empty_like(x)
    s_used = torch.empty(1, dtype=torch.float32, device="cuda")
    ws = torch.empty(64, dtype=torch.uint8, device="cuda")
    d_ms = time_events(lambda: H.quantize_act(x, H.IN_I8, 0.05, 64, 0.0, y=y, s_used=s_used, workspace=ws),
                       args.steps, args.warmup)
    del x
    xf = torch.randn(shape, device="cuda", generator=g).to(torch.float16)
    f_ms = time_events(lambda: H.quantize_act(xf, H.IN_F16, 1.0, 64, 0.05, y=y), args.steps, args.warmup)
    H.sync_status()
    n = y.numel()
    print(json.dumps({"mode": "fwht", "shape": list(shape), "hb": 64, "ms": ms, "GB/s": gbs, "peak_hbm_gbs": peak,
                      "frac": gbs / peak,
                      "i8_dynamic": {"ms": d_ms, "GB/s": 3 * n / (d_ms / 1000) / 1e9,
                                     "frac": 3 * n / (d_ms / 1000) / 1e9 / peak},
                      "f16_static": {"ms": f_ms, "GB/s": 3 * n / (f_ms / 1000) / 1e9,
                                     "frac": 3 * n / (f_ms / 1000) / 1e9 / peak}}), flush=True)


def run_orders_mode(args, cfg, scales):
    """The paper's single order on the config-4 ga2 layer: the activation-side
    transform into the Paley-I order 192 as a 1x1 tensor-core layer on the
    8 x 1080 x 1920 x 192 INT8 input, then ga2 (5x5 s2, 192 -> 192) prepared
    in that basis. CUDA events, inputs larger than L2."""
    import torch
    from paper_2608_01653_gb300 import hatq as H
    H.load()
    ch = cfg.chains[0]
    L = ch.layers[1]
    n, h, w = ch.shapes()[1]
    g = torch.Generator(device="cuda")
    g.manual_seed(11)
    x = torch.randint(-127, 128, (n, h, w, L.c_in), dtype=torch.int8, device="cuda", generator=g)
    sc = scales[ch.name][1]
    T = H.prepare_order_transform(L.c_in, 0.05, sc["s_x"])
    m = T.c_out
    op = torch.empty((n, h, w, m), dtype=torch.int8, device="cuda")
    w_, b_ = C.chain_params(ch)[1]
    P = H.prepare_weights_order(H.make_desc(L.c_in, L.c_out, L.k, L.stride, L.pad, "DH"), w_, b_, sc["s_x"],
                                sc["s_out"], L.act, 0)
    y = torch.empty(P.out_shape(n, h, w), dtype=torch.int8, device="cuda")
    t_ms = time_events(lambda: H.conv2d_i8(x, T, y=op), args.steps, args.warmup)
    c_ms = time_events(lambda: H.conv2d_i8(op, P, y=y), args.steps, args.warmup)
    H.sync_status()
    peaks = json.load(open(PEAKS)) if os.path.exists(PEAKS) else {}
    tc, hbm = peaks.get("bf16_tflops", FALLBACK_BF16_TFLOPS), peaks.get("hbm_gbs", FALLBACK_HBM_GBS)
    t_flops, t_bytes = 2 * n * h * w * L.c_in * m, n * h * w * (L.c_in + m) + m * L.c_in
    ho, wo = L.out_hw(h, w)
    c_flops = 2 * n * ho * wo * L.c_out * L.k * L.k * L.c_in
    print(json.dumps({
        "mode": "orders", "order": m, "construction": "Paley-I q = %d" % (m - 1), "batch": n, "in_hw": [h, w],
        "transform": {"ms": t_ms, "tflops": t_flops / (t_ms / 1000) / 1e12, "gbs": t_bytes / (t_ms / 1000) / 1e9,
                      "bound": "hbm" if t_bytes / hbm / 1e9 > t_flops / tc / 1e12 else "tensor",
                      "frac": max(t_bytes / (hbm * 1e9), t_flops / (tc * 1e12)) * 1000 / t_ms},
        "ga2_order": {"ms": c_ms, "tflops": c_flops / (c_ms / 1000) / 1e12,
                      "frac": c_flops / (tc * 1e12) * 1000 / c_ms},
        "peaks": {"bf16_tflops": tc, "hbm_gbs": hbm}}), flush=True)


def run_decoder_mode(args):
    """Decoder-side operators at the config-4 latent size (batch 8): a
    synthesis transposed convolution 320 -> 192 (5x5, stride 2, pad 2, output
    padding 1, WH 64 output block, ReLU) on the 8 x 135 x 240 latent, and a
    sub-pixel layer 192 -> 768 (3x3, DH 64, ReLU) with factor 2 on its
    8 x 270 x 480 output. Random INT8 operands, CUDA events."""
    import torch
    from paper_2608_01653_gb300 import hatq as H
    H.load()
    peaks = json.load(open(PEAKS)) if os.path.exists(PEAKS) else {}
    tc = peaks.get("bf16_tflops", FALLBACK_BF16_TFLOPS)
    g = torch.Generator(device="cuda")
    g.manual_seed(13)
    n, h, w = 8, 135, 240
    Lt = C.layer("gs1", 320, 192, 5, 2, 2, "WH", "relu", hb_out=64)
    T = H.prepare_weights_transposed(H.desc_from_spec(Lt), 1, I.weights(192, 5, 5, 320, 31), I.bias(192, 32), 0.1,
                                     0.05, "relu", 0)
    x = torch.randint(-127, 128, (n, h, w, 320), dtype=torch.int8, device="cuda", generator=g)
    y = torch.empty(T.out_shape(n, h, w), dtype=torch.int8, device="cuda")
    t_ms = time_events(lambda: H.conv_transpose2d_i8(x, T, y=y), args.steps, args.warmup)
    _, ho, wo, _ = y.shape
    t_flops = 2 * n * h * w * 320 * 192 * 25                   # every input pixel meets every tap once
    Ls = C.layer("gs2", 192, 768, 3, 1, 1, "DH", "relu", hb_in=64)
    P = H.prepare_weights(H.desc_from_spec(Ls), I.weights(768, 3, 3, 192, 33), I.bias(768, 34), 0.1, 0.05, "relu", 0)
    z = torch.empty((n, ho * 2, wo * 2, 192), dtype=torch.int8, device="cuda")
    s_ms = time_events(lambda: H.conv2d_i8_subpixel(y, P, 2, y=z), args.steps, args.warmup)
    H.sync_status()
    s_flops = 2 * n * ho * wo * 768 * 9 * 192
    print(json.dumps({
        "mode": "decoder", "batch": n,
        "transposed": {"layer": "320->192 5x5 s2 p2 q1 WH64 ReLU", "in_hw": [h, w], "out_hw": [ho, wo], "ms": t_ms,
                       "tflops": t_flops / (t_ms / 1000) / 1e12, "frac": t_flops / (tc * 1e12) * 1000 / t_ms},
        "subpixel": {"layer": "192->768 3x3 DH64 ReLU, r = 2", "in_hw": [ho, wo], "out_hw": [2 * ho, 2 * wo],
                     "ms": s_ms, "tflops": s_flops / (s_ms / 1000) / 1e12, "frac": s_flops / (tc * 1e12) * 1000 / s_ms},
        "peak_bf16_burst": tc}), flush=True)


def run_gdn_mode(args):
    """A GDN analysis layer at the config-4 ga2 output size (batch 8): ga2
    (5x5 s2, 192 -> 192, DH 64) emitting the integer preactivation z, then
    the GDN transition (pool on the tensor cores, phi_int, the next layer's
    DH 64 input transition) on the 8 x 540 x 960 x 192 codes. Random INT8
    operands, seeded beta / gamma of GDN's usual shape (beta ~ 1, small
    non-negative gamma), CUDA events."""
    import torch
    from paper_2608_01653_gb300 import hatq as H
    H.load()
    peaks = json.load(open(PEAKS)) if os.path.exists(PEAKS) else {}
    tc, hbm = peaks.get("bf16_tflops", FALLBACK_BF16_TFLOPS), peaks.get("hbm_gbs", FALLBACK_HBM_GBS)
    n, h, w, c = 8, 1080, 1920, 192
    g = torch.Generator(device="cuda")
    g.manual_seed(19)
    rng = np.random.default_rng(19)
    beta, gamma = 0.5 + rng.random(c), np.abs(rng.standard_normal((c, c))) * 0.01
    L = C.layer("ga2", 192, 192, 5, 2, 2, "DH", "none", hb_in=64)
    P = H.prepare_weights(H.desc_from_spec(L), I.weights(192, 5, 5, 192, 2001), I.bias(192, 2051), 0.1, 0.05, "none", 0)
    G = H.prepare_gdn(c, beta, gamma, 0.05, 0.02, False, 0.05, 64)
    x = torch.randint(-127, 128, (n, h, w, c), dtype=torch.int8, device="cuda", generator=g)
    z = torch.empty(P.out_shape(n, h, w), dtype=torch.int8, device="cuda")
    y = torch.empty_like(z)
    c_ms = time_events(lambda: H.conv2d_i8(x, P, y=z), args.steps, args.warmup)
    g_ms = time_events(lambda: H.gdn(z, G, y=y), args.steps, args.warmup)
    H.sync_status()
    pix = z.numel() // c
    g_bytes = 2 * z.numel()                                   # z read, x written
    g_flops = 2 * 2 * pix * c * c                             # two limbs of the pool contraction
    c_flops = 2 * pix * c * 25 * c
    print(json.dumps({
        "mode": "gdn", "batch": n, "z_shape": list(z.shape),
        "conv": {"layer": "ga2 192->192 5x5 s2 DH64, emits z", "ms": c_ms,
                 "tflops": c_flops / (c_ms / 1000) / 1e12, "frac": c_flops / (tc * 1e12) * 1000 / c_ms},
        "gdn": {"ms": g_ms, "Mpixel_per_s": pix / (g_ms / 1000) / 1e6,
                "hbm_gbs": g_bytes / (g_ms / 1000) / 1e9, "hbm_frac": g_bytes / (g_ms / 1000) / 1e9 / hbm,
                "pool_tflops": g_flops / (g_ms / 1000) / 1e12, "tensor_frac": g_flops / (g_ms / 1000) / 1e12 / tc},
        "peak_bf16_burst": tc, "peak_hbm_gbs": hbm}), flush=True)


def run_affine_mode(args):
    """ga2 (5x5 s2, 192 -> 192, DH 64) with dynamic affine activations at
    batch 8 on the 1080 x 1920 fp16 input: the range + quantize passes
    (fp16 in, centred int16 out) and the convolution on the centred codes."""
    import torch
    from paper_2608_01653_gb300 import hatq as H
    H.load()
    peaks = json.load(open(PEAKS)) if os.path.exists(PEAKS) else {}
    tc, hbm = peaks.get("bf16_tflops", FALLBACK_BF16_TFLOPS), peaks.get("hbm_gbs", FALLBACK_HBM_GBS)
    n, h, w = 8, 1080, 1920
    g = torch.Generator(device="cuda")
    g.manual_seed(17)
    x = (torch.randn((n, h, w, 192), device="cuda", generator=g) + 0.5).to(torch.float16)
    codes = torch.empty((n, h, w, 192), dtype=torch.int16, device="cuda")
    params = torch.empty(2, dtype=torch.float32, device="cuda")
    ws = torch.empty(64, dtype=torch.uint8, device="cuda")
    L = C.layer("ga2", 192, 192, 5, 2, 2, "DH", "relu", hb_in=64)
    P = H.prepare_weights_affine(H.desc_from_spec(L), I.weights(192, 5, 5, 192, 2001), I.bias(192, 2051), "relu")
    y = torch.empty(P.out_shape(n, h, w), dtype=torch.float32, device="cuda")
    q_ms = time_events(lambda: H.quantize_act_affine(x, 64, y=codes, params=params, workspace=ws), args.steps,
                       args.warmup)
    c_ms = time_events(lambda: H.conv2d_affine(codes, P, params, y=y), args.steps, args.warmup)
    H.sync_status()
    q_bytes = x.numel() * (2 + 2 + 2)                         # fp16 read twice (range, quantize) + int16 write
    ho, wo = L.out_hw(h, w)
    c_flops = 2 * n * ho * wo * 192 * 25 * 192
    print(json.dumps({"mode": "affine", "batch": n, "in_hw": [h, w],
                      "quantize": {"ms": q_ms, "gbs": q_bytes / (q_ms / 1000) / 1e9,
                                   "frac": q_bytes / (hbm * 1e9) * 1000 / q_ms},
                      "conv": {"ms": c_ms, "tflops": c_flops / (c_ms / 1000) / 1e12,
                               "frac": c_flops / (tc * 1e12) * 1000 / c_ms}}), flush=True)


def run_int8mm_mode(args):
    """torch._int_mm (the library INT8 GEMM, int32 output) on 8192^3, CUDA
    events: the measured INT8 tensor-core reference point of this GPU."""
    import torch
    n = 8192
    a = torch.randint(-127, 128, (n, n), dtype=torch.int8, device="cuda")
    b = torch.randint(-127, 128, (n, n), dtype=torch.int8, device="cuda")
    ms = time_events(lambda: torch._int_mm(a, b), args.steps, args.warmup)
    af = a.to(torch.float16)
    bf = b.to(torch.float16)
    ms16 = time_events(lambda: torch.matmul(af, bf), args.steps, args.warmup)
    print(json.dumps({"mode": "int8mm", "n": n, "int8_ms": ms, "int8_tops": 2 * n ** 3 / (ms / 1000) / 1e12,
                      "f16_ms": ms16, "f16_tflops": 2 * n ** 3 / (ms16 / 1000) / 1e12}), flush=True)


def run_profile_mode(args):
    """The range-expansion profiling pass (Eq. hadamard_sensitivity, hb 64) over
    a batch shaped like the config-4 ga2 input: 1 byte read per element."""
    import torch
    from paper_2608_01653_gb300 import hatq as H
    H.load()
    shape = (args.batch, 1080, 1920, 192)
    x = torch.from_numpy(I.uniform_codes(shape, seed=9)).cuda()
    ms = time_events(lambda: H.profile_range(x, 64), args.steps, args.warmup)
    H.sync_status()
    nbytes = x.numel()
    peaks = json.load(open(PEAKS)) if os.path.exists(PEAKS) else {}
    peak = peaks.get("hbm_gbs", FALLBACK_HBM_GBS)
    gbs = nbytes / (ms / 1000) / 1e9
    print(json.dumps({"mode": "profile", "shape": list(shape), "hb": 64, "ms": ms, "GB/s": gbs,
                      "peak_hbm_gbs": peak, "frac": gbs / peak}), flush=True)


# ------------------------------------------------------------------ GPU arm

def main():
    args = parse()
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    cfg, scales = workload_chains("cfg4" if args.workload in ("cfg4", "fwht", "profile", "int8mm", "orders", "decoder",
                                                              "affine", "gdn") else args.workload)
    if args.impl == "reference":
        run_reference(args, cfg, scales)
        return
    if args.layer:
        run_layer_mode(args, cfg, scales)
        return
    if args.workload == "fwht":
        run_fwht_mode(args)
        return
    if args.workload == "profile":
        run_profile_mode(args)
        return
    if args.workload == "int8mm":
        run_int8mm_mode(args)
        return
    if args.workload == "orders":
        run_orders_mode(args, cfg, scales)
        return
    if args.workload == "decoder":
        run_decoder_mode(args)
        return
    if args.workload == "gdn":
        run_gdn_mode(args)
        return
    if args.workload == "affine":
        run_affine_mode(args)
        return

    import torch
    from paper_2608_01653_gb300 import hatq as H
    from paper_2608_01653_gb300.chain import Chain
    torch.cuda.set_device(local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    H.load()
    dev = torch.device("cuda", local)

    # --- setup (untimed): weights, inputs, buffers
    chains = []
    for ch in cfg.chains:
        params = C.chain_params(ch)
        plan = C.plan_chain(ch)
        chain = Chain(ch.layers, params, scales[ch.name], plan, ch.out_f32, device=dev)
        kind = H.IN_F16 if ch.input_kind == "f16" else H.IN_I8
        x_host = C.chain_input(ch.with_batch(ch.n, ch.h, ch.w, replica_seed(ch.input_seed, rank)))
        x_pin = torch.from_numpy(x_host).pin_memory()
        x_dev = x_pin.to(dev)
        outs, scratch = chain.alloc(ch.n, ch.h, ch.w, dev)
        chains.append(dict(spec=ch, chain=chain, kind=kind, x_pin=x_pin, x_dev=x_dev, outs=outs,
                           scratch=scratch, out_pin=torch.empty(outs[-1].shape, dtype=outs[-1].dtype).pin_memory()))
    stream = torch.cuda.current_stream(dev)
    macs_step = sum(c["spec"].macs() for c in chains)
    images_step = cfg.images

    # conv launches of one step, each timed by an event pair on the launching stream
    def step(record=None):
        for ci, c in enumerate(chains):
            chain, ch = c["chain"], c["spec"]
            kinds = chain.input_kinds(c["kind"], ch.s_in)
            cur = c["x_dev"]
            n, h, w = ch.n, ch.h, ch.w
            for i, P in enumerate(chain.prepared):
                k, s_in = kinds[i]
                if H.layer_launches(k, s_in, P) > 1:
                    hb = ch.layers[i].hb_in if ch.layers[i].form == "DH" else 1
                    op = c["scratch"][: n * h * w * P.c_in].view(n, h, w, P.c_in)
                    H.quantize_act(cur, k, s_in, hb, P.s_x, y=op)
                    cur = op
                if record is not None:
                    e0 = torch.cuda.Event(enable_timing=True)
                    e1 = torch.cuda.Event(enable_timing=True)
                    e0.record(stream)
                H.conv2d_i8(cur, P, y=c["outs"][i])
                if record is not None:
                    e1.record(stream)
                    record.append((ci, i, e0, e1))
                cur = c["outs"][i]
                _, h, w, _ = c["outs"][i].shape

    launches_step = sum(c["chain"].launches(c["kind"], c["spec"].s_in) for c in chains)

    for _ in range(max(3, args.warmup)):
        step()
    H.sync_status()
    torch.cuda.synchronize()

    sampler = ClockSampler(local)
    sampler.start()
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    records = []
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    t0.record(stream)
    for _ in range(args.steps):
        step(records)
    t1.record(stream)
    torch.cuda.synchronize()
    ms = job_step_time(t0.elapsed_time(t1) / args.steps, dist, dev)
    if dist:
        dist.barrier()
    clocks = sampler.stop()
    H.sync_status()

    peaks = json.load(open(PEAKS)) if os.path.exists(PEAKS) else {}
    tc_peak, tc_src = peaks.get("bf16_tflops"), "measured bf16 burst (fp16 operands run at the bf16 rate)"
    if tc_peak is None:
        tc_peak, tc_src = FALLBACK_BF16_TFLOPS, "fallback bf16"
    hbm_peak, hbm_src = peaks.get("hbm_gbs"), "measured HBM copy"
    if hbm_peak is None:
        hbm_peak, hbm_src = FALLBACK_HBM_GBS, "fallback HBM"

    # per layer: algorithmic flops (2 MACs of the unpadded reduction) and bytes
    # (INT8 input + INT8 output + INT8 weights, each once); its roofline is the
    # larger of the tensor-core and the HBM time
    per_layer = {}
    for ci, i, e0, e1 in records:
        per_layer.setdefault((ci, i), []).append(e0.elapsed_time(e1))
    layers = []
    for (ci, i), times in sorted(per_layer.items()):
        ch = chains[ci]["spec"]
        L = ch.layers[i]
        n, h, w = ch.shapes()[i]
        ho, wo = L.out_hw(h, w)
        flops = 2 * L.macs(n, h, w)
        nbytes = n * h * w * L.c_in + n * ho * wo * L.c_out + L.c_out * L.k * L.k * L.c_in
        lms = sum(times) / len(times)
        int_ops = n * ho * wo * L.c_out * epilogue_int_ops(L, chains[ci]["chain"].plan[i])
        t_tc, t_hbm, t_int = flops / (tc_peak * 1e12), nbytes / (hbm_peak * 1e9), int_ops / INT_OPS_PEAK
        bound = max((t_tc, "tensor"), (t_hbm, "hbm"), (t_int, "alu"))[1]
        layers.append({"layer": L.name, "chain": ch.name, "ms": lms, "bound": bound,
                       "tflops": flops / (lms / 1000) / 1e12, "gbs": nbytes / (lms / 1000) / 1e9,
                       "int_tops": int_ops / (lms / 1000) / 1e12,
                       "flops": flops, "bytes": nbytes, "int_ops": int_ops,
                       "frac": max(t_tc, t_hbm, t_int) * 1000 / lms})
    conv_ms = sum(x["ms"] for x in layers)
    conv_flops = sum(x["flops"] for x in layers)
    n_conv = len(layers)
    achieved = conv_flops / (conv_ms / 1000.0) / 1e12
    traffic = None
    prof = os.path.join(ROOT, "profiles", "conv_cfg4_traffic.json")
    if os.path.exists(prof):
        # the captured counters stand for the kernel source they were taken on, and for no later one
        rec = json.load(open(prof))
        if conv_source_sha() == rec.get("kernel_source_sha256_16"):
            traffic = rec.get("dram_bytes_per_launch")
    roofline_peaks = {"tensor_tflops": tc_peak, "hbm_gbs": hbm_peak, "int_tops": INT_OPS_PEAK / 1e12,
                      "int_source": "derived: 152 SMs x 4 sub-partitions x 32 lanes x 2.07 GHz (half-rate ALU + "
                                    "FMA-heavy integer pipes)"}
    roofline = {"bound": "tensor", "achieved": achieved, "peak": tc_peak, "unit": "TFLOP/s", "frac": achieved / tc_peak,
                "traffic": traffic, "kernel": "hatq conv_kernel (tcgen05 kind::f16, exact INT8)",
                "launches": n_conv, "avg_launch_ms": conv_ms / max(n_conv, 1), "peak_source": tc_src,
                "note": "all conv launches of the step; per-layer bounds in roofline_layers"}

    # the INT8-entry transform + requantize pass on the config-4 ga2-shaped input (not part of the step:
    # every transition inside a chain is fused into its producer)
    f_ms, f_bytes, f_shape = fwht_pass(8, max(5, args.steps), 3, dev)
    roofline_fwht = {"bound": "hbm", "achieved": f_bytes / (f_ms / 1000) / 1e9, "peak": hbm_peak, "unit": "GB/s",
                     "frac": f_bytes / (f_ms / 1000) / 1e9 / hbm_peak, "ms": f_ms, "bytes": f_bytes,
                     "shape": list(f_shape), "hb": 64, "peak_source": hbm_src,
                     "kernel": "hatq act_quant_i8_swar_kernel (INT8 entry, two 16-bit lanes per word, 32-bit requantization)"}

    # --- end to end through the public API (Chain.forward) with pinned host buffers: every step copies its
    # inputs in and its chain outputs back. Two input and two output slots per chain; copies run on their own
    # streams (host-to-device and device-to-host each on its own, so neither waits behind the other), and
    # step k's copies overlap the compute of steps k - 1 and k + 1.
    e2e = None
    if not args.no_e2e:
        in_stream = torch.cuda.Stream(dev)
        out_stream = torch.cuda.Stream(dev)
        for c in chains:
            c["x_slots"] = [c["x_dev"], torch.empty_like(c["x_dev"])]
            c["y_slots"] = [c["outs"][-1], torch.empty_like(c["outs"][-1])]
            c["out_pins"] = [c["out_pin"], torch.empty_like(c["out_pin"]).pin_memory()]
        ev = lambda: torch.cuda.Event()  # noqa: E731
        x_free = [ev(), ev()]
        y_free = [ev(), ev()]
        for e in x_free + y_free:
            e.record(stream)

        def e2e_steps(k_steps):
            for k in range(k_steps):
                sl = k % 2
                loaded = ev()
                with torch.cuda.stream(in_stream):
                    in_stream.wait_event(x_free[sl])
                    for c in chains:
                        c["x_slots"][sl].copy_(c["x_pin"], non_blocking=True)
                    loaded.record(in_stream)
                stream.wait_event(loaded)
                stream.wait_event(y_free[sl])
                for c in chains:
                    outs = c["outs"][:-1] + [c["y_slots"][sl]]
                    c["chain"].forward(c["x_slots"][sl], c["kind"], c["spec"].s_in, outs, c["scratch"], stream)
                done = ev()
                done.record(stream)
                x_free[sl] = done
                with torch.cuda.stream(out_stream):
                    out_stream.wait_event(done)
                    for c in chains:
                        c["out_pins"][sl].copy_(c["y_slots"][sl], non_blocking=True)
                    fin = ev()
                    fin.record(out_stream)
                y_free[sl] = fin
        e2e_steps(2)
        torch.cuda.synchronize()
        if dist:
            dist.barrier()
        s0 = torch.cuda.Event(enable_timing=True)
        s1 = torch.cuda.Event(enable_timing=True)
        s0.record(stream)
        in_stream.wait_stream(stream)
        out_stream.wait_stream(stream)
        e2e_steps(args.steps)
        stream.wait_stream(in_stream)
        stream.wait_stream(out_stream)
        s1.record(stream)
        torch.cuda.synchronize()
        e2e_ms = job_step_time(s0.elapsed_time(s1) / args.steps, dist, dev)
        H.sync_status()
        h2d = sum(c["x_pin"].numel() * c["x_pin"].element_size() for c in chains)
        d2h = sum(c["out_pin"].numel() * c["out_pin"].element_size() for c in chains)
        e2e = {"value": job_throughput(images_step, world, e2e_ms), "unit": "images/s", "h2d_bytes_per_step": h2d,
               "d2h_bytes_per_step": d2h, "ms_per_step": e2e_ms,
               "api": "Chain.forward -> hatq_layer (C ABI); H2D and D2H on their own streams, double-buffered"}

    if rank != 0:
        if dist:
            dist.destroy_process_group()
        return

    cpu = None
    if not args.no_cpu and world >= 1:
        try:
            t, frac, ops, threads = oracle_sample(cfg, scales)
            cpu = {"value": frac / t, "unit": "images/s", "cores": threads, "kind": "oracle",
                   "sample": (f"oracle as it stands on one {CPU_SAMPLE_HW[1]}x{CPU_SAMPLE_HW[0]} crop of image 0 "
                              f"plus {CPU_SAMPLE_LATENT[1]}x{CPU_SAMPLE_LATENT[0]} latent crops for every chain "
                              f"({t:.1f} s, {ops / 1e9:.1f} GOP), scaled to 3840x2160 images"),
                   "effective_tops": ops / t / 1e12}
        except Exception as ex:  # the oracle is a reported baseline only
            cpu = {"value": None, "unit": "images/s", "cores": None, "kind": "oracle", "sample": f"failed: {ex}"}

    value = job_throughput(images_step, world, ms)
    line = {
        "metric": METRIC, "value": value, "unit": "images/s", "n_gpus": world, "steps": args.steps,
        "warmup": max(3, args.warmup), "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "int8",
        "arithmetic": "INT8 codes as exact fp16 tensor-core operands, fp32 chunk sums below 2^24, int32 totals, "
                      "int64 requantization",
        "data": "synthetic (seeded LIC-shaped inputs, random-init weights)",
        "effective_tops": world * 2 * macs_step / (ms / 1000.0) / 1e12,
        "config": {"workload": workload_name(cfg), "global_batch": world * images_step,
                   "parallelism": f"replicas x{world}", "l2": "inputs larger than L2 (199 MB image batch)"},
        "roofline": roofline, "roofline_layers": layers, "roofline_peaks": roofline_peaks,
        "roofline_fwht": roofline_fwht,
        "cpu_baseline": cpu, "e2e": e2e, "clocks": clocks,
        "gpu_launches": launches_step * args.steps,
    }
    print(json.dumps(line), flush=True)
    if dist:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
