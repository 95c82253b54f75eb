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
    p.add_argument("--workload", default="cfg4", choices=["cfg4", "cfg2", "cfg1", "fwht", "profile"],
                   help="fwht: the INT8 transform+requantize pass alone on the config-4 ga2 input; "
                        "profile: the range-expansion profiling pass on the same tensor")
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
                                          "--format=csv,noheader,nounits", "-lms", "200"],
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
        plan = C.plan_chain(ch)
        preps = O.prepare_chain(ch.layers, params, scales[ch.name], plan, ch.out_f32)
        t0 = time.perf_counter()
        O.chain_forward(ch.layers, preps, plan, x, ch.input_kind, ch.s_in)
        t_total += time.perf_counter() - t0
        ops += 2 * sub.macs()
        if ch.name == "analysis":
            frac_img = (h * w) / (ch.h * ch.w)
    return t_total, frac_img, ops, threads


def run_reference(args, cfg, scales):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    for _ in range(args.warmup if args.warmup < 1 else 1):
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


def run_fwht_mode(args):
    """The INT8-entry transform + requantize pass (hb 64) on an NHWC tensor
    shaped like the config-4 ga2 input: 1 byte read + 1 byte written per element."""
    import torch
    from paper_2608_01653_gb300 import hatq as H
    H.load()
    shape = (args.batch, 1080, 1920, 192)
    x = torch.from_numpy(I.uniform_codes(shape, seed=9)).cuda()
    y = torch.empty_like(x)
    ms = time_events(lambda: H.quantize_act(x, H.IN_I8, 0.05, 64, 0.07, y=y), args.steps, args.warmup)
    H.sync_status()
    nbytes = 2 * x.numel()
    peaks = json.load(open(PEAKS)) if os.path.exists(PEAKS) else {}
    peak = peaks.get("hbm_gbs", FALLBACK_HBM_GBS)
    gbs = nbytes / (ms / 1000) / 1e9
    print(json.dumps({"mode": "fwht", "shape": list(shape), "hb": 64, "ms": ms, "GB/s": gbs, "peak_hbm_gbs": peak,
                      "frac": gbs / peak}), flush=True)


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
    cfg, scales = workload_chains("cfg4" if args.workload in ("cfg4", "fwht", "profile") else args.workload)
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

    # conv launches of one step with their algorithmic flops, timed by event pairs
    def step(record=None):
        for c in chains:
            chain, ch = c["chain"], c["spec"]
            kinds = chain.input_kinds(c["kind"], ch.s_in)
            cur = c["x_dev"]
            n, h, w = ch.n, ch.h, ch.w
            for i, (P, L) in enumerate(zip(chain.prepared, ch.layers)):
                k, s_in = kinds[i]
                if H.layer_launches(k, s_in, P) > 1:
                    hb = L.hb_in if L.form == "DH" else 1
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
                    record.append((e0, e1, 2 * L.macs(n, h, w)))
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
    conv_ms = sum(e0.elapsed_time(e1) for e0, e1, _ in records)
    conv_flops = sum(f for _, _, f in records)
    n_conv = len(records)

    # --- end to end through the public API with host buffers
    e2e = None
    if not args.no_e2e:
        def e2e_step():
            for c in chains:
                c["x_dev"].copy_(c["x_pin"], non_blocking=True)
                c["chain"].forward(c["x_dev"], c["kind"], c["spec"].s_in, c["outs"], c["scratch"])
                c["out_pin"].copy_(c["outs"][-1], non_blocking=True)
        for _ in range(2):
            e2e_step()
        torch.cuda.synchronize()
        if dist:
            dist.barrier()
        s0 = torch.cuda.Event(enable_timing=True)
        s1 = torch.cuda.Event(enable_timing=True)
        s0.record(stream)
        for _ in range(args.steps):
            e2e_step()
        s1.record(stream)
        torch.cuda.synchronize()
        e2e_ms = job_step_time(s0.elapsed_time(s1) / args.steps, dist, dev)
        H.sync_status()
        h2d = sum(c["x_pin"].numel() * c["x_pin"].element_size() for c in chains)
        d2h = sum(c["out_pin"].numel() * c["out_pin"].element_size() for c in chains)
        e2e = {"value": job_throughput(images_step, world, e2e_ms), "unit": "images/s", "h2d_bytes_per_step": h2d,
               "d2h_bytes_per_step": d2h, "ms_per_step": e2e_ms}

    if rank != 0:
        if dist:
            dist.destroy_process_group()
        return

    peaks = json.load(open(PEAKS)) if os.path.exists(PEAKS) else {}
    peak = peaks.get("bf16_tflops_sustained")
    peak_src = "measured bf16 sustained (fp16 operands run at the bf16 rate)"
    if peak is None:
        peak, peak_src = FALLBACK_BF16_TFLOPS, "fallback bf16"
    achieved = conv_flops / (conv_ms / 1000.0) / 1e12
    traffic = None
    prof = os.path.join(ROOT, "profiles", "conv_cfg4_traffic.json")
    if os.path.exists(prof):
        traffic = json.load(open(prof)).get("dram_bytes_per_launch")
    roofline = {"bound": "tensor", "achieved": achieved, "peak": peak, "unit": "TFLOP/s", "frac": achieved / peak,
                "traffic": traffic, "kernel": "hatq conv_kernel (tcgen05 kind::f16, exact INT8)",
                "launches": n_conv, "avg_launch_ms": conv_ms / max(n_conv, 1), "peak_source": peak_src}

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
        "roofline": roofline, "cpu_baseline": cpu, "e2e": e2e, "clocks": clocks,
        "gpu_launches": launches_step * args.steps,
    }
    print(json.dumps(line), flush=True)
    if dist:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
