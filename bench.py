"""Throughput of the fully binary BMLP training rule (arXiv 2412.00119) on GB300.

Workload (default): the 8192 -> 8192 x4 -> 10 throughput-stress network, bs 100,
trained on a seeded 1,000,000-sample stream of i.i.d. +-1 inputs labelled by a
+-1 teacher 8192 -> 1024 -> 10.  One bench step = one bmlp_train call over
100,000 consecutive samples (1,000 mini-batches: forward, local classifiers,
selection, CP + R + repack of every layer); every 10th step closes the epoch
(p_r rescale), so ten steps are one pass over the stream.  The stream (1 GB
packed) and the model state (256 MiB of hidden weights, bit-sliced at one
byte per weight for h_max = 255) are far larger than L2, so no flush is needed
between steps.

Printed (rank 0, one JSON line): samples/s over all ranks, XNOR-popcount
Gbop/s, the roofline of the dominant kernel measured live with CUDA events on
a sample of the timed mini-batches, the whole training step against its
roofline (HBM bytes the step touches and the forward's bit-pairs at the peak
of the engine that runs them), the oracle's CPU throughput on a bounded
sample, the end-to-end number through the C-ABI with host (pinned) buffers,
SM clocks sampled during the timed region, the forward-only evaluation sweep
(65,536 samples at batch 65,536), the comparison of the units that can run
the forward contraction (peaks and one 8192 x 8192 layer at 100 and 65,536
patterns), and the same figures for the four other workloads.

--impl reference times the CPU oracle (plain C, all host cores) on the same
workload, one 100-sample mini-batch per step.

Multi-GPU (torchrun): every rank trains an independent replica (model seed +
rank) on the same stream -- the paper's "realizations of the initial
conditions" -- with no collective on the data path; the value is the sum over
ranks (weak scaling) and the time the max over ranks.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import workloads as W  # noqa: E402

CONFIG_KEY = "C5"
SAMPLES_PER_STEP = 100_000
STEPS_PER_EPOCH = 10
EVAL_BATCH = 65_536
# sampled mini-batches for the per-kernel figures: one in 100, i.e. 10 per
# step of 1,000 mini-batches (a sampled mini-batch runs kernel by kernel
# between CUDA events instead of inside the captured graphs)
PROFILE_EVERY = 100
# the other workloads: oracle mini-batches timed for their CPU baseline
CONFIG_ORACLE_MINIBATCHES = {"C1": 20, "C2": 10, "C3": 4, "C4": 2}

# HBM traffic of one k_update_ws launch of the timed region, from an ncu
# capture of this bench (dram__bytes_read.sum + dram__bytes_write.sum, one
# pass; see profiles/k_update_ws_c5.md), valid while the kernel sources hash to
# UPDATE_TRAFFIC_SRC_SHA; otherwise reported as null.
UPDATE_TRAFFIC_BYTES = 262_359_808 + 179_019_776  # dram read + write of one timed-region launch (ncu)
UPDATE_TRAFFIC_SRC_SHA = "5de9071d4dacc413"
UPDATE_SOURCES = ("kern_update_ws.cu", "update_common.cuh")
# The same for one 8192 -> 8192 k_forward_eval_tc launch at 65,536 patterns
# (profiles/k_forward_eval_tc_c5eval.md), keyed to the kernel and its shared
# tcgen05 header.  Part of the 67 MB output is still in the write-back L2 when
# the launch ends, so the write figure is below the output's size.
EVAL_TRAFFIC_BYTES = 75_599_360 + 32_936_448
EVAL_TRAFFIC_SRC_SHA = "f8b34ceea49eb88e"
# The same for one 8192 -> 8192 k_train_forward_tc launch at bs 100 (a layer
# >= 2; profiles/k_train_forward_tc_c5.md): the layer's 8 MiB of visible
# weights and the activation words read, z and the sign bits still in the
# write-back L2 when the launch ends.
FWD_TRAFFIC_BYTES = 8_560_384 + 0
FWD_TRAFFIC_SRC_SHA = "63ee748cad5467c0"


def bitpairs_per_sample(widths, classes):
    """Forward XNOR bit-pairs per pattern: sum_l K_l (K_{l-1} + c) (Table 3)."""
    return sum(widths[l] * (widths[l - 1] + classes) for l in range(1, len(widths)))


def forward_weight_bytes(widths):
    """Packed visible weights the forward passes of one mini-batch read."""
    return sum(widths[l] * ((widths[l - 1] + 63) // 64) * 8 for l in range(1, len(widths)))


def step_roofline(ms_per_mb, upd_bytes_per_mb, widths, classes, hbm_gbs, mac_peak, popc_peak,
                  engine):
    """The whole training step (one mini-batch of 100) against its roofline:
    HBM bytes = what the update touched (H of the rows with a CP tuple read and
    written, their W rows written, the sparse reinforcement events of the
    other rows; counted by the kernel) + the packed weights the forward reads;
    compute = the forward's bit-pairs at the peak of the engine that runs
    them.  t_roof = max(HBM time, compute time); frac = t_roof / measured.
    The same step against the CUDA-core popcount peak is reported beside it."""
    nbytes = upd_bytes_per_mb + forward_weight_bytes(widths)
    bp = 100 * bitpairs_per_sample(widths, classes)
    t_meas = ms_per_mb * 1e-3
    t_hbm = nbytes / (hbm_gbs * 1e9)
    t_cmp = bp / mac_peak
    t_popc = bp / popc_peak
    t_roof = max(t_hbm, t_cmp)
    return {"bound": "hbm" if t_hbm >= t_cmp else engine, "frac": t_roof / t_meas,
            "us_measured": t_meas * 1e6, "us_roof": t_roof * 1e6, "hbm_bytes": nbytes,
            "us_hbm": t_hbm * 1e6, "us_compute": t_cmp * 1e6, "engine": engine,
            "achieved_gbs": nbytes / t_meas / 1e9, "peak_gbs": hbm_gbs,
            "vs_popcount_peak": {"us_popc": t_popc * 1e6,
                                 "frac": max(t_hbm, t_popc) / t_meas}}


def hidden_planes(h_max):
    """Bit-planes stored per group of 32 hidden weights: the bits of h_max
    rounded up to a power of two."""
    nbits = max(1, int(h_max).bit_length())
    p = 1
    while p < nbits:
        p *= 2
    return p


def update_bytes_per_launch(widths, h_max=255):
    """Algorithmic HBM bytes of one update launch (all layers active): the
    bit-sliced H of every row read and written (rows padded to 16 bytes),
    the packed W row written."""
    b = 0
    for l in range(1, len(widths)):
        ngrp = (widths[l - 1] + 31) // 32
        ldh = (ngrp * hidden_planes(h_max) + 3) // 4 * 4
        nw = (widths[l - 1] + 63) // 64
        b += widths[l] * (2 * 4 * ldh + nw * 8)
    return b


def peaks():
    """(HBM GB/s, SM max MHz, bf16 TFLOP/s burst, bf16 TFLOP/s sustained, source)."""
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return (d.get("hbm_gbs", 6800.0), d.get("sm_max_mhz", 2070.0), d.get("bf16_tflops", 1900.0),
                d.get("bf16_tflops_sustained", 1700.0), "measured")
    except OSError:
        return 6800.0, 2070.0, 1900.0, 1700.0, "fallback"


# dense fp8 (e4m3) / bf16 tensor throughput, nominal (4.5 / 2.25 PFLOP/s)
FP8_PER_BF16 = 2.0


def popc_peak_bitpairs(sm_mhz, sms=152, popc_per_clk=16):
    """CUDA-core popcount peak: SMs x 16 POPC results/clock/SM x 32 bit-pairs."""
    return sms * popc_per_clk * 32 * sm_mhz * 1e6


def src_sha(*names):
    h = hashlib.sha256()
    for n in names:
        with open(os.path.join(ROOT, "paper_2412_00119_gb300", "csrc", n), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


# -- distributed helpers (also exercised by the gloo tests) ----------------------

def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def replica_seed(base_seed, rank):
    return base_seed + rank


def max_over_ranks(value, device=None):
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()):
        return value
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def sum_over_ranks(value, device=None):
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()):
        return value
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.SUM)
    return float(t.item())


def barrier():
    import torch.distributed as dist
    if dist.is_available() and dist.is_initialized():
        dist.barrier()


# -- clocks ------------------------------------------------------------------------

class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.idx = gpu_index
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.idx), "--query-gpu=" + self.FIELDS,
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
        return self

    def __exit__(self, *exc):
        self.lines = []
        if self.proc is not None:
            self.proc.terminate()
            try:
                out, _ = self.proc.communicate(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
                out, _ = self.proc.communicate()
            self.lines = [ln for ln in out.splitlines() if ln.strip()]
        return False

    def summary(self):
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in getattr(self, "lines", []):
            p = [v.strip() for v in ln.split(",")]
            if len(p) < 9:
                continue
            try:
                sm.append(float(p[1]))
                mx = float(p[2])
            except ValueError:
                continue
            for name, v in zip(names, p[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(name)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": mx,
                "reasons": sorted(reasons), "samples": len(sm)}


# -- workload ----------------------------------------------------------------------

def make_stream(cfg, n, device):
    import torch
    xp = W.make_inputs(cfg, "train", n)
    xd = torch.from_numpy(xp.view(np.int64)).to(device)
    yd = W.teacher_labels_packed_torch(W.make_teacher(cfg), xd, cfg.widths[0], chunk=16384)
    return xp, xd, yd


def cpu_baseline(cfg, x_pm1, y, threads):
    """The oracle, as it stands, on one 100-sample mini-batch of the stream."""
    import oracle as O
    cores = O.set_threads(threads)
    m = O.OracleModel(list(cfg.widths), cfg.classes, seed=cfg.model_seed, bs=100)
    t0 = time.perf_counter()
    m.train(x_pm1[:100], y[:100])
    dt = time.perf_counter() - t0
    m.close()
    return {"value": 100.0 / dt, "unit": "samples/s", "cores": cores, "kind": "oracle",
            "sample": "1 mini-batch (100 samples) of the 8192->8192x4->10 stream, "
                      "forward + local classifiers + selection + CP + R of all 4 layers",
            "seconds": dt}


def run_reference(args):
    """--impl reference: the CPU oracle on the host cores, same config/metric."""
    rank, world, _ = dist_env()
    if rank != 0:
        return 0
    import oracle as O
    cfg = W.CONFIGS[CONFIG_KEY]
    threads = os.cpu_count() or 1
    cores = O.set_threads(threads)
    n = 100 * (args.steps + args.warmup)
    xp = W.make_inputs(cfg, "train", n)
    xpm = W.unpack(xp, cfg.widths[0])
    y = W.teacher_labels_pm1(W.make_teacher(cfg), xpm)
    m = O.OracleModel(list(cfg.widths), cfg.classes, seed=cfg.model_seed, bs=100)
    for s in range(args.warmup):
        m.train(xpm[100 * s:100 * s + 100], y[100 * s:100 * s + 100])
    t0 = time.perf_counter()
    for s in range(args.warmup, args.warmup + args.steps):
        m.train(xpm[100 * s:100 * s + 100], y[100 * s:100 * s + 100])
    dt = time.perf_counter() - t0
    value = 100.0 * args.steps / dt
    line = {
        "impl": "reference", "metric": "training samples/sec", "value": value,
        "unit": "samples/s", "n_gpus": 0, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": 1000.0 * dt / args.steps, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "int8/int32", "data": "synthetic",
        "config": {"workload": "C5 train 8192->8192x4->10, bs 100 (one mini-batch per step)",
                   "model": cfg.name, "global_batch": 100, "seq_len": 0, "parallelism": "none"},
        "cpu_baseline": {"value": value, "unit": "samples/s", "cores": cores, "kind": "oracle",
                         "sample": "%d mini-batches of 100 samples" % args.steps},
        "e2e": {"value": value, "unit": "samples/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


def run_ours(args):
    import torch
    import torch.distributed as dist

    from paper_2412_00119_gb300 import bmlp as B

    rank, world, local = dist_env()
    if world > 1 and not dist.is_initialized():
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    cfg = W.CONFIGS[CONFIG_KEY]
    stream = torch.cuda.current_stream()
    hbm_gbs, sm_max_mhz, bf16_tf, bf16_tf_sus, peak_src = peaks()

    n_stream = cfg.n_train
    xp, xd, yd = make_stream(cfg, n_stream, dev)
    seed = replica_seed(cfg.model_seed, rank)
    model = B.BMLP(cfg.widths, cfg.classes, seed=seed, bs=100)
    h = model.h
    tc = model.info["fwd_impl"] == B.BMLP_FWD_TCGEN05
    steps_total = args.warmup + args.steps

    def train_step(i, x, y):
        s0 = (i % STEPS_PER_EPOCH) * SAMPLES_PER_STEP
        end = (i % STEPS_PER_EPOCH) == STEPS_PER_EPOCH - 1
        B.bmlp_train(h, x[s0:s0 + SAMPLES_PER_STEP], y[s0:s0 + SAMPLES_PER_STEP], SAMPLES_PER_STEP,
                     B.BMLP_EPOCH_END if end else 0, stream)

    for i in range(args.warmup):
        train_step(i, xd, yd)
    torch.cuda.synchronize()

    # timed region: every PROFILE_EVERY-th mini-batch is launched kernel by
    # kernel between CUDA events (the per-kernel figures below); the others
    # run as captured graphs
    B.bmlp_set_profiling(h, PROFILE_EVERY)
    B.bmlp_reset_profile(h)
    B.bmlp_update_stats(h, reset=True)
    launches0 = B.bmlp_launch_count(h)
    ev0 = torch.cuda.Event(enable_timing=True)
    ev1 = torch.cuda.Event(enable_timing=True)
    barrier()
    torch.cuda.synchronize()
    with ClockSampler(local) as clk:
        ev0.record(stream)
        for i in range(args.warmup, steps_total):
            train_step(i, xd, yd)
        ev1.record(stream)
        torch.cuda.synchronize()
    barrier()
    ms = ev0.elapsed_time(ev1)
    launches = B.bmlp_launch_count(h) - launches0
    upd_rows, upd_streamed, upd_bytes_total = B.bmlp_update_stats(h, reset=True)
    prof = B.bmlp_get_profile(h)
    B.bmlp_set_profiling(h, 0)
    ms_max = max_over_ranks(ms, dev)
    total_samples = sum_over_ranks(args.steps * SAMPLES_PER_STEP, dev)
    value = total_samples / (ms_max / 1000.0)

    # per-kernel device time per mini-batch, from the sampled launches
    L = len(cfg.widths) - 1
    per_mb = {}
    for kind, (n, tot) in prof.items():
        if n:
            per_mb[kind] = tot / n * (L if kind == "train_forward" else 1)
    dominant = max(per_mb, key=per_mb.get)
    step_ms_mb = ms / (args.steps * SAMPLES_PER_STEP / 100)
    upd_avg_s = prof["update"][1] / max(prof["update"][0], 1) / 1000.0
    fwd_avg_s = prof["train_forward"][1] / max(prof["train_forward"][0], 1) / 1000.0
    # algorithmic bytes per update launch: what the rule touched in the timed
    # region (rows with CP tuples streamed, sparse reinforcement elsewhere),
    # averaged over its mini-batches; update_bytes_per_launch is the all-rows bound
    n_mb = args.steps * SAMPLES_PER_STEP // 100
    upd_bytes = upd_bytes_total / n_mb if upd_bytes_total > 0 else update_bytes_per_launch(cfg.widths)
    bp_layer = 100 * cfg.widths[1] * cfg.widths[0]  # bit-pairs of one 8192x8192 forward launch
    popc_peak = popc_peak_bitpairs(sm_max_mhz)
    traffic = None
    if UPDATE_TRAFFIC_BYTES is not None and UPDATE_TRAFFIC_SRC_SHA == src_sha(*UPDATE_SOURCES):
        traffic = UPDATE_TRAFFIC_BYTES
    kernels = {
        "update": {"bound": "hbm", "achieved": upd_bytes / upd_avg_s / 1e9, "peak": hbm_gbs,
                   "unit": "GB/s", "frac": upd_bytes / upd_avg_s / 1e9 / hbm_gbs,
                   "traffic": traffic, "avg_us": upd_avg_s * 1e6,
                   "algorithmic_bytes": upd_bytes,
                   "all_rows_bytes": update_bytes_per_launch(cfg.widths),
                   "rows_streamed_frac": upd_streamed / max(upd_rows, 1)},
    }
    if tc:
        fp8_sus = FP8_PER_BF16 * bf16_tf_sus
        ftraffic = None
        if (FWD_TRAFFIC_BYTES is not None and cfg.widths[0] == cfg.widths[1] == 8192
                and FWD_TRAFFIC_SRC_SHA == src_sha("kern_forward_tc.cu", "tc_common.cuh")):
            ftraffic = FWD_TRAFFIC_BYTES
        kernels["train_forward"] = {
            "bound": "tensor", "achieved": 2 * bp_layer / fwd_avg_s / 1e12, "peak": fp8_sus,
            "unit": "TFLOP/s", "frac": 2 * bp_layer / fwd_avg_s / 1e12 / fp8_sus, "traffic": ftraffic,
            "avg_us": fwd_avg_s * 1e6, "algorithmic_flops": 2 * bp_layer,
            "peak_source": peak_src + " bf16 sustained x 2 (e4m3 / bf16 nominal)"}
    else:
        kernels["train_forward"] = {
            "bound": "alu", "achieved": bp_layer / fwd_avg_s / 1e12, "peak": popc_peak / 1e12,
            "unit": "Tbitpair/s", "frac": bp_layer / fwd_avg_s / popc_peak, "traffic": None,
            "avg_us": fwd_avg_s * 1e6, "algorithmic_bitpairs": bp_layer,
            "peak_source": "SM max clock x 152 SMs x 16 POPC/clk x 32"}
    kernels["update"]["peak_source"] = peak_src + " (HBM copy)"
    dom_key = "update" if dominant == "update" else "train_forward"
    roofline = {k: v for k, v in kernels[dom_key].items() if k in
                ("bound", "achieved", "peak", "unit", "frac", "traffic", "peak_source")}
    roofline["kernel"] = {"update": "k_update_ws",
                          "train_forward": "k_train_forward_tc" if tc else "k_train_forward"}[dom_key]

    # end-to-end through the C-ABI with host (pinned) buffers
    x_host = torch.from_numpy(xp.view(np.int64)).pin_memory()
    y_host = yd.cpu().pin_memory()
    n_e2e = max(1, args.steps)
    barrier()
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for i in range(n_e2e):
        s0 = ((args.warmup + i) % STEPS_PER_EPOCH) * SAMPLES_PER_STEP
        B.bmlp_train(h, x_host[s0:s0 + SAMPLES_PER_STEP], y_host[s0:s0 + SAMPLES_PER_STEP],
                     SAMPLES_PER_STEP, 0, stream, count_errors=True)
    torch.cuda.synchronize()
    e2e_s = max_over_ranks(time.perf_counter() - t0, dev)
    e2e_value = sum_over_ranks(n_e2e * SAMPLES_PER_STEP, dev) / e2e_s

    # forward-only evaluation sweep: 65,536 samples at batch 65,536
    xe = torch.from_numpy(W.make_inputs(cfg, "test", EVAL_BATCH).view(np.int64)).to(dev)
    out = torch.empty(EVAL_BATCH, dtype=torch.int32, device=dev)
    B.bmlp_predict(h, xe, out, EVAL_BATCH, stream)
    B.bmlp_set_profiling(h, 1)
    B.bmlp_reset_profile(h)
    reps = 3
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(reps):
        B.bmlp_predict(h, xe, out, EVAL_BATCH, stream)
    e1.record(stream)
    torch.cuda.synchronize()
    B.bmlp_set_profiling(h, 0)
    eprof = B.bmlp_get_profile(h)
    eval_ms = e0.elapsed_time(e1) / reps
    eval_bp = EVAL_BATCH * bitpairs_per_sample(cfg.widths, cfg.classes)
    efwd_s = eprof["eval_forward"][1] / max(eprof["eval_forward"][0], 1) / 1000.0
    efwd_bp = EVAL_BATCH * cfg.widths[1] * cfg.widths[0]
    if tc:
        fp8 = FP8_PER_BF16 * bf16_tf
        etraffic = None
        if (EVAL_TRAFFIC_BYTES is not None and cfg.widths[0] == cfg.widths[1] == 8192
                and EVAL_TRAFFIC_SRC_SHA == src_sha("kern_eval_tc.cu", "tc_common.cuh")):
            etraffic = EVAL_TRAFFIC_BYTES
        eroof = {"bound": "tensor", "kernel": "k_forward_eval_tc",
                 "achieved": 2 * efwd_bp / efwd_s / 1e12, "peak": fp8, "unit": "TFLOP/s",
                 "frac": 2 * efwd_bp / efwd_s / 1e12 / fp8, "traffic": etraffic,
                 "peak_source": peak_src + " bf16 burst x 2 (e4m3 / bf16 nominal)"}
    else:
        eroof = {"bound": "alu", "kernel": "k_forward_eval",
                 "achieved": efwd_bp / efwd_s / 1e12, "peak": popc_peak / 1e12,
                 "unit": "Tbitpair/s", "frac": efwd_bp / efwd_s / popc_peak, "traffic": None,
                 "peak_source": "SM max clock x 152 SMs x 16 POPC/clk x 32"}
    eval_info = {
        "samples_per_s": EVAL_BATCH / (eval_ms / 1000.0), "ms_per_sweep": eval_ms,
        "gbops": 2 * eval_bp / (eval_ms / 1000.0) / 1e9, "avg_us_per_layer": efwd_s * 1e6,
        "roofline": eroof,
    }

    mac_peak = (FP8_PER_BF16 * bf16_tf_sus if tc else 0.0) * 1e12 / 2.0
    sroof = step_roofline(step_ms_mb, upd_bytes, cfg.widths, cfg.classes, hbm_gbs,
                          mac_peak if tc else popc_peak, popc_peak,
                          "tensor (e4m3)" if tc else "alu (popcount)")
    sroof["peak_source"] = (peak_src + " HBM copy; compute: bf16 sustained x 2 (e4m3 / bf16 nominal)"
                            if tc else peak_src + " HBM copy; compute: SM max clock x 152 x 16 POPC x 32")

    engines = engine_bakeoff(dev) if not args.no_extras else None
    configs = ({k: config_figures(k, dev, hbm_gbs, mac_peak if tc else popc_peak, popc_peak,
                                  None if args.no_cpu_baseline else os.cpu_count() or 1)
                for k in ("C1", "C2", "C3", "C4")} if not args.no_extras else None)

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(cfg, W.unpack(xp[:100], cfg.widths[0]),
                           yd[:100].cpu().numpy().astype(np.int32), os.cpu_count() or 1)

    bp = bitpairs_per_sample(cfg.widths, cfg.classes)
    line = {
        "metric": "training samples/sec", "value": value, "unit": "samples/s",
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_max / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": ("b1 (+-1 bits; forward as e4m3 x e4m3 -> fp32 on tcgen05, exact) + bit-sliced "
                  "integer hidden weights (8 planes)" if tc else
                  "b1 (u64-packed XOR/popcount) + bit-sliced integer hidden weights (8 planes)"),
        "data": "synthetic",
        "config": {"workload": "C5 train: 8192->8192x4->10, bs 100, 1,000,000-sample i.i.d. "
                               "stream, teacher 8192->1024->10; step = 100,000 samples",
                   "model": cfg.name, "global_batch": 100 * world, "seq_len": 0,
                   "parallelism": "replicas x%d (independent seeds)" % world,
                   "l2": "inputs larger than L2 (1 GB stream, 256 MiB hidden weights)"},
        "gbops": 2 * bp * value / 1e9,
        "roofline": roofline,
        "step_roofline": sroof,
        "kernels": {k: {kk: vv for kk, vv in v.items()} for k, v in kernels.items()},
        "kernel_ms_per_minibatch": per_mb, "ms_per_minibatch": step_ms_mb,
        "cpu_baseline": cpu,
        "e2e": {"value": e2e_value, "unit": "samples/s",
                "h2d_bytes_per_step": SAMPLES_PER_STEP * (8 * xp.shape[1] + 4),
                "d2h_bytes_per_step": 24},
        "gpu_launches": launches,
        "clocks": clk.summary(),
        "eval": eval_info,
        "engines": engines,
        "configs": configs,
    }
    if rank == 0:
        print(json.dumps(line), flush=True)
    model.close()
    if world > 1:
        dist.destroy_process_group()
    return 0


def config_figures(key, dev, hbm_gbs, mac_peak, popc_peak, threads):
    """Throughput of one of the other workloads on this GPU: its whole
    training set for one epoch (after an untimed epoch that captures the
    graphs), timed between CUDA events; the step roofline as for the stress
    workload; and the CPU oracle on a bounded number of its mini-batches."""
    import torch

    from paper_2412_00119_gb300 import bmlp as B

    cfg = W.CONFIGS[key]
    st = torch.cuda.current_stream(dev)
    xp = W.make_inputs(cfg, "train")
    xd = torch.from_numpy(xp.view(np.int64)).to(dev)
    yd = W.teacher_labels_packed_torch(W.make_teacher(cfg), xd, cfg.widths[0])
    n = cfg.n_train
    model = B.BMLP(cfg.widths, cfg.classes, seed=cfg.model_seed, bs=100)
    B.bmlp_train(model.h, xd, yd, n, B.BMLP_EPOCH_END, st)
    B.bmlp_update_stats(model.h, reset=True)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    e0.record(st)
    B.bmlp_train(model.h, xd, yd, n, B.BMLP_EPOCH_END, st)
    e1.record(st)
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1)
    _, _, ubytes = B.bmlp_update_stats(model.h, reset=True)
    engine = ("tensor (e4m3)" if model.info["fwd_impl"] == B.BMLP_FWD_TCGEN05 else "alu (popcount)")
    model.close()
    n_mb = n // 100
    out = {"workload": "%s train: %s->%d, bs 100, %d training samples; timed: the second epoch"
                       % (key, "->".join(map(str, cfg.widths)), cfg.classes, n),
           "samples_per_s": n / (ms / 1e3), "ms_per_epoch": ms,
           "gbops": 2 * bitpairs_per_sample(cfg.widths, cfg.classes) * n / (ms / 1e3) / 1e9,
           "step_roofline": step_roofline(ms / n_mb, ubytes / n_mb, cfg.widths, cfg.classes,
                                          hbm_gbs, mac_peak, popc_peak, engine)}
    if threads:
        import oracle as O
        cores = O.set_threads(threads)
        mbs = CONFIG_ORACLE_MINIBATCHES[key]
        xo = W.unpack(xp[:100 * mbs], cfg.widths[0])
        yo = yd[:100 * mbs].cpu().numpy().astype(np.int32)
        ref = O.OracleModel(list(cfg.widths), cfg.classes, seed=cfg.model_seed, bs=100)
        t0 = time.perf_counter()
        ref.train(xo, yo)
        dt = time.perf_counter() - t0
        ref.close()
        out["cpu_baseline"] = {"value": 100 * mbs / dt, "unit": "samples/s", "cores": cores,
                               "kind": "oracle", "sample": "first %d mini-batches of 100" % mbs}
    return out


ENGINE_NAMES = {1: "popc", 2: "tcgen05_e4m3", 3: "b1_mma_sync", 4: "s8_mma_sync"}
# iterations of each peak kernel's timed launch (tens of milliseconds each)
PEAK_ITERS = {1: 20000, 2: 20000, 3: 20000, 4: 20000}


def engine_bakeoff(dev, reps=20):
    """The forward contraction (Alg. 1 l.8, Table 3's XNOR/popcount term) on
    every unit sm_103a offers: each unit's measured peak (bit-pairs/s over the
    device), and one 8192 -> 8192 layer at the training batch (100 patterns)
    and at the evaluation sweep's batch (65,536 patterns) on each engine that
    has a layer kernel, timed between CUDA events (average of `reps`
    launches after 3 untimed ones).  tcgen05.mma.kind::i8 does not exist on
    sm_103a, so +-1 as int8 runs only on the legacy mma.sync path, which has a
    peak kernel here but no layer kernel."""
    import torch

    from paper_2412_00119_gb300 import bmlp as B

    out = {"peaks": {}, "layer_8192x8192": {}}
    for e, name in ENGINE_NAMES.items():
        rate, ms = B.bmlp_engine_peak(e, PEAK_ITERS[e])
        out["peaks"][name] = {"bitpairs_per_s": rate, "tbitpairs_per_s": rate / 1e12, "ms": ms}
    widths = (8192, 8192)
    model = B.BMLP(widths, 10, seed=1, bs=100)
    st = torch.cuda.current_stream(dev)
    for M in (100, EVAL_BATCH):
        xa = torch.from_numpy(W.random_packed(77, M, widths[0]).view(np.int64)).to(dev)
        ya = torch.empty((M, W.words(widths[1])), dtype=torch.int64, device=dev)
        bp = float(M) * widths[0] * widths[1]
        row = {}
        for e in (1, 2, 3):
            name = ENGINE_NAMES[e]
            for _ in range(3):
                B.bmlp_layer_forward_engine(model.h, 1, e, xa, ya, stream=st)
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(st)
            for _ in range(reps if M <= 128 else 3):
                B.bmlp_layer_forward_engine(model.h, 1, e, xa, ya, stream=st)
            e1.record(st)
            torch.cuda.synchronize()
            us = e0.elapsed_time(e1) * 1e3 / (reps if M <= 128 else 3)
            pk = out["peaks"][name]["bitpairs_per_s"]
            row[name] = {"us": us, "tbitpairs_per_s": bp / us / 1e6,
                         "frac_of_engine_peak": bp / (us * 1e-6) / pk}
        out["layer_8192x8192"]["M%d" % M] = row
    model.close()
    return out


def run_bakeoff(args):
    import torch
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    print(json.dumps({"engines": engine_bakeoff(dev)}), flush=True)
    return 0


def run_ncu_case(args):
    """Small case for profiler captures: the 8192->8192x4->10 model trained on
    N mini-batches twice (the second pass is the one to capture)."""
    import torch

    from paper_2412_00119_gb300 import bmlp as B

    cfg = W.CONFIGS[CONFIG_KEY]
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    n = 100 * args.ncu_case
    xp, xd, yd = make_stream(cfg, n, dev)
    model = B.BMLP(cfg.widths, cfg.classes, seed=cfg.model_seed, bs=100)
    for _ in range(2):
        model.train(xd, yd)
    out = torch.empty(n, dtype=torch.int32, device=dev)
    model.predict(xd, out)
    torch.cuda.synchronize()
    print(json.dumps({"ncu_case_minibatches": args.ncu_case, "launches": B.bmlp_launch_count(model.h)}))
    model.close()
    return 0


def run_frontend_case(args):
    """The expansion front end alone (for timing and profiler captures): N x 1000
    uint8 patterns of D inputs through a fixed random K-wide expansion layer,
    the weight stream drawn once, the layer run twice (the second launch is
    the one to time or capture)."""
    import torch

    from paper_2412_00119_gb300 import bmlp as B

    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    D, K = (int(v) for v in args.frontend_shape.split(","))
    n = 1000 * args.frontend_case
    x = torch.from_numpy(W.pixel_bytes(1, n, D, "pixels")).to(dev)
    E = torch.empty((K, W.words(D)), dtype=torch.int64, device=dev)
    out = torch.empty((n, W.words(K)), dtype=torch.int64, device=dev)
    st = torch.cuda.current_stream(dev)
    B.bmlp_expand_weights(7, K, D, E, stream=st)
    B.bmlp_expand_sign(x, E, K, out, stream=st)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    e0.record(st)
    B.bmlp_expand_sign(x, E, K, out, stream=st)
    e1.record(st)
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1)
    print(json.dumps({"frontend_case": {"n": n, "D": D, "K": K, "expand_ms": ms,
                                        "patterns_per_s": n / ms * 1e3,
                                        "multiply_adds_per_s": n * D * K / ms * 1e3}}))
    return 0


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-extras", action="store_true",
                    help="skip the engine comparison and the other workloads' figures")
    ap.add_argument("--ncu-case", type=int, default=0, metavar="N",
                    help="run only a small N-mini-batch case (for profiler captures)")
    ap.add_argument("--frontend-case", type=int, default=0, metavar="N",
                    help="run only the expansion front end on N x 1000 uint8 patterns")
    ap.add_argument("--frontend-shape", default="784,1024", metavar="D,K",
                    help="inputs and width of the expansion layer for --frontend-case")
    ap.add_argument("--bakeoff", action="store_true",
                    help="run only the contraction-engine comparison (peaks and layer times)")
    args = ap.parse_args(argv)
    if args.bakeoff:
        return run_bakeoff(args)
    if args.ncu_case:
        return run_ncu_case(args)
    if args.frontend_case:
        return run_frontend_case(args)
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    if args.impl == "reference":
        return run_reference(args)
    return run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
