"""Throughput of the fused commit step (LM head + mask-suppressed softmax
confidence + multi-threshold commit) on GB300, as masked positions per second.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                    [--config NAME] [--no-graph] [--no-configs]

One step = one bd_commit_step over one window of the workload (compaction,
packing, LM head with the online softmax epilogue, merge and commit for the
whole threshold grid). The headline workload is the largest that fits one
GPU: 256 sequences x 8 slots x 64 positions, d = 5120, V = 157184, an E4M3
head with per-row scales and bf16 hidden states (W8A16). The line's
`configs` object reports each of the other four workloads the same way (its
own positions/s, LM-head time and roofline fractions), and `sustained` runs
two of them back to back for seconds, in the power-capped steady state.

With N > 1 (torchrun, one rank per GPU) every rank runs its own independent
window: the step shards by sequence with no data exchange, so scaling is
weak. Rank 0 prints one JSON line.

The reference arm (--impl reference) times the float64 CPU oracle on the
host cores, one bounded sample of whole blocks per step.
"""

from __future__ import annotations

import argparse
import contextlib
import hashlib
import json
import os
import statistics
import subprocess
import sys
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from workloads import B256X8X64_E4M3, B64X4X64_BF16, B8X2X32_BF16, CONFIGS, by_name, generate  # noqa: E402

DEFAULT_CONFIG = B256X8X64_E4M3.name
METRIC = "masked positions/s through fused LM-head+confidence+commit"
UNIT = "positions/s"
# the arithmetic type the path computes in, per head format
DTYPE_OF = {"f32": "f32", "bf16": "bf16", "e4m3": "e4m3xbf16", "nvfp4": "nvfp4xbf16"}
# workloads also run back to back for seconds (power-capped steady state)
SUSTAINED = (B8X2X32_BF16.name, B64X4X64_BF16.name)
# sources of the LM-head kernels (the traffic records name the hash of these)
KERNEL_SOURCES = ["paper_2609_33887_gb300/csrc/k_lmhead_pair.cu", "paper_2609_33887_gb300/csrc/k_lmhead_tc.cu",
                  "paper_2609_33887_gb300/csrc/common.cuh"]
TRAFFIC_FILE = os.path.join(ROOT, "profiles", "lmhead_traffic.txt")
# Idle seconds before each side measurement (other workloads, precision
# levers): the headline's seconds-long legs leave the board at its power limit
# with lowered clocks, which the next short measurement would otherwise inherit.
COOLDOWN_S = 2.0


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=1000)  # about 48 s of timed steps on the largest window
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--config", default=DEFAULT_CONFIG)
    ap.add_argument("--no-graph", dest="graph", action="store_false",
                    help="launch every step eagerly instead of replaying the K steps as one CUDA graph")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-verify", action="store_true",
                    help="skip the speculative-verification and precision-lever (NVFP4, E4M3, W8A8) measurements")
    ap.add_argument("--no-configs", action="store_true",
                    help="skip the other workloads and the sustained legs")
    return ap.parse_args()


# --------------------------------------------------------------- helpers --
def timing_events(n, stream):
    """n (begin, end) pairs of timing events whose CUDA handles exist (torch
    creates them lazily, at the first record)."""
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(n)]
    for a, b in evs:
        a.record(stream)
        b.record(stream)
    return evs


def aggregate_over_ranks(elapsed_ms, n_masked, dist=None, device="cpu"):
    """Weak-scaling aggregation: the slowest rank's time and every rank's
    masked positions (each rank serves its own independent window)."""
    if dist is None:
        return float(elapsed_ms), float(n_masked)
    t = torch.tensor([float(elapsed_ms)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    n = torch.tensor([float(n_masked)], dtype=torch.float64, device=device)
    dist.all_reduce(n, op=dist.ReduceOp.SUM)
    return float(t.item()), float(n.item())


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return d["hbm_gbs"], d["bf16_tflops"], d.get("bf16_tflops_sustained"), "measured"
    return 6800.0, 1900.0, 1700.0, "fallback"


def kernel_hash():
    h = hashlib.sha256()
    for f in KERNEL_SOURCES:
        with open(os.path.join(ROOT, f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def recorded_traffic(config_name):
    """DRAM bytes per LM-head launch from a committed ncu summary (records of
    `key: value` lines separated by blank lines), if one was taken on the
    current kernel sources for this workload; else None."""
    if not os.path.exists(TRAFFIC_FILE):
        return None
    recs, rec = [], {}
    with open(TRAFFIC_FILE) as f:
        for line in f:
            if not line.strip():
                if rec:
                    recs.append(rec)
                rec = {}
            elif ":" in line and not line.startswith("#"):
                k, v = line.split(":", 1)
                rec[k.strip()] = v.strip()
    if rec:
        recs.append(rec)
    h = kernel_hash()
    for rec in recs:
        if rec.get("kernel_sha256_16") == h and rec.get("workload") == config_name:
            try:
                return float(rec["dram_bytes_per_launch"])
            except (KeyError, ValueError):
                return None
    return None


class ClockSampler:
    """nvidia-smi clock / throttle samples while the timed region runs."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def start(self):
        import tempfile

        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), "--query-gpu=" + self.FIELDS, "--format=csv,noheader,nounits",
                 "-lms", "50"], stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None
        time.sleep(0.3)

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"], "samples": 0}
        time.sleep(0.1)
        self.proc.terminate()
        self.proc.wait()
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
        os.unlink(self.path)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i].lower().startswith("active")})
        loaded = [x for x in sm if mx and x >= 0.3 * max(mx)] or sm
        return {"sm_mhz": statistics.median(loaded) if loaded else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": reasons, "samples": len(rows),
                "power_w_max": max((float(r[3]) for r in rows if r[3].replace(".", "").isdigit()), default=None)}


def algorithmic(cfg, n_masked):
    """Algorithmic work of one step: 2*N*d*V FLOPs, and the bytes the method
    must move: the head once, the masked hidden rows, 12 B of outputs and 1 B
    of mask per position (logits are never stored)."""
    wbytes = {"f32": 4, "bf16": 2, "e4m3": 1}[cfg.weight_dtype]
    hbytes = {"f32": 4, "bf16": 2}[cfg.hidden_dtype]
    flops = 2.0 * n_masked * cfg.d * cfg.V
    bytes_ = cfg.V * cfg.d * wbytes + (cfg.V * 4 if cfg.weight_dtype == "e4m3" else 0) \
        + n_masked * cfg.d * hbytes + cfg.P * 13
    return flops, bytes_


# ----------------------------------------------------------- oracle timing --
def oracle_sample_time(wl, n_blocks, seed=7, w64=None):
    """Time the oracle on a sample of whole blocks; returns (seconds, masked positions)."""
    import oracle
    from workloads.rawio import dtype_tag, raw_numpy

    cfg = wl.cfg
    rng = np.random.default_rng(seed)
    blocks = sorted(rng.choice(cfg.n_blocks, size=min(n_blocks, cfg.n_blocks), replace=False).tolist())
    if w64 is None:
        w64 = oracle.weights_f64(raw_numpy(wl.weight), dtype_tag(wl.weight),
                                 None if wl.weight_scale is None else raw_numpy(wl.weight_scale))
    hid = raw_numpy(wl.hidden)
    pm = raw_numpy(wl.pos_masked)
    bf = raw_numpy(wl.block_flags)
    t0 = time.perf_counter()
    out = oracle.commit_step(hid, dtype_tag(wl.hidden), w64, "f64", None, pm, bf, cfg.n_seq, cfg.n_slots,
                             cfg.block_len, wl.mask_token_id, wl.tau, blocks=blocks)
    dt = time.perf_counter() - t0
    return dt, int((out["tokens"] >= 0).sum()), blocks, w64


def cores_used():
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count()


# ---------------------------------------------------------- reference arm --
def run_reference(args):
    rank, world, _ = dist_env()
    if rank != 0:
        return 0
    cfg = by_name(args.config)
    wl = generate(cfg)
    # per step: whole blocks, sized so that warmup + steps stay within a few minutes
    _, _, _, w64 = oracle_sample_time(wl, 1)
    t1, n1, _, _ = oracle_sample_time(wl, 1, w64=w64)
    budget = 150.0
    per_step = budget / max(1, args.steps + args.warmup)
    n_blocks = max(1, min(cfg.n_blocks, int(per_step / max(t1, 1e-3))))
    for i in range(args.warmup):
        oracle_sample_time(wl, n_blocks, seed=100 + i, w64=w64)
    tot_t, tot_n = 0.0, 0
    for i in range(args.steps):
        dt, n, _, _ = oracle_sample_time(wl, n_blocks, seed=1000 + i, w64=w64)
        tot_t += dt
        tot_n += n
    value = tot_n / tot_t if tot_t > 0 else 0.0
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * tot_t / max(1, args.steps),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": config_object(cfg, wl, masked_count(wl), world),
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores_used(), "kind": "oracle",
                         "sample": f"{n_blocks} whole block(s) per step of {cfg.name}; head decoded to float64 "
                                   "once, outside the timed steps"},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


# ---------------------------------------------------------------- our arm --
def redline_timing(with_oracle: bool) -> dict:
    """Host time of the Redline selection (libbdcommit, include/redline.h) on a
    grid shaped like the paper's largest (m = 50 configurations, n = 1012
    prompts, seeded synthetic outcomes): counting + p-values + Holm + deployment
    at one budget, and a sweep over 30 budgets; beside it the exact oracle on
    the same grid at one budget."""
    from paper_2609_33887_gb300 import redline as N
    from workloads.redline_inputs import random_grid

    gr = random_grid(1012, 50, seed=3)
    alphas = [i / 100 for i in range(1, 31)]

    def best_us(fn, min_s=0.2):
        reps, t0 = 0, time.perf_counter()
        while True:
            fn()
            reps += 1
            dt = time.perf_counter() - t0
            if dt >= min_s and reps >= 5:
                return dt / reps * 1e6

    def select():
        V = N.bd_redline_violations(gr.outcomes, gr.ref)
        return N.bd_redline_select(V, gr.cost, 1012, 0.10, gr.ref)["deployed"]

    V = N.bd_redline_violations(gr.outcomes, gr.ref)
    out = {"grid": "m50 n1012 synthetic outcomes, delta 0.10, Holm",
           "select_us": best_us(select),
           "sweep30_us": best_us(lambda: N.bd_redline_sweep(V, gr.cost, 1012, alphas, gr.ref)),
           "deployed": select()}
    if with_oracle:
        from oracle import redline_oracle as RO

        t0 = time.perf_counter()
        Vo = RO.joint_violations(gr.outcomes.tolist(), gr.ref)
        dep = RO.redline(Vo, list(gr.cost), 1012, 0.10, 0.10, gr.ref)["deployed"]
        out["oracle_select_ms"] = (time.perf_counter() - t0) * 1e3
        out["oracle_agrees"] = dep == out["deployed"]
    return out


def verify_timing(dev, stream) -> dict:
    """Speculative-decoding verification (bd_verify_step) at the Llama-3.1-8B
    shape: 64 requests of 4 drafts (320 rows), d = 4096, V = 128256, bf16, the
    paper's eleven typical-acceptance settings. Device time per step (CUDA
    events around 200 back-to-back steps), the LM-head kernel's own time and
    roofline, and the accepted tokens per target forward of each setting on
    these synthetic drafts (agreement 0.905)."""
    import statistics as st_

    import paper_2609_33887_gb300 as bdc
    from paper_2609_33887_gb300 import bdcommit as B
    from workloads.verify_inputs import generate_verify, SPEC_LLAMA8B

    cfg = SPEC_LLAMA8B
    wl = generate_verify(cfg).to(dev)
    R = cfg.rows
    ws = torch.empty(bdc.bd_verify_workspace_size(wl.hidden, wl.weight, None, wl.draft, cfg.n_req, cfg.n_draft,
                                                  cfg.eps), dtype=torch.uint8, device=dev)
    outs = {"tokens": torch.empty(R, dtype=torch.int32, device=dev),
            "p_draft": torch.empty(R, dtype=torch.float32, device=dev),
            "entropy": torch.empty(R, dtype=torch.float32, device=dev),
            "accept": torch.empty(R, dtype=torch.int32, device=dev),
            "accepted": torch.empty((cfg.n_req, len(cfg.eps) + 1), dtype=torch.int32, device=dev)}

    def step(ev=None):
        rc = B.bd_verify_step(wl.hidden, wl.weight, None, wl.draft, cfg.n_req, cfg.n_draft, cfg.eps, outs["tokens"],
                              outs["p_draft"], outs["entropy"], outs["accept"], outs["accepted"], stream=stream,
                              workspace=ws, lmhead_events=ev)
        if rc != 0:
            raise B.BdError(rc, "bd_verify_step")

    for _ in range(5):
        step()
    n = 200
    (e0, e1), = timing_events(1, stream)
    e0.record(stream)
    for _ in range(n):
        step()
    e1.record(stream)
    lm = timing_events(20, stream)
    for ev in lm:
        step(ev)
    torch.cuda.synchronize()
    st = B.bd_get_device_status(stream)
    if st != 0:
        raise B.BdError(st, "verify")
    ms = e0.elapsed_time(e1) / n
    lm_s = st_.mean(a.elapsed_time(b) for a, b in lm) / 1e3
    hbm_gbs, tc_tflops, _, src = peaks()
    flops = 2.0 * R * cfg.d * cfg.V
    abytes = cfg.V * cfg.d * 2 + R * cfg.d * 2 + R * 20
    bound = "tensor" if flops / (tc_tflops * 1e12) >= abytes / (hbm_gbs * 1e9) else "hbm"
    achieved = flops / lm_s / 1e12 if bound == "tensor" else abytes / lm_s / 1e9
    peak = tc_tflops if bound == "tensor" else hbm_gbs
    acc = outs["accepted"].float().mean(dim=0).cpu().tolist()
    tpf = {("lossless" if k == len(cfg.eps) else f"eps={cfg.eps[k]}"): 1.0 + acc[k] for k in range(len(acc))}
    return {"workload": cfg.name, "rows": R, "requests": cfg.n_req, "ms_per_step": ms,
            "rows_per_s": R / (ms / 1e3), "lmhead_us": lm_s * 1e6,
            "roofline": {"bound": bound, "achieved": achieved, "peak": peak,
                         "unit": "TFLOP/s" if bound == "tensor" else "GB/s", "frac": achieved / peak,
                         "peak_source": src, "algorithmic_flops": flops, "algorithmic_bytes": abytes},
            "tokens_per_forward": tpf, "data": "synthetic drafts, agreement 0.905 with the planted argmax"}


LEVERS = {
    # key: (workload, description of the LM-head path and what bounds it)
    "nvfp4": ("b8x2x32_d2048_v151936_nvfp4",
              "codes streamed by TMA and decoded exactly to f16 inside the LM-head kernel (f16 MMA, token rows "
              "scaled by a power of two per row); bound: the converter warps"),
    "e4m3": ("b8x2x32_d2048_v151936_e4m3",
             "W8A16 on the 8-bit tensor path: E4M3 codes read by TMA straight into the MMA operand; each bf16 row "
             "packed as two E4M3 terms (exact above 2^-10 of the row's largest), both multiplied by the head "
             "(tcgen05.mma kind::f8f6f4) into one fp32 accumulator"),
    "w8a8": ("b8x2x32_d2048_v151936_e4m3",
             "W8A8: packed rows quantised to E4M3 per row by the compaction kernel, E4M3 x E4M3 on the "
             "8-bit tensor path (tcgen05.mma kind::f8f6f4), both scales applied to the fp32 logits"),
}


@contextlib.contextmanager
def trace(name: str):
    """An NVTX range around a region (a no-op without a tracer, or where the
    torch build has no NVTX)."""
    try:
        torch.cuda.nvtx.range_push(name)
        pushed = True
    except Exception:  # noqa: BLE001 - tracing is optional
        pushed = False
    try:
        yield
    finally:
        if pushed:
            torch.cuda.nvtx.range_pop()


def fp8_gemm_tflops(dev, stream, n=8192, reps=30):
    """Dense E4M3 x E4M3 -> bf16 GEMM throughput of the vendor library
    (torch._scaled_mm, n x n x n, random codes) on this GPU, for the W8A8
    roofline's FP8 peak; None (with the reason) where the call is unavailable."""
    try:
        g = torch.Generator(device="cpu").manual_seed(5)
        a = torch.randn(n, n, generator=g).to(dev).to(torch.float8_e4m3fn)
        b = torch.randn(n, n, generator=g).to(dev).to(torch.float8_e4m3fn).t()  # column-major operand
        one = torch.ones((), device=dev)
        with torch.cuda.stream(stream):
            for _ in range(5):
                torch._scaled_mm(a, b, scale_a=one, scale_b=one, out_dtype=torch.bfloat16)
            (e0, e1), = timing_events(1, stream)
            e0.record(stream)
            for _ in range(reps):
                torch._scaled_mm(a, b, scale_a=one, scale_b=one, out_dtype=torch.bfloat16)
            e1.record(stream)
        torch.cuda.synchronize()
        return 2.0 * n ** 3 * reps / (e0.elapsed_time(e1) * 1e-3) / 1e12, None
    except Exception as exc:  # noqa: BLE001 - reported, not raised
        return None, f"{type(exc).__name__}: {exc}"[:200]


def lever_timing(dev, stream, lever: str) -> dict:
    """The bench window (8 x 2 x 32, d = 2048, V = 151936) with a quantised
    head (the precision levers): after COOLDOWN_S idle, the LM-head kernel's
    own time (20 event-timed steps), then the device time per commit step
    (CUDA events around 200 back-to-back steps), and the step
    against the lever's algorithmic bytes (the stored head: NVFP4 codes V*d/2
    and block scales V*d/16, or E4M3 codes V*d; row scales 4V; the masked bf16
    rows; 13 B per window position). The tensor fraction of the W8A8 head is
    taken against twice the measured bf16 peak (the nominal FP8 : BF16 ratio)."""
    import statistics as st_

    import paper_2609_33887_gb300 as bdc
    from paper_2609_33887_gb300 import bdcommit as B

    name, path = LEVERS[lever]
    cfg = by_name(name)
    wl = generate(cfg).to(dev)
    head = bdc.Nvfp4Head(wl.weight, wl.weight_block_scale, cfg.d) if lever == "nvfp4" else wl.weight
    flags = B.BD_EXEC_FP8_ACTIVATIONS if lever == "w8a8" else 0
    P = cfg.P
    ws = torch.empty(bdc.bd_workspace_size(wl.hidden, head, wl.weight_scale, wl.pos_masked, wl.block_flags,
                                           cfg.n_seq, cfg.n_slots, cfg.block_len, cfg.mask_token_id, cfg.tau),
                     dtype=torch.uint8, device=dev)
    tokens = torch.empty(P, dtype=torch.int32, device=dev)
    conf = torch.empty(P, dtype=torch.float32, device=dev)
    commit = torch.empty(P, dtype=torch.int32, device=dev)

    def step(ev=None):
        rc = B.bd_commit_step_ex(wl.hidden, head, wl.weight_scale, wl.pos_masked, wl.block_flags, cfg.n_seq,
                                 cfg.n_slots, cfg.block_len, cfg.mask_token_id, cfg.tau, tokens, conf, commit,
                                 stream=stream, workspace=ws, lmhead_events=ev, flags=flags)
        if rc != 0:
            raise B.BdError(rc, f"{lever} step")

    for _ in range(5):
        step()
    n = 200
    (e0, e1), = timing_events(1, stream)
    lm = timing_events(20, stream)
    torch.cuda.synchronize()
    time.sleep(COOLDOWN_S)
    smp = ClockSampler(dev.index if dev.index is not None else 0)
    smp.start()
    for ev in lm:  # the LM head first, from the idle state (see side_config)
        step(ev)
    e0.record(stream)
    for _ in range(n):
        step()
    e1.record(stream)
    torch.cuda.synchronize()
    clk = smp.stop()
    st = B.bd_get_device_status(stream)
    if st != 0:
        raise B.BdError(st, lever)
    ms = e0.elapsed_time(e1) / n
    lm_us = st_.mean(a.elapsed_time(b) for a, b in lm) * 1e3
    n_masked = int(((wl.pos_masked != 0) & (torch.repeat_interleave(wl.block_flags & 1, cfg.block_len) != 0)).sum())
    head_bytes = (cfg.V * cfg.d // 2 + cfg.V * ((cfg.d + 15) // 16)) if lever == "nvfp4" else cfg.V * cfg.d
    abytes = head_bytes + 4 * cfg.V + n_masked * cfg.d * 2 + P * 13
    flops = 2.0 * n_masked * cfg.d * cfg.V
    hbm_gbs, tc_tflops, _, src = peaks()
    tc_peak = 2.0 * tc_tflops if lever == "w8a8" else tc_tflops
    out = {"workload": cfg.name, "ms_per_step": ms, "positions_per_s": n_masked / (ms / 1e3),
           "lmhead_us": lm_us, "algorithmic_bytes": abytes, "algorithmic_flops": flops,
           "step_hbm_frac": abytes / (ms / 1e3) / 1e9 / hbm_gbs,
           "lmhead_tensor_frac": flops / (lm_us * 1e-6) / 1e12 / tc_peak,
           "tensor_peak_tflops": tc_peak,
           "path": path, "clocks": clk, "cooldown_s": COOLDOWN_S,
           "peak_source": src + (" (x2: nominal FP8 : BF16 ratio)" if lever == "w8a8" else "")}
    if lever == "w8a8":
        # the library's own FP8 GEMM on this GPU, measured here, beside the nominal-ratio peak
        fp8, why = fp8_gemm_tflops(dev, stream)
        out["fp8_gemm_tflops_measured"] = fp8
        out["lmhead_tensor_frac_of_measured_fp8"] = (flops / (lm_us * 1e-6) / 1e12 / fp8) if fp8 else None
        if why:
            out["fp8_gemm_unavailable"] = why
    return out


def config_object(cfg, wl_host, n_masked, world):
    """The workload description both arms print (identical keys and values)."""
    wbytes = {"f32": 4, "bf16": 2, "e4m3": 1}[cfg.weight_dtype]
    return {"workload": cfg.name, "n_seq": cfg.n_seq, "n_slots": cfg.n_slots, "block_len": cfg.block_len,
            "masked_positions_per_rank": int(n_masked), "d": cfg.d, "V": cfg.V, "T": len(cfg.tau),
            "head_dtype": cfg.weight_dtype, "hidden_dtype": cfg.hidden_dtype,
            "parallelism": f"independent windows x{world}",
            "l2": ("inputs larger than L2 (the LM head is %.0f MB, read every step)" if cfg.V * cfg.d * wbytes > 129e6
                   else "no flush: the %.0f MB head stays in L2 between steps (a launch-latency-bound workload)")
                  % (cfg.V * cfg.d * wbytes / 1e6),
            "inputs_sha256": wl_host.digests()}


def masked_count(wl_host):
    cfg = wl_host.cfg
    return int(((wl_host.pos_masked != 0) &
                (torch.repeat_interleave(wl_host.block_flags & 1, cfg.block_len) != 0)).sum())


def lmhead_launches(r):
    """LM-head launches per step: the library's kernel count less compaction,
    merge and the head decode where a bf16 copy is made."""
    decoded = r.cfg.weight_dtype == "nvfp4" and r.cfg.P > 8192
    return launches_per_step(r) - 2 - (1 if decoded else 0)


def launches_per_step(r):
    """Library kernels one commit step of runner `r` queues, as the library
    reports them for its arguments (bd_step_kernels): compaction + row packing,
    the decode of a quantised head where a bf16 copy is made, the LM head (one
    launch, or two where spill pairs run beside clusters of two CTA pairs),
    merge + commit. The counts reset is a runtime memset, not a kernel."""
    n = r.kernels_per_step
    if n <= 0:
        raise RuntimeError(f"bd_step_kernels: {n}")
    return n


class StepRunner:
    """One workload resident on the device with its workspace and outputs."""

    def __init__(self, cfg, wl_host, dev):
        import paper_2609_33887_gb300 as bdc

        self.B = bdc.bdcommit
        self.cfg = cfg
        self.wl_host = wl_host
        self.wl = wl_host.to(dev)
        self.dev = dev
        wl, P, T = self.wl, cfg.P, len(cfg.tau)
        ws_bytes = bdc.bd_workspace_size(wl.hidden, wl.weight, wl.weight_scale, wl.pos_masked, wl.block_flags,
                                         cfg.n_seq, cfg.n_slots, cfg.block_len, cfg.mask_token_id, cfg.tau)
        self.workspace = torch.empty(max(ws_bytes, 1), dtype=torch.uint8, device=dev)
        self.kernels_per_step = bdc.bd_step_kernels(wl.hidden, wl.weight, wl.weight_scale, wl.pos_masked,
                                                    wl.block_flags, cfg.n_seq, cfg.n_slots, cfg.block_len,
                                                    cfg.mask_token_id, cfg.tau)
        self.tokens = torch.empty(P, dtype=torch.int32, device=dev)
        self.conf = torch.empty(P, dtype=torch.float32, device=dev)
        self.commit = torch.empty(P, dtype=torch.int32, device=dev)
        self.counts = torch.empty((cfg.n_seq, T), dtype=torch.int32, device=dev)
        self.n_masked = masked_count(wl_host)

    def step(self, ev=None, hidden=None, pm=None, bf=None, outs=None):
        cfg, wl = self.cfg, self.wl
        o = outs or (self.tokens, self.conf, self.commit, self.counts)
        rc = self.B.bd_commit_step_ex(wl.hidden if hidden is None else hidden, wl.weight, wl.weight_scale,
                                      wl.pos_masked if pm is None else pm, wl.block_flags if bf is None else bf,
                                      cfg.n_seq, cfg.n_slots, cfg.block_len, cfg.mask_token_id, cfg.tau,
                                      o[0], o[1], o[2], stream=torch.cuda.current_stream(),
                                      workspace=self.workspace, out_counts=o[3], lmhead_events=ev)
        if rc != 0:
            raise self.B.BdError(rc)

    def check_status(self, where):
        st = self.B.bd_get_device_status(torch.cuda.current_stream())
        if st != 0:
            raise self.B.BdError(st, where)

    def capture(self, n):
        """n steps as one CUDA graph (the serving engine also replays captured graphs)."""
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            for _ in range(n):
                self.step()
        torch.cuda.synchronize()
        return g

    def lmhead_ms(self, n=24):
        """The LM-head kernel's own duration, CUDA events on the launching stream
        around each of n eager steps (outside any graph: an event node between two
        kernels would cancel their programmatic launch overlap in the graph)."""
        stream = torch.cuda.current_stream()
        evs = timing_events(n, stream)
        for ev in evs:
            self.step(ev=ev)
        torch.cuda.synchronize()
        self.check_status("LM-head timing")
        return [a.elapsed_time(b) for a, b in evs]


def roofline_of(cfg, n_masked, lm_ms, traffic=None, lm_launches=1):
    """Roofline of the LM-head kernel: the algorithmic FLOPs (2 N d V) or bytes
    per step over the mean CUDA-event duration of its launches (one, or the
    main and spill launches of clusters of two CTA pairs), against the
    measured peak."""
    hbm_gbs, tc_tflops, tc_sus, peak_src = peaks()
    flops, abytes = algorithmic(cfg, n_masked)
    lm_s = statistics.mean(lm_ms) / 1e3
    t_tc = flops / (tc_tflops * 1e12)
    t_hbm = abytes / (hbm_gbs * 1e9)
    if t_tc >= t_hbm:
        achieved = flops / lm_s / 1e12
        roof = {"bound": "tensor", "achieved": achieved, "peak": tc_tflops, "unit": "TFLOP/s",
                "frac": achieved / tc_tflops, "traffic": traffic,
                "peak_source": f"bf16_tflops (burst) of {peak_src}",
                "frac_of_sustained": (achieved / tc_sus) if tc_sus else None}
    else:
        achieved = abytes / lm_s / 1e9
        roof = {"bound": "hbm", "achieved": achieved, "peak": hbm_gbs, "unit": "GB/s",
                "frac": achieved / hbm_gbs, "traffic": traffic, "peak_source": f"hbm_gbs of {peak_src}"}
    roof["lmhead_ms_avg"] = statistics.mean(lm_ms)
    roof["lmhead_ms_median"] = statistics.median(lm_ms)
    roof["lmhead_launches_timed"] = len(lm_ms)
    roof["lmhead_launches_per_step"] = lm_launches
    roof["hbm_view"] = {"algorithmic_bytes": abytes, "achieved_gbs": abytes / lm_s / 1e9,
                        "frac": abytes / lm_s / 1e9 / hbm_gbs,
                        # against the nominal HBM3e figure, for context (the measured copy is the peak)
                        "frac_of_nominal_7900": abytes / lm_s / 1e9 / 7900.0}
    roof["tensor_view"] = {"algorithmic_flops": flops, "achieved_tflops": flops / lm_s / 1e12,
                           "frac": flops / lm_s / 1e12 / tc_tflops,
                           "frac_of_sustained": (flops / lm_s / 1e12 / tc_sus) if tc_sus else None}
    roof["traffic_over_algorithmic"] = (traffic / abytes) if traffic else None
    roof["kernel_sha256_16"] = kernel_hash()
    return roof


def side_config(cfg, dev, min_s=0.25, steps=20, warmup=5):
    """One of the other workloads: after COOLDOWN_S idle, the LM-head roofline
    from 24 event-timed launches, then positions/s over a graph-replayed timed
    region of at least `steps` steps and ~min_s seconds; clocks sampled over
    both. (The LM head is timed first: after a region of this length the board
    sits at its power limit, which the sustained legs report separately.)"""
    wl_host = generate(cfg)
    r = StepRunner(cfg, wl_host, dev)
    for _ in range(warmup):
        r.step()
    torch.cuda.synchronize()
    r.check_status("warm-up")
    t0 = time.perf_counter()
    for _ in range(3):
        r.step()
    torch.cuda.synchronize()
    est = (time.perf_counter() - t0) / 3
    k = int(min(2000, max(steps, min_s / max(est, 1e-6))))
    g = r.capture(k)
    g.replay()  # warm replay
    torch.cuda.synchronize()
    stream = torch.cuda.current_stream()
    (e0, e1), = timing_events(1, stream)
    time.sleep(COOLDOWN_S)
    smp = ClockSampler(dev.index if dev.index is not None else 0)
    smp.start()
    lm = r.lmhead_ms()
    e0.record(stream)
    g.replay()
    e1.record(stream)
    torch.cuda.synchronize()
    r.check_status("timed region")
    ms = e0.elapsed_time(e1) / k
    clk = smp.stop()
    roof = roofline_of(cfg, r.n_masked, lm, recorded_traffic(cfg.name), lmhead_launches(r))
    out = {"positions_per_s": r.n_masked / (ms / 1e3), "ms_per_step": ms, "steps": k,
           "masked_positions": r.n_masked, "lmhead_us": roof["lmhead_ms_avg"] * 1e3,
           "tensor_frac": roof["tensor_view"]["frac"], "hbm_frac": roof["hbm_view"]["frac"],
           "traffic_over_algorithmic": roof["traffic_over_algorithmic"], "roofline": roof,
           "gpu_launches_per_step": launches_per_step(r), "clocks": clk, "cooldown_s": COOLDOWN_S}
    del g, r
    torch.cuda.empty_cache()
    return out


def sustained_leg(cfg, dev, gpu_index, seconds=3.0):
    """Back-to-back commit steps for >= `seconds` (the power-capped steady
    state a serving loop sees), with the clocks sampled meanwhile; the step's
    tensor rate against the measured sustained bf16 peak."""
    wl_host = generate(cfg)
    r = StepRunner(cfg, wl_host, dev)
    for _ in range(5):
        r.step()
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for _ in range(3):
        r.step()
    torch.cuda.synchronize()
    est = (time.perf_counter() - t0) / 3
    per_graph = int(min(500, max(1, 0.25 / max(est, 1e-6))))
    g = r.capture(per_graph)
    stream = torch.cuda.current_stream()
    sampler = ClockSampler(gpu_index)
    sampler.start()
    (e0, e1), = timing_events(1, stream)
    e0.record(stream)
    n_rep, t_start = 0, time.perf_counter()
    while time.perf_counter() - t_start < seconds or n_rep < 2:
        g.replay()
        n_rep += 1
        if n_rep % 4 == 0:
            torch.cuda.synchronize()
    e1.record(stream)
    torch.cuda.synchronize()
    clocks = sampler.stop()
    r.check_status("sustained leg")
    steps = n_rep * per_graph
    ms = e0.elapsed_time(e1) / steps
    _, tc_tflops, tc_sus, src = peaks()
    flops, abytes = algorithmic(cfg, r.n_masked)
    out = {"workload": cfg.name, "seconds": e0.elapsed_time(e1) / 1e3, "steps": steps, "ms_per_step": ms,
           "positions_per_s": r.n_masked / (ms / 1e3),
           "step_tflops": flops / (ms / 1e3) / 1e12,
           "step_frac_of_sustained_bf16": (flops / (ms / 1e3) / 1e12 / tc_sus) if tc_sus else None,
           "step_frac_of_burst_bf16": flops / (ms / 1e3) / 1e12 / tc_tflops,
           "step_hbm_gbs": abytes / (ms / 1e3) / 1e9, "peak_source": src, "clocks": clocks}
    del g, r
    torch.cuda.empty_cache()
    return out


def e2e_leg(r, K, W, pg, dev):
    """The metric end to end through the public call with host buffers: every
    step copies its inputs (hidden states and mask state) in from pinned host
    memory and its outputs (tokens, conf, commit, counts) out to pinned host
    memory. The copies are double-buffered on two copy streams, ordered by
    events, so the input copy of step i + 1 and the output copy of step i - 1
    overlap the kernels of step i, as a serving loop would run them."""
    cfg, wl_host, P, T = r.cfg, r.wl_host, r.cfg.P, len(r.cfg.tau)
    h_host = wl_host.hidden.pin_memory()
    pm_host = wl_host.pos_masked.pin_memory()
    bf_host = wl_host.block_flags.pin_memory()
    bufs = []
    for _ in range(2):
        bufs.append({
            "h": torch.empty_like(r.wl.hidden), "pm": torch.empty_like(r.wl.pos_masked),
            "bf": torch.empty_like(r.wl.block_flags),
            "out": [torch.empty(P, dtype=torch.int32, device=dev), torch.empty(P, dtype=torch.float32, device=dev),
                    torch.empty(P, dtype=torch.int32, device=dev),
                    torch.empty((cfg.n_seq, T), dtype=torch.int32, device=dev)],
            "host": [torch.empty(P, dtype=torch.int32).pin_memory(),
                     torch.empty(P, dtype=torch.float32).pin_memory(),
                     torch.empty(P, dtype=torch.int32).pin_memory(),
                     torch.empty((cfg.n_seq, T), dtype=torch.int32).pin_memory()],
        })
    c_in, c_out = torch.cuda.Stream(device=dev), torch.cuda.Stream(device=dev)
    evs = [torch.cuda.Event() for _ in range(6)]

    def e2e_steps(n):
        # the stream current at call time: inside a graph capture, the capture stream
        stream = torch.cuda.current_stream()
        comp, outd, inr = evs[0:2], evs[2:4], evs[4:6]
        fork = torch.cuda.Event()
        fork.record(stream)
        c_in.wait_event(fork)
        c_out.wait_event(fork)
        for i in range(n):
            b = i & 1
            u = bufs[b]
            with torch.cuda.stream(c_in):
                if i >= 2:
                    c_in.wait_event(comp[b])  # step i - 2 no longer reads these inputs
                u["h"].copy_(h_host, non_blocking=True)
                u["pm"].copy_(pm_host, non_blocking=True)
                u["bf"].copy_(bf_host, non_blocking=True)
                inr[b].record(c_in)
            stream.wait_event(inr[b])
            if i >= 2:
                stream.wait_event(outd[b])  # the outputs of step i - 2 have been copied out
            r.step(hidden=u["h"], pm=u["pm"], bf=u["bf"], outs=u["out"])
            comp[b].record(stream)
            with torch.cuda.stream(c_out):
                c_out.wait_event(comp[b])
                for hst, d_ in zip(u["host"], u["out"]):
                    hst.copy_(d_, non_blocking=True)
                outd[b].record(c_out)
        stream.wait_stream(c_in)
        stream.wait_stream(c_out)

    e2e_steps(W)
    torch.cuda.synchronize()
    egraph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(egraph):
        e2e_steps(K)
    torch.cuda.synchronize()
    if pg:
        pg.barrier()
    stream = torch.cuda.current_stream()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    egraph.replay()
    e1.record(stream)
    torch.cuda.synchronize()
    r.check_status("e2e")
    e_ms, total = aggregate_over_ranks(e0.elapsed_time(e1), r.n_masked, pg, dev)
    h2d = h_host.numel() * h_host.element_size() + pm_host.numel() + bf_host.numel()
    d2h = sum(o.numel() * o.element_size() for o in bufs[0]["host"])
    # the results of the last step really arrived in host memory
    last = bufs[(K - 1) & 1]
    assert torch.equal(last["host"][0], last["out"][0].cpu())
    out = {"value": total * K / (e_ms / 1e3), "unit": UNIT, "h2d_bytes_per_step": int(h2d),
           "d2h_bytes_per_step": int(d2h),
           "note": "pinned host hidden states + mask state in, tokens/conf/commit/counts out, every step; "
                   "double-buffered on two copy streams so copies overlap the neighbouring steps' kernels; "
                   "LM-head weights stay resident in HBM; the K steps replayed as one CUDA graph"}
    del egraph, bufs
    return out


def run_ours(args):
    import paper_2609_33887_gb300 as bdc

    rank, world, local = dist_env()
    if not torch.cuda.is_available():
        raise SystemExit("bench.py needs a CUDA device (no CPU fallback)")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    pg = None
    if world > 1:
        import torch.distributed as dist

        dist.init_process_group("nccl", device_id=dev)
        pg = dist
    bdc.load_library()
    vis = [x for x in os.environ.get("CUDA_VISIBLE_DEVICES", "").split(",") if x]
    gpu_index = vis[local] if local < len(vis) else str(local)

    cfg = by_name(args.config)
    # each rank serves its own window (independent sequences): weak scaling
    from dataclasses import replace

    wl_host = generate(replace(cfg, seed=cfg.seed + 1000 * rank) if rank else cfg)
    r = StepRunner(cfg, wl_host, dev)
    K, W = args.steps, args.warmup
    for _ in range(W):
        r.step()
    torch.cuda.synchronize()
    r.check_status("warm-up")
    graph = r.capture(K) if args.graph else None

    # ---- device-resident timed region: exactly K steps
    sampler = ClockSampler(gpu_index)
    sampler.start()
    if pg:
        pg.barrier()
    stream = torch.cuda.current_stream()
    torch.cuda.synchronize()
    t_start, t_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with trace(f"timed region: {K} steps"):
        t_start.record(stream)
        if graph is None:
            for _ in range(K):
                r.step()
        else:
            graph.replay()
        t_end.record(stream)
    torch.cuda.synchronize()
    if pg:
        pg.barrier()
    clocks = sampler.stop()
    elapsed_ms = t_start.elapsed_time(t_end)
    r.check_status("timed region")
    elapsed_ms, total_masked = aggregate_over_ranks(elapsed_ms, r.n_masked, pg, dev)
    ms_per_step = elapsed_ms / K
    value = total_masked * K / (elapsed_ms / 1e3)
    del graph

    # ---- the LM head's own duration (roofline), outside the timed region
    with trace("LM-head events"):
        lm = r.lmhead_ms(max(24, min(K, 200)))
    roof = roofline_of(cfg, r.n_masked, lm, recorded_traffic(cfg.name), lmhead_launches(r))

    # ---- end to end through the public call with host buffers
    e2e = None
    if not args.no_e2e:
        with trace("e2e"):
            e2e = e2e_leg(r, K, W, pg, dev)

    # ---- CPU baseline: the oracle on a bounded sample, rank 0 at N = 1 only
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        dt, n, blocks, w64 = oracle_sample_time(wl_host, 1)
        target = 12.0  # seconds of oracle work
        nb = max(1, min(cfg.n_blocks, int(target / 4 / max(dt, 1e-3))))
        tot_t, tot_n, passes = 0.0, 0, 0
        while tot_t < target and passes < 1000:
            dt, n, blocks, _ = oracle_sample_time(wl_host, nb, seed=11 + passes, w64=w64)
            tot_t += dt
            tot_n += n
            passes += 1
        del w64
        cpu = {"value": tot_n / tot_t, "unit": UNIT, "cores": cores_used(), "kind": "oracle",
               "sample": f"{passes} pass(es) over {len(blocks)} whole blocks of {cfg.name} ({tot_n} masked "
                         f"positions, {tot_t:.1f} s); head decoded to float64 once outside the timed calls"}

    conf_obj = config_object(cfg, wl_host, r.n_masked, world)
    kernels = launches_per_step(r)
    del r
    torch.cuda.empty_cache()

    # ---- every other workload, the sustained legs and the side measurements (rank 0)
    configs, sustained = {}, {}
    if rank == 0 and not args.no_configs:
        for other in CONFIGS:
            if other.name != cfg.name:
                with trace(f"workload {other.name}"):
                    configs[other.name] = side_config(other, dev)
        for name in SUSTAINED:
            with trace(f"sustained {name}"):
                sustained[name] = sustained_leg(by_name(name), dev, gpu_index)
    with trace("redline"):
        redline = redline_timing(with_oracle=cpu is not None) if rank == 0 else None
    with trace("sweep"):
        sweep = sweep_timing(dev) if rank == 0 and not args.no_verify else None
    with trace("verify"):
        verify = verify_timing(dev, stream) if rank == 0 and not args.no_verify else None
    with trace("precision levers"):
        levers = {k: lever_timing(dev, stream, k) for k in LEVERS} if rank == 0 and not args.no_verify else {}

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": K, "warmup": W,
            "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": DTYPE_OF[cfg.weight_dtype], "data": "synthetic",
            "config": conf_obj,
            "timing": {"graph": bool(args.graph),
                       "region": f"{K} steps" + (" replayed as one CUDA graph" if args.graph else " launched eagerly"),
                       "lmhead": f"{len(lm)} eager steps with CUDA events around the LM-head launches, "
                                 "after the timed region"},
            "roofline": roof,
            "cpu_baseline": cpu,
            "e2e": e2e,
            "gpu_launches": kernels * K,
            "clocks": clocks,
            "configs": configs or None,
            "sustained": sustained or None,
            "redline": redline,
            "sweep": sweep,
            "verify": verify,
            "nvfp4": levers.get("nvfp4"),
            "e4m3": levers.get("e4m3"),
            "w8a8": levers.get("w8a8"),
        }
        print(json.dumps(line), flush=True)
    if pg:
        pg.destroy_process_group()
    return 0


def sweep_timing(dev):
    """bd_commit_sweep (the block-buffer update that follows the step in a
    decode loop) on the 8 x 2 x 32 window, back to back on one stream."""
    import paper_2609_33887_gb300 as bdc

    B = bdc.bdcommit
    cfg = B8X2X32_BF16
    r = StepRunner(cfg, generate(cfg), dev)
    r.step()
    torch.cuda.synchronize()
    P = cfg.P
    stream = torch.cuda.current_stream()
    tok_w = torch.full((P,), -1, dtype=torch.int32, device=dev)
    pm_w, fl_w = r.wl.pos_masked.clone(), r.wl.block_flags.clone()
    cache_w = torch.empty(P, dtype=torch.int32, device=dev)
    ncom_w = torch.empty(cfg.n_seq, dtype=torch.int32, device=dev)

    def sweep_once():
        rc = B.bd_commit_sweep(tok_w, pm_w, fl_w, cfg.n_seq, cfg.n_slots, cfg.block_len, cfg.mask_token_id,
                               r.tokens, r.commit, len(cfg.tau) - 1, B.BD_SWEEP_ADMIT | B.BD_SWEEP_ELIGIBLE_OLDEST,
                               cache_w, ncom_w, None, stream=stream)
        if rc != 0:
            raise B.BdError(rc, "bd_commit_sweep")

    for _ in range(10):
        sweep_once()
    n_sw = 500
    (e0, e1), = timing_events(1, stream)
    e0.record(stream)
    for _ in range(n_sw):
        sweep_once()
    e1.record(stream)
    torch.cuda.synchronize()
    return {"workload": cfg.name, "us_per_launch": e0.elapsed_time(e1) * 1e3 / n_sw, "launches_timed": n_sw,
            "window_positions": P, "ctas": cfg.n_seq, "bound": "latency (one CTA per sequence)",
            "note": "bd_commit_sweep after one commit step, back to back on one stream"}


def main():
    args = parse_args()
    if args.impl == "reference":
        return run_reference(args)
    return run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
