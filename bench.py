#!/usr/bin/env python3
"""Benchmark of the W8A8 SmoothQuant hot path on GB300.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

Prints ONE JSON line (rank 0).  The headline workload is the lm_head of a Gemma-3-1B-shaped
model at decode (1152 -> 262144, W8A8, M = 1 token, fp32 logits + top-1), the paper's largest
single operation.  A step is one lm_head call on a fresh token; L2 is flushed (a 512 MiB
write) before every timed step, and each step is timed on the device with CUDA events.
``value`` = ms per token (max over ranks; replicas only, every rank runs the same workload).

The same line carries:
  * ``kernels``: per-call time, TOPS and algorithmic GB/s of the single W8A8 linear
    (M = 16, 1152 -> 6912), the FFN block (M in 1, 8, 64, 512, 2048) and lm_head
    (M in 1, 16, 128, 512), W8A8 and bf16, with the fraction of the measured HBM peak;
  * ``roofline`` of the headline kernel against the measured HBM copy bandwidth;
  * ``e2e``: the same metric through the public API from pinned host buffers (input copy in,
    top-1 copy out, host wall clock);
  * ``cpu_baseline``: the oracle on this host's cores for a bounded sample.
``--impl reference`` times the oracle (CPU) on the same workload and metric.
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

METRIC = "W8A8 linear TOPS & HBM GB/s vs GB300 roofline; decode ms/token per mask vs bf16"
HIDDEN, INTER, VOCAB = 1152, 6912, 262144
FALLBACK_HBM_GBS = 6800.0
FALLBACK_BF16_TFLOPS = 1900.0


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--no-sweep", action="store_true", help="skip the per-kernel sweep")
    return ap.parse_args()


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return {"hbm_gbs": float(d["hbm_gbs"]), "bf16_tflops": float(d["bf16_tflops"]),
                "bf16_tflops_sustained": float(d.get("bf16_tflops_sustained", d["bf16_tflops"])), "source": "measured"}
    return {"hbm_gbs": FALLBACK_HBM_GBS, "bf16_tflops": FALLBACK_BF16_TFLOPS, "bf16_tflops_sustained": 1700.0,
            "source": "fallback"}


# ----------------------------------------------------------------------------- distributed
class Dist:
    def __init__(self, backend):
        self.world = int(os.environ.get("WORLD_SIZE", "1"))
        self.rank = int(os.environ.get("RANK", "0"))
        self.local = int(os.environ.get("LOCAL_RANK", "0"))
        self.pg = None
        if self.world > 1:
            import torch.distributed as dist
            os.environ.setdefault("MASTER_ADDR", "127.0.0.1")
            dist.init_process_group(backend=backend)
            self.pg = dist

    def barrier(self):
        if self.pg:
            self.pg.barrier()

    def max(self, x: float) -> float:
        if not self.pg:
            return x
        import torch
        t = torch.tensor([x], dtype=torch.float64, device="cuda" if self.pg.get_backend() == "nccl" else "cpu")
        self.pg.all_reduce(t, op=self.pg.ReduceOp.MAX)
        return float(t.item())

    def close(self):
        if self.pg:
            self.pg.destroy_process_group()


# ------------------------------------------------------------------------------ clocks
class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled every 200 ms during the timed region."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.idx = gpu_index
        self.proc = None
        self.path = None

    def start(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                                          "-lms", "200", "-i", str(self.idx)], stdout=open(self.path, "w"),
                                         stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None
        time.sleep(0.3)

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        time.sleep(0.25)
        self.proc.terminate()
        self.proc.wait()
        rows = [r.split(",") for r in open(self.path).read().strip().splitlines() if r.count(",") >= 8]
        os.unlink(self.path)
        sm = [float(r[1]) for r in rows if r[1].strip().replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].strip().replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i].strip() == "Active"})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(rows)}


# --------------------------------------------------------------------------- GPU timing
def timed_steps(fn, steps: int, warmup: int, flush, stream, kernel_events=None):
    """Run `warmup` untimed calls, then `steps` calls each preceded by an L2 flush; return the
    per-step device times (ms) from CUDA events recorded on `stream`.  A GPU-side sleep is queued
    first so that the host enqueues every step before the GPU reaches them: the events then time
    device work only, not host launch gaps."""
    import torch
    for _ in range(warmup):
        fn()
    torch.cuda.synchronize()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
    kev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
    for ka, kb in kev:  # torch creates CUDA events lazily: record once so that their handles exist
        ka.record(stream)
        kb.record(stream)
    torch.cuda.synchronize()
    with torch.cuda.stream(stream):
        torch.cuda._sleep(int(4e7 + 2e6 * steps))  # ~20 ms + 1 ms per step at 2 GHz
        for (a, b), (ka, kb) in zip(ev, kev):
            flush()
            a.record(stream)
            if kernel_events is not None:
                kernel_events(ka, kb)
            fn()
            b.record(stream)
    torch.cuda.synchronize()
    if kernel_events is not None:
        timed_steps.kernel_ms = [ka.elapsed_time(kb) for ka, kb in kev]
    return [a.elapsed_time(b) for a, b in ev]


def w8a8_bytes(M, N, K, out_bytes=2):
    """Algorithmic bytes of one W8A8 linear: INT8 weights, bf16 input, output, fp32 scales."""
    return N * K + M * K * 2 + M * N * out_bytes + 4 * (N + M + K)


def bf16_bytes(M, N, K, out_bytes=2):
    return N * K * 2 + M * K * 2 + M * N * out_bytes


def ffn_bytes(M, int8):
    H, F = HIDDEN, INTER
    if int8:  # both linears; the intermediate counts as an INT8 write plus read
        return (2 * F * H + H * F) + M * H * 2 + 2 * M * F + M * H * 2 + 4 * (3 * F + 2 * H + 2 * M)
    return (2 * F * H + H * F) * 2 + M * H * 2 + 2 * M * F * 2 + M * H * 2


def run_ours(args, dist: Dist):
    import torch
    import synth
    from paper_2608_28003_gb300 import build as _build
    _build.build()
    from paper_2608_28003_gb300 import binding as B

    torch.cuda.set_device(dist.local)
    dev = torch.device("cuda", dist.local)
    stream = torch.cuda.current_stream()
    peaks = load_peaks()
    flush_buf = torch.empty(512 << 20, dtype=torch.uint8, device=dev)
    flush = lambda: flush_buf.zero_()  # noqa: E731  (512 MiB > 129 MB L2)

    # ---- lm_head weights (tied table) and its calibration statistic
    hc = synth.lm_head_case(512, seed=0)
    head_w = hc["w"].to(dev)
    q = B.prepare_weights(head_w, B.act_absmax(hc["calib"].to(dev)))
    head = B.HeadWeights(VOCAB, HIDDEN, q, head_w)
    x_all = hc["x"].to(dev)
    logits = torch.empty(512, VOCAB, dtype=torch.float32, device=dev)
    top1 = torch.empty(512 * 4, dtype=torch.int32, device=dev)  # slot i at 16 * i bytes (16-byte aligned)
    ws = B.Workspace(dev)

    # ---- headline: lm_head W8A8, M = 1, a different token row per step
    counter = [0]

    def head_step():
        i = counter[0] % 512
        counter[0] += 1
        B.lm_head(head, B.W8A8_PREC_W8A8, x_all[i:i + 1], logits=logits[i:i + 1], top1=top1[4 * i:4 * i + 1], ws=ws)

    head_step()
    torch.cuda.synchronize()
    clocks = ClockSampler(dist.local)
    dist.barrier()
    torch.cuda.synchronize()
    clocks.start()
    per_step = timed_steps(head_step, args.steps, args.warmup, flush, stream, kernel_events=B.set_kernel_events)
    kernel_ms = statistics.mean(timed_steps.kernel_ms)
    clk = clocks.stop()
    torch.cuda.synchronize()
    dist.barrier()
    ms_local = statistics.mean(per_step)
    ms = dist.max(ms_local)
    launches_per_step = 2  # per-token quantiser + weight-streaming GEMV

    hb = w8a8_bytes(1, VOCAB, HIDDEN, out_bytes=4)
    achieved = hb / (kernel_ms * 1e-3) / 1e9
    roofline = {"bound": "hbm", "achieved": round(achieved, 1), "peak": peaks["hbm_gbs"], "unit": "GB/s",
                "frac": round(achieved / peaks["hbm_gbs"], 4), "traffic": None,
                "peak_source": peaks["source"], "kernel": "gemv_dp4a_kernel<1,16> (W8A8 lm_head GEMV, M=1)",
                "kernel_us": round(kernel_ms * 1e3, 2), "algorithmic_bytes_per_launch": hb}

    # ---- e2e through the public API from pinned host memory
    x_host = hc["x"][:64].pin_memory()
    top_host = torch.empty(1, dtype=torch.int32).pin_memory()
    x_dev = torch.empty(1, HIDDEN, dtype=torch.bfloat16, device=dev)
    e2e_times = []
    for s in range(args.warmup + args.steps):
        flush()
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        x_dev.copy_(x_host[s % 64:s % 64 + 1], non_blocking=True)
        B.lm_head(head, B.W8A8_PREC_W8A8, x_dev, logits=logits[:1], top1=top1[:1], ws=ws)
        top_host.copy_(top1[:1], non_blocking=True)
        torch.cuda.current_stream().synchronize()
        if s >= args.warmup:
            e2e_times.append((time.perf_counter() - t0) * 1e3)
    e2e_ms = dist.max(statistics.mean(e2e_times))

    kernels = {} if args.no_sweep else sweep(B, dev, head, hc, flush, stream, peaks)

    return {
        "ms": ms, "per_step": per_step, "clocks": clk, "roofline": roofline, "launches": launches_per_step * args.steps,
        "e2e": {"value": round(e2e_ms, 4), "unit": "ms/token", "h2d_bytes_per_step": HIDDEN * 2,
                "d2h_bytes_per_step": 4, "clock": "host wall clock incl. copies and stream sync"},
        "kernels": kernels, "peaks": peaks,
    }


def sweep(B, dev, head, hc, flush, stream, peaks):
    """Per-call device time of every workload shape, W8A8 and bf16 (3 warm-up, 10 timed)."""
    import torch
    import synth
    out = {}
    hbm = peaks["hbm_gbs"]

    def rec(name, ms, flops, nbytes, kernel=False):
        """Per-call time; for single linears also the GEMM kernel alone (hook events) and the
        kernel's algorithmic GB/s against the measured HBM peak."""
        r = {"us": round(ms * 1e3, 2), "TOPS": round(flops / (ms * 1e-3) / 1e12, 3),
             "GBps": round(nbytes / (ms * 1e-3) / 1e9, 1), "hbm_frac": round(nbytes / (ms * 1e-3) / 1e9 / hbm, 4)}
        if kernel:
            km = statistics.mean(timed_steps.kernel_ms)
            r.update({"kernel_us": round(km * 1e3, 2), "kernel_GBps": round(nbytes / (km * 1e-3) / 1e9, 1),
                      "kernel_hbm_frac": round(nbytes / (km * 1e-3) / 1e9 / hbm, 4)})
        out[name] = r
    kev = B.set_kernel_events

    ws = B.Workspace(dev)
    # single linear (M = 16, 1152 -> 6912)
    c = synth.linear_case()
    q = B.prepare_weights(c["w"].to(dev), B.act_absmax(c["calib"].to(dev)))
    x = c["x"].to(dev)
    w = c["w"].to(dev)
    y = torch.empty(16, INTER, dtype=torch.bfloat16, device=dev)
    t = statistics.mean(timed_steps(lambda: B.linear(q, x, out=y, ws=ws), 10, 3, flush, stream, kev))
    rec("linear_w8a8_M16", t, 2 * 16 * INTER * HIDDEN, w8a8_bytes(16, INTER, HIDDEN), True)
    t = statistics.mean(timed_steps(lambda: B.linear_bf16(w, x, out=y, ws=ws), 10, 3, flush, stream, kev))
    rec("linear_bf16_M16", t, 2 * 16 * INTER * HIDDEN, bf16_bytes(16, INTER, HIDDEN), True)
    # FFN block
    fc = synth.ffn_case(2048, seed=0)
    gu = B.prepare_gate_up(fc["wg"].to(dev), fc["wu"].to(dev), B.act_absmax(fc["calib"].to(dev)))
    dn = B.prepare_weights(fc["wd"].to(dev), torch.from_numpy(fc["stat_h"]).to(dev))
    f = B.FfnWeights(HIDDEN, INTER, gu, dn, B.interleave_gate_up(fc["wg"].to(dev), fc["wu"].to(dev)), fc["wd"].to(dev))
    xf = fc["x"].to(dev)
    yf = torch.empty(2048, HIDDEN, dtype=torch.bfloat16, device=dev)
    for M in (1, 8, 64, 512, 2048):
        flops = 2 * M * 3 * INTER * HIDDEN
        for prec, tag in ((B.W8A8_PREC_W8A8, "w8a8"), (B.W8A8_PREC_BF16, "bf16")):
            t = statistics.mean(timed_steps(lambda: B.ffn_block(f, prec, xf[:M], out=yf[:M], ws=ws), 10, 3, flush, stream))
            rec(f"ffn_{tag}_M{M}", t, flops, ffn_bytes(M, prec == B.W8A8_PREC_W8A8))
    # lm_head
    xh = hc["x"].to(dev)
    lg = torch.empty(512, VOCAB, dtype=torch.float32, device=dev)
    tp = torch.empty(512, dtype=torch.int32, device=dev)
    for M in (1, 16, 128, 512):
        flops = 2 * M * VOCAB * HIDDEN
        t = statistics.mean(timed_steps(lambda: B.lm_head(head, B.W8A8_PREC_W8A8, xh[:M], logits=lg[:M], top1=tp[:M],
                                                          ws=ws), 10, 3, flush, stream, kev))
        rec(f"lm_head_w8a8_M{M}", t, flops, w8a8_bytes(M, VOCAB, HIDDEN, 4), True)
        t = statistics.mean(timed_steps(lambda: B.lm_head(head, B.W8A8_PREC_BF16, xh[:M], logits=lg[:M], top1=tp[:M],
                                                          ws=ws), 10, 3, flush, stream, kev))
        rec(f"lm_head_bf16_M{M}", t, flops, bf16_bytes(M, VOCAB, HIDDEN, 4), True)
    return out


# ------------------------------------------------------------------------- CPU oracle
def oracle_threads():
    try:
        from threadpoolctl import threadpool_info
        n = [i.get("num_threads", 1) for i in threadpool_info() if i.get("user_api") == "blas"]
        if n:
            return max(n)
    except Exception:
        pass
    return os.cpu_count()


def oracle_lm_head_sample(n_tokens: int):
    """Time the oracle's W8A8 lm_head (quantise, exact INT8 GEMM, dequantise, top-1) for
    `n_tokens` single-token calls.  Returns (ms per token, description)."""
    import synth
    from oracle import blocks as OB
    from oracle import w8a8 as OW
    hc = synth.lm_head_case(n_tokens, seed=0)
    prep = OW.prepare_weights(hc["w32"], OW.act_absmax(hc["calib32"]))
    times = []
    for i in range(n_tokens):
        t0 = time.perf_counter()
        OB.lm_head_w8a8(hc["x32"][i:i + 1], prep)
        times.append((time.perf_counter() - t0) * 1e3)
    return statistics.mean(times), times


def main():
    args = parse()
    if args.impl == "reference":
        dist = Dist("gloo")
        if dist.rank != 0:
            dist.close()
            return
        n = max(1, min(args.steps, 8))
        for _ in range(min(args.warmup, 1)):
            oracle_lm_head_sample(1)
        ms, times = oracle_lm_head_sample(n)
        cores = oracle_threads()
        line = {
            "impl": "reference", "metric": METRIC, "value": round(ms, 3), "unit": "ms/token", "n_gpus": args.gpus,
            "steps": n, "warmup": args.warmup, "ms_per_step": round(ms, 3), "higher_is_better": False,
            "scaling": "weak", "vs_baseline": None, "dtype": "int8/fp32 (f64 exact sums)", "data": "synthetic",
            "config": {"workload": "lm_head 1152->262144 W8A8 decode, M=1 (fp32 logits + top-1)", "global_batch": 1,
                       "seq_len": 1, "parallelism": "replicas"},
            "cpu_baseline": {"value": round(ms, 3), "unit": "ms/token", "cores": cores, "kind": "oracle",
                             "sample": f"{n} single-token lm_head calls of the numpy oracle"},
            "e2e": {"value": round(ms, 3), "unit": "ms/token", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
        }
        print(json.dumps(line))
        dist.close()
        return

    dist = Dist("nccl")
    res = run_ours(args, dist)
    cpu = None
    if dist.rank == 0 and args.gpus == 1:
        ms_cpu, _ = oracle_lm_head_sample(4)
        cpu = {"value": round(ms_cpu, 3), "unit": "ms/token", "cores": oracle_threads(), "kind": "oracle",
               "sample": "4 single-token W8A8 lm_head calls (1152 -> 262144) of the numpy oracle"}
    if dist.rank == 0:
        ms = res["ms"]
        line = {
            "metric": METRIC, "value": round(ms, 5), "unit": "ms/token", "n_gpus": args.gpus, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": round(ms, 5), "higher_is_better": False, "scaling": "weak",
            "vs_baseline": None, "dtype": "int8 (fp16-coded operands, fp32->int32 exact accumulation)",
            "data": "synthetic",
            "config": {"workload": "lm_head 1152->262144 W8A8 decode, M=1 (fp32 logits + top-1)", "global_batch": 1,
                       "seq_len": 1, "parallelism": f"replicas x{args.gpus}", "l2": "flushed (512 MiB write) before every step"},
            "aggregate_tok_s": round(args.gpus * 1e3 / ms, 1),
            "clocks": res["clocks"], "roofline": res["roofline"], "e2e": res["e2e"], "gpu_launches": res["launches"],
            "cpu_baseline": cpu, "kernels": res["kernels"],
        }
        print(json.dumps(line))
    dist.close()


if __name__ == "__main__":
    main()
