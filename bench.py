#!/usr/bin/env python3
"""Benchmark of the W8A8 SmoothQuant hot path on GB300.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference] [--quick]

Prints ONE JSON line (rank 0).  The headline workload is decode of a 26-layer Gemma-3-1B-shaped
decoder (random-init bf16 weights, hidden 1152, 4 query / 1 KV heads of 256, FFN 6912, vocab
262144) under the precision mask "FFN 5+5 + lm_head" (the FFN blocks of the five outermost
layers at each end and lm_head in W8A8, everything else bf16), batch 1: a 128-token prefill,
then one step = one decode token (a CUDA-graph replay of the whole decoder, fp32 logits' top-1
included).  Tokens are seeded uniform ids, teacher-forced.  Every step streams about 1.46 GB of
weights, far more than the 129 MB L2, so no flush is needed between steps.  ``value`` = ms per
decoded token of the whole job (time, max over ranks, / tokens all ranks decoded; replicas only).

The same line carries:
  * ``masks``: per-mask decode ms/token, the latency change against the all-bf16 mask, Top-1
    agreement and perplexity change, for the 16 candidate masks, and the mask the library's
    allocator picks (Top-1 >= 98.9 %, perplexity change <= 1 %);
  * ``batches``: decode ms/step at batch 1, 8 and 32 and prefill of 128 and 2048 tokens for four
    masks;
  * ``kernels``: per-call time, TOPS and algorithmic GB/s of the single W8A8 linear (M = 16,
    1152 -> 6912), the FFN block (M in 1, 8, 64, 512, 2048) and lm_head (M in 1, 16, 128, 512),
    W8A8 and bf16 (L2 flushed before each call);
  * ``roofline`` of the decode step's dominant kernel (the row-owning GEMV on bf16 weights, by
    share of device time) against the measured HBM copy bandwidth, with the lm_head GEMV beside it;
  * ``e2e``: decode through the public API with the token copied in from pinned host memory
    and the top-1 copied back every step (host wall clock);
  * ``cpu_baseline``: the oracle on this host's cores for a bounded sample of the same decode.
``--impl reference`` times the oracle (CPU) decoding the same model under the same mask.
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
HIDDEN, INTER, VOCAB, LAYERS = 1152, 6912, 262144, 26
PREFILL = 128
# DRAM bytes read + written per launch of the decode GEMV, averaged over the roofline mix's launches
# (ncu over one decode step of `--profile-workload decode4`, the same shapes)
GEMV_MIX_TRAFFIC = 11170354
FALLBACK_HBM_GBS = 6800.0
FALLBACK_BF16_TFLOPS = 1900.0
WORKLOAD = ("decode, 26-layer Gemma-3-1B-shaped decoder (H 1152, 4q/1kv x 256, FFN 6912, V 262144), mask FFN 5+5 + "
            "lm_head W8A8, batch 1, prefill 128 then one token per step (teacher-forced)")


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=128)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--quick", action="store_true", help="headline only: skip the mask sweep and the tables")
    ap.add_argument("--profile-workload", choices=["decode4", "gemm", "linear16", "prefill4", "ffn2048", "mid4"], default=None,
                    help="run a small fixed workload for a profiler and exit (no JSON line): 'decode4' = five "
                         "batch-1 decode steps of a 4-layer decoder with the full shapes (FFN layers 0-1 and "
                         "lm_head W8A8); 'gemm' = three bf16, three W8A8 and three FP8 prefill linears, 2048 x 1152 -> 13824; "
                         "'linear16' = the single-linear workload (M 16, 1152 -> 6912) three times each as W8A8 "
                         "on INT8 codes, W8A8 with the fp16 code copy and bf16, then three W8A8 FFN blocks at M 8; "
                         "'prefill4' = a 2048-token prefill of a 4-layer decoder with the full shapes (bf16); "
                         "'ffn2048' = three W8A8 and three bf16 FFN blocks at M 2048; 'mid4' = two 128-token "
                         "prefills (batch 1) and three batch-32 decode steps of a 4-layer decoder with the full "
                         "shapes (bf16)")
    return ap.parse_args()


def profile_workload(name):
    """Small fixed workloads for ncu captures (a few GB on the device at most)."""
    import torch
    import synth
    from paper_2608_28003_gb300 import build
    build.build()
    from paper_2608_28003_gb300 import binding as B
    dev = torch.device("cuda", 0)
    global LAYERS
    if name == "prefill4":
        LAYERS = 4
        f32, bf, norms = synth.decoder_weights(4, seed=0, want_f32=False)
        dec, _ = make_decoder(B, dev, bf, norms, max_batch=1, max_seq=2048, max_tokens=2048)
        toks = torch.from_numpy(synth.tokens(2048, VOCAB, seed=2)).to(dev).view(1, 2048)
        for _ in range(2):
            dec.forward(toks, 0, want_logits=False)
        torch.cuda.synchronize()
        dec.close()
    elif name == "mid4":
        LAYERS = 4
        f32, bf, norms = synth.decoder_weights(4, seed=0, want_f32=False)
        dec, _ = make_decoder(B, dev, bf, norms, max_batch=32, max_seq=512, max_tokens=2048)
        toks = torch.from_numpy(synth.tokens(32 * 128, VOCAB, seed=2)).to(dev).view(32, 128)
        for _ in range(2):
            dec.forward(toks[:1].contiguous(), 0, want_logits=False)
        prefill(dec, toks, 2048)
        top = torch.zeros(32, dtype=torch.int32, device=dev)
        for s in range(3):
            dec.decode_step(top, 128 + s, top1=top)
        torch.cuda.synchronize()
        dec.close()
    elif name == "decode4":
        LAYERS = 4
        f32, bf, norms = synth.decoder_weights(4, seed=0, want_f32=False)
        dec, _ = make_decoder(B, dev, bf, norms, max_batch=1, max_seq=512, max_tokens=256)
        dec.calibrate(torch.from_numpy(synth.tokens(64, VOCAB, seed=1).reshape(1, 64)).to(dev))
        dec.prepare()
        dec.set_mask(0b0011, 0, 1)
        toks = torch.from_numpy(synth.tokens(300, VOCAB, seed=2)).to(dev)
        prefill(dec, toks[:PREFILL].view(1, PREFILL), 256)
        top = torch.zeros(16, dtype=torch.int32, device=dev)
        for s in range(5):
            dec.decode_step(toks[PREFILL + s:PREFILL + s + 1], PREFILL + s, top1=top[s:s + 1])
        torch.cuda.synchronize()
        dec.close()
    elif name == "ffn2048":
        fc = synth.ffn_case(2048, seed=0)
        gu = B.prepare_gate_up(fc["wg"].to(dev), fc["wu"].to(dev), B.act_absmax(fc["calib"].to(dev)), want_f16=True)
        dn = B.prepare_weights(fc["wd"].to(dev), torch.from_numpy(fc["stat_h"]).to(dev), want_f16=True)
        f = B.FfnWeights(HIDDEN, INTER, gu, dn, B.interleave_gate_up(fc["wg"].to(dev), fc["wu"].to(dev)),
                         fc["wd"].to(dev))
        x = fc["x"].to(dev)
        ws = B.Workspace(dev)
        y = torch.empty(2048, HIDDEN, dtype=torch.bfloat16, device=dev)
        for prec in (B.W8A8_PREC_W8A8, B.W8A8_PREC_BF16):
            for _ in range(3):
                B.ffn_block(f, prec, x, out=y, ws=ws)
        torch.cuda.synchronize()
    elif name == "linear16":
        c = synth.linear_case()
        stat = torch.from_numpy(c["calib32"]).abs().amax(0).to(dev)
        q = B.prepare_weights(c["w"].to(dev), stat)
        q16 = B.prepare_weights(c["w"].to(dev), stat, want_f16=True)
        x = c["x"].to(dev)
        ws = B.Workspace(dev)
        y = torch.empty(x.shape[0], q.n, dtype=torch.bfloat16, device=dev)
        for _ in range(3):
            B.linear(q, x, out=y, ws=ws)  # INT8 codes only: the streaming kernel
        for _ in range(3):
            B.linear(q16, x, out=y, ws=ws)  # with the fp16 code copy: the tensor-core GEMM
        for _ in range(3):
            B.linear_bf16(c["w"].to(dev), x, out=y, ws=ws)
        _, wg = synth.weight(INTER, HIDDEN, seed=3)
        _, wu = synth.weight(INTER, HIDDEN, seed=4)
        _, wd = synth.weight(HIDDEN, INTER, seed=5)
        _, x8, _ = synth.activations(8, HIDDEN, 8, seed=6)
        x8 = x8.to(dev)
        ones_h, ones_f = torch.ones(HIDDEN, device=dev), torch.ones(INTER, device=dev)
        f = B.FfnWeights(HIDDEN, INTER, gate_up=B.prepare_gate_up(wg.to(dev), wu.to(dev), ones_h),
                         down=B.prepare_weights(wd.to(dev), ones_f))
        y8 = torch.empty(8, HIDDEN, dtype=torch.bfloat16, device=dev)
        for _ in range(3):
            B.ffn_block(f, B.W8A8_PREC_W8A8, x8, out=y8, ws=ws)
        torch.cuda.synchronize()
    else:
        M, N, K = 2048, 2 * INTER, HIDDEN
        _, w = synth.weight(N, K, seed=1)
        _, x, _ = synth.activations(M, K, 8, seed=2)
        w, x = w.to(dev), x.to(dev)
        ws = B.Workspace(dev)
        y = torch.empty(M, N, dtype=torch.bfloat16, device=dev)
        q = B.prepare_weights(w, B.act_absmax(x), want_f16=True)
        q8 = B.fp8_prepare_weights(w, B.act_absmax(x))
        for _ in range(3):
            B.linear_bf16(w, x, out=y, ws=ws)
        for _ in range(3):
            B.linear(q, x, out=y, ws=ws)
        for _ in range(3):
            B.fp8_linear(q8, x, out=y, ws=ws)
        torch.cuda.synchronize()
    print("ok")


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
    """Replicas: every rank runs the same workload on its own GPU; only timings are reduced."""

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


def whole_job_ms_per_token(max_ms_total: float, tokens_per_rank: int, world: int) -> float:
    """Time-like whole-job figure: the slowest rank's time over the tokens all ranks decoded."""
    return max_ms_total / (tokens_per_rank * world)


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
def _events(n):
    import torch
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(n)]
    s = torch.cuda.current_stream()
    for e in ev:  # torch creates CUDA events lazily: record once so that their handles exist
        e.record(s)
    return ev


def gpu_sleep_for(steps: int, ms_per_step: float):
    """Queue a GPU-side sleep long enough for the host to enqueue every timed step before the
    GPU reaches them, so that the events time device work only, not host launch gaps."""
    import torch
    torch.cuda._sleep(int(2e6 * (20 + steps * max(ms_per_step, 0.05) * 1.5)))  # ~2e6 cycles per ms


def timed_steps(fn, steps: int, warmup: int, flush, stream, kernel_events=None):
    """`warmup` untimed calls, then `steps` calls each preceded by an L2 flush; per-step device
    times (ms) from CUDA events on `stream`."""
    import torch
    for _ in range(warmup):
        fn()
    torch.cuda.synchronize()
    ev = [(a, b) for a, b in zip(_events(steps), _events(steps))]
    kev = [(a, b) for a, b in zip(_events(steps), _events(steps))]
    torch.cuda.synchronize()
    with torch.cuda.stream(stream):
        gpu_sleep_for(steps, 1.0)
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


def decode_weight_bytes(ffn_bits: int, attn_bits: int, lm: int) -> int:
    """Weight bytes one decode token streams under a mask (INT8 = 1 byte, bf16 = 2 bytes)."""
    qkv, o = (4 + 2) * 256 * HIDDEN, HIDDEN * 4 * 256
    ffn = 3 * INTER * HIDDEN
    total = 0
    for l in range(LAYERS):
        total += (qkv + o) * (1 if (attn_bits >> l) & 1 else 2)
        total += ffn * (1 if (ffn_bits >> l) & 1 else 2)
    return total + VOCAB * HIDDEN * (1 if lm else 2)


# -------------------------------------------------------------------------- the decoder
def make_decoder(B, dev, bf, norms, max_batch, max_seq, max_tokens):
    import torch
    w = {k: [t.to(dev) for t in v] if isinstance(v, list) else v.to(dev) for k, v in bf.items()}
    n = {k: [torch.from_numpy(a).to(dev) for a in v] if isinstance(v, list) else torch.from_numpy(v).to(dev)
         for k, v in norms.items()}
    cfg = B.DecoderConfig(layers=LAYERS, max_batch=max_batch, max_seq=max_seq, max_tokens=max_tokens)
    return B.Decoder(cfg, w, n), w


def prefill(dec, toks, max_tokens):
    """Prefill tokens [B, T] from position 0 in chunks of at most max_tokens rows."""
    Bn, T = toks.shape
    chunk = max(1, max_tokens // Bn)
    for t0 in range(0, T, chunk):
        dec.forward(toks[:, t0:t0 + chunk].contiguous(), t0, want_logits=False)


def decode_ms(dec, Bn, steps, warmup, pos0):
    """Greedy decode of Bn sequences after a prefill ending at pos0: per-step device time (ms)."""
    import torch
    dev = torch.device("cuda", torch.cuda.current_device())
    tok = torch.zeros(max(4, Bn), dtype=torch.int32, device=dev)
    for s in range(warmup):
        dec.decode_step(tok[:Bn], pos0 + s, top1=tok[:Bn])
    torch.cuda.synchronize()
    e0, e1 = _events(2)
    torch.cuda.synchronize()
    gpu_sleep_for(steps, 1.0)
    e0.record()
    for s in range(steps):
        dec.decode_step(tok[:Bn], pos0 + warmup + s, top1=tok[:Bn])
    e1.record()
    torch.cuda.synchronize()
    return e0.elapsed_time(e1) / steps


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
    K, W = args.steps, args.warmup
    want_cpu = dist.rank == 0 and args.gpus == 1

    # ---- weights (seeded), calibration (5 x 128 tokens of stream seed 1), preparation
    t_setup = time.time()
    f32, bf, norms = synth.decoder_weights(LAYERS, seed=0, want_f32=want_cpu)
    max_seq = max(2048 + 256 + 64, PREFILL + 2 * (W + K) + 8)  # the mask grid decodes 256 steps after 2048
    dec, wdev = make_decoder(B, dev, bf, norms, max_batch=32, max_seq=max_seq, max_tokens=2048)
    calib = torch.from_numpy(synth.tokens(5 * PREFILL, VOCAB, seed=1).reshape(5, PREFILL)).to(dev)
    dec.calibrate(calib)
    dec.prepare()
    torch.cuda.synchronize()
    setup_s = time.time() - t_setup

    g = B.GROUP_BITS
    head_mask = (g["5+5"], 0, 1)
    dec.set_mask(*head_mask)
    stream_toks = synth.tokens(PREFILL + 2 * (W + K) + 8, VOCAB, seed=2)
    toks_dev = torch.from_numpy(stream_toks).to(dev)
    prefill(dec, toks_dev[:PREFILL].view(1, PREFILL), 2048)
    top = torch.zeros(W + K + 4, dtype=torch.int32, device=dev)

    def step(s):  # token s of the stream after the prefill, at position PREFILL + s
        dec.decode_step(toks_dev[PREFILL + s:PREFILL + s + 1], PREFILL + s, top1=top[s:s + 1])

    # ---- headline: K decode tokens, device-timed
    for s in range(W):
        step(s)
    torch.cuda.synchronize()
    kernels_per_step = dec.decode_kernels(1)
    ev = _events(K + 1)
    torch.cuda.synchronize()
    clocks = ClockSampler(dist.local)
    clocks.start()
    dist.barrier()
    torch.cuda.synchronize()
    gpu_sleep_for(K, 1.0)
    for s in range(K):
        ev[s].record(stream)
        step(W + s)
    ev[K].record(stream)
    torch.cuda.synchronize()
    dist.barrier()
    clk = clocks.stop()
    total_ms = ev[0].elapsed_time(ev[K])
    per_step = [ev[i].elapsed_time(ev[i + 1]) for i in range(K)]
    ms = whole_job_ms_per_token(dist.max(total_ms), K, dist.world)
    wbytes = decode_weight_bytes(*head_mask)

    # ---- e2e: token from pinned host memory in, top-1 back to pinned host memory, every step
    host_tok = torch.from_numpy(stream_toks).pin_memory()
    host_top = torch.zeros(1, dtype=torch.int32).pin_memory()
    tok_in = torch.zeros(4, dtype=torch.int32, device=dev)
    top_out = torch.zeros(4, dtype=torch.int32, device=dev)
    p0 = PREFILL + W + K
    e2e = []
    for s in range(W + K):
        i = p0 + s
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        tok_in[:1].copy_(host_tok[i:i + 1], non_blocking=True)
        dec.decode_step(tok_in[:1], i, top1=top_out[:1])
        host_top.copy_(top_out[:1], non_blocking=True)
        stream.synchronize()
        if s >= W:
            e2e.append((time.perf_counter() - t0) * 1e3)
    e2e_ms = whole_job_ms_per_token(dist.max(sum(e2e)), K, dist.world)

    # ---- roofline: the decode step's dominant kernel by share of device time (the ncu launch list),
    # the row-owning decode GEMV, over every one of its launches in a step under the headline mask:
    # 26 q/k/v (1152 -> 1536) and 26 o (1024 -> 1152) on bf16 weights, gate/up + GeGLU (1152 ->
    # 2 x 6912) and down (6912 -> 1152) on the 16 bf16 and the 10 W8A8 FFN layers (K1 fused into the
    # W8A8 ones).  Each shape is launched as in the decode step, timed alone with events around the
    # kernel, L2 flushed before each launch; achieved = the mix's algorithmic bytes / its kernel time.
    # L2 flush: write 512 MiB (> 129 MB L2), then read another 512 MiB so that the write-backs of the
    # dirty lines happen before the timed kernel, not during it
    flush_buf = torch.empty(512 << 20, dtype=torch.uint8, device=dev)
    flush_rd = torch.ones(128 << 20, dtype=torch.float32, device=dev)
    flush_sum = torch.empty((), dtype=torch.float32, device=dev)

    def flush():
        flush_buf.zero_()
        torch.sum(flush_rd, dim=0, out=flush_sum)

    ws = B.Workspace(dev)
    stats = torch.from_numpy(dec.get_stats()).to(dev)
    stride = 2 * HIDDEN + 1024 + INTER  # per layer: q/k/v, o, gate/up, down input statistics
    st5 = stats[5 * stride:6 * stride]
    gu_stat, down_stat = st5[HIDDEN + 1024:2 * HIDDEN + 1024].contiguous(), st5[2 * HIDDEN + 1024:].contiguous()
    wg, wu, wd = wdev["wg"][5], wdev["wu"][5], wdev["wd"][5]
    f_bf = B.FfnWeights(HIDDEN, INTER, gate_up_bf16=B.interleave_gate_up(wg, wu), down_bf16=wd)
    f_i8 = B.FfnWeights(HIDDEN, INTER, gate_up=B.prepare_gate_up(wg, wu, gu_stat), down=B.prepare_weights(wd, down_stat))
    n_i8 = bin(head_mask[0]).count("1")
    n_bf = LAYERS - n_i8

    def xrow(k, seed):
        return torch.from_numpy(synth.activations(1, k, 8, seed=seed)[0]).to(torch.bfloat16).to(dev)

    x_h, x_q, x_f = xrow(HIDDEN, 1), xrow(1024, 2), xrow(INTER, 3)
    y_h, y_qkv = torch.empty(1, HIDDEN, dtype=torch.bfloat16, device=dev), torch.empty(1, 1536, dtype=torch.bfloat16,
                                                                                       device=dev)
    wq5, wo5 = wdev["wqkv"][5], wdev["wo"][5]
    mix = [("qkv bf16", 26, lambda: B.linear_bf16(wq5, x_h, out=y_qkv, ws=ws), bf16_bytes(1, 1536, HIDDEN)),
           ("o bf16", 26, lambda: B.linear_bf16(wo5, x_q, out=y_h, ws=ws), bf16_bytes(1, HIDDEN, 1024)),
           ("gate/up bf16", n_bf, lambda: B.ffn_block(f_bf, B.W8A8_PREC_BF16, x_h, out=y_h, ws=ws),
            bf16_bytes(1, 2 * INTER, HIDDEN, out_bytes=1)),
           ("down bf16", n_bf, lambda: B.linear_bf16(wd, x_f, out=y_h, ws=ws), bf16_bytes(1, HIDDEN, INTER)),
           ("gate/up W8A8", n_i8, lambda: B.ffn_block(f_i8, B.W8A8_PREC_W8A8, x_h, out=y_h, ws=ws),
            w8a8_bytes(1, 2 * INTER, HIDDEN, out_bytes=1)),
           ("down W8A8", n_i8, lambda: B.linear(f_i8.down, x_f, out=y_h, ws=ws), w8a8_bytes(1, HIDDEN, INTER))]
    parts, tot_bytes, tot_us, n_launch = {}, 0.0, 0.0, 0
    for name, count, fn, nbytes in mix:
        if count == 0:
            continue
        # the hook's events bracket the next library launch: the GEMV itself (for the FFN block, its
        # first launch, gate/up + GeGLU)
        timed_steps(fn, max(K, 20), 3, flush, stream, kernel_events=B.set_kernel_events)
        us = statistics.mean(timed_steps.kernel_ms) * 1e3
        parts[name] = {"launches_per_step": count, "kernel_us": round(us, 2), "bytes": nbytes,
                       "GBps": round(nbytes / (us * 1e-6) / 1e9, 1)}
        tot_bytes += count * nbytes
        tot_us += count * us
        n_launch += count
    isolated = {"GBps": round(tot_bytes / (tot_us * 1e-6) / 1e9, 1), "kernel_us": round(tot_us / n_launch, 2),
                "launch_mix": parts,
                "timing": "CUDA events around the kernel on its stream, each shape launched alone as in the "
                          "decode step, L2 flushed (512 MiB written, then 512 MiB read) before each launch; "
                          "per-launch figures are the mix's averages"}

    # The same 104 launches chained as in the decode step: every layer's q/k/v, o and FFN (gate/up +
    # GeGLU, down) on that layer's own weights (bf16, or W8A8 on the mask's FFN layers), recorded
    # once as a CUDA graph (programmatic dependent launch between the kernels, nothing else in
    # between) and replayed back to back; 1.15 GB of weights per replay stream through the 129 MB
    # L2.  Average launch duration = replay time / 104.
    f_layers = []
    for l in range(LAYERS):
        wgl, wul, wdl = wdev["wg"][l], wdev["wu"][l], wdev["wd"][l]
        if (head_mask[0] >> l) & 1:
            stl = stats[l * stride:(l + 1) * stride]
            f_layers.append(B.FfnWeights(
                HIDDEN, INTER, gate_up=B.prepare_gate_up(wgl, wul, stl[HIDDEN + 1024:2 * HIDDEN + 1024].contiguous()),
                down=B.prepare_weights(wdl, stl[2 * HIDDEN + 1024:].contiguous())))
        else:
            f_layers.append(B.FfnWeights(HIDDEN, INTER, gate_up_bf16=B.interleave_gate_up(wgl, wul), down_bf16=wdl))
    chain_bytes = 0
    for l in range(LAYERS):
        i8 = (head_mask[0] >> l) & 1
        chain_bytes += bf16_bytes(1, 1536, HIDDEN) + bf16_bytes(1, HIDDEN, 1024)
        chain_bytes += (w8a8_bytes(1, 2 * INTER, HIDDEN, out_bytes=1) + w8a8_bytes(1, HIDDEN, INTER) if i8 else
                        bf16_bytes(1, 2 * INTER, HIDDEN, out_bytes=1) + bf16_bytes(1, HIDDEN, INTER))

    def chain():
        for l in range(LAYERS):
            B.linear_bf16(wdev["wqkv"][l], x_h, out=y_qkv, ws=ws)
            B.linear_bf16(wdev["wo"][l], x_q, out=y_h, ws=ws)
            B.ffn_block(f_layers[l], B.W8A8_PREC_W8A8 if (head_mask[0] >> l) & 1 else B.W8A8_PREC_BF16, x_h, out=y_h,
                        ws=ws)

    cap = torch.cuda.Stream()  # graphs are captured on a side stream
    with torch.cuda.stream(cap):
        chain()  # every kernel's attributes set before capture
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=cap):
        chain()
    for _ in range(3):
        graph.replay()
    torch.cuda.synchronize()
    reps = max(K, 20)
    c0, c1 = _events(2)
    with torch.cuda.stream(stream):
        gpu_sleep_for(reps, 1.0)
        c0.record(stream)
        for _ in range(reps):
            graph.replay()
        c1.record(stream)
    torch.cuda.synchronize()
    chain_us = c0.elapsed_time(c1) * 1e3 / reps
    del graph
    achieved = chain_bytes / (chain_us * 1e-6) / 1e9
    roofline = {"bound": "hbm", "achieved": round(achieved, 1), "peak": peaks["hbm_gbs"], "unit": "GB/s",
                "frac": round(achieved / peaks["hbm_gbs"], 4), "traffic": GEMV_MIX_TRAFFIC,
                "peak_source": peaks["source"],
                "kernel": "gemv_small_kernel (decode row-owning GEMV, all %d launches of a step)" % n_launch,
                "kernel_us": round(chain_us / n_launch, 2), "algorithmic_bytes_per_launch": round(chain_bytes / n_launch),
                "timing": "the step's %d GEMV launches chained as in the decode step (each layer's own weights, "
                          "programmatic dependent launch, one CUDA graph) and replayed %d times back to back; CUDA "
                          "events on the launching stream around the replays; average launch duration = replay "
                          "time / %d" % (n_launch, reps, n_launch),
                "isolated_launches": isolated}

    # the lm_head GEMV (W8A8, one token) on the same terms, for comparison
    lm_stat = stats[-HIDDEN:].contiguous()
    q_lm = B.prepare_weights(wdev["embed"], lm_stat, want_f16=True)
    head = B.HeadWeights(VOCAB, HIDDEN, q_lm, wdev["embed"])
    _, xh = synth.normed_rows(512, HIDDEN, seed=0)
    xh = xh.to(dev)
    logits = torch.empty(512, VOCAB, dtype=torch.float32, device=dev)
    top1 = torch.empty(512 * 4, dtype=torch.int32, device=dev)  # slot i at 16 * i bytes (16-byte aligned)
    ctr = [0]

    def head_call():
        i = ctr[0] % 512
        ctr[0] += 1
        B.lm_head(head, B.W8A8_PREC_W8A8, xh[i:i + 1], logits=logits[i:i + 1], top1=top1[4 * i:4 * i + 1], ws=ws)

    timed_steps(head_call, max(K, 20), 3, flush, stream, kernel_events=B.set_kernel_events)
    kernel_ms = statistics.mean(timed_steps.kernel_ms)
    hb = w8a8_bytes(1, VOCAB, HIDDEN, out_bytes=4)
    roofline["lm_head_gemv"] = {"kernel": "gemv_dp4a_kernel<1,16> (lm_head W8A8, M=1, 1152 -> 262144)",
                                "kernel_us": round(kernel_ms * 1e3, 2), "bytes": hb,
                                "GBps": round(hb / (kernel_ms * 1e-3) / 1e9, 1),
                                "frac": round(hb / (kernel_ms * 1e-3) / 1e9 / peaks["hbm_gbs"], 4)}

    out = {"ms": ms, "total_ms": total_ms, "per_step": per_step, "clocks": clk, "roofline": roofline,
           "launches": kernels_per_step * K, "kernels_per_step": kernels_per_step,
           "e2e": {"value": round(e2e_ms, 5), "unit": "ms/token", "h2d_bytes_per_step": 4, "d2h_bytes_per_step": 4,
                   "clock": "host wall clock per step: pinned H2D token copy, decode step, D2H top-1 copy, sync"},
           "weight_gb_per_token": round(wbytes / 1e9, 4),
           "weight_gbps": round(wbytes / (statistics.median(per_step) * 1e-3) / 1e9, 1),
           "setup_s": round(setup_s, 1), "peaks": peaks, "f32": f32, "norms": norms}

    if not args.quick:
        out["masks"] = mask_sweep(B, dec, dev)
        out["masks_grid"] = mask_grid(B, dec, dev)
        out["batches"] = batch_table(B, dec, dev)
        out["kernels"] = sweep(B, dev, head, xh, flush, stream, peaks)
        out["sqnr"] = sqnr_table(B, dec, dev)
    dec.close()
    return out


def mask_sweep(B, dec, dev):
    """The library's allocator over the 16 candidate masks: Top-1 agreement and perplexity change
    against the all-bf16 decoder on 4 x 128 eval tokens (stream seed 2), decode ms/token at
    batch 1 after a 128-token prefill (median of 3 runs of 64 greedy steps); then the
    per-sublayer allocator (single-sublayer masks timed over 3 runs of 32 steps, greedy additions
    under the same budget)."""
    import torch
    import synth
    names, cands = zip(*B.candidate_masks())
    ev = torch.from_numpy(synth.tokens(4 * PREFILL, VOCAB, seed=2, stream=1).reshape(4, PREFILL)).to(dev)
    t0 = time.time()
    rep = dec.allocate(list(cands), ev, decode_B=1, prefill_T=PREFILL, decode_steps=64, reps=3)
    base = rep["latency_ms"][0]  # candidate 0: all bf16
    rows = []
    for i, (n, (f, a, l)) in enumerate(zip(names, cands)):
        t = rep["latency_ms"][i]
        rows.append({"mask": n, "ms_per_token": round(t, 5), "latency_change_pct": round(100 * (t / base - 1), 2),
                     "speedup_vs_bf16": round(base / t, 4), "top1": round(rep["top1"][i], 5),
                     "ppl_delta": round(rep["ppl_delta"][i], 5), "weight_gb": round(decode_weight_bytes(f, a, l) / 1e9, 4)})
    ch = rep["chosen"]
    out = {"rows": rows, "chosen": names[ch] if ch >= 0 else None, "rule": "Top-1 >= 0.989, ppl change <= 0.01",
           "seconds": round(time.time() - t0, 1)}
    # below the groups: the per-sublayer allocator on the same stream and budget
    t0 = time.time()
    lr = dec.allocate_layers(ev, decode_B=1, prefill_T=PREFILL, decode_steps=32, reps=3)
    f, a, l = lr["chosen"]
    out["per_sublayer"] = {
        "ffn_layers": [i for i in range(LAYERS) if f >> i & 1], "attn_layers": [i for i in range(LAYERS) if a >> i & 1],
        "lm_head": bool(l), "ranked": len(lr["order"]), "accepted": lr["n_accepted"],
        "bf16_ms_per_token": round(lr["base_ms"], 5), "ms_per_token": round(lr["chosen_ms"], 5),
        "speedup_vs_bf16": round(lr["base_ms"] / lr["chosen_ms"], 4), "top1": round(lr["chosen_top1"], 5),
        "ppl_delta": round(lr["chosen_ppl_delta"], 5), "weight_gb": round(decode_weight_bytes(f, a, l) / 1e9, 4),
        "seconds": round(time.time() - t0, 1)}
    return out


def mask_grid(B, dec, dev):
    """The allocation sweep's grid: the 16 candidate masks timed at decode batch 1, 8 and 32 after a
    prefill of 128 and of 2048 tokens (256 greedy decode steps, one run each), with the allocator's
    choice per cell at the paper's budget (Top-1 >= 98.9 %, perplexity change <= 1 %) and, marked
    synthetic, at a budget a random-init decoder can meet (Top-1 >= 85 %, perplexity change <= 5 %):
    its flat logits put every quantised mask below the paper's budget."""
    import torch
    import synth
    names, cands = zip(*B.candidate_masks())
    n_int8 = [bin(f).count("1") + bin(a).count("1") + int(l) for f, a, l in cands]
    ev = torch.from_numpy(synth.tokens(4 * PREFILL, VOCAB, seed=2, stream=1).reshape(4, PREFILL)).to(dev)
    t0 = time.time()
    out = {}
    for Bn in (1, 8, 32):
        for T in (128, 2048):
            rep = dec.allocate(list(cands), ev, decode_B=Bn, prefill_T=T, decode_steps=256, reps=1)
            lat = rep["latency_ms"]
            base = lat[0]
            syn = B.choose_mask(lat, rep["top1"], rep["ppl_delta"], n_int8, min_top1=0.85, max_ppl_delta=0.05)
            out[f"B{Bn}_prefill{T}"] = {
                "ms_per_step": {nm: round(t, 4) for nm, t in zip(names, lat)},
                "speedup_vs_bf16": {nm: round(base / t, 4) for nm, t in zip(names, lat)},
                "chosen": names[rep["chosen"]] if rep["chosen"] >= 0 else None,
                "chosen_synthetic_budget": names[syn] if syn >= 0 else None}
    out["top1"] = {nm: round(v, 5) for nm, v in zip(names, rep["top1"])}
    out["ppl_delta"] = {nm: round(v, 5) for nm, v in zip(names, rep["ppl_delta"])}
    out["budget"] = "paper: Top-1 >= 0.989, ppl change <= 0.01; synthetic: Top-1 >= 0.85, ppl change <= 0.05"
    out["seconds"] = round(time.time() - t0, 1)
    dec.set_mask(B.GROUP_BITS["5+5"], 0, 1)  # the headline mask again
    return out


def sqnr_table(B, dec, dev):
    """SQNR diagnostics (Eq. sqnr-block per decoder layer, Eq. sqnr-ffn on the logits) of four
    masks over a 4 x 128-token prefill of the evaluation stream, isolated and propagated, with
    SmoothQuant (alpha 0.5) and with delta = 1 (no smoothing); the model is re-prepared with
    smoothing afterwards."""
    import torch
    import synth
    g = B.GROUP_BITS
    masks = {"ffn 5+5 + lm": (g["5+5"], 0, 1), "ffn all26 + lm": (g["all26"], 0, 1),
             "att all26": (0, g["all26"], 0), "ffn all26 + att all26 + lm": (g["all26"], g["all26"], 1)}
    toks = torch.from_numpy(synth.tokens(4 * PREFILL, VOCAB, seed=2, stream=1).reshape(4, PREFILL)).to(dev)
    t0 = time.time()
    out = {}
    r2 = lambda v: round(v, 2) if v != float("inf") else None  # noqa: E731  (None: layer left in bf16)
    for smooth in (True, False):
        dec.prepare(0.5, smooth)
        rows = {}
        for name, m in masks.items():
            row = {}
            for mode in ("isolated", "propagated"):
                layer, lm = dec.sqnr_profile(toks, m, isolated=mode == "isolated")
                fin = [v for v in layer if v != float("inf")]
                row[mode] = {"layers_db": [r2(v) for v in layer], "min_db": r2(min(fin)) if fin else None,
                             "lm_head_logits_db": r2(lm)}
            rows[name] = row
        out["smoothquant_alpha_0.5" if smooth else "delta_1"] = rows
    dec.prepare(0.5, True)
    # the single linear (M 16, 1152 -> 6912, 8 outlier channels x20, delta from its own input):
    # the W8A8 output against the bf16 pass-through's, with and without smoothing
    c = synth.linear_case()
    x, w = c["x"].to(dev), c["w"].to(dev)
    stat = torch.from_numpy(c["calib32"]).abs().amax(0).to(dev)
    y_ref = B.linear_bf16(w, x).float()
    lin = {}
    for smooth in (True, False):
        q = B.prepare_weights(w, stat, 0.5, smooth)
        lin["smoothquant_alpha_0.5" if smooth else "delta_1"] = round(B.sqnr_db(y_ref, B.linear(q, x).float()), 2)
    out["single_linear_db"] = lin
    out["seconds"] = round(time.time() - t0, 1)
    return out


def batch_table(B, dec, dev):
    """Decode ms/step at batch 1, 8, 32 (prefill 128, 16 greedy steps after 3 warm-ups) and prefill
    time of 128 and 2048 tokens (batch 1), for four masks."""
    import torch
    import synth
    g = B.GROUP_BITS
    masks = {"bf16": (0, 0, 0), "ffn 5+5 + lm": (g["5+5"], 0, 1), "ffn all26 + lm": (g["all26"], 0, 1),
             "ffn all26 + att all26 + lm": (g["all26"], g["all26"], 1)}
    out = {}
    pre = torch.from_numpy(synth.tokens(32 * 2048, VOCAB, seed=3).reshape(32, 2048)).to(dev)
    for name, m in masks.items():
        dec.set_mask(*m)
        r = {}
        for Bn in (1, 8, 32):
            prefill(dec, pre[:Bn, :PREFILL], 2048)
            t = decode_ms(dec, Bn, 16, 3, PREFILL)
            r[f"decode_B{Bn}_ms_per_step"] = round(t, 4)
            r[f"decode_B{Bn}_tok_s"] = round(Bn * 1e3 / t, 1)
        for T in (PREFILL, 2048):
            x = pre[:1, :T].contiguous()
            dec.forward(x, 0, want_logits=False)
            e0, e1 = _events(2)
            torch.cuda.synchronize()
            e0.record()
            for _ in range(3):
                dec.forward(x, 0, want_logits=False)
            e1.record()
            torch.cuda.synchronize()
            t = e0.elapsed_time(e1) / 3
            r[f"prefill_T{T}_ms"] = round(t, 3)
            r[f"prefill_T{T}_tok_s"] = round(T * 1e3 / t, 1)
        out[name] = r
    dec.set_mask(g["5+5"], 0, 1)
    return out


def sweep(B, dev, head, xh, flush, stream, peaks):
    """Per-call device time of the single linear, FFN block and lm_head shapes, W8A8 and bf16
    (3 warm-up, 10 timed, L2 flushed before each call)."""
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
    c = synth.linear_case()
    q = B.prepare_weights(c["w"].to(dev), B.act_absmax(c["calib"].to(dev)), want_f16=True)
    x = c["x"].to(dev)
    w = c["w"].to(dev)
    y = torch.empty(16, INTER, dtype=torch.bfloat16, device=dev)
    t = statistics.mean(timed_steps(lambda: B.linear(q, x, out=y, ws=ws), 10, 3, flush, stream, kev))
    rec("linear_w8a8_M16", t, 2 * 16 * INTER * HIDDEN, w8a8_bytes(16, INTER, HIDDEN), True)
    t = statistics.mean(timed_steps(lambda: B.linear_bf16(w, x, out=y, ws=ws), 10, 3, flush, stream, kev))
    rec("linear_bf16_M16", t, 2 * 16 * INTER * HIDDEN, bf16_bytes(16, INTER, HIDDEN), True)
    q8 = B.fp8_prepare_weights(w, B.act_absmax(c["calib"].to(dev)))
    t = statistics.mean(timed_steps(lambda: B.fp8_linear(q8, x, out=y, ws=ws), 10, 3, flush, stream, kev))
    rec("linear_fp8_M16", t, 2 * 16 * INTER * HIDDEN, w8a8_bytes(16, INTER, HIDDEN), True)
    fc = synth.ffn_case(2048, seed=0)
    gu = B.prepare_gate_up(fc["wg"].to(dev), fc["wu"].to(dev), B.act_absmax(fc["calib"].to(dev)), want_f16=True)
    dn = B.prepare_weights(fc["wd"].to(dev), torch.from_numpy(fc["stat_h"]).to(dev), want_f16=True)
    f = B.FfnWeights(HIDDEN, INTER, gu, dn, B.interleave_gate_up(fc["wg"].to(dev), fc["wu"].to(dev)), fc["wd"].to(dev))
    xf = fc["x"].to(dev)
    yf = torch.empty(2048, HIDDEN, dtype=torch.bfloat16, device=dev)
    stat_in = B.act_absmax(fc["calib"].to(dev))
    f8 = B.Fp8FfnWeights(HIDDEN, INTER, B.fp8_prepare_gate_up(fc["wg"].to(dev), fc["wu"].to(dev), stat_in),
                         B.fp8_prepare_weights(fc["wd"].to(dev), torch.from_numpy(fc["stat_h"]).to(dev)))
    cmp = {}
    for M in (1, 8, 64, 512, 2048):
        flops = 2 * M * 3 * INTER * HIDDEN
        row = {}
        for tag, fn in (("w8a8", lambda: B.ffn_block(f, B.W8A8_PREC_W8A8, xf[:M], out=yf[:M], ws=ws)),
                        ("bf16", lambda: B.ffn_block(f, B.W8A8_PREC_BF16, xf[:M], out=yf[:M], ws=ws)),
                        ("fp8", lambda: B.fp8_ffn_block(f8, xf[:M], out=yf[:M], ws=ws))):
            t = statistics.mean(timed_steps(fn, 10, 3, flush, stream))
            rec(f"ffn_{tag}_M{M}", t, flops, ffn_bytes(M, tag != "bf16"))
            row[f"{tag}_us"] = out[f"ffn_{tag}_M{M}"]["us"]
        row["w8a8_vs_bf16"] = round(row["bf16_us"] / row["w8a8_us"], 3)
        row["fp8_vs_bf16"] = round(row["bf16_us"] / row["fp8_us"], 3)
        cmp[f"M{M}"] = row
    out["ffn_fp8_int8_bf16"] = cmp
    # the exact integer routes' sustained rates (the rooflines of the INT8 paths): best of three
    rp = {}
    for route, name in ((0, "dp4a"), (1, "mma_sync_s8"), (2, "mma_sync_f16_on_int8_codes")):
        rp[name] = round(max(B.route_peak(route) for _ in range(3)), 1)
    rp["tcgen05_kind_f16_on_int8_codes"] = peaks.get("bf16_tflops")
    rp["note"] = ("TOPS; tcgen05 kind::f16 runs fp16 operands at the bf16 rate, so the W8A8 prefill GEMM's "
                  "route peak is the measured bf16 GEMM peak; FP8 (kind::f8f6f4) is twice it (nominal ratio)")
    out["int8_route_peaks"] = rp
    # the prefill GEMM alone (gate/up shape as a plain linear, 2048 x 1152 -> 13824): its kernel's
    # tensor rate against its route's peak (bf16 and INT8-as-fp16: the measured bf16 peak; FP8: twice it)
    Mg, Ng = 2048, 2 * INTER
    _, wg = synth.weight(Ng, HIDDEN, seed=1)
    _, xg, _ = synth.activations(Mg, HIDDEN, 8, seed=2)
    wg, xg = wg.to(dev), xg.to(dev)
    yg = torch.empty(Mg, Ng, dtype=torch.bfloat16, device=dev)
    qg = B.prepare_weights(wg, B.act_absmax(xg), want_f16=True)
    q8g = B.fp8_prepare_weights(wg, B.act_absmax(xg))
    flops = 2 * Mg * Ng * HIDDEN
    bf = peaks["bf16_tflops"]
    for tag, fn, pk in (("w8a8", lambda: B.linear(qg, xg, out=yg, ws=ws), bf),
                        ("bf16", lambda: B.linear_bf16(wg, xg, out=yg, ws=ws), bf),
                        ("fp8", lambda: B.fp8_linear(q8g, xg, out=yg, ws=ws), 2 * bf)):
        t = statistics.mean(timed_steps(fn, 10, 3, flush, stream, kev))
        nm = f"gemm_{tag}_2048x1152x13824"
        rec(nm, t, flops, (w8a8_bytes if tag != "bf16" else bf16_bytes)(Mg, Ng, HIDDEN), True)
        kt = out[nm]["kernel_us"] * 1e-6
        out[nm].update({"kernel_TOPS": round(flops / kt / 1e12, 1), "route_peak_TOPS": round(pk, 1),
                        "route_frac": round(flops / kt / 1e12 / pk, 4)})
    del wg, xg, yg, qg, q8g
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


def oracle_decode_sample(f32, norms, n_tokens: int, warmup: int = 1, prefill_T: int = 16):
    """The oracle decoder (26 layers, full Gemma-3-1B shapes, the bench's weights) under the
    FFN 5+5 + lm_head mask: statistics from 16 calibration tokens (stream seed 1), a prefill of
    `prefill_T` tokens, then `warmup` untimed and `n_tokens` timed single-token decode steps.
    Returns per-token times (ms)."""
    import synth
    from oracle import decoder as OD
    from oracle import masks as OM
    if f32 is None:
        f32, _, norms = synth.decoder_weights(LAYERS, seed=0)
    ow = dict(f32)
    ow.update(norms)
    cfg = OD.DecoderConfig(layers=LAYERS)
    od = OD.OracleDecoder(cfg, ow, batch=1, max_len=prefill_T + warmup + n_tokens + 1)
    od.calibrate([synth.tokens(16, VOCAB, seed=1).reshape(1, 16)])
    od.prepare()
    mask = OM.make_mask("5+5", "none", True)
    toks = synth.tokens(prefill_T + warmup + n_tokens, VOCAB, seed=2)
    od.forward(toks[None, :prefill_T], 0, mask=mask, want_logits=False)
    times = []
    for s in range(warmup + n_tokens):
        p = prefill_T + s
        t0 = time.perf_counter()
        od.forward(toks[None, p:p + 1], p, mask=mask)
        if s >= warmup:
            times.append((time.perf_counter() - t0) * 1e3)
    return times


def reference_line(args, times, n):
    ms = statistics.mean(times)
    cores = oracle_threads()
    sample = (f"oracle decoder, 26 layers at full shapes, mask FFN 5+5 + lm_head: prefill 16 tokens, "
              f"{min(args.warmup, 1)} untimed + {n} timed decode tokens")
    return {
        "impl": "reference", "metric": METRIC, "value": round(ms, 3), "unit": "ms/token", "n_gpus": args.gpus,
        "steps": n, "warmup": min(args.warmup, 1), "ms_per_step": round(ms, 3), "higher_is_better": False,
        "scaling": "weak", "vs_baseline": None, "dtype": "int8/fp32 (f64 exact sums)", "data": "synthetic",
        "config": {"workload": WORKLOAD, "global_batch": 1, "seq_len": 1, "parallelism": "replicas"},
        "cpu_baseline": {"value": round(ms, 3), "unit": "ms/token", "cores": cores, "kind": "oracle", "sample": sample},
        "e2e": {"value": round(ms, 3), "unit": "ms/token", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }


def main():
    args = parse()
    if args.profile_workload:
        profile_workload(args.profile_workload)
        return
    if args.impl == "reference":
        dist = Dist("gloo")
        if dist.rank != 0:
            dist.close()
            return
        n = max(1, min(args.steps, 16))
        times = oracle_decode_sample(None, None, n, warmup=min(args.warmup, 1))
        print(json.dumps(reference_line(args, times, n)))
        dist.close()
        return

    dist = Dist("nccl")
    res = run_ours(args, dist)
    cpu = None
    if dist.rank == 0 and args.gpus == 1:
        times = oracle_decode_sample(res["f32"], res["norms"], 4)
        cpu = {"value": round(statistics.mean(times), 3), "unit": "ms/token", "cores": oracle_threads(),
               "kind": "oracle",
               "sample": "oracle decoder, 26 layers at full shapes, same weights and mask: prefill 16 tokens, "
                         "1 untimed + 4 timed decode tokens"}
    if dist.rank == 0:
        ms = res["ms"]
        line = {
            "metric": METRIC, "value": round(ms, 5), "unit": "ms/token", "n_gpus": args.gpus, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": round(res["total_ms"] / args.steps, 5), "higher_is_better": False,
            "scaling": "weak", "vs_baseline": None,
            "dtype": "int8 W8A8 (exact int32 sums) on the masked sublayers, bf16 (fp32 sums) elsewhere",
            "data": "synthetic",
            "config": {"workload": WORKLOAD, "global_batch": args.gpus, "seq_len": 1, "prefill": PREFILL,
                       "parallelism": f"replicas x{args.gpus}",
                       "l2": "not flushed: each step streams the mask's weights (1.46 GB) through the 129 MB L2",
                       "weights": "random-init bf16 N(0, 0.02), seed 0; calibration 5 x 128 tokens (seed 1)"},
            "median_step_ms": round(statistics.median(res["per_step"]), 5),
            "weight_gb_per_token": res["weight_gb_per_token"], "weight_gbps_median_step": res["weight_gbps"],
            "clocks": res["clocks"], "roofline": res["roofline"], "e2e": res["e2e"], "gpu_launches": res["launches"],
            "kernels_per_step": res["kernels_per_step"], "cpu_baseline": cpu,
            "masks": res.get("masks"), "masks_grid": res.get("masks_grid"), "batches": res.get("batches"),
            "kernels": res.get("kernels"),
            "sqnr": res.get("sqnr"), "setup_s": res["setup_s"],
        }
        print(json.dumps(line))
    dist.close()


if __name__ == "__main__":
    main()
