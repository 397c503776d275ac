"""Thin ctypes binding of libw8a8.so (argument marshalling only).

Every computation runs in the library's CUDA kernels; this module only turns torch tensors
(device memory owned by the caller) into the pointers and descriptors of ``include/w8a8.h``,
allocates output tensors and workspaces with torch, and raises on a non-OK status.  There is
no CPU fallback: if the library is missing or the device is not sm_103, calls raise.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass
from typing import Optional

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libw8a8.so")

W8A8_PREC_BF16 = 0
W8A8_PREC_W8A8 = 1
WS_RESERVED = 65536

STATUS = {0: "OK", 1: "ERR_INVALID_ARG", 2: "ERR_SHAPE", 3: "ERR_ALIGN", 4: "ERR_CUDA", 5: "ERR_UNSUPPORTED",
          6: "ERR_TIMEOUT", 7: "ERR_WORKSPACE"}


class W8A8Error(RuntimeError):
    def __init__(self, name, status, msg):
        super().__init__(f"{name} -> {STATUS.get(status, status)}: {msg}")
        self.status = status


_vp = ctypes.c_void_p
_i32 = ctypes.c_int
_f32 = ctypes.c_float
_sz = ctypes.c_size_t


class QWeightC(ctypes.Structure):
    _fields_ = [("n", ctypes.c_int32), ("k", ctypes.c_int32), ("wq", _vp), ("s_w", _vp), ("inv_delta", _vp),
                ("wq_f16", _vp)]


class DebugC(ctypes.Structure):
    _fields_ = [("xq", _vp), ("s_x", _vp), ("acc", _vp)]


class FfnC(ctypes.Structure):
    _fields_ = [("hidden", ctypes.c_int32), ("inter", ctypes.c_int32), ("gate_up", QWeightC), ("down", QWeightC),
                ("gate_up_bf16", _vp), ("down_bf16", _vp)]


class Fp8WeightC(ctypes.Structure):
    _fields_ = [("n", ctypes.c_int32), ("k", ctypes.c_int32), ("wq", _vp), ("s_w", _vp), ("inv_delta", _vp)]


class Fp8FfnC(ctypes.Structure):
    _fields_ = [("hidden", ctypes.c_int32), ("inter", ctypes.c_int32), ("gate_up", Fp8WeightC), ("down", Fp8WeightC)]


class HeadC(ctypes.Structure):
    _fields_ = [("vocab", ctypes.c_int32), ("hidden", ctypes.c_int32), ("q", QWeightC), ("bf16", _vp)]


class ModelCfgC(ctypes.Structure):
    _fields_ = [("layers", ctypes.c_int32), ("hidden", ctypes.c_int32), ("inter", ctypes.c_int32),
                ("n_q", ctypes.c_int32), ("n_kv", ctypes.c_int32), ("head_dim", ctypes.c_int32),
                ("vocab", ctypes.c_int32), ("eps", ctypes.c_float), ("rope_local", ctypes.c_float),
                ("rope_global", ctypes.c_float), ("window", ctypes.c_int32), ("n_global", ctypes.c_int32),
                ("global_layers", ctypes.c_int32 * 32), ("qk_norm", ctypes.c_int32), ("max_batch", ctypes.c_int32),
                ("max_seq", ctypes.c_int32), ("max_tokens", ctypes.c_int32)]


class LayerBf16C(ctypes.Structure):
    _fields_ = [("wqkv", _vp), ("wo", _vp), ("wgate", _vp), ("wup", _vp), ("wdown", _vp), ("ln_in", _vp),
                ("ln_post_attn", _vp), ("ln_pre_ffn", _vp), ("ln_post_ffn", _vp), ("q_norm", _vp), ("k_norm", _vp)]


class TraceC(ctypes.Structure):
    _fields_ = [("a_in", _vp), ("qkv", _vp), ("attn", _vp), ("y_o", _vp), ("a_ffn", _vp), ("h", _vp), ("y_f", _vp),
                ("r", _vp), ("a_fin", _vp), ("max_rows", ctypes.c_int32)]


class MaskC(ctypes.Structure):
    _fields_ = [("ffn_bits", ctypes.c_uint32), ("attn_bits", ctypes.c_uint32), ("lm", ctypes.c_int32)]


class AllocOptsC(ctypes.Structure):
    _fields_ = [("candidates", ctypes.POINTER(MaskC)), ("n_candidates", ctypes.c_int32), ("eval_tokens", _vp),
                ("eval_B", ctypes.c_int32), ("eval_T", ctypes.c_int32), ("decode_B", ctypes.c_int32),
                ("prefill_T", ctypes.c_int32), ("decode_steps", ctypes.c_int32), ("reps", ctypes.c_int32),
                ("min_top1", ctypes.c_float), ("max_ppl_delta", ctypes.c_float)]


class AllocReportC(ctypes.Structure):
    _fields_ = [("chosen", ctypes.c_int32), ("latency_ms", ctypes.POINTER(ctypes.c_float)),
                ("top1", ctypes.POINTER(ctypes.c_float)), ("ppl_delta", ctypes.POINTER(ctypes.c_float))]


class LayerAllocOptsC(ctypes.Structure):
    _fields_ = [("eval_tokens", _vp), ("eval_B", ctypes.c_int32), ("eval_T", ctypes.c_int32),
                ("decode_B", ctypes.c_int32), ("prefill_T", ctypes.c_int32), ("decode_steps", ctypes.c_int32),
                ("reps", ctypes.c_int32), ("min_top1", ctypes.c_float), ("max_ppl_delta", ctypes.c_float)]


class LayerAllocReportC(ctypes.Structure):
    _fields_ = [("chosen", MaskC), ("base_ms", ctypes.c_float), ("chosen_ms", ctypes.c_float),
                ("chosen_top1", ctypes.c_float), ("chosen_ppl_delta", ctypes.c_float),
                ("gain_ms", ctypes.POINTER(ctypes.c_float)), ("top1", ctypes.POINTER(ctypes.c_float)),
                ("ppl_delta", ctypes.POINTER(ctypes.c_float)), ("order", ctypes.POINTER(ctypes.c_int32)),
                ("n_order", ctypes.c_int32), ("n_accepted", ctypes.c_int32)]


_fp = ctypes.POINTER(ctypes.c_float)

# name -> (restype, argtypes)
SIGNATURES = {
    "w8a8_abi_version": (_i32, []),
    "w8a8_last_error": (ctypes.c_char_p, []),
    "w8a8_workspace_check": (_i32, [_vp, _vp]),
    "w8a8_set_kernel_events": (_i32, [_vp, _vp]),
    "w8a8_route_peak": (_i32, [_i32, ctypes.POINTER(ctypes.c_double), _vp]),
    "w8a8_act_absmax": (_i32, [_vp, _i32, _i32, _vp, _vp]),
    "w8a8_prepare_weights": (_i32, [_vp, _i32, _i32, _vp, _f32, _i32, _vp, _vp, _vp, _vp, _vp, _vp]),
    "w8a8_prepare_gate_up": (_i32, [_vp, _vp, _i32, _i32, _vp, _f32, _i32, _vp, _vp, _vp, _vp, _vp, _vp]),
    "w8a8_interleave_gate_up": (_i32, [_vp, _vp, _i32, _i32, _vp, _vp]),
    "w8a8_quantize_activations": (_i32, [_vp, _i32, _i32, _vp, _vp, _vp, _vp, _vp]),
    "w8a8_linear_workspace_size": (_i32, [_i32, _i32, _i32, ctypes.POINTER(_sz)]),
    "w8a8_linear": (_i32, [ctypes.POINTER(QWeightC), _vp, _i32, _vp, _vp, ctypes.POINTER(DebugC), _vp, _sz, _vp]),
    "w8a8_linear_noalloc_capacity": (_sz, []),
    "w8a8_linear_noalloc": (_i32, [ctypes.POINTER(QWeightC), _vp, _i32, _vp, _vp, _vp]),
    "w8a8_linear_noalloc_check": (_i32, [_vp]),
    "w8a8_linear_bf16_workspace_size": (_i32, [_i32, _i32, _i32, ctypes.POINTER(_sz)]),
    "w8a8_linear_bf16": (_i32, [_vp, _i32, _i32, _vp, _i32, _vp, _vp, _vp, _sz, _vp]),
    "w8a8_ffn_workspace_size": (_i32, [_i32, _i32, _i32, ctypes.POINTER(_sz)]),
    "w8a8_ffn_block": (_i32, [ctypes.POINTER(FfnC), _i32, _vp, _i32, _vp, _vp, _vp, _sz, _vp]),
    "w8a8_fp8_prepare_weights": (_i32, [_vp, _i32, _i32, _vp, _f32, _i32, _vp, _vp, _vp, _vp, _vp]),
    "w8a8_fp8_prepare_gate_up": (_i32, [_vp, _vp, _i32, _i32, _vp, _f32, _i32, _vp, _vp, _vp, _vp, _vp]),
    "w8a8_fp8_quantize_activations": (_i32, [_vp, _i32, _i32, _vp, _vp, _vp, _vp]),
    "w8a8_fp8_linear": (_i32, [ctypes.POINTER(Fp8WeightC), _vp, _i32, _vp, _vp, _vp, _vp, _vp, _sz, _vp]),
    "w8a8_fp8_ffn_block": (_i32, [ctypes.POINTER(Fp8FfnC), _vp, _i32, _vp, _vp, _vp, _sz, _vp]),
    "w8a8_lm_head_workspace_size": (_i32, [_i32, _i32, _i32, ctypes.POINTER(_sz)]),
    "w8a8_lm_head": (_i32, [ctypes.POINTER(HeadC), _i32, _vp, _i32, _vp, _vp, _vp, _sz, _vp]),
    "w8a8_model_create": (_i32, [ctypes.POINTER(ModelCfgC), ctypes.POINTER(LayerBf16C), _vp, _vp,
                                 ctypes.POINTER(_vp)]),
    "w8a8_model_destroy": (_i32, [_vp]),
    "w8a8_model_calibrate": (_i32, [_vp, _vp, _i32, _i32, _vp]),
    "w8a8_model_reset_calibration": (_i32, [_vp, _vp]),
    "w8a8_model_prepare": (_i32, [_vp, _f32, _i32, _vp]),
    "w8a8_model_stats_count": (_sz, [_vp]),
    "w8a8_model_get_stats": (_i32, [_vp, _fp]),
    "w8a8_model_set_stats": (_i32, [_vp, _fp]),
    "w8a8_set_layer_precision": (_i32, [_vp, _i32, _i32, _i32]),
    "w8a8_set_mask": (_i32, [_vp, ctypes.c_uint32, ctypes.c_uint32, _i32]),
    "w8a8_get_mask": (_i32, [_vp, ctypes.POINTER(ctypes.c_uint32), ctypes.POINTER(ctypes.c_uint32),
                             ctypes.POINTER(_i32)]),
    "w8a8_decoder_forward": (_i32, [_vp, _vp, _i32, _i32, _i32, _vp, _vp, _vp]),
    "w8a8_decoder_decode_step": (_i32, [_vp, _vp, _i32, _i32, _vp, _vp, _vp]),
    "w8a8_model_decode_kernels": (_i32, [_vp, _i32, _i32, ctypes.POINTER(ctypes.c_int32)]),
    "w8a8_decode_gemv_plan": (_i32, [_i32, _i32, _i32, _i32, _i32, _i32, _i32, ctypes.POINTER(ctypes.c_int32)]),
    "w8a8_stream_gemm_plan": (_i32, [_i32, _i32, _i32, _i32, _i32, ctypes.POINTER(ctypes.c_int32)]),
    "w8a8_tc_gemm_plan": (_i32, [_i32, _i32, _i32, _i32, _i32, _i32, _i32, ctypes.POINTER(ctypes.c_int32)]),
    "w8a8_model_set_trace": (_i32, [_vp, ctypes.POINTER(TraceC)]),
    "w8a8_token_nll": (_i32, [_vp, _vp, _i32, _i32, _vp, _vp]),
    "w8a8_choose_mask": (_i32, [_fp, _fp, _fp, ctypes.POINTER(ctypes.c_int32), _i32, _f32, _f32]),
    "w8a8_allocate_mask": (_i32, [_vp, ctypes.POINTER(AllocOptsC), ctypes.POINTER(AllocReportC), _vp]),
    "w8a8_greedy_order": (_i32, [_fp, _fp, _fp, _i32, _f32, _f32, ctypes.POINTER(ctypes.c_int32)]),
    "w8a8_sqnr_db": (_i32, [_vp, _vp, ctypes.c_size_t, ctypes.POINTER(ctypes.c_double), _vp]),
    "w8a8_sqnr_profile": (_i32, [_vp, _vp, _i32, _i32, ctypes.POINTER(MaskC), _i32, _fp, _fp, _vp]),
    "w8a8_allocate_layers": (_i32, [_vp, ctypes.POINTER(LayerAllocOptsC), ctypes.POINTER(LayerAllocReportC), _vp]),
}

_LIB = None


def lib() -> ctypes.CDLL:
    """Load libw8a8.so (built by ``paper_2608_28003_gb300.build.build()``); raise if it is absent."""
    global _LIB
    if _LIB is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is not built: run paper_2608_28003_gb300.build.build() "
                               "(the W8A8 path has no CPU fallback)")
        L = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in SIGNATURES.items():
            fn = getattr(L, name)
            fn.restype = res
            fn.argtypes = args
        _LIB = L
    return _LIB


def _check(name: str, status: int) -> None:
    if status != 0:
        raise W8A8Error(name, status, lib().w8a8_last_error().decode())


def _p(t: Optional[torch.Tensor]):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream=None):
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


def _bits(t: torch.Tensor) -> torch.Tensor:
    assert t.is_cuda and t.is_contiguous(), "tensors must be contiguous CUDA tensors"
    return t


# ------------------------------------------------------------------------------ workspace
class Workspace:
    """A zero-initialised device byte buffer, grown on demand (re-zeroed when regrown)."""

    def __init__(self, device=None):
        self.device = device or torch.device("cuda")
        self.buf = torch.zeros(WS_RESERVED, dtype=torch.uint8, device=self.device)

    def get(self, nbytes: int) -> torch.Tensor:
        if self.buf.numel() < nbytes:
            self.buf = torch.zeros(int(nbytes * 1.25) + 256, dtype=torch.uint8, device=self.device)
        return self.buf


_DEFAULT_WS = {}


def default_workspace() -> Workspace:
    dev = torch.cuda.current_device()
    if dev not in _DEFAULT_WS:
        _DEFAULT_WS[dev] = Workspace(torch.device("cuda", dev))
    return _DEFAULT_WS[dev]


def workspace_check(ws: "Workspace", stream=None) -> None:
    """Raise W8A8Error(ERR_TIMEOUT) if a kernel using `ws` recorded a device-side timeout."""
    _check("w8a8_workspace_check", lib().w8a8_workspace_check(_p(ws.buf), _stream(stream)))


def route_peak(route: int, stream=None) -> float:
    """Sustained TOPS of an exact integer route (0 dp4a, 1 mma.sync s8, 2 mma.sync fp16)."""
    out = ctypes.c_double(0.0)
    _check("w8a8_route_peak", lib().w8a8_route_peak(int(route), ctypes.byref(out), _stream(stream)))
    return out.value


def set_kernel_events(start, stop) -> None:
    """Record the torch.cuda.Events `start`/`stop` around the next weight-streaming GEMM kernel
    launched by this thread (measurement aid)."""
    _check("w8a8_set_kernel_events", lib().w8a8_set_kernel_events(
        ctypes.c_void_p(start.cuda_event) if start is not None else None,
        ctypes.c_void_p(stop.cuda_event) if stop is not None else None))


def _size(fn_name, *args) -> int:
    out = ctypes.c_size_t(0)
    _check(fn_name, getattr(lib(), fn_name)(*args, ctypes.byref(out)))
    return out.value


# ---------------------------------------------------------------------------- descriptors
@dataclass
class QWeight:
    """A prepared W8A8 weight (tensors owned here; the C descriptor points into them)."""
    wq: torch.Tensor
    s_w: torch.Tensor
    delta: torch.Tensor
    inv_delta: torch.Tensor
    wq_f16: Optional[torch.Tensor] = None

    @property
    def n(self):
        return self.wq.shape[0]

    @property
    def k(self):
        return self.wq.shape[1]

    def c(self) -> QWeightC:
        return QWeightC(self.n, self.k, self.wq.data_ptr(), self.s_w.data_ptr(), self.inv_delta.data_ptr(),
                        self.wq_f16.data_ptr() if self.wq_f16 is not None else None)


# ---------------------------------------------------------------------------- entry points
def abi_version() -> int:
    return lib().w8a8_abi_version()


def act_absmax(X: torch.Tensor, absmax: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
    T, K = X.shape
    if absmax is None:
        absmax = torch.zeros(K, dtype=torch.float32, device=X.device)
    _check("w8a8_act_absmax", lib().w8a8_act_absmax(_p(_bits(X)), T, K, _p(absmax), _stream(stream)))
    return absmax


def prepare_weights(W: torch.Tensor, act_stat: Optional[torch.Tensor], alpha: float = 0.5, smooth: bool = True,
                    want_f16: bool = False, stream=None) -> QWeight:
    N, K = W.shape
    dev = W.device
    q = QWeight(torch.empty(N, K, dtype=torch.int8, device=dev), torch.empty(N, dtype=torch.float32, device=dev),
                torch.empty(K, dtype=torch.float32, device=dev), torch.empty(K, dtype=torch.float32, device=dev),
                torch.empty(N, K, dtype=torch.float16, device=dev) if want_f16 else None)
    _check("w8a8_prepare_weights", lib().w8a8_prepare_weights(
        _p(_bits(W)), N, K, _p(act_stat), float(alpha), int(smooth), _p(q.wq), _p(q.s_w), _p(q.delta),
        _p(q.inv_delta), _p(q.wq_f16), _stream(stream)))
    return q


def prepare_gate_up(W_gate: torch.Tensor, W_up: torch.Tensor, act_stat: Optional[torch.Tensor], alpha: float = 0.5,
                    smooth: bool = True, want_f16: bool = False, stream=None) -> QWeight:
    F, H = W_gate.shape
    dev = W_gate.device
    q = QWeight(torch.empty(2 * F, H, dtype=torch.int8, device=dev),
                torch.empty(2 * F, dtype=torch.float32, device=dev),
                torch.empty(H, dtype=torch.float32, device=dev), torch.empty(H, dtype=torch.float32, device=dev),
                torch.empty(2 * F, H, dtype=torch.float16, device=dev) if want_f16 else None)
    _check("w8a8_prepare_gate_up", lib().w8a8_prepare_gate_up(
        _p(_bits(W_gate)), _p(_bits(W_up)), F, H, _p(act_stat), float(alpha), int(smooth), _p(q.wq), _p(q.s_w),
        _p(q.delta), _p(q.inv_delta), _p(q.wq_f16), _stream(stream)))
    return q


def interleave_gate_up(W_gate: torch.Tensor, W_up: torch.Tensor, stream=None) -> torch.Tensor:
    F, H = W_gate.shape
    out = torch.empty(2 * F, H, dtype=W_gate.dtype, device=W_gate.device)
    _check("w8a8_interleave_gate_up", lib().w8a8_interleave_gate_up(
        _p(_bits(W_gate)), _p(_bits(W_up)), F, H, _p(out), _stream(stream)))
    return out


def quantize_activations(X: torch.Tensor, inv_delta: torch.Tensor, stream=None):
    M, K = X.shape
    xq = torch.empty(M, K, dtype=torch.int8, device=X.device)
    xf = torch.empty(M, K, dtype=torch.float16, device=X.device)
    s_x = torch.empty(M, dtype=torch.float32, device=X.device)
    _check("w8a8_quantize_activations", lib().w8a8_quantize_activations(
        _p(_bits(X)), M, K, _p(inv_delta), _p(xq), _p(xf), _p(s_x), _stream(stream)))
    return xq, xf, s_x


def linear(w: QWeight, X: torch.Tensor, bias: Optional[torch.Tensor] = None, debug: bool = False,
           out: Optional[torch.Tensor] = None, ws: Optional[Workspace] = None, stream=None):
    M = X.shape[0]
    Y = out if out is not None else torch.empty(M, w.n, dtype=torch.bfloat16, device=X.device)
    nbytes = _size("w8a8_linear_workspace_size", M, w.n, w.k)
    buf = (ws or default_workspace()).get(nbytes)
    dbg = None
    dbg_t = None
    if debug:
        dbg_t = (torch.empty(M, w.k, dtype=torch.int8, device=X.device),
                 torch.empty(M, dtype=torch.float32, device=X.device),
                 torch.empty(M, w.n, dtype=torch.int32, device=X.device))
        dbg = DebugC(*(t.data_ptr() for t in dbg_t))
    wc = w.c()
    _check("w8a8_linear", lib().w8a8_linear(ctypes.byref(wc), _p(_bits(X)), M, _p(bias), _p(Y),
                                            ctypes.byref(dbg) if dbg is not None else None, _p(buf),
                                            buf.numel(), _stream(stream)))
    if debug:
        return Y, {"xq": dbg_t[0], "s_x": dbg_t[1], "acc": dbg_t[2]}
    return Y


def linear_noalloc(w: QWeight, X: torch.Tensor, bias: Optional[torch.Tensor] = None,
                   out: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
    """W8A8 linear on the library's built-in scratch array: for callers that cannot give a workspace.
    Calls on one device must not overlap on the GPU (they share the array)."""
    M = X.shape[0]
    Y = out if out is not None else torch.empty(M, w.n, dtype=torch.bfloat16, device=X.device)
    wc = w.c()
    _check("w8a8_linear_noalloc", lib().w8a8_linear_noalloc(ctypes.byref(wc), _p(_bits(X)), M, _p(bias), _p(Y),
                                                            _stream(stream)))
    return Y


def linear_bf16(W: torch.Tensor, X: torch.Tensor, bias: Optional[torch.Tensor] = None,
                out: Optional[torch.Tensor] = None, ws: Optional[Workspace] = None, stream=None) -> torch.Tensor:
    N, K = W.shape
    M = X.shape[0]
    Y = out if out is not None else torch.empty(M, N, dtype=torch.bfloat16, device=X.device)
    nbytes = _size("w8a8_linear_bf16_workspace_size", M, N, K)
    buf = (ws or default_workspace()).get(nbytes)
    _check("w8a8_linear_bf16", lib().w8a8_linear_bf16(_p(_bits(W)), N, K, _p(_bits(X)), M, _p(bias), _p(Y), _p(buf),
                                                      buf.numel(), _stream(stream)))
    return Y


@dataclass
class FfnWeights:
    hidden: int
    inter: int
    gate_up: Optional[QWeight] = None
    down: Optional[QWeight] = None
    gate_up_bf16: Optional[torch.Tensor] = None
    down_bf16: Optional[torch.Tensor] = None

    def c(self) -> FfnC:
        empty = QWeightC(0, 0, None, None, None, None)
        return FfnC(self.hidden, self.inter, self.gate_up.c() if self.gate_up else empty,
                    self.down.c() if self.down else empty,
                    self.gate_up_bf16.data_ptr() if self.gate_up_bf16 is not None else None,
                    self.down_bf16.data_ptr() if self.down_bf16 is not None else None)


def ffn_block(f: FfnWeights, precision: int, X: torch.Tensor, want_h: bool = False,
              out: Optional[torch.Tensor] = None, ws: Optional[Workspace] = None, stream=None):
    M = X.shape[0]
    Y = out if out is not None else torch.empty(M, f.hidden, dtype=torch.bfloat16, device=X.device)
    h = torch.empty(M, f.inter, dtype=torch.bfloat16, device=X.device) if want_h else None
    nbytes = _size("w8a8_ffn_workspace_size", M, f.hidden, f.inter)
    buf = (ws or default_workspace()).get(nbytes)
    fc = f.c()
    _check("w8a8_ffn_block", lib().w8a8_ffn_block(ctypes.byref(fc), int(precision), _p(_bits(X)), M, _p(Y), _p(h),
                                                  _p(buf), buf.numel(), _stream(stream)))
    return (Y, h) if want_h else Y


# ------------------------------------------------------------------------ FP8 (e4m3) variant
@dataclass
class Fp8Weight:
    """A prepared FP8 weight: e4m3 codes (uint8 bytes), per-channel scales, smoothing factors."""
    wq: torch.Tensor
    s_w: torch.Tensor
    delta: torch.Tensor
    inv_delta: torch.Tensor

    @property
    def n(self):
        return self.wq.shape[0]

    @property
    def k(self):
        return self.wq.shape[1]

    def c(self) -> Fp8WeightC:
        return Fp8WeightC(self.n, self.k, self.wq.data_ptr(), self.s_w.data_ptr(), self.inv_delta.data_ptr())


def _fp8_weight(rows: int, K: int, dev) -> Fp8Weight:
    return Fp8Weight(torch.empty(rows, K, dtype=torch.uint8, device=dev),
                     torch.empty(rows, dtype=torch.float32, device=dev),
                     torch.empty(K, dtype=torch.float32, device=dev), torch.empty(K, dtype=torch.float32, device=dev))


def fp8_prepare_weights(W: torch.Tensor, act_stat: Optional[torch.Tensor], alpha: float = 0.5, smooth: bool = True,
                        stream=None) -> Fp8Weight:
    N, K = W.shape
    q = _fp8_weight(N, K, W.device)
    _check("w8a8_fp8_prepare_weights", lib().w8a8_fp8_prepare_weights(
        _p(_bits(W)), N, K, _p(act_stat), float(alpha), int(smooth), _p(q.wq), _p(q.s_w), _p(q.delta),
        _p(q.inv_delta), _stream(stream)))
    return q


def fp8_prepare_gate_up(W_gate: torch.Tensor, W_up: torch.Tensor, act_stat: Optional[torch.Tensor],
                        alpha: float = 0.5, smooth: bool = True, stream=None) -> Fp8Weight:
    F, H = W_gate.shape
    q = _fp8_weight(2 * F, H, W_gate.device)
    _check("w8a8_fp8_prepare_gate_up", lib().w8a8_fp8_prepare_gate_up(
        _p(_bits(W_gate)), _p(_bits(W_up)), F, H, _p(act_stat), float(alpha), int(smooth), _p(q.wq), _p(q.s_w),
        _p(q.delta), _p(q.inv_delta), _stream(stream)))
    return q


def fp8_quantize_activations(X: torch.Tensor, inv_delta: torch.Tensor, stream=None):
    M, K = X.shape
    xq = torch.empty(M, K, dtype=torch.uint8, device=X.device)
    s_x = torch.empty(M, dtype=torch.float32, device=X.device)
    _check("w8a8_fp8_quantize_activations", lib().w8a8_fp8_quantize_activations(
        _p(_bits(X)), M, K, _p(inv_delta), _p(xq), _p(s_x), _stream(stream)))
    return xq, s_x


def fp8_linear(w: Fp8Weight, X: torch.Tensor, bias: Optional[torch.Tensor] = None, debug: bool = False,
               out: Optional[torch.Tensor] = None, ws: Optional[Workspace] = None, stream=None):
    M = X.shape[0]
    Y = out if out is not None else torch.empty(M, w.n, dtype=torch.bfloat16, device=X.device)
    buf = (ws or default_workspace()).get(_size("w8a8_linear_workspace_size", M, w.n, w.k))
    xq = torch.empty(M, w.k, dtype=torch.uint8, device=X.device) if debug else None
    s_x = torch.empty(M, dtype=torch.float32, device=X.device) if debug else None
    wc = w.c()
    _check("w8a8_fp8_linear", lib().w8a8_fp8_linear(ctypes.byref(wc), _p(_bits(X)), M, _p(bias), _p(Y), _p(xq),
                                                    _p(s_x), _p(buf), buf.numel(), _stream(stream)))
    return (Y, {"xq": xq, "s_x": s_x}) if debug else Y


@dataclass
class Fp8FfnWeights:
    hidden: int
    inter: int
    gate_up: Fp8Weight
    down: Fp8Weight

    def c(self) -> Fp8FfnC:
        return Fp8FfnC(self.hidden, self.inter, self.gate_up.c(), self.down.c())


def fp8_ffn_block(f: Fp8FfnWeights, X: torch.Tensor, want_h: bool = False, out: Optional[torch.Tensor] = None,
                  ws: Optional[Workspace] = None, stream=None):
    M = X.shape[0]
    Y = out if out is not None else torch.empty(M, f.hidden, dtype=torch.bfloat16, device=X.device)
    h = torch.empty(M, f.inter, dtype=torch.bfloat16, device=X.device) if want_h else None
    buf = (ws or default_workspace()).get(_size("w8a8_ffn_workspace_size", M, f.hidden, f.inter))
    fc = f.c()
    _check("w8a8_fp8_ffn_block", lib().w8a8_fp8_ffn_block(ctypes.byref(fc), _p(_bits(X)), M, _p(Y), _p(h), _p(buf),
                                                          buf.numel(), _stream(stream)))
    return (Y, h) if want_h else Y


@dataclass
class HeadWeights:
    vocab: int
    hidden: int
    q: Optional[QWeight] = None
    bf16: Optional[torch.Tensor] = None

    def c(self) -> HeadC:
        empty = QWeightC(0, 0, None, None, None, None)
        return HeadC(self.vocab, self.hidden, self.q.c() if self.q else empty,
                     self.bf16.data_ptr() if self.bf16 is not None else None)


def lm_head(hd: HeadWeights, precision: int, X: torch.Tensor, want_logits: bool = True,
            logits: Optional[torch.Tensor] = None, top1: Optional[torch.Tensor] = None,
            ws: Optional[Workspace] = None, stream=None):
    M = X.shape[0]
    if want_logits and logits is None:
        logits = torch.empty(M, hd.vocab, dtype=torch.float32, device=X.device)
    if top1 is None:
        top1 = torch.empty(M, dtype=torch.int32, device=X.device)
    nbytes = _size("w8a8_lm_head_workspace_size", M, hd.vocab, hd.hidden)
    buf = (ws or default_workspace()).get(nbytes)
    hc = hd.c()
    _check("w8a8_lm_head", lib().w8a8_lm_head(ctypes.byref(hc), int(precision), _p(_bits(X)), M,
                                              _p(logits) if want_logits else None, _p(top1), _p(buf), buf.numel(),
                                              _stream(stream)))
    return (logits if want_logits else None), top1


# ------------------------------------------------------------------------------- decoder
W8A8_SUB_FFN, W8A8_SUB_ATTN, W8A8_SUB_LM = 0, 1, 2


def _layer_bits(layers) -> int:
    return sum(1 << l for l in layers)


# Layer groups of the paper's precision masks (bit l = layer l of the 26): outer 5 + 5 layers,
# outer 10 + 10 layers, all 26 layers.
GROUP_BITS = {
    "none": 0,
    "5+5": _layer_bits(list(range(0, 5)) + list(range(21, 26))),
    "10+10": _layer_bits(list(range(0, 10)) + list(range(16, 26))),
    "all26": _layer_bits(range(26)),
}


def candidate_masks():
    """The 16 candidate masks of the allocation sweep: FFN group x attention group (none / all26)
    x lm_head (bf16 / W8A8), as (name, (ffn_bits, attn_bits, lm))."""
    out = []
    for ffn in ("none", "5+5", "10+10", "all26"):
        for att in ("none", "all26"):
            for lm in (0, 1):
                name = f"ffn={ffn} att={att} lm={'int8' if lm else 'bf16'}"
                out.append((name, (GROUP_BITS[ffn], GROUP_BITS[att], lm)))
    return out


def sqnr_db(y_ref: torch.Tensor, y_q: torch.Tensor, stream=None) -> float:
    """Eq. sqnr-ffn / sqnr-block of two fp32 device tensors of the same size (fp64 sums on the GPU)."""
    assert y_ref.dtype == torch.float32 and y_q.dtype == torch.float32 and y_ref.numel() == y_q.numel()
    out = ctypes.c_double()
    _check("w8a8_sqnr_db", lib().w8a8_sqnr_db(_p(y_ref.contiguous()), _p(y_q.contiguous()), y_ref.numel(),
                                              ctypes.byref(out), _stream(stream)))
    return out.value


def greedy_order(gain_ms, top1, ppl_delta, min_top1: float = 0.989, max_ppl_delta: float = 0.01) -> list:
    """The library's per-sublayer ranking rule on host arrays: the ranked sublayer indices."""
    n = len(gain_ms)
    arr = lambda v, t: (t * n)(*v)  # noqa: E731
    order = (ctypes.c_int32 * max(n, 1))()
    k = lib().w8a8_greedy_order(arr(gain_ms, ctypes.c_float), arr(top1, ctypes.c_float),
                                arr(ppl_delta, ctypes.c_float), n, float(min_top1), float(max_ppl_delta), order)
    return list(order[:k])


PLAN_FIELDS = ("taken", "slots", "rows_per_warp", "ctas", "ctas_per_sm", "consumer_warps", "subslices_per_stage",
               "steps", "stages", "stage_bytes", "x_bytes", "resid_bytes", "partial_bytes", "smem_bytes", "kpad",
               "subslices")
WEIGHT_KINDS = {"bf16": 0, "int8": 1, "fp8": 2}


def decode_gemv_plan(weight_kind: str, M: int, N: int, K: int, geglu: bool = False, fused_norm: bool = False,
                     sms: int = 152) -> dict:
    """The decode GEMV's launch plan for an [N, K] linear over M tokens (host only)."""
    out = (ctypes.c_int32 * len(PLAN_FIELDS))()
    _check("w8a8_decode_gemv_plan", lib().w8a8_decode_gemv_plan(WEIGHT_KINDS[weight_kind], M, N, K, int(geglu),
                                                                int(fused_norm), sms, out))
    return dict(zip(PLAN_FIELDS, list(out)))


STREAM_PLAN_FIELDS = ("dp4a", "whole", "slots", "blocks", "tokens_per_group", "token_groups", "row_groups",
                      "kc", "k_chunks", "ctas", "ctas_per_sm", "stages", "stage_bytes", "smem_bytes",
                      "partial_bytes")


def stream_gemm_plan(int8_weights: bool, M: int, N: int, K: int, sms: int = 152) -> dict:
    """The weight-streaming kernel's plan for an [N, K] linear over M tokens (host only)."""
    out = (ctypes.c_int32 * len(STREAM_PLAN_FIELDS))()
    _check("w8a8_stream_gemm_plan", lib().w8a8_stream_gemm_plan(int(int8_weights), M, N, K, sms, out))
    return dict(zip(STREAM_PLAN_FIELDS, list(out)))


TC_MODES = {"bf16": 0, "int8": 1, "fp8": 2}
EPILOGUES = {"bf16": 0, "geglu": 1, "f32": 2}


def tc_gemm_plan(mode: str, M: int, N: int, K: int, kind: str = "bf16", split_ok: bool = True,
                 sms: int = 152) -> tuple:
    """(pair, channels per tile, k parts) the tcgen05 GEMM takes for an [N, K] linear over M tokens."""
    out = (ctypes.c_int32 * 3)()
    _check("w8a8_tc_gemm_plan", lib().w8a8_tc_gemm_plan(TC_MODES[mode], M, N, K, EPILOGUES[kind], int(split_ok),
                                                        sms, out))
    return tuple(out)


def choose_mask(latency, top1, ppl_delta, n_int8, min_top1: float = 0.989, max_ppl_delta: float = 0.01) -> int:
    """The library's allocation rule on host arrays (index, or -1 if nothing is feasible)."""
    n = len(latency)
    arr = lambda v, t: (t * n)(*v)  # noqa: E731
    return lib().w8a8_choose_mask(arr(latency, ctypes.c_float), arr(top1, ctypes.c_float),
                                  arr(ppl_delta, ctypes.c_float), arr(n_int8, ctypes.c_int32), n,
                                  float(min_top1), float(max_ppl_delta))


@dataclass
class DecoderConfig:
    layers: int = 26
    hidden: int = 1152
    inter: int = 6912
    n_q: int = 4
    n_kv: int = 1
    head_dim: int = 256
    vocab: int = 262144
    eps: float = 1e-6
    rope_local: float = 10000.0
    rope_global: float = 1000000.0
    window: int = 1024
    global_layers: tuple = (0, 6, 12, 18)
    qk_norm: bool = True
    max_batch: int = 1
    max_seq: int = 2048
    max_tokens: int = 2048

    def c(self) -> ModelCfgC:
        g = (ctypes.c_int32 * 32)(*list(self.global_layers))
        return ModelCfgC(self.layers, self.hidden, self.inter, self.n_q, self.n_kv, self.head_dim, self.vocab,
                         self.eps, self.rope_local, self.rope_global, self.window, len(self.global_layers), g,
                         int(self.qk_norm), self.max_batch, self.max_seq, self.max_tokens)


class Decoder:
    """Handle on a w8a8_model.  Keeps the caller-owned weight tensors alive while the model lives.

    weights: dict of per-layer lists of bf16 CUDA tensors (wqkv, wo, wg, wu, wd) and "embed";
    norms: dict of per-layer lists of fp32 CUDA tensors (ln_in, ln_post_attn, ln_pre_ffn,
    ln_post_ffn, q_norm, k_norm) and "final_norm"."""

    def __init__(self, cfg: DecoderConfig, weights: dict, norms: dict):
        self.cfg = cfg
        self._keep = (weights, norms)
        layers = (LayerBf16C * cfg.layers)()
        for l in range(cfg.layers):
            layers[l] = LayerBf16C(*(t.data_ptr() for t in (
                weights["wqkv"][l], weights["wo"][l], weights["wg"][l], weights["wu"][l], weights["wd"][l],
                norms["ln_in"][l], norms["ln_post_attn"][l], norms["ln_pre_ffn"][l], norms["ln_post_ffn"][l],
                norms["q_norm"][l], norms["k_norm"][l])))
        h = ctypes.c_void_p()
        cc = cfg.c()
        _check("w8a8_model_create", lib().w8a8_model_create(ctypes.byref(cc), layers, _p(weights["embed"]),
                                                            _p(norms["final_norm"]), ctypes.byref(h)))
        self.h = h

    def close(self):
        if self.h:
            _check("w8a8_model_destroy", lib().w8a8_model_destroy(self.h))
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def calibrate(self, tokens: torch.Tensor, stream=None):
        B, T = tokens.shape
        _check("w8a8_model_calibrate", lib().w8a8_model_calibrate(self.h, _p(_bits(tokens)), B, T, _stream(stream)))

    def reset_calibration(self, stream=None):
        _check("w8a8_model_reset_calibration", lib().w8a8_model_reset_calibration(self.h, _stream(stream)))

    def get_stats(self):
        """Calibration statistics (host numpy fp32; layout of w8a8_model_get_stats)."""
        import numpy as np
        n = lib().w8a8_model_stats_count(self.h)
        out = np.zeros(n, dtype=np.float32)
        _check("w8a8_model_get_stats", lib().w8a8_model_get_stats(self.h, out.ctypes.data_as(_fp)))
        return out

    def set_stats(self, stats):
        import numpy as np
        s = np.ascontiguousarray(stats, dtype=np.float32)
        assert s.size == lib().w8a8_model_stats_count(self.h)
        _check("w8a8_model_set_stats", lib().w8a8_model_set_stats(self.h, s.ctypes.data_as(_fp)))

    def prepare(self, alpha: float = 0.5, smooth: bool = True, stream=None):
        _check("w8a8_model_prepare", lib().w8a8_model_prepare(self.h, float(alpha), int(smooth), _stream(stream)))

    def set_mask(self, ffn_bits: int = 0, attn_bits: int = 0, lm: bool = False):
        _check("w8a8_set_mask", lib().w8a8_set_mask(self.h, ffn_bits, attn_bits, int(lm)))

    def get_mask(self):
        f, a, l = ctypes.c_uint32(), ctypes.c_uint32(), ctypes.c_int32()
        _check("w8a8_get_mask", lib().w8a8_get_mask(self.h, ctypes.byref(f), ctypes.byref(a), ctypes.byref(l)))
        return f.value, a.value, l.value

    def set_layer_precision(self, layer: int, sublayer: int, precision: int):
        _check("w8a8_set_layer_precision", lib().w8a8_set_layer_precision(self.h, layer, sublayer, precision))

    def forward(self, tokens: torch.Tensor, start_pos: int = 0, want_logits: bool = True, stream=None):
        B, T = tokens.shape
        dev = tokens.device
        logits = torch.empty(B * T, self.cfg.vocab, dtype=torch.float32, device=dev) if want_logits else None
        top1 = torch.empty(B * T, dtype=torch.int32, device=dev)
        _check("w8a8_decoder_forward", lib().w8a8_decoder_forward(self.h, _p(_bits(tokens)), B, T, int(start_pos),
                                                                  _p(logits), _p(top1), _stream(stream)))
        return logits, top1

    def decode_step(self, tokens: torch.Tensor, pos: int, logits: Optional[torch.Tensor] = None,
                    top1: Optional[torch.Tensor] = None, stream=None):
        B = tokens.shape[0]
        if top1 is None:
            top1 = torch.empty(B, dtype=torch.int32, device=tokens.device)
        _check("w8a8_decoder_decode_step", lib().w8a8_decoder_decode_step(self.h, _p(_bits(tokens)), B, int(pos),
                                                                          _p(logits), _p(top1), _stream(stream)))
        return logits, top1

    TRACE_FIELDS = ("a_in", "qkv", "attn", "y_o", "a_ffn", "h", "y_f", "r", "a_fin")

    def set_trace(self, max_rows: Optional[int]):
        """Start tracing every layer's intermediate tensors of the following forward / decode calls
        (rows [0, M) of each call) into fresh device tensors, returned as a dict; None stops."""
        if max_rows is None:
            _check("w8a8_model_set_trace", lib().w8a8_model_set_trace(self.h, None))
            self._trace = None
            return None
        c, L, R = self.cfg, self.cfg.layers, int(max_rows)
        qkv = (c.n_q + 2 * c.n_kv) * c.head_dim
        dev = self._keep[0]["embed"].device
        bf = lambda w: torch.empty(L, R, w, dtype=torch.bfloat16, device=dev)  # noqa: E731
        t = {"a_in": bf(c.hidden), "qkv": bf(qkv), "attn": bf(c.n_q * c.head_dim), "y_o": bf(c.hidden),
             "a_ffn": bf(c.hidden), "h": bf(c.inter), "y_f": bf(c.hidden),
             "r": torch.empty(L, R, c.hidden, dtype=torch.float32, device=dev),
             "a_fin": torch.empty(R, c.hidden, dtype=torch.bfloat16, device=dev)}
        tc = TraceC(*(t[k].data_ptr() for k in self.TRACE_FIELDS), R)
        _check("w8a8_model_set_trace", lib().w8a8_model_set_trace(self.h, ctypes.byref(tc)))
        self._trace = t
        return t

    def decode_kernels(self, B: int, want_logits: bool = False) -> int:
        """Kernel launches of one decode step of B sequences under the current mask."""
        n = ctypes.c_int32()
        _check("w8a8_model_decode_kernels", lib().w8a8_model_decode_kernels(self.h, int(B), int(want_logits),
                                                                            ctypes.byref(n)))
        return n.value

    def allocate(self, candidates, eval_tokens: torch.Tensor, decode_B: int, prefill_T: int, decode_steps: int,
                 reps: int = 3, min_top1: float = 0.989, max_ppl_delta: float = 0.01, stream=None) -> dict:
        """Run the allocator over candidate masks [(ffn_bits, attn_bits, lm), ...]."""
        n = len(candidates)
        masks = (MaskC * n)(*[MaskC(f, a, int(l)) for f, a, l in candidates])
        eB, eT = eval_tokens.shape
        opts = AllocOptsC(masks, n, _bits(eval_tokens).data_ptr(), eB, eT, decode_B, prefill_T, decode_steps, reps,
                          float(min_top1), float(max_ppl_delta))
        lat, t1, pd = (ctypes.c_float * n)(), (ctypes.c_float * n)(), (ctypes.c_float * n)()
        rep = AllocReportC(-1, lat, t1, pd)
        _check("w8a8_allocate_mask", lib().w8a8_allocate_mask(self.h, ctypes.byref(opts), ctypes.byref(rep),
                                                              _stream(stream)))
        return {"chosen": rep.chosen, "latency_ms": list(lat), "top1": list(t1), "ppl_delta": list(pd)}

    def sqnr_profile(self, tokens: torch.Tensor, mask, isolated: bool, stream=None):
        """Per-layer block-output SQNR (dB, length L) and the lm_head logits' SQNR of mask =
        (ffn_bits, attn_bits, lm) over a prefill of tokens [B, T], isolated or propagated."""
        B, T = tokens.shape
        L = self.cfg.layers
        layer, lm = (ctypes.c_float * L)(), (ctypes.c_float * 1)()
        mk = MaskC(int(mask[0]), int(mask[1]), int(mask[2]))
        _check("w8a8_sqnr_profile", lib().w8a8_sqnr_profile(self.h, _p(_bits(tokens)), B, T, ctypes.byref(mk),
                                                            int(bool(isolated)), layer, lm, _stream(stream)))
        return list(layer), lm[0]

    def allocate_layers(self, eval_tokens: torch.Tensor, decode_B: int, prefill_T: int, decode_steps: int,
                        reps: int = 3, min_top1: float = 0.989, max_ppl_delta: float = 0.01, stream=None) -> dict:
        """Run the per-sublayer allocator (sublayer i: FFN of layer i for i < L, attention of layer
        i - L for i < 2L, lm_head for i = 2L); leaves the chosen mask set."""
        n = 2 * self.cfg.layers + 1
        eB, eT = eval_tokens.shape
        opts = LayerAllocOptsC(_bits(eval_tokens).data_ptr(), eB, eT, decode_B, prefill_T, decode_steps, reps,
                               float(min_top1), float(max_ppl_delta))
        gain, t1, pd = (ctypes.c_float * n)(), (ctypes.c_float * n)(), (ctypes.c_float * n)()
        order = (ctypes.c_int32 * n)()
        rep = LayerAllocReportC(MaskC(0, 0, 0), 0.0, 0.0, 0.0, 0.0, gain, t1, pd, order, 0, 0)
        _check("w8a8_allocate_layers", lib().w8a8_allocate_layers(self.h, ctypes.byref(opts), ctypes.byref(rep),
                                                                  _stream(stream)))
        c = rep.chosen
        return {"chosen": (c.ffn_bits, c.attn_bits, c.lm), "base_ms": rep.base_ms, "chosen_ms": rep.chosen_ms,
                "chosen_top1": rep.chosen_top1, "chosen_ppl_delta": rep.chosen_ppl_delta, "gain_ms": list(gain),
                "top1": list(t1), "ppl_delta": list(pd), "order": list(order[:rep.n_order]),
                "n_accepted": rep.n_accepted}


def token_nll(logits: torch.Tensor, targets: torch.Tensor, stream=None) -> torch.Tensor:
    M, V = logits.shape
    out = torch.empty(M, dtype=torch.float32, device=logits.device)
    _check("w8a8_token_nll", lib().w8a8_token_nll(_p(_bits(logits)), _p(_bits(targets)), M, V, _p(out),
                                                  _stream(stream)))
    return out
