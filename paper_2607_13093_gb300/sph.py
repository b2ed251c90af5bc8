"""Thin Python binding of libsph (include/sph.h) over ctypes.

Argument marshalling only: tensors are passed as device pointers with their
leading dimensions, PyTorch supplies the device memory and the stream, and
every step of the computation runs in the library's CUDA kernels.  There is
no fallback: if the library is not built, importing this module raises.

Functions carry the C names (sph_partial_logits, sph_fuse_sample,
sph_verify_draft, ...) and take torch tensors; `Context` bundles a context
handle with the current torch stream.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional

import torch

_LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "_lib",
                         "libsph.so")

SPH_OK = 0
STATUS_NAMES = {0: "SPH_OK", 1: "SPH_ERR_INVALID_ARG", 2: "SPH_ERR_UNSUPPORTED",
                3: "SPH_ERR_CUDA", 4: "SPH_ERR_TIMEOUT", 5: "SPH_ERR_OOM"}
SPH_DTYPE_BF16, SPH_DTYPE_FP8_E4M3 = 0, 1
SPH_ACT_FP32, SPH_ACT_BF16 = 0, 1
SPH_OPT_TC_MIN_ROWS, SPH_OPT_SPIN_LIMIT = 0, 1
SPH_OPT_TC_SCHEDULE, SPH_OPT_TC_STAGES, SPH_OPT_TC_BLOCK_K, SPH_OPT_TC_MAX_BN = 2, 3, 4, 5
SPH_OPT_TC_TILE_M = 6
SPH_OPT_TC_FINISH_WAIT = 7
SPH_OPT_SAMPLER = 8
SPH_OPT_CHECK_IDS = 9
SPH_OPT_SPLIT_QUANTIZE = 10
SPH_OPT_TC_PAIR = 11
SPH_OPT_ENDPOINT_Z = 12
SPH_OPT_ENDPOINT_ROWS_M = 13
SPH_OPT_GEMV_QUANTIZE = 14
SPH_SAMPLER_CDF, SPH_SAMPLER_GUMBEL = 0, 1

_c_void_p = ctypes.c_void_p
_i64 = ctypes.c_int64
_u64 = ctypes.c_uint64
_int = ctypes.c_int
_f32 = ctypes.c_float
_sz = ctypes.c_size_t

PROF_CLASSES = 8
PROF_NAMES = ("cloud_gemm", "quantize", "local_gemm", "sample", "verify",
              "prep", "reserved6", "reserved7")


class sph_profile(ctypes.Structure):
    _fields_ = [("ms", ctypes.c_double * PROF_CLASSES),
                ("calls", ctypes.c_int64 * PROF_CLASSES),
                ("launches", ctypes.c_int64)]


PLAN_FIELDS = ("tensor_core", "row_blocks", "block_rows", "tile_ids", "tiles",
               "k_blocks", "stages", "grid", "whole_tiles", "planes", "gemv_rows", "pair",
               "rows_m", "epilogue_stats")


class sph_plan(ctypes.Structure):
    _fields_ = [(f, ctypes.c_int32) for f in PLAN_FIELDS]


# name -> (restype, argtypes), mirroring include/sph.h
_SIGNATURES = {
    "sph_status_string": (ctypes.c_char_p, [_int]),
    "sph_last_error": (ctypes.c_char_p, [_c_void_p]),
    "sph_create": (_int, [_int, _c_void_p, ctypes.POINTER(_c_void_p)]),
    "sph_destroy": (_int, [_c_void_p]),
    "sph_set_stream": (_int, [_c_void_p, _c_void_p]),
    "sph_sync": (_int, [_c_void_p]),
    "sph_reserve": (_int, [_c_void_p, _i64, _i64, _i64]),
    "sph_set_option": (_int, [_c_void_p, _int, _i64]),
    "sph_buffer_alloc": (_int, [_c_void_p, _sz, ctypes.POINTER(_c_void_p)]),
    "sph_buffer_free": (_int, [_c_void_p, _c_void_p]),
    "sph_buffer_ptr": (_c_void_p, [_c_void_p]),
    "sph_profile_enable": (_int, [_c_void_p, _int]),
    "sph_profile_read": (_int, [_c_void_p, ctypes.POINTER(sph_profile)]),
    "sph_payload_bytes": (_sz, [_i64, _i64]),
    "sph_keep_ids_from_mask": (_int, [_c_void_p, _i64, _c_void_p,
                                      ctypes.POINTER(_i64)]),
    "sph_check_keep_ids": (_int, [_c_void_p, _i64, _i64, ctypes.POINTER(_i64)]),
    "sph_plan_query": (_int, [_c_void_p, _int, _i64, _i64, _i64, _int, _int, _int,
                              ctypes.POINTER(sph_plan)]),
    "sph_partial_logits": (_int, [_c_void_p, _c_void_p, _i64, _i64, _c_void_p,
                                  _int, _i64, _i64, _i64, _c_void_p, _c_void_p,
                                  _c_void_p, _i64, _f32, _int, _c_void_p,
                                  _c_void_p, _c_void_p, ctypes.POINTER(_sz)]),
    "sph_partial_logits_noalloc": (_int, [_int, _c_void_p, _c_void_p, _i64, _i64,
                                          _c_void_p, _int, _i64, _i64, _i64,
                                          _c_void_p, _c_void_p, _c_void_p, _i64,
                                          _f32, _int, _c_void_p, _c_void_p,
                                          _c_void_p, ctypes.POINTER(_sz),
                                          ctypes.c_char_p, _sz]),
    "sph_fuse_sample": (_int, [_c_void_p, _c_void_p, _c_void_p, _i64, _c_void_p,
                               _i64, _c_void_p, _i64, _i64, _i64, _c_void_p,
                               _i64, _f32, _u64, _u64, _c_void_p, _c_void_p]),
    "sph_split_step": (_int, [_c_void_p, _c_void_p, _i64, _i64, _i64, _i64, _c_void_p, _int,
                              _c_void_p, _i64, _c_void_p, _i64, _i64, _c_void_p, _c_void_p,
                              _i64, _f32, _int, _f32, _u64, _u64, _i64, _c_void_p,
                              _c_void_p, _c_void_p, _c_void_p, _c_void_p,
                              ctypes.POINTER(_sz)]),
    "sph_verify_draft": (_int, [_c_void_p, _c_void_p, _i64, _i64, _c_void_p,
                                _i64, _f32, _c_void_p, _c_void_p, _u64, _u64,
                                _c_void_p, _c_void_p]),
}


def _load() -> ctypes.CDLL:
    if not os.path.exists(_LIB_PATH):
        raise RuntimeError(
            f"libsph.so is not built ({_LIB_PATH}); run "
            "`python -c 'import __graft_entry__ as g; g.build()'` first")
    lib = ctypes.CDLL(_LIB_PATH)
    for name, (res, args) in _SIGNATURES.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    return lib


lib = _load()
LIB_PATH = _LIB_PATH


class SphError(RuntimeError):
    def __init__(self, status: int, detail: str):
        self.status = status
        super().__init__(f"{STATUS_NAMES.get(status, status)}: {detail}")


def _check(ctx, status: int):
    if status != SPH_OK:
        detail = lib.sph_last_error(ctx).decode() if ctx else ""
        raise SphError(status, detail)


def _ptr(t: Optional[torch.Tensor]):
    return None if t is None else t.data_ptr()


def _ld(t: torch.Tensor) -> int:
    if t.dim() != 2 or t.stride(1) != 1:
        raise ValueError("expected a 2-D tensor with unit inner stride")
    return t.stride(0)


def _need(t, dtype, name):
    if t is None:
        return
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if dtype is not None and t.dtype != dtype:
        raise ValueError(f"{name} must be {dtype}, got {t.dtype}")


def _dense(dev, *specs):
    """Buffers the kernels index densely, (tensor, name, elements) each:
    every one given must be on `dev`, contiguous, and hold at least that
    many elements, so that no read or write of the call leaves it.  A count
    of None checks the device alone (operands with a row stride)."""
    for t, name, count in specs:
        if t is None:
            continue
        if t.device != dev:
            raise ValueError(f"{name} is on {t.device}, not on {dev}")
        if count is None:
            continue
        if not t.is_contiguous():
            raise ValueError(f"{name} must be contiguous")
        if t.numel() < count:
            raise ValueError(f"{name} holds {t.numel()} elements; the call needs {count}")


# ---------------------------------------------------------------------------
# C functions with torch arguments
# ---------------------------------------------------------------------------

def sph_create(device: int = 0, stream: Optional[int] = None):
    h = ctypes.c_void_p()
    st = lib.sph_create(int(device), ctypes.c_void_p(stream or 0), ctypes.byref(h))
    if st != SPH_OK:
        raise SphError(st, "sph_create failed")
    return h


def sph_destroy(ctx):
    _check(None, lib.sph_destroy(ctx))


def sph_set_stream(ctx, stream: int):
    _check(ctx, lib.sph_set_stream(ctx, ctypes.c_void_p(stream)))


def sph_sync(ctx):
    _check(ctx, lib.sph_sync(ctx))


def sph_reserve(ctx, max_rows: int, max_n_keep: int, max_d: int):
    _check(ctx, lib.sph_reserve(ctx, max_rows, max_n_keep, max_d))


def sph_set_option(ctx, option: int, value: int):
    _check(ctx, lib.sph_set_option(ctx, int(option), int(value)))


def sph_profile_enable(ctx, on: bool = True):
    _check(ctx, lib.sph_profile_enable(ctx, 1 if on else 0))


def sph_profile_read(ctx) -> dict:
    """Accumulated device time (ms) and timed groups per kernel class, and
    the number of kernels launched since tracing was enabled."""
    p = sph_profile()
    _check(ctx, lib.sph_profile_read(ctx, ctypes.byref(p)))
    return dict(ms={PROF_NAMES[i]: p.ms[i] for i in range(PROF_CLASSES)},
                calls={PROF_NAMES[i]: p.calls[i] for i in range(PROF_CLASSES)},
                launches=int(p.launches))


def sph_payload_bytes(rows: int, n_keep: int) -> int:
    return int(lib.sph_payload_bytes(rows, n_keep))


def sph_keep_ids_from_mask(mask_bits, V: int):
    """Host helper: bitmask bytes (numpy uint8, ceil(V/8)) -> sorted ids."""
    import numpy as np
    mask = np.ascontiguousarray(mask_bits, dtype=np.uint8)
    if mask.size * 8 < V:
        raise ValueError("mask too short")
    out = np.empty(V, dtype=np.int32)
    n = _i64(0)
    st = lib.sph_keep_ids_from_mask(mask.ctypes.data_as(ctypes.c_void_p), V,
                                    out.ctypes.data_as(ctypes.c_void_p),
                                    ctypes.byref(n))
    if st != SPH_OK:
        raise SphError(st, "sph_keep_ids_from_mask failed")
    return out[: n.value].copy()


def sph_check_keep_ids(keep_ids, V: int):
    """Host helper: check a host id list (numpy int32) against the id
    conventions; returns (ok, first bad position or -1)."""
    import numpy as np
    ids = np.ascontiguousarray(keep_ids, dtype=np.int32)
    bad = _i64(-1)
    st = lib.sph_check_keep_ids(ids.ctypes.data_as(ctypes.c_void_p), ids.size, int(V),
                                ctypes.byref(bad))
    return st == SPH_OK, int(bad.value)


def sph_plan_query(ctx, call: int, rows: int, n_keep: int, K: int, *,
                   w_dtype=SPH_DTYPE_BF16, act_mode=SPH_ACT_FP32, gather=True) -> dict:
    """The work split the context would choose for one call (call 0: cloud,
    1: endpoint), without launching anything."""
    p = sph_plan()
    _check(ctx, lib.sph_plan_query(ctx, int(call), int(rows), int(n_keep), int(K),
                                   int(w_dtype), int(act_mode), 1 if gather else 0,
                                   ctypes.byref(p)))
    return {f: int(getattr(p, f)) for f in PLAN_FIELDS}


def sph_partial_logits(ctx, h_cloud, W_h, *, keep_ids=None, clip=30.0,
                       w_row_scale=None, bias=None, act_mode=SPH_ACT_FP32,
                       codes=None, row_scale=None, partial_out=None):
    """Cloud call.  Returns (codes int8 [R, n], row_scale fp32 [R],
    payload_bytes).  h_cloud fp32 [R, d_h] (any row stride); W_h bf16 or
    float8_e4m3fn [V, d_h]."""
    _need(h_cloud, torch.float32, "h_cloud")
    if W_h.dtype == torch.bfloat16:
        wdt = SPH_DTYPE_BF16
    elif W_h.dtype == torch.float8_e4m3fn:
        wdt = SPH_DTYPE_FP8_E4M3
    else:
        raise ValueError("W_h must be bfloat16 or float8_e4m3fn")
    _need(W_h, None, "W_h")
    _need(keep_ids, torch.int32, "keep_ids")
    _need(w_row_scale, torch.float32, "w_row_scale")
    _need(bias, torch.float32, "bias")
    R, d_h = h_cloud.shape
    V = W_h.shape[0]
    n = V if keep_ids is None else keep_ids.numel()
    dev = h_cloud.device
    if codes is None:
        codes = torch.empty(R, n, dtype=torch.int8, device=dev)
    if row_scale is None:
        row_scale = torch.empty(R, dtype=torch.float32, device=dev)
    _need(codes, torch.int8, "codes")
    _need(row_scale, torch.float32, "row_scale")
    _need(partial_out, torch.float32, "partial_out")
    _dense(dev, (W_h, "W_h", None), (keep_ids, "keep_ids", n), (w_row_scale, "w_row_scale", V),
           (bias, "bias", V), (codes, "codes", R * n), (row_scale, "row_scale", R),
           (partial_out, "partial_out", R * n))
    pb = _sz(0)
    _check(ctx, lib.sph_partial_logits(
        ctx, _ptr(h_cloud), R, _ld(h_cloud), _ptr(W_h), wdt, V, d_h, _ld(W_h),
        _ptr(w_row_scale), _ptr(bias), _ptr(keep_ids), n, float(clip),
        int(act_mode), _ptr(codes), _ptr(row_scale), _ptr(partial_out),
        ctypes.byref(pb)))
    return codes, row_scale, pb.value


NOALLOC_SCRATCH_BYTES = 8 << 20


def sph_partial_logits_noalloc(h_cloud, W_h, *, codes, row_scale,
                               keep_ids=None, clip=30.0, w_row_scale=None,
                               bias=None, act_mode=SPH_ACT_FP32,
                               partial_out=None, device=None, stream=None):
    """Allocation-free cloud call for callers that cannot allocate device
    memory while they run (see include/sph.h): no context, caller-provided
    outputs, scratch in the library's fixed device array.  Returns the
    payload byte count; raises SphError with the library's message."""
    if W_h.dtype == torch.bfloat16:
        wdt = SPH_DTYPE_BF16
    elif W_h.dtype == torch.float8_e4m3fn:
        wdt = SPH_DTYPE_FP8_E4M3
    else:
        raise ValueError("W_h must be bfloat16 or float8_e4m3fn")
    for t, dt, name in ((h_cloud, torch.float32, "h_cloud"), (W_h, None, "W_h"),
                        (keep_ids, torch.int32, "keep_ids"),
                        (w_row_scale, torch.float32, "w_row_scale"),
                        (bias, torch.float32, "bias"), (codes, torch.int8, "codes"),
                        (row_scale, torch.float32, "row_scale"),
                        (partial_out, torch.float32, "partial_out")):
        _need(t, dt, name)
    R, d_h = h_cloud.shape
    V = W_h.shape[0]
    n = V if keep_ids is None else keep_ids.numel()
    dev = h_cloud.device.index if device is None else int(device)
    # the kernels write codes[r * n + j], partial_out[r * n + j] and
    # row_scale[r] densely, on `dev`: every tensor must live there and the
    # outputs must be contiguous and of exactly these shapes
    for t, name, shape in ((h_cloud, "h_cloud", None), (W_h, "W_h", None),
                           (keep_ids, "keep_ids", (n,)), (w_row_scale, "w_row_scale", (V,)),
                           (bias, "bias", (V,)), (codes, "codes", (R, n)),
                           (row_scale, "row_scale", (R,)), (partial_out, "partial_out", (R, n))):
        if t is None:
            continue
        if t.device.index != dev:
            raise ValueError(f"{name} is on {t.device}, not on cuda:{dev}")
        if shape is not None:
            if tuple(t.shape) != shape:
                raise ValueError(f"{name} must have shape {shape}, got {tuple(t.shape)}")
            if not t.is_contiguous():
                raise ValueError(f"{name} must be contiguous")
    if stream is None:
        stream = torch.cuda.current_stream(dev).cuda_stream
    pb = _sz(0)
    msg = ctypes.create_string_buffer(256)
    st = lib.sph_partial_logits_noalloc(
        dev, ctypes.c_void_p(stream), _ptr(h_cloud), R, _ld(h_cloud), _ptr(W_h),
        wdt, V, d_h, _ld(W_h), _ptr(w_row_scale), _ptr(bias), _ptr(keep_ids), n,
        float(clip), int(act_mode), _ptr(codes), _ptr(row_scale),
        _ptr(partial_out), ctypes.byref(pb), msg, len(msg))
    if st != SPH_OK:
        raise SphError(st, msg.value.decode())
    return pb.value


def sph_fuse_sample(ctx, codes, row_scale, h_local, W_l, *, keep_ids=None,
                    temperature=1.0, seed=0, offset=0, tokens=None,
                    fused_logits_out=None, draw=True):
    """Endpoint call.  Returns tokens int32 [R] (vocabulary ids); with
    draw=False only z is computed (into fused_logits_out, required) and the
    call returns None."""
    _need(codes, torch.int8, "codes")
    _need(row_scale, torch.float32, "row_scale")
    _need(h_local, torch.float32, "h_local")
    _need(W_l, torch.bfloat16, "W_l")
    _need(keep_ids, torch.int32, "keep_ids")
    _need(fused_logits_out, torch.float32, "fused_logits_out")
    R, d_l = h_local.shape
    V = W_l.shape[0]
    n = V if keep_ids is None else keep_ids.numel()
    if not draw:
        if fused_logits_out is None or tokens is not None:
            raise ValueError("draw=False needs fused_logits_out and no tokens")
    elif tokens is None:
        tokens = torch.empty(R, dtype=torch.int32, device=h_local.device)
    _need(tokens, torch.int32, "tokens")
    _dense(h_local.device, (W_l, "W_l", None), (keep_ids, "keep_ids", n),
           (codes, "codes", R * n), (row_scale, "row_scale", R), (tokens, "tokens", R),
           (fused_logits_out, "fused_logits_out", R * n))
    _check(ctx, lib.sph_fuse_sample(
        ctx, _ptr(codes), _ptr(row_scale), R, _ptr(h_local), _ld(h_local),
        _ptr(W_l), V, d_l, _ld(W_l), _ptr(keep_ids), n, float(temperature),
        int(seed) & 0xFFFFFFFFFFFFFFFF, int(offset) & 0xFFFFFFFFFFFFFFFF,
        _ptr(tokens), _ptr(fused_logits_out)))
    return tokens


def sph_split_step(ctx, h, d_l: int, W_h, W_l, *, keep_ids=None, clip=30.0,
                   w_row_scale=None, bias=None, act_mode=SPH_ACT_FP32, temperature=1.0,
                   seed=0, offset=0, chunk=0, endpoint_stream=None, codes=None,
                   scales=None, tokens=None, fused_logits_out=None):
    """The whole split step from the full hidden state h [R, d] (h[:, :d_l]
    the endpoint's part, h[:, d_l:] the cloud's) to tokens.  Returns
    (codes, scales, tokens, payload_bytes): the payload that would cross,
    chunk-major (int8 [R * n] flat, fp32 [nchunk * R])."""
    _need(h, torch.float32, "h")
    if W_h.dtype == torch.bfloat16:
        wdt = SPH_DTYPE_BF16
    elif W_h.dtype == torch.float8_e4m3fn:
        wdt = SPH_DTYPE_FP8_E4M3
    else:
        raise ValueError("W_h must be bfloat16 or float8_e4m3fn")
    _need(W_h, None, "W_h")
    _need(W_l, torch.bfloat16, "W_l")
    _need(keep_ids, torch.int32, "keep_ids")
    _need(w_row_scale, torch.float32, "w_row_scale")
    _need(bias, torch.float32, "bias")
    R = h.shape[0]
    V, d_h = W_h.shape
    n = V if keep_ids is None else keep_ids.numel()
    L = n if (chunk == 0 or chunk >= n) else int(chunk)
    nchunk = (n + L - 1) // L
    dev = h.device
    if codes is None:
        codes = torch.empty(R * n, dtype=torch.int8, device=dev)
    if scales is None:
        scales = torch.empty(nchunk * R, dtype=torch.float32, device=dev)
    if tokens is None:
        tokens = torch.empty(R, dtype=torch.int32, device=dev)
    _need(codes, torch.int8, "codes")
    _need(scales, torch.float32, "scales")
    _need(tokens, torch.int32, "tokens")
    _need(fused_logits_out, torch.float32, "fused_logits_out")
    _dense(dev, (W_h, "W_h", None), (W_l, "W_l", None), (keep_ids, "keep_ids", n),
           (w_row_scale, "w_row_scale", V), (bias, "bias", V), (codes, "codes", R * n),
           (scales, "scales", nchunk * R), (tokens, "tokens", R))
    if fused_logits_out is not None and (tuple(fused_logits_out.shape) != (R, n)
                                         or not fused_logits_out.is_contiguous()):
        raise ValueError("fused_logits_out must be a contiguous (R, n) tensor")
    _dense(dev, (fused_logits_out, "fused_logits_out", R * n))
    pb = _sz(0)
    _check(ctx, lib.sph_split_step(
        ctx, _ptr(h), R, _ld(h), int(d_l), d_h, _ptr(W_h), wdt, _ptr(w_row_scale),
        _ld(W_h), _ptr(W_l), _ld(W_l), V, _ptr(bias), _ptr(keep_ids), n, float(clip),
        int(act_mode), float(temperature), int(seed) & 0xFFFFFFFFFFFFFFFF,
        int(offset) & 0xFFFFFFFFFFFFFFFF, int(chunk),
        ctypes.c_void_p(endpoint_stream or 0), _ptr(codes), _ptr(scales), _ptr(tokens),
        _ptr(fused_logits_out), ctypes.byref(pb)))
    return codes, scales, tokens, pb.value


def sph_verify_draft(ctx, target_logits, sessions: int, k: int, draft_tokens,
                     *, keep_ids=None, draft_probs=None, temperature=1.0,
                     seed=0, offset=0, n_accepted=None, next_token=None):
    """Speculative verification.  Returns (n_accepted, next_token)."""
    _need(target_logits, torch.float32, "target_logits")
    _need(draft_tokens, torch.int32, "draft_tokens")
    _need(draft_probs, torch.float32, "draft_probs")
    _need(keep_ids, torch.int32, "keep_ids")
    n = target_logits.shape[-1]
    dev = target_logits.device
    if n_accepted is None:
        n_accepted = torch.empty(sessions, dtype=torch.int32, device=dev)
    if next_token is None:
        next_token = torch.empty(sessions, dtype=torch.int32, device=dev)
    _need(n_accepted, torch.int32, "n_accepted")
    _need(next_token, torch.int32, "next_token")
    S, K = max(int(sessions), 0), max(int(k), 0)
    _dense(dev, (target_logits, "target_logits", S * (K + 1) * n),
           (draft_tokens, "draft_tokens", S * K), (draft_probs, "draft_probs", S * K * n),
           (keep_ids, "keep_ids", n), (n_accepted, "n_accepted", S),
           (next_token, "next_token", S))
    _check(ctx, lib.sph_verify_draft(
        ctx, _ptr(target_logits), sessions, k, _ptr(keep_ids), n,
        float(temperature), _ptr(draft_tokens), _ptr(draft_probs),
        int(seed) & 0xFFFFFFFFFFFFFFFF, int(offset) & 0xFFFFFFFFFFFFFFFF,
        _ptr(n_accepted), _ptr(next_token)))
    return n_accepted, next_token


class Context:
    """A library context on `device`, issuing work on torch's current
    stream of that device (re-read at every call)."""

    def __init__(self, device: int = 0):
        self.device = int(device)
        self._stream = torch.cuda.current_stream(self.device).cuda_stream
        self.handle = sph_create(self.device, self._stream)

    def _follow_stream(self):
        s = torch.cuda.current_stream(self.device).cuda_stream
        if s != self._stream:
            sph_set_stream(self.handle, s)
            self._stream = s

    def reserve(self, max_rows, max_n_keep, max_d):
        sph_reserve(self.handle, max_rows, max_n_keep, max_d)

    def set_option(self, option: int, value: int):
        sph_set_option(self.handle, option, value)

    def plan(self, call: int, rows: int, n_keep: int, K: int, **kw) -> dict:
        return sph_plan_query(self.handle, call, rows, n_keep, K, **kw)

    def partial_logits(self, *a, **kw):
        self._follow_stream()
        return sph_partial_logits(self.handle, *a, **kw)

    def fuse_sample(self, *a, **kw):
        self._follow_stream()
        return sph_fuse_sample(self.handle, *a, **kw)

    def verify_draft(self, *a, **kw):
        self._follow_stream()
        return sph_verify_draft(self.handle, *a, **kw)

    def split_step(self, *a, **kw):
        self._follow_stream()
        return sph_split_step(self.handle, *a, **kw)

    def sync(self):
        sph_sync(self.handle)

    def profile_enable(self, on: bool = True):
        self._follow_stream()
        sph_profile_enable(self.handle, on)

    def profile_read(self) -> dict:
        return sph_profile_read(self.handle)

    def close(self):
        if self.handle is not None:
            sph_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
