"""AViTS resolution-transition hot path for GB300 (sm_103a).

A thin ctypes binding over ``libavits.so`` (include/avits.h).  Each function
has the name of its C entry point and only marshals arguments: torch tensors
become device pointers, the current torch stream becomes the cudaStream_t, a
non-OK status becomes an ``AvitsError``.  Every step of the path runs in the
library's CUDA kernels; there is no CPU fallback, and importing the functions
fails loudly when the library has not been built (``build()``).

Calls:
  avits_score_spatial       Eq. 3-5  text attention mass per image token
                            (text_mask=: interleaved text keys)
  avits_score_spatial_lse   Eq. 5  from the model attention's logsumexp over
                            all keys and the text keys only
  avits_score_temporal      Sec. 3.3.2  relative step change per token
  avits_score_spatiotemporal  both scores in one call
  avits_score_temporal_var  Eq. 6-7  step variance over N_T snapshots
  avits_fuse_select         Eq. 8-9  min-max fuse + deterministic top-k
                            (perturb=: caller's tie-break noise)
  avits_selective_upsample  Sec. 3.2 Stage 2  packed mixed-resolution sequence
  avits_select_upsample     selection + upsample in one launch
  avits_merge_final         Sec. 3.2 Stage 3  dense full-resolution latent
  avits_device_status       device-side error word (read and cleared)
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional, Sequence

from . import _build

__all__ = [
    "AvitsError", "build", "lib", "library_path",
    "avits_score_spatial", "avits_score_spatial_workspace", "avits_score_spatial_lse",
    "avits_score_temporal",
    "avits_score_spatiotemporal",
    "avits_score_spatial_noalloc", "avits_score_spatial_noalloc_limit",
    "avits_score_temporal_var", "avits_fuse_select",
    "avits_selective_upsample", "avits_select_upsample",
    "avits_merge_final", "avits_merge_final_workspace", "avits_device_status",
    "avits_selftest_bounded_wait", "avits_status_string", "avits_version", "SpatialWorkspace",
]

F32, BF16 = 0, 1
NEAREST, BILINEAR = 0, 1
STATUS = {0: "ok", 1: "invalid argument", 2: "unsupported", 3: "CUDA error",
          4: "device wait timed out", 5: "NaN in fused score", 6: "coverage"}

_lib = None


class AvitsError(RuntimeError):
    def __init__(self, fn: str, code: int, detail: str = ""):
        self.code = code
        super().__init__("%s failed: %s%s" % (fn, STATUS.get(code, code),
                                               (" (" + detail + ")") if detail else ""))


def library_path() -> str:
    return _build.LIB


def build(force: bool = False) -> str:
    """Compile libavits.so for sm_103a (in-tree)."""
    return _build.build(force=force)


def lib():
    """Load libavits.so; raise if it is missing (no fallback path exists)."""
    global _lib
    if _lib is not None:
        return _lib
    path = _build.LIB
    if not os.path.exists(path):
        raise RuntimeError("libavits.so is not built (%s); run paper_2608_17995_gb300.build()" % path)
    L = ctypes.CDLL(path)
    vp, i32, i64, f32, sz = ctypes.c_void_p, ctypes.c_int, ctypes.c_int64, ctypes.c_float, ctypes.c_size_t
    sig = {
        "avits_score_spatial": [vp, vp, i32, i32, i32, i32, i32, i32, i32, i64, i64, i64, i64, i64,
                                i64, f32, f32, i32, vp, vp, vp, sz, vp],
        "avits_score_spatial_workspace": [i32, i32, i32, i32, i32, i32],
        "avits_score_spatial_keymask": [vp, vp, i32, i32, i32, i32, i32, i32, i64, i64, i64, i64,
                                        i64, i64, vp, f32, f32, i32, vp, vp, vp, sz, vp],
        "avits_score_spatial_lse": [vp, vp, i32, i32, i32, i32, i32, i32, i64, i64, i64, i64,
                                    i64, i64, vp, f32, f32, i32, vp, vp, vp, sz, vp],
        "avits_score_temporal": [vp, vp, i32, i32, i32, i32, f32, vp, vp],
        "avits_attention_forward": [vp, vp, vp, i32, i32, i32, i32, i32, i32, i32, vp, vp, vp, vp,
                                    f32, vp, vp, f32, i32, vp, vp, sz, vp],
        "avits_attention_forward_workspace": [i32, i32, i32],
        "avits_score_spatiotemporal": [vp, vp, i32, i32, i32, i32, i32, i32, i32, i64, i64, i64,
                                       i64, i64, i64, f32, f32, i32, vp, vp, vp, sz, vp, vp, i32,
                                       f32, vp, vp],
        "avits_score_temporal_var": [vp, i32, i32, i32, i32, i32, vp, vp],
        "avits_fuse_select": [vp, vp, i32, i32, f32, f32, i32, vp, vp, vp, vp, vp],
        "avits_fuse_select_perturbed": [vp, vp, vp, i32, i32, f32, f32, i32, vp, vp, vp, vp, vp],
        "avits_selective_upsample": [vp, i32, i32, i32, i32, i32, i32, i32, vp, vp, vp, vp, i32,
                                     i32, vp, vp, vp, vp, vp, vp, sz, vp],
        "avits_selective_upsample_workspace": [i32, i32, i32, i32],
        "avits_select_upsample": [vp, vp, vp, i32, i32, f32, f32, i32, vp, vp, vp, vp, vp, i32,
                                  i32, i32, i32, i32, vp, vp, i32, vp, vp, vp, vp, vp, vp, sz,
                                  vp],
        "avits_merge_final": [vp, i32, i32, i32, vp, vp, i32, i32, i32, i32, i32, vp, vp, sz, vp],
        "avits_merge_final_workspace": [i32, i32, i32, i32],
        "avits_score_spatial_noalloc": [vp, vp, i32, i32, i32, i32, i32, i32, i32, i64, i64, i64,
                                        i64, i64, i64, f32, f32, i32, vp, vp, vp],
        "avits_score_spatial_noalloc_limit": [],
        "avits_score_spatial_noalloc_error": [],
        "avits_device_status": [vp],
        "avits_selftest_bounded_wait": [ctypes.c_ulonglong, vp, vp],
        "avits_status_string": [i32],
        "avits_last_error_string": [],
        "avits_version": [],
    }
    for name, args in sig.items():
        fn = getattr(L, name)
        fn.argtypes = args
        fn.restype = ctypes.c_int
    for name in ("avits_score_spatial_workspace", "avits_merge_final_workspace",
                 "avits_score_spatial_noalloc_limit", "avits_attention_forward_workspace",
                 "avits_selective_upsample_workspace"):
        getattr(L, name).restype = ctypes.c_size_t
    for name in ("avits_status_string", "avits_last_error_string", "avits_version",
                 "avits_score_spatial_noalloc_error"):
        getattr(L, name).restype = ctypes.c_char_p
    _lib = L
    return L


# ------------------------------------------------------------- marshalling --
def _torch():
    import torch
    return torch


def _ptr(t) -> Optional[int]:
    if t is None:
        return None
    if isinstance(t, int):
        return t
    if not t.is_cuda:
        raise ValueError("device tensor expected, got a %s tensor" % t.device)
    return t.data_ptr()


def _stream(stream) -> Optional[int]:
    if stream is None:
        return _torch().cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _dtype_code(t) -> int:
    torch = _torch()
    if t.dtype == torch.bfloat16:
        return BF16
    if t.dtype == torch.float32:
        return F32
    raise TypeError("bfloat16 or float32 expected, got %s" % t.dtype)


def _check(fn: str, rc: int):
    if rc != 0:
        detail = lib().avits_last_error_string().decode() if rc == 3 else ""
        raise AvitsError(fn, rc, detail)


def avits_version() -> str:
    return lib().avits_version().decode()


def avits_status_string(code: int) -> str:
    return lib().avits_status_string(code).decode()


def avits_device_status(stream=None) -> int:
    """Synchronise the stream; return and clear the device error code (0 = ok)."""
    return lib().avits_device_status(_stream(stream))


def avits_selftest_bounded_wait(limit_ns: int, result, stream=None):
    """Run the bounded-wait failure path on barriers nothing arrives at (a
    test hook): result (cuda int64[5]) receives completion flags and wait
    times of the timing-out warp and of the warp the abort flag releases."""
    _check("avits_selftest_bounded_wait",
           lib().avits_selftest_bounded_wait(int(limit_ns), _ptr(result), _stream(stream)))


def avits_score_spatial_workspace(dtype, B, H, M, Nk, d) -> int:
    code = dtype if isinstance(dtype, int) else _dtype_code(_torch().empty(0, dtype=dtype))
    return int(lib().avits_score_spatial_workspace(code, B, H, M, Nk, d))


class SpatialWorkspace:
    """Device scratch for avits_score_spatial, grown on demand (reused by
    calls on one stream).  Allocated zero-filled: the counters at its start
    must be zero before a call, and every completed call leaves them zero;
    after a call that reported a device timeout, call reset()."""

    def __init__(self, device=None):
        self.buf = None
        self.device = device

    def get(self, nbytes: int):
        torch = _torch()
        if nbytes == 0:
            return None, 0
        if self.buf is None or self.buf.numel() < nbytes:
            self.buf = torch.zeros(nbytes, dtype=torch.uint8, device=self.device or "cuda")
        return self.buf, self.buf.numel()

    def reset(self):
        if self.buf is not None:
            self.buf.zero_()


_default_ws = {}


def avits_score_spatial(q_img, k_all, L: int, softmax_scale: float, A, weight: float = 1.0,
                        accumulate: bool = False, lse=None, workspace: Optional[SpatialWorkspace] = None,
                        stream=None, text_mask=None):
    """Eq. 3-5.  q_img [B,H,M,d] (any strides, d contiguous), k_all [B,H,Nk,d]
    with the L text keys first; A [B,M] fp32 written (or accumulated).  With
    ``text_mask`` ([B,Nk] uint8 / bool on the device, nonzero = text key) the
    text keys are the masked ones instead (avits_score_spatial_keymask; L is
    ignored)."""
    B, H, M, d = q_img.shape
    Nk = k_all.shape[2]
    if k_all.shape[0] != B or k_all.shape[1] != H or k_all.shape[3] != d:
        raise ValueError("q_img / k_all shapes disagree")
    if q_img.stride(3) != 1 or k_all.stride(3) != 1:
        raise ValueError("the head-dim axis must be contiguous")
    dt = _dtype_code(q_img)
    if _dtype_code(k_all) != dt:
        raise TypeError("q_img and k_all dtypes differ")
    need = int(lib().avits_score_spatial_workspace(dt, B, H, M, Nk, d))
    if workspace is None:
        key = (q_img.device.index, _torch().cuda.current_stream().cuda_stream if stream is None else _stream(stream))
        workspace = _default_ws.setdefault(key, SpatialWorkspace(q_img.device))
    wbuf, wbytes = workspace.get(need)
    if text_mask is not None:
        if tuple(text_mask.shape) != (B, Nk) or text_mask.element_size() != 1 or \
                not text_mask.is_contiguous():
            raise ValueError("text_mask must be a contiguous [B,Nk] byte tensor")
        rc = lib().avits_score_spatial_keymask(
            _ptr(q_img), _ptr(k_all), dt, B, H, M, Nk, d,
            q_img.stride(0), q_img.stride(1), q_img.stride(2),
            k_all.stride(0), k_all.stride(1), k_all.stride(2), _ptr(text_mask),
            float(softmax_scale), float(weight), 1 if accumulate else 0,
            _ptr(A), _ptr(lse), _ptr(wbuf), wbytes, _stream(stream))
        _check("avits_score_spatial_keymask", rc)
        return A
    rc = lib().avits_score_spatial(
        _ptr(q_img), _ptr(k_all), dt, B, H, M, Nk, L, d,
        q_img.stride(0), q_img.stride(1), q_img.stride(2),
        k_all.stride(0), k_all.stride(1), k_all.stride(2),
        float(softmax_scale), float(weight), 1 if accumulate else 0,
        _ptr(A), _ptr(lse), _ptr(wbuf), wbytes, _stream(stream))
    _check("avits_score_spatial", rc)
    return A


def avits_score_spatial_lse(q_img, k_txt, lse_all, softmax_scale: float, A, weight: float = 1.0,
                            accumulate: bool = False, lse=None,
                            workspace: Optional[SpatialWorkspace] = None, stream=None):
    """Eq. 5 from the caller's logsumexp over all keys: q_img [B,H,M,d],
    k_txt [B,H,L,d] (the text keys only, any strides with d contiguous),
    lse_all [B,H,M] fp32 contiguous (natural log, e.g. from the model's
    attention forward); A [B,M] written (or accumulated)."""
    B, H, M, d = q_img.shape
    L = k_txt.shape[2]
    if k_txt.shape[0] != B or k_txt.shape[1] != H or k_txt.shape[3] != d:
        raise ValueError("q_img / k_txt shapes disagree")
    if q_img.stride(3) != 1 or k_txt.stride(3) != 1:
        raise ValueError("the head-dim axis must be contiguous")
    if tuple(lse_all.shape) != (B, H, M) or not lse_all.is_contiguous():
        raise ValueError("lse_all must be a contiguous [B,H,M] tensor")
    dt = _dtype_code(q_img)
    if _dtype_code(k_txt) != dt:
        raise TypeError("q_img and k_txt dtypes differ")
    need = int(lib().avits_score_spatial_workspace(dt, B, H, M, L, d))
    if workspace is None:
        key = (q_img.device.index, _torch().cuda.current_stream().cuda_stream if stream is None else _stream(stream))
        workspace = _default_ws.setdefault(key, SpatialWorkspace(q_img.device))
    wbuf, wbytes = workspace.get(need)
    rc = lib().avits_score_spatial_lse(
        _ptr(q_img), _ptr(k_txt), dt, B, H, M, L, d,
        q_img.stride(0), q_img.stride(1), q_img.stride(2),
        k_txt.stride(0), k_txt.stride(1), k_txt.stride(2), _ptr(lse_all),
        float(softmax_scale), float(weight), 1 if accumulate else 0,
        _ptr(A), _ptr(lse), _ptr(wbuf), wbytes, _stream(stream))
    _check("avits_score_spatial_lse", rc)
    return A


def avits_score_spatiotemporal(q_img, k_all, L: int, softmax_scale: float, A, h_t, h_prev, V,
                               weight: float = 1.0, accumulate: bool = False, lse=None,
                               eps: float = 1e-6, workspace: Optional[SpatialWorkspace] = None,
                               stream=None):
    """avits_score_spatial + avits_score_temporal in one call (the temporal
    kernel overlaps the spatial one on the tensor-core path)."""
    B, H, M, d = q_img.shape
    Nk = k_all.shape[2]
    D = h_t.shape[2]
    if q_img.stride(3) != 1 or k_all.stride(3) != 1:
        raise ValueError("the head-dim axis must be contiguous")
    if not (h_t.is_contiguous() and h_prev.is_contiguous()) or tuple(h_t.shape[:2]) != (B, M):
        raise ValueError("h_t / h_prev must be contiguous [B, M, D]")
    dt = _dtype_code(q_img)
    need = int(lib().avits_score_spatial_workspace(dt, B, H, M, Nk, d))
    if workspace is None:
        key = (q_img.device.index, _stream(stream))
        workspace = _default_ws.setdefault(key, SpatialWorkspace(q_img.device))
    wbuf, wbytes = workspace.get(need)
    rc = lib().avits_score_spatiotemporal(
        _ptr(q_img), _ptr(k_all), dt, B, H, M, Nk, L, d,
        q_img.stride(0), q_img.stride(1), q_img.stride(2),
        k_all.stride(0), k_all.stride(1), k_all.stride(2),
        float(softmax_scale), float(weight), 1 if accumulate else 0,
        _ptr(A), _ptr(lse), _ptr(wbuf), wbytes, _ptr(h_t), _ptr(h_prev), D, float(eps), _ptr(V),
        _stream(stream))
    _check("avits_score_spatiotemporal", rc)
    return A, V


def avits_attention_forward_workspace(B: int, H: int, Mq: int) -> int:
    return int(lib().avits_attention_forward_workspace(B, H, Mq))


def _strides3(t):
    arr = (ctypes.c_int64 * 3)(t.stride(0), t.stride(1), t.stride(2))
    return arr


def avits_attention_forward(q, k, v, L: int, softmax_scale: float, o, lse=None, A=None,
                            weight: float = 1.0, accumulate: bool = False,
                            workspace: Optional[SpatialWorkspace] = None, stream=None):
    """Eq. 4-5 + Eq. 3: the joint-attention forward O = softmax(scale Q K^T) V
    of a double-stream block (q [B,H,Mq,d], k / v [B,H,Nk,d], bf16, any
    strides with d contiguous, the L text keys first) into o [B,H,Mq,d]
    bf16, with lse [B,H,Mq,2] (all keys, text keys) and the spatial score A
    [B,Mq] (written or accumulated) when given."""
    B, H, Mq, d = q.shape
    Nk = k.shape[2]
    if tuple(k.shape) != (B, H, Nk, d) or tuple(v.shape) != (B, H, Nk, d) or \
            tuple(o.shape) != (B, H, Mq, d):
        raise ValueError("q / k / v / o shapes disagree")
    for t in (q, k, v, o):
        if t.stride(3) != 1:
            raise ValueError("the head-dim axis must be contiguous")
    dt = _dtype_code(q)
    if _dtype_code(k) != dt or _dtype_code(v) != dt or _dtype_code(o) != dt:
        raise TypeError("q, k, v and o dtypes differ")
    wbuf, wbytes = None, 0
    if A is not None:
        need = avits_attention_forward_workspace(B, H, Mq)
        if workspace is None:
            key = ("attn", q.device.index,
                   _torch().cuda.current_stream().cuda_stream if stream is None else _stream(stream))
            workspace = _default_ws.setdefault(key, SpatialWorkspace(q.device))
        wbuf, wbytes = workspace.get(need)
    qs, ks, vs, os_ = _strides3(q), _strides3(k), _strides3(v), _strides3(o)
    rc = lib().avits_attention_forward(
        _ptr(q), _ptr(k), _ptr(v), dt, B, H, Mq, Nk, L, d, qs, ks, vs, os_,
        float(softmax_scale), _ptr(o), _ptr(lse), float(weight), 1 if accumulate else 0,
        _ptr(A), _ptr(wbuf), wbytes, _stream(stream))
    _check("avits_attention_forward", rc)
    return o


def avits_score_temporal(h_t, h_prev, V, eps: float = 1e-6, stream=None):
    B, N, D = h_t.shape
    if not (h_t.is_contiguous() and h_prev.is_contiguous()):
        raise ValueError("h_t and h_prev must be contiguous")
    rc = lib().avits_score_temporal(_ptr(h_t), _ptr(h_prev), _dtype_code(h_t), B, N, D,
                                    float(eps), _ptr(V), _stream(stream))
    _check("avits_score_temporal", rc)
    return V


def avits_score_temporal_var(snaps: Sequence, V, stream=None):
    B, N, D = snaps[0].shape
    arr = (ctypes.c_void_p * len(snaps))(*[_ptr(s) for s in snaps])
    rc = lib().avits_score_temporal_var(arr, len(snaps), _dtype_code(snaps[0]), B, N, D, _ptr(V),
                                        _stream(stream))
    _check("avits_score_temporal_var", rc)
    return V


def avits_fuse_select(A, V, alpha: float, k: int, sel_idx, tok_offset, S=None, sel_mask=None,
                      eps_norm: float = 1e-6, stream=None, perturb=None):
    """Eq. 8-9; ``perturb`` ([B,M] fp32, optional): the caller's tie-breaking
    noise, added to S before the selection (avits_fuse_select_perturbed)."""
    B, M = A.shape
    if perturb is None:
        rc = lib().avits_fuse_select(_ptr(A), _ptr(V), B, M, float(alpha), float(eps_norm),
                                     int(k), _ptr(S), _ptr(sel_idx), _ptr(sel_mask),
                                     _ptr(tok_offset), _stream(stream))
        _check("avits_fuse_select", rc)
    else:
        if tuple(perturb.shape) != (B, M):
            raise ValueError("perturb must be [B,M]")
        rc = lib().avits_fuse_select_perturbed(_ptr(A), _ptr(V), _ptr(perturb), B, M,
                                               float(alpha), float(eps_norm), int(k), _ptr(S),
                                               _ptr(sel_idx), _ptr(sel_mask), _ptr(tok_offset),
                                               _stream(stream))
        _check("avits_fuse_select_perturbed", rc)
    return sel_idx


def avits_selective_upsample_workspace(mode: int, B: int, grid_h: int, grid_w: int) -> int:
    return int(lib().avits_selective_upsample_workspace(int(mode), B, grid_h, grid_w))


def _upsample_ws(mode, pos_in, B, grid_h, grid_w, workspace, device):
    """The cell-map workspace a mixed bilinear upsample needs (else none)."""
    if mode != BILINEAR or pos_in is None:
        return None, 0
    need = avits_selective_upsample_workspace(mode, B, grid_h, grid_w)
    if workspace is None:
        workspace = _torch().empty(need, dtype=_torch().uint8, device=device)
    return workspace, workspace.numel() * workspace.element_size()


def avits_select_upsample(A, V, alpha: float, k: int, sel_idx, tok_offset, sel_mask, latent,
                          grid_h: int, grid_w: int, out_latent, out_pos, out_span, out_src_tok,
                          out_src_sub, S=None, perturb=None, mode: int = NEAREST, pos_in=None,
                          span_in=None, eps_norm: float = 1e-6, workspace=None, stream=None):
    """avits_fuse_select(_perturbed) + avits_selective_upsample in one launch;
    the same outputs as the two calls."""
    B, M = A.shape
    T = latent.shape[2]
    ws, wb = _upsample_ws(mode, pos_in, B, grid_h, grid_w, workspace, latent.device)
    rc = lib().avits_select_upsample(
        _ptr(A), _ptr(V), _ptr(perturb), B, M, float(alpha), float(eps_norm), int(k), _ptr(S),
        _ptr(sel_idx), _ptr(sel_mask), _ptr(tok_offset), _ptr(latent), _dtype_code(latent),
        grid_h, grid_w, T // 4, 2, _ptr(pos_in), _ptr(span_in), int(mode), _ptr(out_latent),
        _ptr(out_pos), _ptr(out_span), _ptr(out_src_tok), _ptr(out_src_sub), _ptr(ws), wb,
        _stream(stream))
    _check("avits_select_upsample", rc)
    return sel_idx


def avits_selective_upsample(latent, grid_h: int, grid_w: int, sel_mask, tok_offset, k: int,
                             out_latent, out_pos, out_span, out_src_tok, out_src_sub,
                             mode: int = NEAREST, pos_in=None, span_in=None, workspace=None,
                             stream=None):
    """Sec. 3.2 Stage 2.  A mixed bilinear input (pos_in given) needs
    avits_selective_upsample_workspace() bytes of scratch (allocated here when
    ``workspace`` is None)."""
    B, M, T = latent.shape
    ws, wb = _upsample_ws(mode, pos_in, B, grid_h, grid_w, workspace, latent.device)
    rc = lib().avits_selective_upsample(
        _ptr(latent), _dtype_code(latent), B, M, grid_h, grid_w, T // 4, 2, _ptr(pos_in),
        _ptr(span_in), _ptr(sel_mask), _ptr(tok_offset), int(k), int(mode), _ptr(out_latent),
        _ptr(out_pos), _ptr(out_span), _ptr(out_src_tok), _ptr(out_src_sub), _ptr(ws), wb,
        _stream(stream))
    _check("avits_selective_upsample", rc)
    return out_latent


def avits_merge_final_workspace(mode: int, B: int, full_h: int, full_w: int) -> int:
    return int(lib().avits_merge_final_workspace(int(mode), B, full_h, full_w))


def avits_merge_final(mixed, pos, span, full_h: int, full_w: int, out_full, mode: int = NEAREST,
                      workspace=None, stream=None):
    B, N, T = mixed.shape
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    rc = lib().avits_merge_final(_ptr(mixed), _dtype_code(mixed), B, N, _ptr(pos), _ptr(span),
                                 full_h, full_w, T // 4, 2, int(mode), _ptr(out_full),
                                 _ptr(workspace), ws_bytes, _stream(stream))
    _check("avits_merge_final", rc)
    return out_full


def avits_score_spatial_noalloc(q_img, k_all, L: int, softmax_scale: float, A, weight: float = 1.0,
                                accumulate: bool = False, lse=None, stream=None):
    """avits_score_spatial without a workspace: the library's fixed device
    scratch is used instead (for callers that cannot allocate where they call
    this, e.g. inside an engine plugin's enqueue).  Same arguments otherwise;
    bf16 tensor-core shapes only.  Calls on one device must not overlap."""
    L_ = lib()
    fn = L_.avits_score_spatial_noalloc
    B, H, M, d = q_img.shape
    Nk = k_all.shape[2]
    rc = fn(_ptr(q_img), _ptr(k_all), _dtype_code(q_img), B, H, M, Nk, L, d,
            q_img.stride(0), q_img.stride(1), q_img.stride(2),
            k_all.stride(0), k_all.stride(1), k_all.stride(2),
            float(softmax_scale), float(weight), 1 if accumulate else 0,
            _ptr(A), _ptr(lse), _stream(stream))
    if rc != 0:
        err = L_.avits_score_spatial_noalloc_error()
        raise AvitsError("avits_score_spatial_noalloc", rc,
                         err.decode() if isinstance(err, bytes) else "")
    return A


def avits_score_spatial_noalloc_limit() -> int:
    """Bytes of the fixed scratch array behind avits_score_spatial_noalloc."""
    return int(lib().avits_score_spatial_noalloc_limit())
