"""CPU oracle of the AViTS transition (test infrastructure).

Only the tests, ``__graft_entry__.smoke()`` and bench.py's CPU-baseline arm
may import this package.  The product path (the CUDA library and its binding)
never does; the two share no code.

The arithmetic lives in ``avits_oracle.c`` (plain C, fp64, built with
``-ffp-contract=off`` and OpenMP over independent tokens); this module builds
it and wraps each function for numpy arrays.  bf16 tensors are passed as their
uint16 bit patterns.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from typing import Optional, Sequence

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "avits_oracle.c")
_OUT_DIR = os.path.join(_HERE, "_lib")
_LIB_PATH = os.path.join(_OUT_DIR, "libavits_oracle.so")
_lib = None

F32, BF16 = 0, 1


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (plain -O2, no fast-math, no contraction)."""
    os.makedirs(_OUT_DIR, exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + ".tmp%d" % os.getpid()
    cmd = ["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math", "-fopenmp",
           "-fPIC", "-shared", _SRC, "-o", tmp, "-lm"]
    subprocess.check_call(cmd)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    if _lib is None:
        _lib = ctypes.CDLL(build())
    return _lib


def _p(a: Optional[np.ndarray]):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _dtype_code(a: np.ndarray) -> int:
    if a.dtype == np.float32:
        return F32
    if a.dtype == np.uint16:
        return BF16
    raise TypeError("oracle inputs are float32 or bf16 bit patterns (uint16), got %s" % a.dtype)


def _c(a: np.ndarray) -> np.ndarray:
    if not a.flags["C_CONTIGUOUS"]:
        raise ValueError("oracle arrays must be C-contiguous")
    return a


_threads_set = None


def threads() -> int:
    """OpenMP threads the oracle runs on (set_threads(), else OMP_NUM_THREADS,
    else all cores)."""
    if _threads_set is not None:
        return _threads_set
    env = os.environ.get("OMP_NUM_THREADS")
    return int(env) if env else (os.cpu_count() or 1)


def set_threads(n: int) -> None:
    """Run the oracle's parallel loops on n threads from now on (the OpenMP
    runtime's omp_set_num_threads; the arithmetic and its order per token do
    not depend on it).  Used by the bench to time one thread and all cores."""
    global _threads_set
    fn = _load().omp_set_num_threads
    fn.argtypes = [ctypes.c_int]
    fn.restype = None
    fn(int(n))
    _threads_set = int(n)


def score_spatial(q_img: np.ndarray, k_all: np.ndarray, L: int, softmax_scale: float,
                  weight: float = 1.0, A_in: Optional[np.ndarray] = None,
                  rows: Optional[Sequence[int]] = None, l2norm: bool = False,
                  q_strides: Optional[Sequence[int]] = None,
                  k_strides: Optional[Sequence[int]] = None, shape=None,
                  text_mask: Optional[np.ndarray] = None):
    """Eq. 3 / Eq. 5.  q_img [B,H,M,d], k_all [B,H,Nk,d] (or flat buffers with
    explicit element strides and shape=(B,H,M,Nk,d)).  Returns (A [B,M] fp32,
    mass [B,H,M] fp64, lse [B,H,M,2] fp64); with ``rows`` only those flat
    b*M+i entries are computed (others are 0).  ``text_mask`` ([B,Nk], nonzero
    = text key) replaces the first-L rule for interleaved sequences."""
    lib = _load()
    dt = _dtype_code(q_img)
    if _dtype_code(k_all) != dt:
        raise TypeError("q and k dtypes differ")
    if shape is None:
        B, H, M, d = q_img.shape
        Nk = k_all.shape[2]
        q_strides = q_strides or (H * M * d, M * d, d)
        k_strides = k_strides or (H * Nk * d, Nk * d, d)
        q_img = _c(q_img)
        k_all = _c(k_all)
    else:
        B, H, M, Nk, d = shape
    A = np.zeros((B, M), np.float32) if A_in is None else np.array(A_in, np.float32, copy=True)
    mass = np.zeros((B, H, M), np.float64)
    lse = np.zeros((B, H, M, 2), np.float64)
    rows_arr = None if rows is None else np.ascontiguousarray(np.asarray(rows, np.int32))
    tm = None
    if text_mask is not None:
        tm = np.ascontiguousarray((np.asarray(text_mask) != 0).astype(np.uint8).reshape(B, Nk))
    fn = lib.avits_oracle_score_spatial
    fn.restype = ctypes.c_int
    i64 = ctypes.c_int64
    rc = fn(_p(q_img), _p(k_all), dt, B, H, M, Nk, L, d,
            i64(q_strides[0]), i64(q_strides[1]), i64(q_strides[2]),
            i64(k_strides[0]), i64(k_strides[1]), i64(k_strides[2]),
            ctypes.c_double(softmax_scale), ctypes.c_double(weight),
            0 if A_in is None else 1, 1 if l2norm else 0,
            _p(rows_arr), 0 if rows_arr is None else len(rows_arr), _p(tm), _p(A), _p(mass),
            _p(lse))
    if rc != 0:
        raise ValueError("oracle score_spatial: bad arguments (%d)" % rc)
    return A, mass, lse


def attention(q: np.ndarray, k: np.ndarray, v: np.ndarray, L: int, softmax_scale: float,
              weight: float = 1.0, A_in: Optional[np.ndarray] = None,
              rows: Optional[Sequence[int]] = None):
    """Eq. 4-5: the joint-attention forward O = softmax(scale Q K^T) V of a
    double-stream block, q [B,H,Mq,d], k and v [B,H,Nk,d] (contiguous), the
    text keys first.  Returns (O [B,H,Mq,d] fp64, lse [B,H,Mq,2] fp64 (all
    keys, text keys), mass [B,H,Mq] fp64 (Eq. 5), A [B,Mq] fp32 (Eq. 3)).
    With ``rows`` only those flat b*Mq+i rows are computed (others are 0)."""
    lib = _load()
    dt = _dtype_code(q)
    if _dtype_code(k) != dt or _dtype_code(v) != dt:
        raise TypeError("q, k and v dtypes differ")
    B, H, Mq, d = q.shape
    Nk = k.shape[2]
    if k.shape != (B, H, Nk, d) or v.shape != (B, H, Nk, d):
        raise ValueError("k and v must be [B,H,Nk,d] with the q's B, H and d")
    q, k, v = _c(q), _c(k), _c(v)
    O = np.zeros((B, H, Mq, d), np.float64)
    lse = np.zeros((B, H, Mq, 2), np.float64)
    mass = np.zeros((B, H, Mq), np.float64)
    A = np.zeros((B, Mq), np.float32) if A_in is None else np.array(A_in, np.float32, copy=True)
    rows_arr = None if rows is None else np.ascontiguousarray(np.asarray(rows, np.int32))
    fn = lib.avits_oracle_attention
    fn.restype = ctypes.c_int
    rc = fn(_p(q), _p(k), _p(v), dt, B, H, Mq, Nk, L, d, ctypes.c_double(softmax_scale),
            ctypes.c_double(weight), 0 if A_in is None else 1, _p(rows_arr),
            0 if rows_arr is None else len(rows_arr), _p(O), _p(lse), _p(mass), _p(A))
    if rc != 0:
        raise ValueError("oracle attention: bad arguments (%d)" % rc)
    return O, lse, mass, A


def score_temporal(h_t: np.ndarray, h_prev: np.ndarray, eps: float = 1e-6) -> np.ndarray:
    lib = _load()
    dt = _dtype_code(h_t)
    B, N, D = h_t.shape
    V = np.zeros((B, N), np.float32)
    rc = lib.avits_oracle_score_temporal(_p(_c(h_t)), _p(_c(h_prev)), dt, B, N, D,
                                         ctypes.c_double(eps), _p(V))
    if rc != 0:
        raise ValueError("oracle score_temporal: bad arguments")
    return V


def score_temporal_var(snaps: Sequence[np.ndarray]) -> np.ndarray:
    """Eq. 6-7 over N_T snapshots [B,N,D] (oldest first)."""
    lib = _load()
    dt = _dtype_code(snaps[0])
    B, N, D = snaps[0].shape
    arr = (ctypes.c_void_p * len(snaps))(*[s.ctypes.data for s in snaps])
    for s in snaps:
        _c(s)
    V = np.zeros((B, N), np.float32)
    rc = lib.avits_oracle_score_temporal_var(arr, len(snaps), dt, B, N, D, _p(V))
    if rc != 0:
        raise ValueError("oracle score_temporal_var: bad arguments")
    return V


def fuse(A: np.ndarray, V: np.ndarray, alpha: float, eps: float = 1e-6,
         perturb: Optional[np.ndarray] = None) -> np.ndarray:
    """Min-max normalisation and Eq. 8; with ``perturb`` the caller's
    tie-breaking noise of Eq. 9 is added to S (one rounded fp32 addition)."""
    lib = _load()
    A = _c(np.asarray(A, np.float32))
    V = _c(np.asarray(V, np.float32))
    B, M = A.shape
    P = None if perturb is None else _c(np.asarray(perturb, np.float32).reshape(B, M))
    S = np.zeros((B, M), np.float32)
    rc = lib.avits_oracle_fuse(_p(A), _p(V), B, M, ctypes.c_float(alpha), ctypes.c_float(eps),
                               _p(P), _p(S))
    if rc != 0:
        raise ValueError("oracle fuse: bad arguments")
    return S


def topk(S: np.ndarray, k: int):
    """Eq. 9 -> (sel_idx [B,k] ascending, mask [B,M] u8, tok_offset [B,M])."""
    lib = _load()
    S = _c(np.asarray(S, np.float32))
    B, M = S.shape
    sel = np.zeros((B, k), np.int32)
    mask = np.zeros((B, M), np.uint8)
    off = np.zeros((B, M), np.int32)
    rc = lib.avits_oracle_topk(_p(S), B, M, k, _p(sel), _p(mask), _p(off))
    if rc != 0:
        raise ValueError("oracle topk: bad arguments")
    return sel, mask, off


def fuse_select(A, V, alpha: float, k: int, eps: float = 1e-6, perturb=None):
    S = fuse(A, V, alpha, eps, perturb)
    sel, mask, off = topk(S, k)
    return S, sel, mask, off


def selective_upsample(latent: np.ndarray, grid_h: int, grid_w: int, mask: np.ndarray,
                       mode: str = "nearest", pos_in: Optional[np.ndarray] = None,
                       span_in: Optional[np.ndarray] = None):
    """Sec. 3.2 Stage 2 -> (out [B,N_out,C*4], pos [B,N_out,2], span, src_tok, src_sub)."""
    lib = _load()
    dt = _dtype_code(latent)
    B, M, T = latent.shape
    C = T // 4
    mask = _c(np.asarray(mask, np.uint8))
    k = int(mask[0].sum())
    NO = M + 3 * k
    out = np.zeros((B, NO, T), latent.dtype)
    pos = np.zeros((B, NO, 2), np.int32)
    span = np.zeros((B, NO), np.int32)
    src_tok = np.zeros((B, NO), np.int32)
    src_sub = np.zeros((B, NO), np.int8)
    n_out = ctypes.c_int(0)
    rc = lib.avits_oracle_selective_upsample(
        _p(_c(latent)), dt, B, M, grid_h, grid_w, C,
        _p(None if pos_in is None else _c(np.asarray(pos_in, np.int32))),
        _p(None if span_in is None else _c(np.asarray(span_in, np.int32))),
        _p(mask), 0 if mode == "nearest" else 1, _p(out), _p(pos), _p(span), _p(src_tok),
        _p(src_sub), ctypes.byref(n_out))
    if rc != 0:
        raise ValueError("oracle selective_upsample: bad arguments (%d)" % rc)
    return out, pos, span, src_tok, src_sub


def merge_final(mixed: np.ndarray, pos: np.ndarray, span: np.ndarray, full_h: int, full_w: int,
                mode: str = "nearest", check: bool = True):
    """Sec. 3.2 Stage 3 -> (out [B,full_h*full_w,C*4], cover_count [B,full_h*full_w]).
    Raises ValueError when the tokens do not tile the frame exactly (if check)."""
    lib = _load()
    dt = _dtype_code(mixed)
    B, N, T = mixed.shape
    out = np.zeros((B, full_h * full_w, T), mixed.dtype)
    cover = np.zeros((B, full_h * full_w), np.int32)
    rc = lib.avits_oracle_merge_final(_p(_c(mixed)), dt, B, N, _p(_c(np.asarray(pos, np.int32))),
                                      _p(_c(np.asarray(span, np.int32))), full_h, full_w, T // 4,
                                      0 if mode == "nearest" else 1, _p(out), _p(cover))
    if rc != 0 and check:
        raise ValueError("oracle merge_final: %s" % ("coverage" if rc == 6 else "bad arguments"))
    return out, cover
