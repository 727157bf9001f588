"""Seeded synthetic inputs for the AViTS transition (shared by the CUDA path,
the oracle tests and the bench).

This module only DRAWS inputs.  It contains none of the method's arithmetic:
no softmax, no score, no selection, no resampling.  Both sides receive the
same bytes from here and never import each other.

The paper measures on FLUX.1-dev / FLUX.1-Kontext-dev / Qwen-Image-Edit
activations over DrawBench and GEdit-Bench prompts (Sec. 4.1).  None of those
models or suites is available, so these seeded tensors stand in for them with
the shapes those models use at 1024^2 / 2048^2 (Sec. 4.1, Appendix A): a
32x32 (64x64) grid of 2x2-patchified 16-channel latent tokens, 512 text
tokens, 24 heads of width 128 and a 3072-wide hidden state.

Value recipe (documented draw order, numpy PCG64 ``default_rng(seed)``):
  1. Q_img, K_img, K_txt ~ N(0,1)/sqrt(d) (float64 draws, in that order).
  2. Relevance blobs: for each blob, a centre uniform on the grid, a text key
     index uniform in [0,L); q[h,i] += 1.5 * exp(-r^2 / (2 sigma^2)) * unit(
     k_txt[h, j_b]) with sigma = 2 tokens.  This makes a few regions attend
     strongly to a few text tokens: the long-tailed spatial importance the
     paper reports (Sec. 1, Fig. 2).
  3. For the FLUX-shaped configs Q and K are multiplied by one common factor
     chosen so that the std of softmax_scale * q.k over a fixed sample of
     image-query rows against all keys is ~3 (computed in float64 before the
     bf16 cast).
  4. h_prev ~ N(0,1) [B,N,D]; h_t = h_prev + N(0,1) * (0.05 + 0.5 f_i), with
     f a smooth field: white noise on the grid blurred by a Gaussian of
     sigma = G/8 tokens (reflect boundary), min-max scaled to [0,1].
  5. latent ~ N(0,1) [B, M, C*4].
  6. Editing config: R reference keys on the doubled grid,
     K_ref(Y,X) = 0.6 K_img(Y//2, X//2) + 0.8 N(0, var(K_img)), placed after
     the image keys.
  7. Joint-attention forward (make_joint_attention): one query per key of
     the joint sequence, Q = [Q_txt; Q_img; Q_ref]; Q_img is step 1-3's,
     Q_txt and Q_ref ~ N(0, var(K)) (the keys' scale after step 3), and the
     values V ~ N(0,1) [B,H,Nk,d], drawn from default_rng(seed + 7) in the
     order Q_txt, Q_ref, V per batch element.
bf16 tensors are float values rounded to nearest-even bf16 and kept as their
uint16 bit patterns (numpy has no bfloat16).
"""
from __future__ import annotations

import dataclasses
import math
from typing import Dict, List, Optional

import numpy as np

__all__ = [
    "Transition", "CONFIGS", "make_transition", "make_batched_stage2", "make_joint_attention",
    "to_bf16_bits", "bf16_bits_to_f32", "smooth_field",
]


def to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """float -> bf16 bit patterns (uint16), round to nearest even."""
    f = np.ascontiguousarray(x, dtype=np.float32)
    u = f.view(np.uint32).astype(np.uint64)
    rounding = ((u >> 16) & 1) + 0x7FFF
    out = ((u + rounding) >> 16).astype(np.uint16)
    nan = np.isnan(f)
    if nan.any():
        out[nan] = 0x7FC0
    return out


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (np.ascontiguousarray(b, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def _gauss_blur_1d(a: np.ndarray, sigma: float, axis: int) -> np.ndarray:
    r = max(1, int(math.ceil(3.0 * sigma)))
    t = np.arange(-r, r + 1, dtype=np.float64)
    w = np.exp(-0.5 * (t / sigma) ** 2)
    w /= w.sum()
    pad = [(0, 0)] * a.ndim
    pad[axis] = (r, r)
    ap = np.pad(a, pad, mode="reflect" if a.shape[axis] > r else "symmetric")
    out = np.zeros_like(a, dtype=np.float64)
    n = a.shape[axis]
    for o, wv in zip(range(2 * r + 1), w):
        sl = [slice(None)] * a.ndim
        sl[axis] = slice(o, o + n)
        out += wv * ap[tuple(sl)]
    return out


def smooth_field(rng: np.random.Generator, gh: int, gw: int) -> np.ndarray:
    """Smooth random field on a gh x gw grid, values in [0,1]."""
    noise = rng.standard_normal((gh, gw))
    sigma = max(gh, gw) / 8.0
    f = _gauss_blur_1d(_gauss_blur_1d(noise, sigma, 0), sigma, 1)
    lo, hi = f.min(), f.max()
    return (f - lo) / (hi - lo) if hi > lo else np.zeros_like(f)


@dataclasses.dataclass
class Transition:
    """One transition's inputs.  Arrays are float32 or bf16 bit patterns."""
    name: str
    dtype: str                 # "f32" or "bf16"
    B: int
    H: int
    M: int                     # image tokens scored (and upsampled)
    L: int                     # text keys
    R: int                     # reference keys (editing), 0 otherwise
    d: int
    D: int
    C: int
    grid_h: int
    grid_w: int
    k: int
    alpha: float
    mode: str                  # "nearest" or "bilinear"
    softmax_scale: float
    q_img: np.ndarray          # [B,H,M,d]
    k_all: np.ndarray          # [B,H,L+M+R,d]
    h_t: np.ndarray            # [B,M,D]
    h_prev: np.ndarray         # [B,M,D]
    latent: np.ndarray         # [B,M,C*4]
    pos_in: Optional[np.ndarray] = None    # [B,M,2] int32 (mixed input)
    span_in: Optional[np.ndarray] = None   # [B,M] int32
    frame_h: int = 0           # input frame (== grid when pos_in is None)
    frame_w: int = 0

    @property
    def Nk(self) -> int:
        return self.L + self.M + self.R

    @property
    def n_out(self) -> int:
        return self.M + 3 * self.k


# name -> parameters.  Sizes follow the FLUX-family shapes of Sec. 4.1.
CONFIGS: Dict[str, dict] = {
    "tiny": dict(seed=0, dtype="f32", B=1, H=2, G=16, L=32, R=0, d=64, D=128, C=16,
                 blobs=3, logit_std=None, k=64, alpha=0.5, mode="nearest"),
    "flux1024": dict(seed=1, dtype="bf16", B=1, H=24, G=32, L=512, R=0, d=128, D=3072,
                     C=16, blobs=3, logit_std=3.0, k=307, alpha=0.5, mode="nearest"),
    "flux2048": dict(seed=2, dtype="bf16", B=1, H=24, G=64, L=512, R=0, d=128, D=3072,
                     C=16, blobs=6, logit_std=3.0, k=1024, alpha=0.5, mode="nearest"),
    "edit": dict(seed=3, dtype="bf16", B=1, H=24, G=32, L=512, R=4096, d=128, D=3072,
                 C=16, blobs=3, logit_std=3.0, k=205, alpha=0.6, mode="nearest"),
    # batched multi-stage schedule, first transition (16x16 -> 32x32)
    "batched": dict(seed=100, dtype="bf16", B=8, H=24, G=16, L=512, R=0, d=128, D=3072,
                    C=16, blobs=3, logit_std=3.0, k=128, alpha=0.5, mode="nearest"),
}


def _gauss_env(cy: float, cx: float, ys: np.ndarray, xs: np.ndarray, sigma: float) -> np.ndarray:
    return np.exp(-((ys - cy) ** 2 + (xs - cx) ** 2) / (2.0 * sigma * sigma))


def _draw_qk(rng, H, M, L, d, blobs, ys, xs, grid_h, grid_w):
    """Steps 1-2 of the recipe for one batch element (float64)."""
    inv = 1.0 / math.sqrt(d)
    q = rng.standard_normal((H, M, d)) * inv
    k_img = rng.standard_normal((H, M, d)) * inv
    k_txt = rng.standard_normal((H, L, d)) * inv
    for _ in range(blobs):
        cy = rng.uniform(0, grid_h)
        cx = rng.uniform(0, grid_w)
        jb = int(rng.integers(0, max(L, 1))) if L > 0 else 0
        if L == 0:
            continue
        g = _gauss_env(cy, cx, ys, xs, 2.0)                    # [M]
        kt = k_txt[:, jb, :]                                  # [H,d]
        kt = kt / np.linalg.norm(kt, axis=1, keepdims=True)
        q += 1.5 * g[None, :, None] * kt[:, None, :]
    return q, k_img, k_txt


def _logit_std(q, k_all, scale, rows):
    """Std of scale*q.k over a fixed row sample (input calibration only)."""
    vals = []
    for h in range(q.shape[0]):
        vals.append((q[h, rows, :] @ k_all[h].T) * scale)
    return float(np.std(np.concatenate([v.ravel() for v in vals])))


def _finish(arr: np.ndarray, dtype: str) -> np.ndarray:
    if dtype == "bf16":
        return to_bf16_bits(arr.astype(np.float32))
    return np.ascontiguousarray(arr, dtype=np.float32)


def make_transition(name: str, seed: Optional[int] = None, **overrides) -> Transition:
    """Build a named configuration (``overrides`` replace any parameter)."""
    p = dict(CONFIGS[name])
    p.update(overrides)
    if seed is not None:
        p["seed"] = seed
    B, H, G, L, R, d, D, C = (p[x] for x in ("B", "H", "G", "L", "R", "d", "D", "C"))
    gh = gw = G
    M = gh * gw
    ys = (np.arange(M) // gw).astype(np.float64) + 0.5
    xs = (np.arange(M) % gw).astype(np.float64) + 0.5
    qs, ks, hts, hps, lats = [], [], [], [], []
    for b in range(B):
        rng = np.random.default_rng(p["seed"] + (b if name == "batched" else 1000 * b))
        q, k_img, k_txt = _draw_qk(rng, H, M, L, d, p["blobs"], ys, xs, gh, gw)
        parts = [k_txt, k_img]
        if R > 0:
            rg = 2 * G
            Y = np.arange(rg * rg) // rg
            X = np.arange(rg * rg) % rg
            src = (Y // 2) * gw + (X // 2)
            sd = float(np.std(k_img))
            parts.append(0.6 * k_img[:, src, :] + 0.8 * sd * rng.standard_normal((H, rg * rg, d)))
        k_all = np.concatenate(parts, axis=1)
        scale = 1.0 / math.sqrt(d)
        if p["logit_std"] is not None:
            rows = np.arange(0, M, max(1, M // 64))
            s0 = _logit_std(q, k_all, scale, rows)
            c = math.sqrt(p["logit_std"] / s0)
            q = q * c
            k_all = k_all * c
        f = smooth_field(rng, gh, gw).reshape(M)
        hp = rng.standard_normal((M, D))
        ht = hp + rng.standard_normal((M, D)) * (0.05 + 0.5 * f)[:, None]
        lat = rng.standard_normal((M, C * 4))
        qs.append(q); ks.append(k_all); hts.append(ht); hps.append(hp); lats.append(lat)
    dt = p["dtype"]
    return Transition(
        name=name, dtype=dt, B=B, H=H, M=M, L=L, R=R, d=d, D=D, C=C, grid_h=gh, grid_w=gw,
        k=p["k"], alpha=p["alpha"], mode=p["mode"], softmax_scale=1.0 / math.sqrt(d),
        q_img=_finish(np.stack(qs), dt), k_all=_finish(np.stack(ks), dt),
        h_t=_finish(np.stack(hts), dt), h_prev=_finish(np.stack(hps), dt),
        latent=_finish(np.stack(lats), dt), frame_h=gh, frame_w=gw)


def make_joint_attention(tr: "Transition", seed: Optional[int] = None):
    """Step 7 of the recipe: (q_all [B,H,Nk,d], v_all [B,H,Nk,d]) of the joint
    sequence of transition ``tr``, rows ordered as its keys (text, image,
    reference).  Same dtype convention as ``tr``."""
    s = (CONFIGS[tr.name]["seed"] if seed is None else seed) + 7
    B, H, L, M, R, d = tr.B, tr.H, tr.L, tr.M, tr.R, tr.d
    k = bf16_bits_to_f32(tr.k_all) if tr.dtype == "bf16" else tr.k_all
    q_img = bf16_bits_to_f32(tr.q_img) if tr.dtype == "bf16" else tr.q_img
    qs, vs = [], []
    for b in range(B):
        rng = np.random.default_rng(s + 1000 * b)
        sd = float(np.std(k[b].astype(np.float64)))
        q_txt = rng.standard_normal((H, L, d)) * sd
        q_ref = rng.standard_normal((H, R, d)) * sd
        v = rng.standard_normal((H, L + M + R, d))
        qs.append(np.concatenate([q_txt, q_img[b].astype(np.float64), q_ref], axis=1))
        vs.append(v)
    return _finish(np.stack(qs), tr.dtype), _finish(np.stack(vs), tr.dtype)


def make_batched_stage2(pos: np.ndarray, span: np.ndarray, frame: int, seed: int = 100,
                        H: int = 24, L: int = 512, d: int = 128, D: int = 3072,
                        k: int = 192, alpha: float = 0.5, blobs: int = 3,
                        logit_std: float = 3.0, dtype: str = "bf16",
                        latent: Optional[np.ndarray] = None) -> Transition:
    """Second transition of the batched multi-stage schedule.

    pos [B,N,2] / span [B,N] describe the mixed sequence left by the first
    transition (frame x frame cells).  Q, K and the hidden states are drawn
    fresh for those N tokens; blobs and the smooth field are evaluated at each
    token's footprint centre.  ``latent`` (the first transition's output) is
    passed through unchanged.
    """
    B, N = span.shape
    qs, ks, hts, hps = [], [], [], []
    for b in range(B):
        rng = np.random.default_rng(seed + 500 + b)
        ys = pos[b, :, 0].astype(np.float64) + span[b].astype(np.float64) / 2.0
        xs = pos[b, :, 1].astype(np.float64) + span[b].astype(np.float64) / 2.0
        q, k_img, k_txt = _draw_qk(rng, H, N, L, d, blobs, ys, xs, frame, frame)
        k_all = np.concatenate([k_txt, k_img], axis=1)
        scale = 1.0 / math.sqrt(d)
        rows = np.arange(0, N, max(1, N // 64))
        c = math.sqrt(logit_std / _logit_std(q, k_all, scale, rows))
        q = q * c
        k_all = k_all * c
        f = smooth_field(rng, frame, frame)
        fy = np.clip(ys.astype(np.int64), 0, frame - 1)
        fx = np.clip(xs.astype(np.int64), 0, frame - 1)
        fv = f[fy, fx]
        hp = rng.standard_normal((N, D))
        ht = hp + rng.standard_normal((N, D)) * (0.05 + 0.5 * fv)[:, None]
        qs.append(q); ks.append(k_all); hts.append(ht); hps.append(hp)
    C = 16 if latent is None else latent.shape[2] // 4
    if latent is None:
        latent = _finish(np.random.default_rng(seed + 900).standard_normal((B, N, C * 4)), dtype)
    return Transition(
        name="batched_t2", dtype=dtype, B=B, H=H, M=N, L=L, R=0, d=d, D=D, C=C,
        grid_h=frame, grid_w=frame, k=k, alpha=alpha, mode="nearest",
        softmax_scale=1.0 / math.sqrt(d), q_img=_finish(np.stack(qs), dtype),
        k_all=_finish(np.stack(ks), dtype), h_t=_finish(np.stack(hts), dtype),
        h_prev=_finish(np.stack(hps), dtype), latent=latent,
        pos_in=np.ascontiguousarray(pos, dtype=np.int32),
        span_in=np.ascontiguousarray(span, dtype=np.int32), frame_h=frame, frame_w=frame)


def random_scores(seed: int, B: int, M: int, ties: bool = False) -> List[np.ndarray]:
    """Score vectors A, V in [0,1) for selection tests; with ``ties`` many
    values repeat (quantised to 1/16) to exercise the lower-index rule."""
    rng = np.random.default_rng(seed)
    A = rng.random((B, M))
    V = rng.random((B, M))
    if ties:
        A = np.floor(A * 16) / 16
        V = np.floor(V * 16) / 16
    return [A.astype(np.float32), V.astype(np.float32)]
