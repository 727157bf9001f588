"""GPU parity: the CUDA path (through the C ABI) against the CPU oracle.

Tolerances: scores from bf16 inputs rel 2e-3; fp32 scores 1e-5; the fused
score, top-k indices, masks, offsets, nearest resampling, maps and positions
bit-exact; bilinear outputs within 1e-6 (bit-exact in practice: both sides
round the same fp32 operations); end-to-end selected sets may differ only at
tokens whose oracle score is within 1e-3 of the oracle's k-th score.
"""
import json
import math
import os

import numpy as np
import pytest

from helpers import as_f32

pytestmark = pytest.mark.gpu

BF16_RTOL = 2e-3
F32_TOL = 1e-5


@pytest.fixture(scope="module")
def av():
    import torch
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    import paper_2608_17995_gb300 as av
    av.build()
    av.lib()
    return av


@pytest.fixture(scope="module")
def orc():
    import oracle
    oracle.build()
    return oracle


def _dev(arr, dtype="f32"):
    from paper_2608_17995_gb300.pipeline import to_device
    return to_device(arr, dtype)


def _np(t):
    from paper_2608_17995_gb300.pipeline import to_numpy
    return to_numpy(t)


def _status(av):
    return av.avits_device_status()


def _sample_rows(B, M, n, seed=0):
    rng = np.random.default_rng(seed)
    rows = set(rng.choice(B * M, size=min(n, B * M), replace=False).tolist())
    rows |= {0, B * M - 1, M - 1}          # ends of the first element and of the batch
    return sorted(rows)


# ------------------------------------------------------------- spatial ----

def _check_spatial(av, orc, q, k, L, scale, dtype, rows=None, rtol=BF16_RTOL, weight=1.0,
                   A_in=None, q_t=None, k_t=None):
    import torch
    B, H, M, d = q.shape
    qd = _dev(q, dtype) if q_t is None else q_t
    kd = _dev(k, dtype) if k_t is None else k_t
    A = torch.zeros(B, M, dtype=torch.float32, device="cuda") if A_in is None else _dev(A_in)
    lse = torch.zeros(B, H, M, 2, dtype=torch.float32, device="cuda")
    av.avits_score_spatial(qd, kd, L, scale, A, weight=weight, accumulate=A_in is not None, lse=lse)
    assert _status(av) == 0
    A_o, mass_o, lse_o = orc.score_spatial(q, k, L, scale, weight=weight, A_in=A_in, rows=rows)
    A_g = _np(A)
    lse_g = _np(lse)
    idx = np.arange(B * M) if rows is None else np.asarray(rows)
    np.testing.assert_allclose(A_g.ravel()[idx], A_o.ravel()[idx], rtol=rtol, atol=1e-6)
    # per-head text mass through the lse pair (mass = exp(lse_txt - lse_all))
    b_i = np.stack([idx // M, idx % M], 1)
    for h in range(H):
        mg = np.exp(lse_g[b_i[:, 0], h, b_i[:, 1], 1] - lse_g[b_i[:, 0], h, b_i[:, 1], 0])
        mo = mass_o[b_i[:, 0], h, b_i[:, 1]]
        np.testing.assert_allclose(mg, mo, rtol=max(rtol, 1e-5) * 2, atol=1e-6)
    return A_g


@pytest.mark.parametrize("name,nrows", [("tiny", None), ("flux1024", 40), ("edit", 24), ("batched", 32)])
def test_spatial_from_lse_all(av, orc, name, nrows):
    """Eq. 5 from the logsumexp over all keys (as a model's attention forward
    returns it) and the text keys only: A against the oracle on the same
    rows, lse_all taken from the oracle (fp64 rounded to fp32)."""
    import torch
    from paper_2608_17995_gb300.workloads import make_transition, to_bf16_bits
    tr = make_transition(name)
    q, k = tr.q_img, tr.k_all
    if q.dtype == np.float32:   # the fp32 config: the same bf16 values on both sides
        q, k = to_bf16_bits(q), to_bf16_bits(k)
    B, H, M, d = q.shape
    rows = None if nrows is None else _sample_rows(B, M, nrows, seed=3)
    A_o, mass_o, lse_o = orc.score_spatial(q, k, tr.L, tr.softmax_scale, rows=rows)
    lse_all = torch.from_numpy(np.ascontiguousarray(lse_o[..., 0].astype(np.float32))).cuda()
    qd, kd = _dev(q, "bf16"), _dev(k, "bf16")
    A = torch.zeros(B, M, dtype=torch.float32, device="cuda")
    lse = torch.zeros(B, H, M, 2, dtype=torch.float32, device="cuda")
    av.avits_score_spatial_lse(qd, kd[:, :, :tr.L], lse_all, tr.softmax_scale, A, lse=lse)
    assert _status(av) == 0
    idx = np.arange(B * M) if rows is None else np.asarray(rows)
    np.testing.assert_allclose(_np(A).ravel()[idx], A_o.ravel()[idx], rtol=BF16_RTOL, atol=1e-6)
    # lse_opt: the given lse_all, and lse_txt against the oracle's
    lg = _np(lse)
    b_i = (idx // M, idx % M)
    for h in range(H):
        assert np.array_equal(lg[b_i[0], h, b_i[1], 0], lse_o[b_i[0], h, b_i[1], 0].astype(np.float32))
        np.testing.assert_allclose(lg[b_i[0], h, b_i[1], 1], lse_o[b_i[0], h, b_i[1], 1],
                                   rtol=1e-3, atol=2e-3)


def test_spatial_from_lse_all_matches_full_pass(av):
    """With lse_all from the full pass's own lse output, the text-key pass
    gives the full pass's A (weight and accumulate included)."""
    import torch
    from paper_2608_17995_gb300.workloads import make_transition
    tr = make_transition("flux1024")
    qd, kd = _dev(tr.q_img, "bf16"), _dev(tr.k_all, "bf16")
    B, H, M, d = tr.q_img.shape
    A1 = torch.full((B, M), 0.5, dtype=torch.float32, device="cuda")
    lse = torch.zeros(B, H, M, 2, dtype=torch.float32, device="cuda")
    av.avits_score_spatial(qd, kd, tr.L, tr.softmax_scale, A1, weight=0.25, accumulate=True, lse=lse)
    A2 = torch.full((B, M), 0.5, dtype=torch.float32, device="cuda")
    av.avits_score_spatial_lse(qd, kd[:, :, :tr.L], lse[..., 0].contiguous(), tr.softmax_scale, A2,
                               weight=0.25, accumulate=True)
    assert _status(av) == 0
    np.testing.assert_allclose(_np(A2), _np(A1), rtol=2e-5, atol=1e-7)


def _check_spatial_mask(av, orc, q, k, mask, scale, dtype, rows=None, rtol=BF16_RTOL):
    """avits_score_spatial_keymask against the masked oracle (A and the
    per-head mass through the lse pair)."""
    import torch
    B, H, M, d = q.shape
    A = torch.zeros(B, M, dtype=torch.float32, device="cuda")
    lse = torch.zeros(B, H, M, 2, dtype=torch.float32, device="cuda")
    md = torch.from_numpy(np.ascontiguousarray(mask.astype(np.uint8))).cuda()
    av.avits_score_spatial(_dev(q, dtype), _dev(k, dtype), 0, scale, A, lse=lse, text_mask=md)
    assert _status(av) == 0
    A_o, mass_o, _ = orc.score_spatial(q, k, 0, scale, rows=rows, text_mask=mask)
    A_g, lse_g = _np(A), _np(lse)
    idx = np.arange(B * M) if rows is None else np.asarray(rows)
    np.testing.assert_allclose(A_g.ravel()[idx], A_o.ravel()[idx], rtol=rtol, atol=1e-6)
    b_i = np.stack([idx // M, idx % M], 1)
    for h in range(H):
        mg = np.exp(lse_g[b_i[:, 0], h, b_i[:, 1], 1] - lse_g[b_i[:, 0], h, b_i[:, 1], 0])
        np.testing.assert_allclose(mg, mass_o[b_i[:, 0], h, b_i[:, 1]],
                                   rtol=max(rtol, 1e-5) * 2, atol=1e-6)
    return A_g


def test_spatial_keymask_fp32(av, orc):
    """Interleaved text keys, CUDA-core path (fp32)."""
    from paper_2608_17995_gb300.workloads import make_transition
    tr = make_transition("tiny")
    rng = np.random.default_rng(3)
    mask = (rng.random((tr.B, tr.Nk)) < 0.2).astype(np.uint8)
    _check_spatial_mask(av, orc, tr.q_img, tr.k_all, mask, tr.softmax_scale, "f32", rtol=F32_TOL)


@pytest.mark.parametrize("B,H,M,Nk,d,kind", [(1, 24, 1024, 1536, 128, "random"),
                                             (2, 4, 300, 1333, 128, "blocks"),
                                             (1, 6, 256, 700, 64, "random"),
                                             (1, 8, 512, 1024, 128, "none"),
                                             (1, 8, 512, 1024, 128, "all")])
def test_spatial_keymask_bf16(av, orc, B, H, M, Nk, d, kind):
    """Interleaved text keys on the tensor-core path: random masks (every
    item mixed), text blocks at arbitrary offsets (full text, full image and
    mixed items), ragged key counts, d = 64, and the empty / full masks."""
    from paper_2608_17995_gb300.workloads import to_bf16_bits
    rng = np.random.default_rng(M + Nk)
    q = to_bf16_bits((rng.standard_normal((B, H, M, d)) * 0.3).astype(np.float32))
    k = to_bf16_bits((rng.standard_normal((B, H, Nk, d)) * 0.3).astype(np.float32))
    if kind == "random":
        mask = (rng.random((B, Nk)) < 0.3).astype(np.uint8)
    elif kind == "blocks":
        mask = np.zeros((B, Nk), np.uint8)
        mask[:, 77:301] = 1
        mask[:, 640:768] = 1          # one whole 128-key tile
        mask[:, 1290:1333] = 1        # up to the ragged end
    elif kind == "none":
        mask = np.zeros((B, Nk), np.uint8)
    else:
        mask = np.ones((B, Nk), np.uint8)
    rows = _sample_rows(B, M, 64, seed=5)
    A = _check_spatial_mask(av, orc, q, k, mask, 1.0 / math.sqrt(d), "bf16", rows=rows)
    if kind == "none":
        assert np.all(A == 0.0)
    if kind == "all":
        np.testing.assert_allclose(A, 1.0, rtol=1e-6)


def test_spatial_keymask_first_l_is_l_form(av, orc):
    """A mask of the first 384 keys (a multiple of the 64-key halves a
    softmax warp reduces per item) takes the same item paths as the L form
    with L = 384: bit-identical A at the FLUX-1024 shape."""
    import torch
    from paper_2608_17995_gb300.workloads import make_transition
    tr = make_transition("flux1024")
    L = 384
    q, k = _dev(tr.q_img, "bf16"), _dev(tr.k_all, "bf16")
    A1 = torch.zeros(tr.B, tr.M, dtype=torch.float32, device="cuda")
    A2 = torch.zeros_like(A1)
    av.avits_score_spatial(q, k, L, tr.softmax_scale, A1)
    mask = torch.zeros(tr.B, tr.Nk, dtype=torch.uint8, device="cuda")
    mask[:, :L] = 1
    av.avits_score_spatial(q, k, 0, tr.softmax_scale, A2, text_mask=mask)
    assert _status(av) == 0
    assert torch.equal(A1.view(torch.int32), A2.view(torch.int32))


def test_spatial_tiny_fp32(av, orc):
    from paper_2608_17995_gb300.workloads import make_transition
    tr = make_transition("tiny")
    _check_spatial(av, orc, tr.q_img, tr.k_all, tr.L, tr.softmax_scale, "f32", rtol=F32_TOL)


@pytest.mark.parametrize("name,nrows", [("flux1024", 160), ("edit", 64), ("flux2048", 64),
                                        ("batched", 96)])
def test_spatial_bf16_configs(av, orc, name, nrows):
    """Full-size shapes in the launch configuration the bench times; the
    oracle evaluates a sample of rows (all heads)."""
    from paper_2608_17995_gb300.workloads import make_transition
    tr = make_transition(name)
    rows = _sample_rows(tr.B, tr.M, nrows, seed=len(name))
    _check_spatial(av, orc, tr.q_img, tr.k_all, tr.L, tr.softmax_scale, "bf16", rows=rows)


@pytest.mark.parametrize("B,H,M,L,R,d", [
    (2, 3, 200, 77, 45, 128),    # ragged rows, text boundary inside a key tile, ragged keys
    (1, 2, 100, 300, 0, 64),     # d = 64 tiles, fewer rows than one tile
    (1, 1, 513, 128, 130, 128),  # H = 1 (no head reduction), 3 row tiles
    (3, 2, 64, 1, 5, 128),       # one text key
    (1, 2, 129, 0, 7, 64),       # no text: mass 0
    (1, 2, 40, 60, 0, 128),      # Nk < 128
    (2, 3, 400, 77, 45, 128),    # CTA pairs (two row units per head), ragged second unit
    (1, 5, 1000, 256, 3, 128),   # CTA pairs, 4 row units per head, odd head count
])
def test_spatial_tc_ragged_shapes(av, orc, B, H, M, L, R, d):
    from paper_2608_17995_gb300.workloads import to_bf16_bits
    rng = np.random.default_rng(B * 1000 + M)
    Nk = L + M + R
    q = to_bf16_bits(rng.standard_normal((B, H, M, d)) * 1.3)
    k = to_bf16_bits(rng.standard_normal((B, H, Nk, d)) * 1.3)
    _check_spatial(av, orc, q, k, L, 1.0 / math.sqrt(d), "bf16")


@pytest.mark.parametrize("amp,L_all", [(4.0, False), (16.0, False), (1.0, True)])
def test_spatial_tc_large_logits_and_all_text(av, orc, amp, L_all):
    """Logits spread far beyond the lazy running maximum's 64 log2-unit
    window (amp 4: ~150 log2 units per row; amp 16: ~2,000, near one-hot
    rows), so chunks keep rescuing the maximum; and every key a text key
    (mass 1 for every row and head)."""
    from paper_2608_17995_gb300.workloads import to_bf16_bits
    rng = np.random.default_rng(int(amp) + 10 * L_all)
    B, H, M, R, d = 2, 3, 300, 37, 128
    L = M + R + 90 if L_all else 90
    Nk = L if L_all else L + M + R
    q = to_bf16_bits(rng.standard_normal((B, H, M, d)) * amp)
    k = to_bf16_bits(rng.standard_normal((B, H, Nk, d)) * amp)
    A = _check_spatial(av, orc, q, k, L, 1.0 / math.sqrt(d), "bf16")
    if L_all:
        np.testing.assert_allclose(A, 1.0, rtol=0, atol=1e-6)


def test_spatial_strided_views_and_accumulate(av, orc):
    """Q as the image rows of a token-major joint [B, L+M, H, d] projection,
    K token-major too; accumulate with a weight (aggregation over blocks and
    steps)."""
    import torch
    from paper_2608_17995_gb300.workloads import to_bf16_bits
    rng = np.random.default_rng(5)
    B, H, M, L, d = 2, 4, 300, 96, 128
    Nk = L + M
    q_all = to_bf16_bits(rng.standard_normal((B, L + M, H, d)) * 1.5)
    k_tok = to_bf16_bits(rng.standard_normal((B, Nk, H, d)) * 1.5)
    q = np.ascontiguousarray(q_all[:, L:].transpose(0, 2, 1, 3))
    k = np.ascontiguousarray(k_tok.transpose(0, 2, 1, 3))
    qa_t = _dev(q_all, "bf16")
    q_t = qa_t[:, L:].permute(0, 2, 1, 3)          # strides (Nq*H*d, d, H*d, 1)
    k_t = _dev(k_tok, "bf16").permute(0, 2, 1, 3)
    A_in = rng.random((B, M)).astype(np.float32)
    _check_spatial(av, orc, q, k, L, 1.0 / math.sqrt(d), "bf16", weight=0.25, A_in=A_in,
                   q_t=q_t, k_t=k_t)


def test_spatial_deterministic_and_workspace_clean(av):
    """Repeated calls on one workspace give bit-identical A.  A is refilled
    with NaN before every call: a ticket left non-zero by the previous call
    would keep the last-arriver merge from running and leave NaN behind."""
    import torch
    from paper_2608_17995_gb300 import SpatialWorkspace
    from paper_2608_17995_gb300.workloads import make_transition
    tr = make_transition("flux1024")
    q, k = _dev(tr.q_img, "bf16"), _dev(tr.k_all, "bf16")
    ws = SpatialWorkspace()
    outs = []
    for _ in range(4):
        A = torch.full((tr.B, tr.M), float("nan"), dtype=torch.float32, device="cuda")
        av.avits_score_spatial(q, k, tr.L, tr.softmax_scale, A, workspace=ws)
        outs.append(A.cpu())
    assert _status(av) == 0
    for o in outs:
        assert not torch.isnan(o).any()
        assert torch.equal(o, outs[0])


@pytest.mark.parametrize("name", ["flux1024", "tiny", "batched"])
def test_spatiotemporal_matches_separate_calls(av, orc, name):
    """One call for both scores (temporal overlapped with spatial on the
    tensor-core path) gives the separate calls' results, and the oracle's."""
    import torch
    from paper_2608_17995_gb300.workloads import make_transition
    tr = make_transition(name)
    q, k = _dev(tr.q_img, tr.dtype), _dev(tr.k_all, tr.dtype)
    ht, hp = _dev(tr.h_t, tr.dtype), _dev(tr.h_prev, tr.dtype)
    for _ in range(2):
        A = torch.full((tr.B, tr.M), float("nan"), device="cuda")
        V = torch.full((tr.B, tr.M), float("nan"), device="cuda")
        av.avits_score_spatiotemporal(q, k, tr.L, tr.softmax_scale, A, ht, hp, V)
        A2 = torch.empty_like(A)
        V2 = torch.empty_like(V)
        av.avits_score_spatial(q, k, tr.L, tr.softmax_scale, A2)
        av.avits_score_temporal(ht, hp, V2)
        assert _status(av) == 0
        assert torch.equal(A, A2) and torch.equal(V, V2)
    rtol = F32_TOL if tr.dtype == "f32" else BF16_RTOL
    np.testing.assert_allclose(_np(V), orc.score_temporal(tr.h_t, tr.h_prev), rtol=rtol, atol=1e-7)
    rows = _sample_rows(tr.B, tr.M, 48, seed=3)
    A_o, _, _ = orc.score_spatial(tr.q_img, tr.k_all, tr.L, tr.softmax_scale, rows=rows)
    np.testing.assert_allclose(_np(A).ravel()[rows], A_o.ravel()[rows], rtol=rtol, atol=1e-6)


# ------------------------------------------------------------ temporal ----

@pytest.mark.parametrize("name", ["tiny", "flux1024", "edit", "flux2048", "batched"])
def test_temporal_configs(av, orc, name):
    import torch
    from paper_2608_17995_gb300.workloads import make_transition
    tr = make_transition(name)
    V = torch.empty(tr.B, tr.M, dtype=torch.float32, device="cuda")
    av.avits_score_temporal(_dev(tr.h_t, tr.dtype), _dev(tr.h_prev, tr.dtype), V)
    V_o = orc.score_temporal(tr.h_t, tr.h_prev)
    rtol = F32_TOL if tr.dtype == "f32" else BF16_RTOL
    np.testing.assert_allclose(_np(V), V_o, rtol=rtol, atol=1e-7)


@pytest.mark.parametrize("dtype,D", [("bf16", 100), ("f32", 33), ("bf16", 8), ("f32", 4096)])
def test_temporal_odd_widths(av, orc, dtype, D):
    import torch
    from paper_2608_17995_gb300.workloads import to_bf16_bits
    rng = np.random.default_rng(D)
    B, N = 3, 37
    hp = rng.standard_normal((B, N, D)).astype(np.float32)
    ht = (hp + 0.1 * rng.standard_normal((B, N, D))).astype(np.float32)
    if dtype == "bf16":
        hp, ht = to_bf16_bits(hp), to_bf16_bits(ht)
    V = torch.empty(B, N, dtype=torch.float32, device="cuda")
    av.avits_score_temporal(_dev(ht, dtype), _dev(hp, dtype), V)
    rtol = F32_TOL if dtype == "f32" else BF16_RTOL
    np.testing.assert_allclose(_np(V), orc.score_temporal(ht, hp), rtol=rtol, atol=1e-7)


@pytest.mark.parametrize("dtype,n_t,D", [("f32", 2, 96), ("f32", 5, 96), ("bf16", 3, 96),
                                         ("bf16", 4, 3072), ("bf16", 8, 200), ("f32", 12, 64),
                                         ("bf16", 16, 40), ("bf16", 3, 30), ("f32", 6, 7)])
def test_temporal_variance_eq7(av, orc, dtype, n_t, D):
    """Eq. 6-7 over n_t snapshots: the 16-byte vector path (4, 8 and 16
    snapshot variants) and the scalar path (rows not a multiple of 16 bytes)."""
    import torch
    from paper_2608_17995_gb300.workloads import to_bf16_bits
    rng = np.random.default_rng(n_t + D)
    B, N = 2, 50
    snaps = [rng.standard_normal((B, N, D)).astype(np.float32) for _ in range(n_t)]
    if dtype == "bf16":
        snaps = [to_bf16_bits(s) for s in snaps]
    V = torch.empty(B, N, dtype=torch.float32, device="cuda")
    av.avits_score_temporal_var([_dev(s, dtype) for s in snaps], V)
    np.testing.assert_allclose(_np(V), orc.score_temporal_var(snaps), rtol=1e-5, atol=1e-7)


# ---------------------------------------------------------- fuse/select ----


@pytest.mark.parametrize("M,k,ties", [(1024, 307, True), (3000, 900, False), (9000, 2000, True)])
def test_fuse_select_perturbed_bitexact(av, orc, M, k, ties):
    """Eq. 9 with caller-supplied tie-breaking noise: S' and the selection
    bit-exact against the oracle (register and shared-memory key paths)."""
    import torch
    from paper_2608_17995_gb300.workloads import random_scores
    A, V = random_scores(40 + M, 2, M, ties=ties)
    rng = np.random.default_rng(M)
    d = (1e-6 * rng.standard_normal((2, M))).astype(np.float32)
    S_o = orc.fuse(A, V, 0.5, perturb=d)
    sel_o, mask_o, off_o = orc.topk(S_o, k)
    dev = lambda x: torch.from_numpy(np.ascontiguousarray(x)).cuda()
    S = torch.empty(2, M, dtype=torch.float32, device="cuda")
    sel = torch.empty(2, k, dtype=torch.int32, device="cuda")
    mask = torch.empty(2, M, dtype=torch.uint8, device="cuda")
    off = torch.empty(2, M, dtype=torch.int32, device="cuda")
    av.avits_fuse_select(dev(A), dev(V), 0.5, k, sel, off, S=S, sel_mask=mask, perturb=dev(d))
    assert np.array_equal(_np(S).view(np.uint32), S_o.view(np.uint32))
    assert np.array_equal(_np(sel), sel_o)
    assert np.array_equal(_np(mask), mask_o)
    assert np.array_equal(_np(off), off_o)
    # zero noise: exactly the unperturbed call
    S2 = torch.empty_like(S)
    sel2 = torch.empty_like(sel)
    off2 = torch.empty_like(off)
    av.avits_fuse_select(dev(A), dev(V), 0.5, k, sel2, off2, S=S2,
                         perturb=torch.zeros(2, M, dtype=torch.float32, device="cuda"))
    S3 = torch.empty_like(S)
    sel3 = torch.empty_like(sel)
    off3 = torch.empty_like(off)
    av.avits_fuse_select(dev(A), dev(V), 0.5, k, sel3, off3, S=S3)
    assert torch.equal(S2.view(torch.int32), S3.view(torch.int32))
    assert torch.equal(sel2, sel3) and torch.equal(off2, off3)

def _run_select(av, A, V, alpha, k):
    import torch
    B, M = A.shape
    S = torch.empty(B, M, dtype=torch.float32, device="cuda")
    sel = torch.empty(B, max(k, 1), dtype=torch.int32, device="cuda")
    mask = torch.empty(B, M, dtype=torch.uint8, device="cuda")
    off = torch.empty(B, M, dtype=torch.int32, device="cuda")
    av.avits_fuse_select(_dev(A), _dev(V), alpha, k, sel, off, S=S, sel_mask=mask)
    st = _status(av)
    return _np(S), _np(sel)[:, :k], _np(mask), _np(off), st


@pytest.mark.parametrize("seed,B,M,k,ties,alpha", [
    (0, 1, 1024, 307, False, 0.5), (1, 3, 1024, 307, True, 0.5), (2, 1, 4096, 1024, True, 0.25),
    (3, 2, 640, 192, True, 1.0), (4, 1, 1, 1, False, 0.5), (5, 2, 5, 0, False, 0.5),
    (6, 1, 100, 100, True, 0.0), (7, 1, 32768, 9000, True, 0.6), (8, 4, 1000, 1, True, 0.5),
    (9, 1, 3000, 2999, True, 0.5), (10, 2, 1600, 500, True, 0.5), (11, 1, 2048, 700, False, 0.3),
    (12, 3, 257, 80, True, 0.5),
])
def test_select_bit_exact(av, orc, seed, B, M, k, ties, alpha):
    from paper_2608_17995_gb300.workloads import random_scores
    A, V = random_scores(seed, B, M, ties=ties)
    S, sel, mask, off, st = _run_select(av, A, V, alpha, k)
    assert st == 0
    S_o = orc.fuse(A, V, alpha)
    assert np.array_equal(S.view(np.uint32), S_o.view(np.uint32))
    sel_o, mask_o, off_o = orc.topk(S_o, k)
    assert np.array_equal(sel, sel_o)
    assert np.array_equal(mask, mask_o)
    assert np.array_equal(off, off_o)


def test_select_golden_ties_and_nan(av, orc):
    with open(os.path.join(os.path.dirname(__file__), "golden", "p6_select_ties.json")) as f:
        g = json.load(f)["topk_case"]
    # alpha = 1 with A = S keeps the order and the ties of S (min-max is monotone)
    A = np.array([g["S"]], np.float32)
    _, sel, _, off, st = _run_select(av, A, np.zeros_like(A), 1.0, g["k"])
    assert sel[0].tolist() == g["sel_idx"] and off[0].tolist() == g["tok_offset"] and st == 0
    A = np.array([[0.3, np.nan, 0.9, -0.0, 0.0, 0.9]], np.float32)
    S, sel, _, _, st = _run_select(av, A, np.zeros_like(A), 1.0, 3)
    assert st == 5                                   # AVITS_ERR_NAN raised on the device
    assert sel[0].tolist() == orc.topk(S, 3)[0][0].tolist() == [0, 2, 5]


@pytest.mark.parametrize("n_bucket", [1, 31, 32, 33, 200])
@pytest.mark.parametrize("ties", [False, True])
def test_select_threshold_bucket_sizes(av, orc, n_bucket, ties):
    """The k-th score inside a value bucket of width 1/256 holding n_bucket
    scores: up to 32 they are ranked by one warp, beyond that the radix
    select decides; ties inside the bucket take the lower index first."""
    rng = np.random.default_rng(100 + n_bucket + 7 * ties)
    B, M = 2, 1024
    lo_b, hi_b = 100.0 / 256, 101.0 / 256
    A = np.empty((B, M), np.float32)
    for b in range(B):
        rest = M - 2 - n_bucket
        n_hi = rest // 3
        below = rng.uniform(0.0, lo_b - 1e-3, rest - n_hi)
        above = rng.uniform(hi_b + 1e-3, 1.0, n_hi)
        inside = lo_b + 1e-3 + (hi_b - lo_b - 2e-3) * rng.uniform(0, 1, n_bucket)
        if ties:
            inside = np.round(inside * 4096) / 4096   # exact repeats within the bucket
        vals = np.concatenate([[0.0, 1.0], below, above, inside]).astype(np.float32)
        A[b] = vals[rng.permutation(M)]
    k = 1 + (M - 2 - n_bucket) // 3 + (n_bucket + 1) // 2   # the k-th lands in the bucket
    S, sel, mask, off, st = _run_select(av, A, np.zeros_like(A), 1.0, k)
    assert st == 0
    S_o = orc.fuse(A, np.zeros_like(A), 1.0)
    assert np.array_equal(S.view(np.uint32), S_o.view(np.uint32))
    kth = np.sort(S_o, axis=1)[:, ::-1][:, k - 1]
    assert np.all(np.floor(kth * 256) == 100)
    sel_o, mask_o, off_o = orc.topk(S_o, k)
    assert np.array_equal(sel, sel_o)
    assert np.array_equal(mask, mask_o)
    assert np.array_equal(off, off_o)


@pytest.mark.parametrize("M,k", [(1024, 307), (2048, 700), (4096, 1)])
def test_select_clustered_scores(av, orc, M, k):
    """Scores packed into one bucket apart from the two extremes: the radix
    path over keys in registers, bit-exact."""
    rng = np.random.default_rng(M + k)
    A = (0.5 + 1e-4 * rng.standard_normal((2, M))).astype(np.float32)
    A[:, 3] = 0.0
    A[:, 7] = 1.0
    S, sel, mask, off, st = _run_select(av, A, np.zeros_like(A), 1.0, k)
    assert st == 0
    S_o = orc.fuse(A, np.zeros_like(A), 1.0)
    sel_o, mask_o, off_o = orc.topk(S_o, k)
    assert np.array_equal(sel, sel_o)
    assert np.array_equal(mask, mask_o)
    assert np.array_equal(off, off_o)


# ---------------------------------------------------- upsample / merge ----

def _upsample(av, lat, dtype, gh, gw, mask, off, k, mode, pos_in=None, span_in=None):
    import torch
    B, M, T = lat.shape
    NO = M + 3 * k
    tdt = torch.bfloat16 if dtype == "bf16" else torch.float32
    out = torch.full((B, NO, T), float("nan"), dtype=tdt, device="cuda")
    pos = torch.full((B, NO, 2), -7, dtype=torch.int32, device="cuda")
    span = torch.full((B, NO), -7, dtype=torch.int32, device="cuda")
    st_ = torch.full((B, NO), -7, dtype=torch.int32, device="cuda")
    ss = torch.full((B, NO), -7, dtype=torch.int8, device="cuda")
    av.avits_selective_upsample(_dev(lat, dtype), gh, gw, _dev(mask), _dev(off), k, out, pos,
                                span, st_, ss, mode=mode,
                                pos_in=None if pos_in is None else _dev(pos_in),
                                span_in=None if span_in is None else _dev(span_in))
    assert _status(av) == 0
    return _np(out), _np(pos), _np(span), _np(st_), _np(ss)


def _merge(av, mixed, dtype, pos, span, fh, fw, mode, expect_status=0):
    import torch
    B, N, T = mixed.shape
    tdt = torch.bfloat16 if dtype == "bf16" else torch.float32
    out = torch.full((B, fh * fw, T), float("nan"), dtype=tdt, device="cuda")
    nb = av.avits_merge_final_workspace(mode, B, fh, fw)
    ws = torch.zeros(max(nb, 16), dtype=torch.uint8, device="cuda")
    av.avits_merge_final(_dev(mixed, dtype), _dev(pos), _dev(span), fh, fw, out, mode=mode,
                         workspace=ws)
    assert _status(av) == expect_status
    return _np(out)


def _bits(a):
    return a.view(np.uint16) if a.dtype == np.uint16 else a.view(np.uint32)


@pytest.mark.parametrize("name,mode", [("tiny", 0), ("tiny", 1), ("flux1024", 0),
                                       ("flux1024", 1), ("flux2048", 0), ("edit", 1)])
def test_upsample_and_merge_bit_exact(av, orc, name, mode):
    from paper_2608_17995_gb300.workloads import make_transition, random_scores
    tr = make_transition(name)
    A, V = random_scores(11, tr.B, tr.M, ties=True)
    S_o = orc.fuse(A, V, tr.alpha)
    _, mask, off = orc.topk(S_o, tr.k)
    mname = "nearest" if mode == 0 else "bilinear"
    g = _upsample(av, tr.latent, tr.dtype, tr.grid_h, tr.grid_w, mask, off, tr.k, mode)
    o = orc.selective_upsample(tr.latent, tr.grid_h, tr.grid_w, mask, mode=mname)
    for a, b in zip(g, o):
        assert np.array_equal(_bits(a) if a.dtype.kind == "f" or a.dtype == np.uint16 else a,
                              _bits(b) if b.dtype.kind == "f" or b.dtype == np.uint16 else b)
    fh, fw = 2 * tr.grid_h, 2 * tr.grid_w
    full_g = _merge(av, o[0], tr.dtype, o[1], o[2], fh, fw, mode)
    full_o, cover = orc.merge_final(o[0], o[1], o[2], fh, fw, mode=mname)
    assert np.all(cover == 1)
    assert np.array_equal(_bits(full_g), _bits(full_o))


def test_upsample_golden_4x4(av):
    with open(os.path.join(os.path.dirname(__file__), "golden", "p5_upsample_4x4.json")) as f:
        g = json.load(f)
    A = np.array([g["S"]], np.float32)
    _, sel, mask, off, st = _run_select(av, A, np.zeros_like(A), 1.0, g["k"])
    assert st == 0 and sel[0].tolist() == g["sel_idx"] and off[0].tolist() == g["tok_offset"]
    lat = np.array([[[10 * i + 1, 10 * i + 2, 10 * i + 3, 10 * i + 4] for i in range(16)]],
                   np.float32)
    out, pos, span, src_tok, src_sub = _upsample(av, lat, "f32", 4, 4, mask, off, g["k"], 0)
    assert out.shape[1] == g["n_out"]
    for e in g["out_tokens"]:
        o = e["o"]
        assert pos[0, o].tolist() == e["pos"] and span[0, o] == e["span"]
        assert src_tok[0, o] == e["src_tok"] and src_sub[0, o] == e["src_sub"]
        assert out[0, o].tolist() == e["val"]


@pytest.mark.parametrize("mode", [0, 1])
def test_merge_detects_bad_tiling(av, orc, mode):
    """Sec. 3.2 Stage 3 expands tokens that tile the frame exactly once.  In
    both modes a token moved onto its neighbour (one cell covered twice, one
    left empty), a duplicated token with the sequence one short of cells (a
    hole alone: here the last token dropped), and a token outside the frame
    each raise AVITS_ERR_COVERAGE; a valid tiling right after each bad one
    still merges cleanly (the workspace state is consistent)."""
    lat = np.random.default_rng(0).standard_normal((1, 16, 8)).astype(np.float32)
    mask = np.zeros((1, 16), np.uint8)
    mask[0, [5, 10]] = 1
    out, pos, span, _, _ = orc.selective_upsample(lat, 4, 4, mask)
    import torch
    B, N, T = out.shape
    nb = av.avits_merge_final_workspace(mode, B, 8, 8)
    ws = torch.zeros(nb, dtype=torch.uint8, device="cuda")

    def run(o, p, s, expect):
        full = torch.full((B, 64, T), float("nan"), dtype=torch.float32, device="cuda")
        av.avits_merge_final(_dev(o), _dev(p), _dev(s), 8, 8, full, mode=mode, workspace=ws)
        assert _status(av) == expect
        return _np(full)

    good, cover = orc.merge_final(out, pos, span, 8, 8,
                                  mode="nearest" if mode == 0 else "bilinear")
    assert np.all(cover == 1)
    moved = pos.copy()
    moved[0, 1] = moved[0, 0]                       # double cover + hole
    run(out, moved, span, 6)
    assert np.array_equal(run(out, pos, span, 0), good)
    run(out[:, :-1], pos[:, :-1], span[:, :-1], 6)  # hole only
    assert np.array_equal(run(out, pos, span, 0), good)
    far = pos.copy()
    far[0, 3] = [7, 7]                              # outside the frame
    run(out, far, span, 6)
    assert np.array_equal(run(out, pos, span, 0), good)
    dup = np.concatenate([out, out[:, :1]], 1)      # one extra token on cell 0
    run(dup, np.concatenate([pos, pos[:, :1]], 1), np.concatenate([span, span[:, :1]], 1), 6)
    assert np.array_equal(run(out, pos, span, 0), good)


@pytest.mark.parametrize("mode", [0, 1])
def test_upsample_reports_offsets_outside_the_sequence(av, orc, mode):
    """avits_selective_upsample writes token i at the caller's tok_offset[i]
    (Sec. 3.2 Stage 2).  An offset whose outputs would leave the sequence of
    N_out = M + 3k tokens (a selected token starting 2 before the end, a
    negative offset, a deferred token at N_out) raises AVITS_ERR_COVERAGE and
    that token is not written; the other tokens are, and a consistent call
    right after is clean and matches the oracle."""
    import torch
    lat = np.random.default_rng(1).standard_normal((1, 16, 8)).astype(np.float32)
    mask = np.zeros((1, 16), np.uint8)
    mask[0, [5, 10]] = 1
    k = 2
    off = (np.arange(16) + 3 * np.concatenate([[0], np.cumsum(mask[0])[:-1]])).astype(np.int32)[None]
    NO = 16 + 3 * k
    ref = orc.selective_upsample(lat, 4, 4, mask, mode="nearest" if mode == 0 else "bilinear")
    bad = off.copy()
    bad[0, 10] = NO - 2      # selected: its 4 children would end 2 past the sequence
    bad[0, 3] = -1
    bad[0, 15] = NO          # deferred: one past the end
    out = torch.full((1, NO, 8), float("nan"), dtype=torch.float32, device="cuda")
    pos = torch.full((1, NO, 2), -7, dtype=torch.int32, device="cuda")
    span = torch.full((1, NO), -7, dtype=torch.int32, device="cuda")
    st_ = torch.full((1, NO), -7, dtype=torch.int32, device="cuda")
    ss = torch.full((1, NO), -7, dtype=torch.int8, device="cuda")
    av.avits_selective_upsample(_dev(lat), 4, 4, _dev(mask), _dev(bad), k, out, pos, span, st_, ss,
                                mode=mode)
    assert _status(av) == 6
    o, po = _np(out), _np(pos)
    for i in range(16):      # every token with a valid offset is written as usual
        if i in (3, 10, 15):
            continue
        n = 4 if mask[0, i] else 1
        sl = slice(off[0, i], off[0, i] + n)
        assert np.array_equal(o[0, sl], ref[0][0, sl]) and np.array_equal(po[0, sl], ref[1][0, sl])
    got = _upsample(av, lat, "f32", 4, 4, mask, off, k, mode)
    for a, b in zip(got, ref):
        assert np.array_equal(a, b)


# ------------------------------------------------------------ end to end ----

@pytest.mark.parametrize("name,mode", [("tiny", "nearest"), ("flux1024", "nearest"),
                                       ("flux1024", "bilinear"), ("flux2048", "nearest"),
                                       ("edit", "nearest"), ("batched", "nearest")])
def test_transition_end_to_end(av, orc, name, mode):
    """The whole path on the device (both scores in one call, selection +
    upsample in one launch, merge) against the oracle's transition computed
    from the same inputs on every image row: A and V within the score
    tolerance; selected sets may differ from the oracle's only at tokens whose
    oracle score is within 1e-3 of the k-th score; the upsample and merge
    are bit-exact given the device's own selection.  Every configuration,
    including the editing shape (alpha = 0.6, k = 205, 4096 reference keys in
    the softmax) and the batched schedule's first transition (B = 8)."""
    from paper_2608_17995_gb300.pipeline import TransitionBuffers
    from paper_2608_17995_gb300.workloads import make_transition
    tr = make_transition(name)
    buf = TransitionBuffers(tr, mode=mode)
    buf.run()
    assert _status(av) == 0
    A_o, _, _ = orc.score_spatial(tr.q_img, tr.k_all, tr.L, tr.softmax_scale)
    V_o = orc.score_temporal(tr.h_t, tr.h_prev)
    rtol = F32_TOL if tr.dtype == "f32" else BF16_RTOL
    np.testing.assert_allclose(_np(buf.A), A_o, rtol=rtol, atol=1e-6)
    np.testing.assert_allclose(_np(buf.V), V_o, rtol=rtol, atol=1e-7)
    S_o = orc.fuse(A_o, V_o, tr.alpha)
    sel_o, _, _ = orc.topk(S_o, tr.k)
    sel_g = _np(buf.sel_idx)[:, :tr.k]
    for b in range(tr.B):
        kth = np.sort(S_o[b])[::-1][tr.k - 1]
        diff = set(sel_g[b].tolist()) ^ set(sel_o[b].tolist())
        for i in diff:
            assert abs(float(S_o[b, i]) - float(kth)) < 1e-3, (b, i, S_o[b, i], kth)
    # the rest of the path is exact given the device's own selection
    o = orc.selective_upsample(tr.latent, tr.grid_h, tr.grid_w, _np(buf.sel_mask), mode=mode)
    assert np.array_equal(_bits(_np(buf.mixed)), _bits(o[0]))
    assert np.array_equal(_np(buf.pos), o[1]) and np.array_equal(_np(buf.span), o[2])
    full_o, cover = orc.merge_final(o[0], o[1], o[2], 2 * tr.grid_h, 2 * tr.grid_w, mode=mode)
    assert np.all(cover == 1)
    assert np.array_equal(_bits(_np(buf.full)), _bits(full_o))


@pytest.mark.parametrize("name,mode", [("flux2048", "nearest"), ("edit", "nearest"),
                                       ("g40", "bilinear"), ("g40", "nearest")])
def test_select_upsample_fused_vs_oracle(av, orc, name, mode):
    """avits_select_upsample (one launch) against the oracle given the same
    scores A, V: the fused score S, sel_idx, mask and tok_offset, the mixed
    sequence and its maps all bit-exact (M = 4096 at FLUX-2048, 1600 at
    G = 40; the editing shape's alpha = 0.6 and k = 205)."""
    from paper_2608_17995_gb300.pipeline import TransitionBuffers
    from paper_2608_17995_gb300.workloads import make_transition
    tr = make_transition("flux1024", G=40, k=480) if name == "g40" else make_transition(name)
    buf = TransitionBuffers(tr, mode=mode)
    buf.spatial()
    buf.temporal()
    buf.select_upsample()
    assert _status(av) == 0
    A, V = _np(buf.A), _np(buf.V)
    S_o = orc.fuse(A, V, tr.alpha)
    assert np.array_equal(_bits(_np(buf.S)), _bits(S_o))
    sel_o, mask_o, off_o = orc.topk(S_o, tr.k)
    assert np.array_equal(_np(buf.sel_idx)[:, :tr.k], sel_o)
    assert np.array_equal(_np(buf.sel_mask), mask_o) and np.array_equal(_np(buf.tok_offset), off_o)
    o = orc.selective_upsample(tr.latent, tr.grid_h, tr.grid_w, mask_o, mode=mode)
    assert np.array_equal(_bits(_np(buf.mixed)), _bits(o[0]))
    assert np.array_equal(_np(buf.pos), o[1]) and np.array_equal(_np(buf.span), o[2])
    assert np.array_equal(_np(buf.src_tok), o[3]) and np.array_equal(_np(buf.src_sub), o[4])


def _fused_vs_separate(av, buf, perturb=None, k=None):
    """avits_select_upsample against avits_fuse_select + avits_selective_upsample
    on the same inputs: every output bit-identical."""
    import torch
    tr = buf.tr
    k = tr.k if k is None else k
    A, V = buf.A, buf.V
    M = tr.M
    B = tr.B
    NO = M + 3 * k
    dt = buf.latent.dtype
    def outs():
        d = dict(device="cuda")
        return dict(S=torch.full((B, M), float("nan"), **d),
                    sel=torch.full((B, max(k, 1)), -7, dtype=torch.int32, **d),
                    mask=torch.full((B, M), 9, dtype=torch.uint8, **d),
                    off=torch.full((B, M), -7, dtype=torch.int32, **d),
                    mixed=torch.full((B, NO, tr.C * 4), float("nan"), dtype=dt, **d),
                    pos=torch.full((B, NO, 2), -7, dtype=torch.int32, **d),
                    span=torch.full((B, NO), -7, dtype=torch.int32, **d),
                    src=torch.full((B, NO), -7, dtype=torch.int32, **d),
                    sub=torch.full((B, NO), 9, dtype=torch.int8, **d))
    a, f = outs(), outs()
    av.avits_fuse_select(A, V, tr.alpha, k, a["sel"], a["off"], S=a["S"], sel_mask=a["mask"],
                         perturb=perturb)
    av.avits_selective_upsample(buf.latent, tr.frame_h, tr.frame_w, a["mask"], a["off"], k,
                                a["mixed"], a["pos"], a["span"], a["src"], a["sub"],
                                mode=buf.mode, pos_in=buf.pos_in, span_in=buf.span_in)
    av.avits_select_upsample(A, V, tr.alpha, k, f["sel"], f["off"], f["mask"], buf.latent,
                             tr.frame_h, tr.frame_w, f["mixed"], f["pos"], f["span"], f["src"],
                             f["sub"], S=f["S"], perturb=perturb, mode=buf.mode,
                             pos_in=buf.pos_in, span_in=buf.span_in)
    assert _status(av) == 0
    for key in a:
        x, y = a[key], f[key]
        if x.dtype in (torch.float32, torch.bfloat16):
            x = x.view(torch.int32 if x.dtype == torch.float32 else torch.int16)
            y = y.view(torch.int32 if y.dtype == torch.float32 else torch.int16)
        if key == "sel" and k == 0:
            continue
        assert torch.equal(x, y), key


@pytest.mark.parametrize("name,mode", [("tiny", "nearest"), ("flux1024", "nearest"),
                                       ("flux1024", "bilinear"), ("batched", "nearest"),
                                       ("flux2048", "nearest"), ("flux2048", "bilinear"),
                                       ("edit", "nearest"), ("g40", "nearest"),
                                       ("g40", "bilinear")])
def test_select_upsample_fused_matches_separate(av, name, mode):
    """One-launch selection + upsample at 1, 2, 4 and 8 keys per thread
    (M = 256, 1024, 1600, 4096), bit-identical to the two calls."""
    from paper_2608_17995_gb300.pipeline import TransitionBuffers
    from paper_2608_17995_gb300.workloads import make_transition
    tr = make_transition("flux1024", G=40, k=480) if name == "g40" else make_transition(name)
    buf = TransitionBuffers(tr, mode=mode)
    buf.spatial(); buf.temporal()
    _fused_vs_separate(av, buf)


def test_select_upsample_fused_edges(av):
    """k = 0, k = M, ties with a perturbation, multi-level positions (the
    batched schedule's second transition)."""
    import torch
    from paper_2608_17995_gb300.pipeline import TransitionBuffers
    from paper_2608_17995_gb300.workloads import make_batched_stage2, make_transition
    buf = TransitionBuffers(make_transition("flux1024"))
    buf.spatial(); buf.temporal()
    _fused_vs_separate(av, buf, k=0)
    _fused_vs_separate(av, buf, k=buf.tr.M)
    g = torch.Generator(device="cuda"); g.manual_seed(1)
    pert = 1e-6 * torch.randn(buf.tr.B, buf.tr.M, device="cuda", generator=g)
    _fused_vs_separate(av, buf, perturb=pert)
    t1 = make_transition("batched")
    b1 = TransitionBuffers(t1)
    b1.run(merge=False)
    t2 = make_batched_stage2(_np(b1.pos), _np(b1.span), frame=32, latent=_np(b1.mixed))
    b2 = TransitionBuffers(t2)
    b2.spatial(); b2.temporal()
    _fused_vs_separate(av, b2)


def test_batched_two_transitions(av, orc):
    """Batched multi-stage schedule: 8 elements, 16x16 -> 32x32 -> 64x64, the
    second transition re-scores every token of the mixed sequence, then the
    final merge.  Spatial scores on sampled rows; the rest exact."""
    import torch
    from paper_2608_17995_gb300.pipeline import TransitionBuffers
    from paper_2608_17995_gb300.workloads import make_batched_stage2, make_transition
    t1 = make_transition("batched")
    b1 = TransitionBuffers(t1)
    b1.run(merge=False)
    assert _status(av) == 0
    rows = _sample_rows(t1.B, t1.M, 48, seed=1)
    A_o, _, _ = orc.score_spatial(t1.q_img, t1.k_all, t1.L, t1.softmax_scale, rows=rows)
    np.testing.assert_allclose(_np(b1.A).ravel()[rows], A_o.ravel()[rows], rtol=BF16_RTOL, atol=1e-6)
    mixed1, pos1, span1 = _np(b1.mixed), _np(b1.pos), _np(b1.span)
    t2 = make_batched_stage2(pos1, span1, frame=32, latent=mixed1)
    b2 = TransitionBuffers(t2)
    b2.run()
    assert _status(av) == 0
    rows2 = _sample_rows(t2.B, t2.M, 48, seed=2)
    A2_o, _, _ = orc.score_spatial(t2.q_img, t2.k_all, t2.L, t2.softmax_scale, rows=rows2)
    np.testing.assert_allclose(_np(b2.A).ravel()[rows2], A2_o.ravel()[rows2], rtol=BF16_RTOL,
                               atol=1e-6)
    S2 = _np(b2.S)
    sel_o, mask_o, off_o = orc.topk(S2, t2.k)
    assert np.array_equal(_np(b2.sel_mask), mask_o)
    o = orc.selective_upsample(mixed1, 32, 32, mask_o, pos_in=pos1, span_in=span1)
    assert np.array_equal(_bits(_np(b2.mixed)), _bits(o[0]))
    assert np.array_equal(_np(b2.pos), o[1]) and np.array_equal(_np(b2.span), o[2])
    full_o, cover = orc.merge_final(o[0], o[1], o[2], 64, 64)
    assert np.all(cover == 1)
    assert np.array_equal(_bits(_np(b2.full)), _bits(full_o))


# ------------------------------------------- multi-level bilinear (spans 1, 2, 4)

def test_batched_two_transitions_bilinear(av, orc):
    """The batched schedule in bilinear mode: the second transition upsamples
    selected span-1 and span-2 tokens from levels 0 and 1 of the mixed
    frame's pyramid, and the final merge (spans 1, 2 and 4) runs the
    coarse-to-fine cascade; both bit-exact against the oracle (given the
    kernel's own selection, itself checked against the oracle's top-k)."""
    from paper_2608_17995_gb300.pipeline import TransitionBuffers
    from paper_2608_17995_gb300.workloads import make_batched_stage2, make_transition
    t1 = make_transition("batched")
    b1 = TransitionBuffers(t1, mode="bilinear")
    b1.run(merge=False)
    assert _status(av) == 0
    mixed1, pos1, span1 = _np(b1.mixed), _np(b1.pos), _np(b1.span)
    _, mask1_o, _ = orc.topk(_np(b1.S), t1.k)
    o1 = orc.selective_upsample(t1.latent, 16, 16, mask1_o, mode="bilinear")
    assert np.array_equal(_bits(mixed1), _bits(o1[0]))
    t2 = make_batched_stage2(pos1, span1, frame=32, latent=mixed1)
    b2 = TransitionBuffers(t2, mode="bilinear")
    b2.run()
    assert _status(av) == 0
    _, mask_o, _ = orc.topk(_np(b2.S), t2.k)
    assert np.array_equal(_np(b2.sel_mask), mask_o)
    o = orc.selective_upsample(mixed1, 32, 32, mask_o, mode="bilinear", pos_in=pos1,
                               span_in=span1)
    assert set(np.unique(o[2])) == {1, 2, 4}
    assert np.array_equal(_bits(_np(b2.mixed)), _bits(o[0]))
    assert np.array_equal(_np(b2.pos), o[1]) and np.array_equal(_np(b2.span), o[2])
    full_o, cover = orc.merge_final(o[0], o[1], o[2], 64, 64, mode="bilinear")
    assert np.all(cover == 1)
    assert np.array_equal(_bits(_np(b2.full)), _bits(full_o))


@pytest.mark.parametrize("dtype,case", [("f32", "random"), ("bf16", "random"),
                                        ("f32", "all"), ("bf16", "none"), ("f32", "none-all")])
def test_multilevel_bilinear_bit_exact(av, orc, dtype, case):
    """Two transitions in bilinear mode on a 12x10 grid (ragged frame, C = 6):
    random selections (spans 1, 2 and 4 mixed), everything selected, nothing
    selected (span-4 merge), nothing then everything; the second upsample
    through both entry points (avits_selective_upsample and the selection +
    upsample call, which routes a mixed bilinear input through the cell
    map) and the merge, bit-exact against the oracle."""
    import torch
    from paper_2608_17995_gb300.workloads import random_scores, to_bf16_bits
    B, gh, gw, C = 2, 12, 10, 6
    M = gh * gw
    lat = np.random.default_rng(31).standard_normal((B, M, 4 * C)).astype(np.float32)
    if dtype == "bf16":
        lat = to_bf16_bits(lat)
    k1 = {"random": 30, "all": M, "none": 0, "none-all": 0}[case]
    _, m1, off1 = orc.topk(random_scores(41, B, M)[0], k1)
    g1 = _upsample(av, lat, dtype, gh, gw, m1, off1, k1, 1)
    o1 = orc.selective_upsample(lat, gh, gw, m1, mode="bilinear")
    assert np.array_equal(_bits(g1[0]), _bits(o1[0]))
    N1 = o1[0].shape[1]
    k2 = {"random": 70, "all": N1, "none": 0, "none-all": N1}[case]
    A2, V2 = random_scores(42, B, N1)
    S2 = orc.fuse(A2, V2, 0.5)
    _, m2, off2 = orc.topk(S2, k2)
    g2 = _upsample(av, o1[0], dtype, 2 * gh, 2 * gw, m2, off2, k2, 1, pos_in=o1[1],
                   span_in=o1[2])
    o2 = orc.selective_upsample(o1[0], 2 * gh, 2 * gw, m2, mode="bilinear", pos_in=o1[1],
                                span_in=o1[2])
    for a, b in zip(g2, o2):
        assert np.array_equal(_bits(a) if a.dtype.kind == "f" or a.dtype == np.uint16 else a,
                              _bits(b) if b.dtype.kind == "f" or b.dtype == np.uint16 else b)
    # the selection + upsample entry point on the same mixed input
    tdt = torch.bfloat16 if dtype == "bf16" else torch.float32
    NO = N1 + 3 * k2
    outs = [torch.full((B, NO, 4 * C), float("nan"), dtype=tdt, device="cuda"),
            torch.zeros(B, NO, 2, dtype=torch.int32, device="cuda"),
            torch.zeros(B, NO, dtype=torch.int32, device="cuda"),
            torch.zeros(B, NO, dtype=torch.int32, device="cuda"),
            torch.zeros(B, NO, dtype=torch.int8, device="cuda")]
    sel = torch.zeros(B, max(k2, 1), dtype=torch.int32, device="cuda")
    off = torch.zeros(B, N1, dtype=torch.int32, device="cuda")
    msk = torch.zeros(B, N1, dtype=torch.uint8, device="cuda")
    av.avits_select_upsample(_dev(A2), _dev(V2), 0.5, k2, sel, off, msk, _dev(o1[0], dtype),
                             2 * gh, 2 * gw, *outs, mode=1, pos_in=_dev(o1[1]),
                             span_in=_dev(o1[2]))
    assert _status(av) == 0
    assert np.array_equal(_np(msk), m2)
    assert np.array_equal(_bits(_np(outs[0])), _bits(o2[0]))
    assert np.array_equal(_np(outs[1]), o2[1]) and np.array_equal(_np(outs[2]), o2[2])
    if case == "none":
        assert np.all(o2[2] == 4)
    full_g = _merge(av, o2[0], dtype, o2[1], o2[2], 4 * gh, 4 * gw, 1)
    full_o, _ = orc.merge_final(o2[0], o2[1], o2[2], 4 * gh, 4 * gw, mode="bilinear")
    assert np.array_equal(_bits(full_g), _bits(full_o))


def test_multilevel_bilinear_rejects_other_spans(av, orc):
    """Spans outside {1, 2, 4} (or off their alignment) in a bilinear merge or
    a mixed bilinear upsample raise AVITS_ERR_COVERAGE on the device; the
    next valid call is clean."""
    import torch
    lat = np.random.default_rng(2).standard_normal((1, 4, 8)).astype(np.float32)
    out, pos, span, _, _ = orc.selective_upsample(lat, 2, 2, np.zeros((1, 4), np.uint8))
    # one span-8 token over the whole 8x8 frame
    big = np.zeros((1, 1, 8), np.float32)
    _merge(av, big, "f32", np.zeros((1, 1, 2), np.int32), np.full((1, 1), 8, np.int32), 8, 8, 1,
           expect_status=6)
    _merge(av, out, "f32", pos, span, 4, 4, 1)
    # a mixed upsample input whose span-2 token sits off its alignment
    bad = pos.copy()
    bad[0, 1] = (0, 1)
    mask = np.ones((1, 4), np.uint8)
    _, _, off = orc.topk(np.ones((1, 4), np.float32), 4)
    with pytest.raises(AssertionError):
        _upsample(av, out, "f32", 4, 4, mask, off, 4, 1, pos_in=bad, span_in=span)
    assert _status(av) == 0
    _upsample(av, out, "f32", 4, 4, mask, off, 4, 1, pos_in=pos, span_in=span)
