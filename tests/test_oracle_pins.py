"""Pins of the CPU oracle against what the paper and the mathematics fix.

None of these compares the oracle with itself or with the CUDA path: each
checks it against a brute-force re-statement, a closed form, an invariant, a
library routine or a hand-worked fixture (tests/golden/).
"""
import json
import math
import os

import numpy as np
import pytest

from helpers import as_f32, image_to_tokens, tokens_to_image

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def _golden(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)


# ---------------------------------------------------------------- spatial --

@pytest.mark.parametrize("seed,B,H,M,L,R,d,dt", [
    (0, 1, 2, 16, 8, 0, 16, "f32"),
    (1, 2, 3, 37, 11, 5, 24, "f32"),
    (2, 1, 4, 64, 32, 0, 64, "bf16"),
    (3, 2, 1, 7, 1, 0, 8, "bf16"),
    (4, 1, 2, 20, 0, 3, 8, "f32"),      # L = 0: no text mass
    (5, 1, 2, 9, 13, 0, 8, "f32"),      # more text keys than image keys
])
def test_spatial_matches_full_softmax(oracle_mod, seed, B, H, M, L, R, d, dt):
    """P1: the oracle equals a materialised-softmax NumPy computation."""
    from oracle import brute
    from paper_2608_17995_gb300.workloads import to_bf16_bits
    rng = np.random.default_rng(seed)
    Nk = L + M + R
    q = rng.standard_normal((B, H, M, d)).astype(np.float32) * 0.7
    k = rng.standard_normal((B, H, Nk, d)).astype(np.float32) * 0.7
    if dt == "bf16":
        q, k = to_bf16_bits(q), to_bf16_bits(k)
    scale = 1.0 / math.sqrt(d)
    A, mass, lse = oracle_mod.score_spatial(q, k, L, scale)
    A_ref, mass_ref = brute.spatial_full_softmax(q, k, L, scale)
    np.testing.assert_allclose(mass, mass_ref, rtol=1e-12, atol=1e-14)
    np.testing.assert_allclose(A, A_ref.astype(np.float32), rtol=1e-6, atol=1e-7)
    # invariants: text + image mass = 1 and mass = exp(lse_txt - lse_all)
    assert np.all(mass >= 0) and np.all(mass <= 1 + 1e-15)
    if L > 0:
        np.testing.assert_allclose(np.exp(lse[..., 1] - lse[..., 0]), mass, rtol=1e-12)
    else:
        assert np.all(mass == 0) and np.all(np.isneginf(lse[..., 1]))
    # lse over all keys (the value a model's attention forward returns, the
    # input of the lse-based entry point) against a brute-force logsumexp
    qf, kf = brute.as_f64(q), brute.as_f64(k)
    logits = scale * np.einsum("bhmd,bhnd->bhmn", qf, kf)
    mx = logits.max(-1, keepdims=True)
    lse_ref = (mx + np.log(np.exp(logits - mx).sum(-1, keepdims=True)))[..., 0]
    np.testing.assert_allclose(lse[..., 0], lse_ref, rtol=1e-12, atol=1e-12)


def test_spatial_q_zero_uniform(oracle_mod):
    """P2: Q = 0 makes every logit 0, so the text mass is exactly L/Nk (1/9 for
    the tiny shape: 32 text keys of 288)."""
    B, H, M, L, d = 1, 2, 256, 32, 64
    Nk = L + M
    q = np.zeros((B, H, M, d), np.float32)
    k = np.random.default_rng(0).standard_normal((B, H, Nk, d)).astype(np.float32)
    A, mass, _ = oracle_mod.score_spatial(q, k, L, 0.125)
    assert np.allclose(mass, 1.0 / 9.0, rtol=0, atol=1e-15)
    assert np.allclose(A, np.float32(1.0 / 9.0), rtol=0, atol=0)


def test_spatial_one_hot_logit_and_head_mean(oracle_mod):
    """P2: one text logit a (others 0) gives mass (e^a + L-1)/(e^a + Nk-1);
    different a per head checks the mean over heads (Eq. 3) and the scale."""
    L, M, d, scale = 5, 3, 4, 0.5
    Nk = L + M
    a_h = [2.0, -1.0, 0.25]           # a/scale exact in fp32
    H = len(a_h)
    q = np.zeros((1, H, M, d), np.float32)
    k = np.zeros((1, H, Nk, d), np.float32)
    for h, a in enumerate(a_h):
        k[0, h, 0, 0] = 1.0              # text key 0 along e0
        k[0, h, 1:, 1] = 1.0             # every other key along e1
        q[0, h, :, 0] = a / scale        # logit a on key 0, 0 elsewhere
    A, mass, _ = oracle_mod.score_spatial(q, k, L, scale)
    expect = [(math.exp(a) + L - 1) / (math.exp(a) + Nk - 1) for a in a_h]
    for h in range(H):
        np.testing.assert_allclose(mass[0, h], expect[h], rtol=1e-14)
    np.testing.assert_allclose(A[0], np.float32(np.mean(expect)), rtol=1e-7)


def test_spatial_weight_accumulate_rows_and_strides(oracle_mod):
    """Aggregation over blocks/steps: A_in + w * mean_h mass; a row subset and a
    [B,N,H,d]-strided layout give the same numbers."""
    rng = np.random.default_rng(7)
    B, H, M, L, d = 2, 3, 10, 4, 8
    Nk = L + M
    q = rng.standard_normal((B, H, M, d)).astype(np.float32)
    k = rng.standard_normal((B, H, Nk, d)).astype(np.float32)
    A0, mass, _ = oracle_mod.score_spatial(q, k, L, 0.3)
    A_in = rng.random((B, M)).astype(np.float32)
    A1, _, _ = oracle_mod.score_spatial(q, k, L, 0.3, weight=0.25, A_in=A_in)
    np.testing.assert_allclose(A1, (A_in + 0.25 * mass.mean(1)).astype(np.float32), rtol=1e-6)
    rows = [3, 11, 19]
    A2, _, _ = oracle_mod.score_spatial(q, k, L, 0.3, rows=rows)
    np.testing.assert_array_equal(A2.ravel()[rows], A0.ravel()[rows])
    # token-major [B, N, H, d] storage with the image rows after L text rows
    qa = np.zeros((B, L + M, H, d), np.float32)
    qa[:, L:] = q.transpose(0, 2, 1, 3)
    ka = np.ascontiguousarray(k.transpose(0, 2, 1, 3))
    qflat = np.ascontiguousarray(qa[:, L:]).reshape(-1)  # contiguous copy for flat pointer
    A3, _, _ = oracle_mod.score_spatial(
        qflat, ka.reshape(-1), L, 0.3, shape=(B, H, M, Nk, d),
        q_strides=(M * H * d, d, H * d), k_strides=(Nk * H * d, d, H * d))
    np.testing.assert_array_equal(A3, A0)


def test_spatial_l2norm_reading_scale_invariant(oracle_mod):
    """c2 literal reading: with unit-normalised q and k rows the result does not
    change when q rows are rescaled, and a query equal to text key 0 (all other
    keys orthogonal to it) gets logit = scale on that key and 0 elsewhere."""
    rng = np.random.default_rng(3)
    B, H, M, L, d = 1, 2, 6, 3, 8
    q = rng.standard_normal((B, H, M, d)).astype(np.float32)
    k = rng.standard_normal((B, H, L + M, d)).astype(np.float32)
    A, _, _ = oracle_mod.score_spatial(q, k, L, 2.0, l2norm=True)
    q2 = q * rng.uniform(0.5, 4.0, (B, H, M, 1)).astype(np.float32)
    A2, _, _ = oracle_mod.score_spatial(q2, k, L, 2.0, l2norm=True)
    np.testing.assert_allclose(A, A2, rtol=1e-6)
    qe = np.zeros((1, 1, 2, 4), np.float32)
    ke = np.zeros((1, 1, 5, 4), np.float32)
    qe[0, 0, :, 0] = 3.0
    ke[0, 0, 0, 0] = 7.0            # text key 0, parallel to q
    ke[0, 0, 1:, 1] = 2.0           # text key 1 and the image keys, orthogonal
    _, me, _ = oracle_mod.score_spatial(qe, ke, 2, 1.5, l2norm=True)
    np.testing.assert_allclose(me[0, 0], (math.exp(1.5) + 1) / (math.exp(1.5) + 4), rtol=1e-14)


# --------------------------------------------------------------- temporal --

@pytest.mark.parametrize("seed,B,H,M,Nk,d", [(0, 2, 3, 7, 40, 16), (1, 1, 2, 33, 97, 8)])
def test_spatial_text_mask(oracle_mod, seed, B, H, M, Nk, d):
    """Interleaved text keys (MLLM-style sequences): the masked oracle equals
    the materialised softmax with the masked columns summed; a first-L mask
    is the L form bit for bit; a mask and its complement add up to 1; moving
    keys and mask together changes nothing."""
    from oracle import brute
    rng = np.random.default_rng(seed)
    q = rng.standard_normal((B, H, M, d)).astype(np.float32)
    k = rng.standard_normal((B, H, Nk, d)).astype(np.float32)
    mask = (rng.random((B, Nk)) < 0.3).astype(np.uint8)
    A, mass, _ = oracle_mod.score_spatial(q, k, 0, 0.4, text_mask=mask)
    A_b, mass_b = brute.spatial_full_softmax(q, k, 0, 0.4, text_mask=mask)
    np.testing.assert_allclose(mass, mass_b, rtol=0, atol=1e-12)
    np.testing.assert_allclose(A, A_b, rtol=1e-6, atol=1e-7)
    L = Nk // 3
    first = np.zeros((B, Nk), np.uint8)
    first[:, :L] = 1
    _, mass_l, lse_l = oracle_mod.score_spatial(q, k, L, 0.4)
    _, mass_f, lse_f = oracle_mod.score_spatial(q, k, 0, 0.4, text_mask=first)
    assert np.array_equal(mass_l, mass_f) and np.array_equal(lse_l, lse_f)
    _, mass_c, _ = oracle_mod.score_spatial(q, k, 0, 0.4, text_mask=1 - mask)
    np.testing.assert_allclose(mass + mass_c, 1.0, rtol=0, atol=1e-12)
    perm = rng.permutation(Nk)
    _, mass_p, _ = oracle_mod.score_spatial(q, np.ascontiguousarray(k[:, :, perm]), 0, 0.4,
                                            text_mask=np.ascontiguousarray(mask[:, perm]))
    np.testing.assert_allclose(mass_p, mass, rtol=0, atol=1e-12)


# ------------------------------------------------ joint-attention forward (Eq. 4-5)

@pytest.mark.parametrize("seed,B,H,Mq,Nk,L,d,dt", [
    (0, 1, 2, 9, 13, 4, 8, "f32"),
    (1, 2, 3, 17, 40, 12, 16, "bf16"),
    (2, 1, 1, 5, 7, 0, 4, "f32"),       # no text key
    (3, 1, 2, 6, 6, 6, 8, "f32"),       # every key a text key
])
def test_attention_matches_torch_sdpa(oracle_mod, seed, B, H, Mq, Nk, L, d, dt):
    """The forward's O against torch's CPU scaled_dot_product_attention in fp64
    (an independent library routine), its logsumexp against torch.logsumexp of
    the logits, and mass / lse_txt / A against the spatial-score function,
    which is pinned on its own above (Eq. 3, 5)."""
    import torch
    rng = np.random.default_rng(seed)
    q = rng.standard_normal((B, H, Mq, d)).astype(np.float32)
    k = rng.standard_normal((B, H, Nk, d)).astype(np.float32)
    v = rng.standard_normal((B, H, Nk, d)).astype(np.float32)
    if dt == "bf16":
        from paper_2608_17995_gb300.workloads import to_bf16_bits
        q, k, v = to_bf16_bits(q), to_bf16_bits(k), to_bf16_bits(v)
    scale = 1.0 / math.sqrt(d)
    O, lse, mass, A = oracle_mod.attention(q, k, v, L, scale)
    tq, tk, tv = (torch.tensor(as_f32(x), dtype=torch.float64) for x in (q, k, v))
    ref = torch.nn.functional.scaled_dot_product_attention(tq, tk, tv, scale=scale).numpy()
    np.testing.assert_allclose(O, ref, rtol=1e-12, atol=1e-12)
    logits = torch.einsum("bhid,bhjd->bhij", tq, tk) * scale
    np.testing.assert_allclose(lse[..., 0], torch.logsumexp(logits, -1).numpy(), rtol=1e-12,
                               atol=1e-12)
    A_s, mass_s, lse_s = oracle_mod.score_spatial(q, k, L, scale)
    np.testing.assert_allclose(mass, mass_s, rtol=1e-12, atol=1e-15)
    np.testing.assert_allclose(lse[..., 1], lse_s[..., 1], rtol=1e-12, atol=1e-12)
    np.testing.assert_array_equal(A, A_s)
    if L == 0:
        assert np.all(np.isneginf(lse[..., 1])) and np.all(mass == 0)
    if L == Nk:
        np.testing.assert_allclose(mass, 1.0, rtol=0, atol=1e-15)


def test_attention_closed_forms(oracle_mod):
    """Closed forms that catch a missing normalisation, swapped k / v, a wrong
    scale and a transposed product:
      v_j = c for every key -> O_i = c (the softmax weights sum to one);
      Q = 0 -> uniform weights, O_i = mean_j v_j, lse = log Nk, mass = L/Nk;
      one logit a on key 0 (others 0) ->
        O_i = (e^a v_0 + sum_{j>0} v_j) / (e^a + Nk - 1)."""
    rng = np.random.default_rng(11)
    B, H, Mq, Nk, L, d = 1, 2, 4, 6, 2, 4
    q = rng.standard_normal((B, H, Mq, d)).astype(np.float32)
    k = rng.standard_normal((B, H, Nk, d)).astype(np.float32)
    c = np.array([0.5, -2.0, 3.25, 1.0], np.float32)
    v = np.broadcast_to(c, (B, H, Nk, d)).astype(np.float32).copy()
    O, _, _, _ = oracle_mod.attention(q, k, v, L, 0.7)
    np.testing.assert_allclose(O, np.broadcast_to(c, O.shape), rtol=1e-14, atol=1e-14)

    v = rng.standard_normal((B, H, Nk, d)).astype(np.float32)
    O, lse, mass, A = oracle_mod.attention(np.zeros_like(q), k, v, L, 0.7)
    np.testing.assert_allclose(O, np.broadcast_to(v.astype(np.float64).mean(2, keepdims=True),
                                                  O.shape), rtol=1e-13, atol=1e-14)
    np.testing.assert_allclose(lse[..., 0], math.log(Nk), rtol=1e-15)
    np.testing.assert_allclose(mass, L / Nk, rtol=1e-14)

    a, scale = 1.5, 0.5
    q = np.zeros((B, H, Mq, d), np.float32)
    k = np.zeros((B, H, Nk, d), np.float32)
    k[..., 0, 0] = 1.0
    k[..., 1:, 1] = 1.0
    q[..., 0] = a / scale
    O, lse, _, _ = oracle_mod.attention(q, k, v, L, scale)
    vv = v.astype(np.float64)
    expect = (math.exp(a) * vv[:, :, :1] + vv[:, :, 1:].sum(2, keepdims=True)) / (math.exp(a) + Nk - 1)
    np.testing.assert_allclose(O, np.broadcast_to(expect, O.shape), rtol=1e-13, atol=1e-14)
    np.testing.assert_allclose(lse[..., 0], math.log(math.exp(a) + Nk - 1), rtol=1e-14)


def test_attention_permutation_rows_and_accumulate(oracle_mod):
    """Permuting the keys and values together (within the text block and within
    the image block) leaves every output unchanged; permuting the values alone
    changes O.  A row subset gives the same rows; accumulate adds w * A."""
    rng = np.random.default_rng(5)
    B, H, Mq, Nk, L, d = 2, 3, 7, 11, 4, 8
    q = rng.standard_normal((B, H, Mq, d)).astype(np.float32)
    k = rng.standard_normal((B, H, Nk, d)).astype(np.float32)
    v = rng.standard_normal((B, H, Nk, d)).astype(np.float32)
    O, lse, mass, A = oracle_mod.attention(q, k, v, L, 0.3)
    perm = np.concatenate([rng.permutation(L), L + rng.permutation(Nk - L)])
    O2, lse2, mass2, A2 = oracle_mod.attention(q, np.ascontiguousarray(k[:, :, perm]),
                                               np.ascontiguousarray(v[:, :, perm]), L, 0.3)
    np.testing.assert_allclose(O2, O, rtol=1e-12, atol=1e-13)
    np.testing.assert_allclose(lse2, lse, rtol=1e-13)
    np.testing.assert_allclose(mass2, mass, rtol=1e-12)
    O3, _, _, _ = oracle_mod.attention(q, k, np.ascontiguousarray(v[:, :, perm]), L, 0.3)
    assert np.abs(O3 - O).max() > 1e-3
    rows = [3, Mq + 5, 0]
    O4, _, _, A4 = oracle_mod.attention(q, k, v, L, 0.3, rows=rows)
    for f in rows:
        b, i = divmod(f, Mq)
        np.testing.assert_array_equal(O4[b, :, i], O[b, :, i])
        assert A4[b, i] == A[b, i]
    A_in = rng.standard_normal((B, Mq)).astype(np.float32)
    _, _, _, A5 = oracle_mod.attention(q, k, v, L, 0.3, weight=0.25, A_in=A_in)
    np.testing.assert_allclose(A5, A_in + 0.25 * A.astype(np.float64), rtol=1e-6, atol=1e-7)


def test_temporal_closed_forms(oracle_mod):
    """P2: h_t = c h_prev gives |c-1| |h| / (|h| + eps); h_prev = 0 gives |h_t|/eps."""
    rng = np.random.default_rng(1)
    B, N, D = 2, 9, 33
    hp = rng.standard_normal((B, N, D)).astype(np.float32)
    for c in (3.0, 0.5, 1.0, -2.0):
        ht = (hp * np.float32(c)).astype(np.float32)
        V = oracle_mod.score_temporal(ht, hp, 1e-6)
        nrm = np.sqrt((hp.astype(np.float64) ** 2).sum(-1))
        np.testing.assert_allclose(V, abs(c - 1) * nrm / (nrm + 1e-6), rtol=1e-6, atol=1e-12)
    V0 = oracle_mod.score_temporal(hp, np.zeros_like(hp), 1e-6)
    np.testing.assert_allclose(V0, np.sqrt((hp.astype(np.float64) ** 2).sum(-1)) / 1e-6, rtol=1e-6)
    # swapped arguments are not the same function (catches a transposed operand)
    Vs = oracle_mod.score_temporal(hp, (hp * 3).astype(np.float32), 1e-6)
    assert np.allclose(Vs, 2.0 / 3.0, rtol=1e-5)


def test_temporal_variance_closed_forms(oracle_mod):
    """Eq. 6-7: N_T = 2 gives |z1 - z2|^2 / (2D); snapshots (0, x, 2x) give
    mean_d x_d^2; constant snapshots give 0."""
    rng = np.random.default_rng(2)
    B, N, D = 1, 5, 16
    z1 = rng.standard_normal((B, N, D)).astype(np.float32)
    z2 = rng.standard_normal((B, N, D)).astype(np.float32)
    V = oracle_mod.score_temporal_var([z1, z2])
    np.testing.assert_allclose(V, ((z1.astype(np.float64) - z2) ** 2).sum(-1) / (2 * D), rtol=1e-6)
    x = rng.standard_normal((B, N, D)).astype(np.float32)
    V3 = oracle_mod.score_temporal_var([np.zeros_like(x), x, (2 * x).astype(np.float32)])
    np.testing.assert_allclose(V3, (x.astype(np.float64) ** 2).mean(-1), rtol=1e-6)
    assert np.all(oracle_mod.score_temporal_var([x, x, x, x]) == 0)


# ----------------------------------------------------------- fuse / topk --

def test_minmax_and_ties_golden(oracle_mod):
    """P6 (tests/golden/p6_select_ties.json)."""
    g = _golden("p6_select_ties.json")
    tc = g["topk_case"]
    sel, mask, off = oracle_mod.topk(np.array([tc["S"]], np.float32), tc["k"])
    assert sel[0].tolist() == tc["sel_idx"]
    assert off[0].tolist() == tc["tok_offset"]
    mc = g["minmax_case"]
    A = np.array([mc["A"]], np.float32)
    # alpha = 1 gives S = A^ exactly
    S = oracle_mod.fuse(A, np.zeros_like(A), 1.0, mc["eps"])
    den = np.float32(np.float32(2.0) + np.float32(1e-6))
    expect = [np.float32(0.0), np.float32(1.0) / den, np.float32(2.0) / den]
    assert S[0].tolist() == [float(e) for e in expect]


def test_fuse_alpha_arms_and_range(oracle_mod):
    """P7 (the alpha = 1 / alpha = 0 ablation arms): the ranking follows A^ alone
    or V^ alone; every S lies in [0,1]; a constant score normalises to 0."""
    from paper_2608_17995_gb300.workloads import random_scores
    A, V = random_scores(11, 3, 200)
    for alpha, ref in ((1.0, A), (0.0, V)):
        S = oracle_mod.fuse(A, V, alpha)
        for b in range(3):
            assert np.array_equal(np.argsort(-S[b], kind="stable"), np.argsort(-ref[b], kind="stable"))
    S = oracle_mod.fuse(A, V, 0.37)
    assert S.min() >= 0.0 and S.max() <= 1.0
    Sc = oracle_mod.fuse(np.full((1, 10), 0.3, np.float32), V[:1, :10], 0.5)
    np.testing.assert_allclose(Sc, 0.5 * oracle_mod.fuse(V[:1, :10], V[:1, :10], 1.0), rtol=1e-6)


def test_perturbation_breaks_ties_and_is_one_rounded_add(oracle_mod):
    """Eq. 9's tie-breaking noise (caller-supplied): zero noise is the plain
    selection bit for bit; +1e-6 on one of three tied tokens moves it ahead
    of the others (a dropped or sign-flipped term keeps the lower-index
    tokens); S' - S equals the noise to within half an ulp of S'."""
    A = np.array([[0.5, 0.9, 0.5, 0.5, 0.1]], np.float32)
    V = np.zeros_like(A)
    S0 = oracle_mod.fuse(A, V, 1.0)
    Sz = oracle_mod.fuse(A, V, 1.0, perturb=np.zeros_like(A))
    assert np.array_equal(S0.view(np.uint32), Sz.view(np.uint32))
    assert oracle_mod.topk(S0, 3)[0][0].tolist() == [0, 1, 2]
    d = np.array([[0.0, 0.0, 0.0, 1e-6, 0.0]], np.float32)
    S1 = oracle_mod.fuse(A, V, 1.0, perturb=d)
    assert oracle_mod.topk(S1, 3)[0][0].tolist() == [0, 1, 3]
    rng = np.random.default_rng(5)
    Ar, Vr = rng.random((2, 300), dtype=np.float32), rng.random((2, 300), dtype=np.float32)
    dr = (1e-6 * rng.standard_normal((2, 300))).astype(np.float32)
    Sa = oracle_mod.fuse(Ar, Vr, 0.5).astype(np.float64)
    Sb = oracle_mod.fuse(Ar, Vr, 0.5, perturb=dr)
    err = np.abs(Sb.astype(np.float64) - Sa - dr.astype(np.float64))
    assert np.all(err <= 0.5 * np.spacing(Sb).astype(np.float64))


@pytest.mark.parametrize("seed,M,k,ties", [(0, 50, 7, False), (1, 300, 300, True),
                                            (2, 1000, 0, True), (3, 1024, 307, True),
                                            (4, 1, 1, False)])
def test_topk_matches_full_sort(oracle_mod, seed, M, k, ties):
    """P1: TopK equals a full stable sort; |S| = k; tok_offset invariants."""
    from oracle import brute
    from paper_2608_17995_gb300.workloads import random_scores
    S = random_scores(seed, 2, M, ties=ties)[0]
    if M > 4:
        S[0, 3] = np.nan
        S[1, 1] = -0.0
        S[1, 2] = 0.0
    sel, mask, off = oracle_mod.topk(S, k)
    ref = brute.topk_full_sort(S, k)
    assert np.array_equal(sel, ref)
    assert np.all(mask.sum(1) == k)
    for b in range(2):
        assert np.all(np.diff(off[b]) >= 1)
        assert off[b, -1] + 1 + 3 * int(mask[b, -1]) == M + 3 * k
        assert np.array_equal(np.nonzero(mask[b])[0], sel[b])


def test_topk_nan_and_signed_zero(oracle_mod):
    S = np.array([[np.nan, -0.0, 0.0, -1.0, np.nan]], np.float32)
    assert oracle_mod.topk(S, 2)[0][0].tolist() == [1, 2]        # -0 == +0, lower index
    assert oracle_mod.topk(S, 4)[0][0].tolist() == [0, 1, 2, 3]  # NaN after -1


# ------------------------------------------------------ upsample / merge --

def test_upsample_golden_4x4(oracle_mod):
    """P5: hand-worked 4x4 -> 8x8 example (tests/golden/p5_upsample_4x4.json)."""
    g = _golden("p5_upsample_4x4.json")
    S = np.array([g["S"]], np.float32)
    sel, mask, off = oracle_mod.topk(S, g["k"])
    assert sel[0].tolist() == g["sel_idx"]
    assert off[0].tolist() == g["tok_offset"]
    lat = np.array([[[10 * i + 1, 10 * i + 2, 10 * i + 3, 10 * i + 4] for i in range(16)]],
                   np.float32)
    out, pos, span, src_tok, src_sub = oracle_mod.selective_upsample(lat, 4, 4, mask)
    assert out.shape[1] == g["n_out"]
    for e in g["out_tokens"]:
        o = e["o"]
        assert pos[0, o].tolist() == e["pos"], o
        assert span[0, o] == e["span"] and src_tok[0, o] == e["src_tok"]
        assert src_sub[0, o] == e["src_sub"]
        assert out[0, o].tolist() == e["val"], o
    full, cover = oracle_mod.merge_final(out, pos, span, 8, 8)
    assert cover.sum() == g["covered_cells"] and np.all(cover == 1)


def _dense_case(seed, B, gh, gw, C, dtype=np.float32):
    rng = np.random.default_rng(seed)
    return rng.standard_normal((B, gh * gw, C * 4)).astype(dtype)


def test_upsample_nearest_dense_is_repeat(oracle_mod):
    """P4: with every token selected, nearest upsampling is np.repeat x2 of the
    pixel image (torch's nearest resize)."""
    B, gh, gw, C = 2, 5, 7, 3
    lat = _dense_case(0, B, gh, gw, C)
    mask = np.ones((B, gh * gw), np.uint8)
    out, pos, span, _, _ = oracle_mod.selective_upsample(lat, gh, gw, mask)
    full, _ = oracle_mod.merge_final(out, pos, span, 2 * gh, 2 * gw)
    img = tokens_to_image(lat, gh, gw)
    ref = np.repeat(np.repeat(img, 2, axis=2), 2, axis=3)
    assert np.array_equal(tokens_to_image(full, 2 * gh, 2 * gw), ref)


def test_upsample_bilinear_dense_matches_torch(oracle_mod):
    """P4: with every token selected, bilinear upsampling equals
    torch.nn.functional.interpolate(scale 2, bilinear, align_corners=False)."""
    import torch
    g = _golden("p6_select_ties.json")["bilinear_1d_case"]
    src = torch.tensor(g["src"], dtype=torch.float32).view(1, 1, 1, 2)
    t1 = torch.nn.functional.interpolate(src, scale_factor=2, mode="bilinear", align_corners=False)
    assert t1.view(-1).tolist()[:4] == g["out"]
    B, gh, gw, C = 2, 6, 5, 2
    lat = _dense_case(1, B, gh, gw, C)
    mask = np.ones((B, gh * gw), np.uint8)
    out, pos, span, _, _ = oracle_mod.selective_upsample(lat, gh, gw, mask, mode="bilinear")
    full, _ = oracle_mod.merge_final(out, pos, span, 2 * gh, 2 * gw, mode="bilinear")
    img = torch.from_numpy(tokens_to_image(lat, gh, gw))
    ref = torch.nn.functional.interpolate(img, scale_factor=2, mode="bilinear",
                                          align_corners=False).numpy()
    np.testing.assert_allclose(tokens_to_image(full, 2 * gh, 2 * gw), ref, atol=1e-6, rtol=0)
    # the 1-D worked case through the oracle: a 1x1 grid of C=1 holding [[0,4],[0,4]]
    lat1 = np.array([[[0.0, 4.0, 0.0, 4.0]]], np.float32)
    o1, p1, s1, _, _ = oracle_mod.selective_upsample(lat1, 1, 1, np.ones((1, 1), np.uint8),
                                                     mode="bilinear")
    f1, _ = oracle_mod.merge_final(o1, p1, s1, 2, 2, mode="bilinear")
    assert tokens_to_image(f1, 2, 2)[0, 0, 0].tolist() == g["out"]


@pytest.mark.parametrize("mode", ["nearest", "bilinear"])
def test_merge_none_selected_is_plain_resize(oracle_mod, mode):
    """P3: with k = 0 the merge is the plain 2x resize of the low-res latent."""
    import torch
    B, gh, gw, C = 1, 4, 6, 2
    lat = _dense_case(2, B, gh, gw, C)
    mask = np.zeros((B, gh * gw), np.uint8)
    out, pos, span, _, src_sub = oracle_mod.selective_upsample(lat, gh, gw, mask)
    assert np.all(src_sub == -1) and np.array_equal(out, lat)
    full, _ = oracle_mod.merge_final(out, pos, span, 2 * gh, 2 * gw, mode=mode)
    img = torch.from_numpy(tokens_to_image(lat, gh, gw))
    ref = torch.nn.functional.interpolate(img, scale_factor=2, mode=mode,
                                          **({} if mode == "nearest" else {"align_corners": False}))
    np.testing.assert_allclose(tokens_to_image(full, 2 * gh, 2 * gw), ref.numpy(), atol=1e-6, rtol=0)


def test_merge_of_selective_nearest_is_nearest_everywhere(oracle_mod):
    """P3: merge(upsample(x, any selection, nearest), nearest) = nearest 2x of x,
    every cell covered exactly once, N_out = M + 3k."""
    from paper_2608_17995_gb300.workloads import random_scores
    B, gh, gw, C, k = 2, 8, 8, 4, 19
    lat = _dense_case(3, B, gh, gw, C)
    S = random_scores(5, B, gh * gw)[0]
    _, mask, _ = oracle_mod.topk(S, k)
    out, pos, span, src_tok, src_sub = oracle_mod.selective_upsample(lat, gh, gw, mask)
    assert out.shape[1] == gh * gw + 3 * k
    full, cover = oracle_mod.merge_final(out, pos, span, 2 * gh, 2 * gw)
    assert np.all(cover == 1)
    img = tokens_to_image(lat, gh, gw)
    assert np.array_equal(tokens_to_image(full, 2 * gh, 2 * gw),
                          np.repeat(np.repeat(img, 2, axis=2), 2, axis=3))


def test_merge_bilinear_selected_cells_verbatim(oracle_mod):
    """Bilinear merge copies span-1 cells verbatim and resamples span-2 cells
    from the pooled low-res grid; with all tokens deferred except a few, the
    deferred cells equal the bilinear resize of the grid where the selected
    cells are replaced by the pooled children."""
    import torch
    from paper_2608_17995_gb300.workloads import random_scores
    B, gh, gw, C, k = 1, 6, 6, 2, 9
    lat = _dense_case(4, B, gh, gw, C)
    _, mask, _ = oracle_mod.topk(random_scores(9, B, gh * gw)[0], k)
    out, pos, span, src_tok, src_sub = oracle_mod.selective_upsample(lat, gh, gw, mask, "bilinear")
    full, _ = oracle_mod.merge_final(out, pos, span, 2 * gh, 2 * gw, mode="bilinear")
    fimg = tokens_to_image(full, 2 * gh, 2 * gw)
    # selected children appear verbatim
    for o in range(out.shape[1]):
        if span[0, o] == 1:
            Y, X = pos[0, o]
            cell = fimg[0, :, 2 * Y:2 * Y + 2, 2 * X:2 * X + 2].reshape(C, 4)
            assert np.array_equal(cell.reshape(-1), out[0, o].reshape(C, 4).reshape(-1))
    # pooled grid: deferred tokens as-is, selected tokens = 2x2 means of children
    pooled = lat.copy()
    for i in np.nonzero(mask[0])[0]:
        kids = out[0][(src_tok[0] == i)]
        for ch in range(4):
            for c in range(C):
                pooled[0, i, c * 4 + ch] = kids[ch, c * 4:(c + 1) * 4].astype(np.float64).mean()
    ref = torch.nn.functional.interpolate(torch.from_numpy(tokens_to_image(pooled, gh, gw)),
                                          scale_factor=2, mode="bilinear",
                                          align_corners=False).numpy()
    for o in range(out.shape[1]):
        if span[0, o] == 2:
            Y, X = pos[0, o]
            np.testing.assert_allclose(fimg[0, :, 2 * Y:2 * Y + 4, 2 * X:2 * X + 4],
                                       ref[0, :, 2 * Y:2 * Y + 4, 2 * X:2 * X + 4], atol=1e-6)


def test_merge_rejects_bad_tiling(oracle_mod):
    """P3: a sequence that covers a cell twice (or leaves one empty) is refused."""
    lat = _dense_case(5, 1, 2, 2, 1)
    out, pos, span, _, _ = oracle_mod.selective_upsample(lat, 2, 2, np.zeros((1, 4), np.uint8))
    pos2 = pos.copy()
    pos2[0, 1] = pos2[0, 0]
    with pytest.raises(ValueError):
        oracle_mod.merge_final(out, pos2, span, 4, 4)
    _, cover = oracle_mod.merge_final(out, pos2, span, 4, 4, check=False)
    assert cover.max() == 2 and cover.min() == 0


def test_two_level_schedule_is_nearest_4x(oracle_mod):
    """Batched multi-stage reading (two transitions, nearest): with no denoising
    in between, merging the second mixed sequence gives the nearest 4x resize
    of the first latent; spans 1, 2 and 4 appear and tile the frame once."""
    from paper_2608_17995_gb300.workloads import random_scores
    B, g, C = 2, 4, 2
    lat = _dense_case(6, B, g, g, C)
    _, m1, _ = oracle_mod.topk(random_scores(1, B, g * g)[0], 8)
    o1, p1, s1, _, _ = oracle_mod.selective_upsample(lat, g, g, m1)
    N1 = o1.shape[1]
    _, m2, _ = oracle_mod.topk(random_scores(2, B, N1)[0], 12)
    o2, p2, s2, _, _ = oracle_mod.selective_upsample(o1, 2 * g, 2 * g, m2, pos_in=p1, span_in=s1)
    assert set(np.unique(s2)) <= {1, 2, 4} and 4 in set(np.unique(s2))
    full, cover = oracle_mod.merge_final(o2, p2, s2, 4 * g, 4 * g)
    assert np.all(cover == 1)
    img = tokens_to_image(lat, g, g)
    ref = np.repeat(np.repeat(img, 4, axis=2), 4, axis=3)
    assert np.array_equal(tokens_to_image(full, 4 * g, 4 * g), ref)


def test_bf16_rounding_is_nearest_even(oracle_mod):
    """bf16 outputs of the oracle round to nearest even (checked through a
    bilinear case whose fp32 results fall between bf16 neighbours)."""
    import torch
    from paper_2608_17995_gb300.workloads import to_bf16_bits
    B, gh, gw, C = 1, 3, 3, 2
    lat32 = _dense_case(7, B, gh, gw, C)
    latb = to_bf16_bits(lat32)
    mask = np.ones((B, gh * gw), np.uint8)
    outb = oracle_mod.selective_upsample(latb, gh, gw, mask, mode="bilinear")[0]
    out32 = oracle_mod.selective_upsample(as_f32(latb), gh, gw, mask, mode="bilinear")[0]
    ref = torch.from_numpy(out32).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(outb, ref)


# ------------------------------------- multi-level bilinear (Sec. 3.2, Stages 2-3)

def _bil2x(img):
    import torch
    return torch.nn.functional.interpolate(torch.from_numpy(np.ascontiguousarray(img)),
                                           scale_factor=2, mode="bilinear",
                                           align_corners=False).numpy()


def _mixed_image(out, pos, span, fh, fw):
    """Pixel image of a mixed sequence (each token pixel over its s x s footprint)."""
    B, N, T = out.shape
    C = T // 4
    img = np.zeros((B, C, 2 * fh, 2 * fw), np.float32)
    for b in range(B):
        for t in range(N):
            y, x = pos[b, t]
            s = span[b, t]
            pix = out[b, t].reshape(C, 2, 2)
            img[b, :, 2 * y:2 * y + 2 * s, 2 * x:2 * x + 2 * s] = np.repeat(np.repeat(pix, s, 1), s, 2)
    return img


@pytest.mark.parametrize("first", ["all", "none"])
def test_multilevel_bilinear_two_transitions_all_selected(oracle_mod, first):
    """Two transitions in bilinear mode with every token selected at the
    second: after an all-selected first transition the children are the 2x
    bilinear resize of the 2x resize of the latent (torch, twice); after an
    all-deferred first one (span-2 tokens, whose level-1 image is the latent
    itself) they are its single 2x resize.  Merging the all-deferred-then-
    selected sequence (span 2 everywhere) gives the twice-resized latent."""
    B, g, C = 2, 4, 3
    lat = _dense_case(21, B, g, g, C)
    img = tokens_to_image(lat, g, g)
    m1 = np.full((B, g * g), 1 if first == "all" else 0, np.uint8)
    o1, p1, s1, _, _ = oracle_mod.selective_upsample(lat, g, g, m1, mode="bilinear")
    N1 = o1.shape[1]
    o2, p2, s2, _, _ = oracle_mod.selective_upsample(o1, 2 * g, 2 * g, np.ones((B, N1), np.uint8),
                                                     mode="bilinear", pos_in=p1, span_in=s1)
    got = _mixed_image(o2, p2, s2, 4 * g, 4 * g)
    if first == "all":
        ref = _bil2x(_bil2x(img))
        assert np.all(s2 == 1)
    else:
        ref = np.repeat(np.repeat(_bil2x(img), 2, 2), 2, 3)   # span-2 children, one pixel per 2x2
        assert np.all(s2 == 2)
    np.testing.assert_allclose(got, ref, rtol=0, atol=2e-6)
    full, cover = oracle_mod.merge_final(o2, p2, s2, 4 * g, 4 * g, mode="bilinear")
    assert np.all(cover == 1)
    np.testing.assert_allclose(tokens_to_image(full, 4 * g, 4 * g), _bil2x(_bil2x(img)), rtol=0,
                               atol=3e-6)


def test_multilevel_merge_of_span4_tokens_is_two_resizes(oracle_mod):
    """Two all-deferred transitions leave span-4 tokens only; the merge's
    cascade (level 2 = the latent, level 1 its 2x resize, level 0 that one's)
    equals torch's bilinear 2x applied twice."""
    B, g, C = 1, 4, 2
    lat = _dense_case(22, B, g, g, C)
    o1, p1, s1, _, _ = oracle_mod.selective_upsample(lat, g, g, np.zeros((B, g * g), np.uint8))
    o2, p2, s2, _, _ = oracle_mod.selective_upsample(o1, 2 * g, 2 * g, np.zeros((B, g * g), np.uint8),
                                                     pos_in=p1, span_in=s1)
    assert np.all(s2 == 4)
    full, _ = oracle_mod.merge_final(o2, p2, s2, 4 * g, 4 * g, mode="bilinear")
    img = tokens_to_image(lat, g, g)
    np.testing.assert_allclose(tokens_to_image(full, 4 * g, 4 * g), _bil2x(_bil2x(img)), rtol=0,
                               atol=3e-6)


def test_multilevel_bilinear_constant_and_copies(oracle_mod):
    """Random selections at both transitions (spans 1, 2 and 4 mixed): a
    constant latent stays exactly constant through both upsamples and the
    merge (the weights sum to one and 1.5 * 0.25 etc. are exact), and the
    merge copies every span-1 token verbatim."""
    from paper_2608_17995_gb300.workloads import random_scores
    B, g, C = 2, 8, 2
    lat = np.full((B, g * g, 4 * C), 1.5, np.float32)
    _, m1, _ = oracle_mod.topk(random_scores(3, B, g * g)[0], 20)
    o1, p1, s1, _, _ = oracle_mod.selective_upsample(lat, g, g, m1, mode="bilinear")
    _, m2, _ = oracle_mod.topk(random_scores(4, B, o1.shape[1])[0], 40)
    o2, p2, s2, _, _ = oracle_mod.selective_upsample(o1, 2 * g, 2 * g, m2, mode="bilinear",
                                                     pos_in=p1, span_in=s1)
    assert set(np.unique(s2)) == {1, 2, 4}
    assert np.all(o2 == np.float32(1.5))
    full, _ = oracle_mod.merge_final(o2, p2, s2, 4 * g, 4 * g, mode="bilinear")
    assert np.all(full == np.float32(1.5))
    lat = _dense_case(23, B, g, g, C)
    o1, p1, s1, _, _ = oracle_mod.selective_upsample(lat, g, g, m1, mode="bilinear")
    o2, p2, s2, _, _ = oracle_mod.selective_upsample(o1, 2 * g, 2 * g, m2, mode="bilinear",
                                                     pos_in=p1, span_in=s1)
    full, _ = oracle_mod.merge_final(o2, p2, s2, 4 * g, 4 * g, mode="bilinear")
    fw = 4 * g
    for b in range(B):
        for t in np.nonzero(s2[b] == 1)[0]:
            y, x = p2[b, t]
            assert np.array_equal(full[b, y * fw + x], o2[b, t])


def test_multilevel_bilinear_rejects_unaligned_or_odd_frames(oracle_mod):
    """A mixed bilinear input must tile an even frame with aligned power-of-two
    spans: an odd frame and a span-3 token are refused, and so is a merge
    with a token moved off its alignment."""
    lat = _dense_case(24, 1, 2, 2, 1)
    out, pos, span, _, _ = oracle_mod.selective_upsample(lat, 2, 2, np.zeros((1, 4), np.uint8))
    with pytest.raises(ValueError):
        oracle_mod.selective_upsample(out, 3, 4, np.ones((1, 4), np.uint8), mode="bilinear",
                                      pos_in=pos, span_in=span)
    bad = span.copy()
    bad[0, 0] = 3
    with pytest.raises(ValueError):
        oracle_mod.selective_upsample(out, 4, 4, np.ones((1, 4), np.uint8), mode="bilinear",
                                      pos_in=pos, span_in=bad)
    shifted = pos.copy()
    shifted[0, 3] = (1, 3)   # a span-2 token off its alignment (and the tiling)
    with pytest.raises(ValueError):
        oracle_mod.merge_final(out, shifted, span, 4, 4, mode="bilinear")
