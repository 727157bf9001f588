"""GPU parity of the joint-attention forward (Eq. 4-5 with Eq. 3's score read
off the same softmax) against the oracle, through the C ABI.

Tolerances, from the arithmetic of the kernel:
  O    The softmax numerators p_j enter the P V product rounded to bf16
       (8 significant bits: relative error <= 2^-8 each); the row sum, the
       exponentials (ex2, relative error ~2^-22) and the accumulation are
       fp32; O is rounded to bf16 once (2^-8 |O|).  So
       |O - O_ref| <= 2^-8 (sum_j w_j |v_j| + |O_ref|) plus fp32 terms, with
       w the exact softmax weights; sum_j w_j |v_j| is the oracle's attention
       with |v| for v (O_abs).  The test allows 1.01 times that plus 1e-5.
  lse  fp32 sums of up to Nk exponentials: 2e-4 + 2e-5 |lse|.
  A    the same fp32 ratio as the spatial kernel: rel 2e-3, abs 1e-6.
"""
import math

import numpy as np
import pytest

pytestmark = pytest.mark.gpu

A_RTOL = 2e-3


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


def _dev(arr):
    from paper_2608_17995_gb300.pipeline import to_device
    return to_device(arr, "bf16")


def _np(t):
    from paper_2608_17995_gb300.pipeline import to_numpy
    return to_numpy(t)


def _bf16(x):
    from paper_2608_17995_gb300.workloads import to_bf16_bits
    return to_bf16_bits(np.asarray(x, np.float32))


def _rand_qkv(seed, B, H, Mq, Nk, d, logit_std=3.0):
    # q, k ~ N(0, s): q.k / sqrt(d) has standard deviation s = logit_std
    rng = np.random.default_rng(seed)
    c = math.sqrt(logit_std)
    q = rng.standard_normal((B, H, Mq, d)) * c
    k = rng.standard_normal((B, H, Nk, d)) * c
    v = rng.standard_normal((B, H, Nk, d))
    return _bf16(q), _bf16(k), _bf16(v)


def _run(av, q, k, v, L, scale, with_score=True, A_in=None, weight=1.0, qd=None, kd=None,
         vd=None, o=None):
    import torch
    B, H, Mq, d = q.shape
    qd = _dev(q) if qd is None else qd
    kd = _dev(k) if kd is None else kd
    vd = _dev(v) if vd is None else vd
    o = torch.zeros(B, H, Mq, d, dtype=torch.bfloat16, device="cuda") if o is None else o
    lse = torch.zeros(B, H, Mq, 2, dtype=torch.float32, device="cuda") if with_score else None
    A = None
    if with_score:
        A = torch.zeros(B, Mq, dtype=torch.float32, device="cuda") if A_in is None else \
            torch.from_numpy(np.ascontiguousarray(A_in)).cuda()
    av.avits_attention_forward(qd, kd, vd, L, scale, o, lse=lse, A=A, weight=weight,
                               accumulate=A_in is not None)
    assert av.avits_device_status() == 0
    return o, lse, A


def _compare(orc, q, k, v, L, scale, o, lse, A, rows=None, A_in=None, weight=1.0):
    B, H, Mq, d = q.shape
    O_r, lse_r, _, A_r = orc.attention(q, k, v, L, scale, rows=rows, A_in=A_in, weight=weight)
    v_abs = _bf16(np.abs(_f32(v)))
    O_abs, _, _, _ = orc.attention(q, k, v_abs, L, scale, rows=rows)
    idx = np.arange(B * Mq) if rows is None else np.asarray(rows)
    bi, ii = idx // Mq, idx % Mq
    og = _f32(_np(o))[bi, :, ii]
    err = np.abs(og - O_r[bi, :, ii])
    tol = 1.01 * 2.0 ** -8 * (O_abs[bi, :, ii] + np.abs(O_r[bi, :, ii])) + 1e-5
    assert np.all(err <= tol), "O: max excess %g, max err/tol %g" % ((err - tol).max(),
                                                                     (err / tol).max())
    if lse is not None:
        lg = _np(lse)[bi, :, ii]
        lr = lse_r[bi, :, ii]
        np.testing.assert_allclose(lg[..., 0], lr[..., 0], rtol=2e-5, atol=2e-4)
        fin = np.isfinite(lr[..., 1])
        assert np.array_equal(np.isfinite(lg[..., 1]), fin)
        np.testing.assert_allclose(lg[..., 1][fin], lr[..., 1][fin], rtol=2e-5, atol=2e-4)
    if A is not None:
        np.testing.assert_allclose(_np(A).ravel()[idx], A_r.ravel()[idx], rtol=A_RTOL, atol=1e-6)
    return float(err.max())


def _f32(a):
    from helpers import as_f32
    return as_f32(np.asarray(a))


@pytest.mark.parametrize("B,H,Mq,Nk,L,d", [
    (1, 2, 300, 333, 77, 128),     # ragged query and key tiles, text boundary inside a chunk
    (2, 3, 256, 200, 64, 64),      # d = 64, one key tile and a ragged one
    (1, 1, 1, 1, 1, 128),          # one query, one (text) key
    (1, 2, 130, 129, 0, 128),      # no text key: lse_txt = -inf, A = 0
    (1, 2, 64, 256, 256, 128),     # every key a text key: A = 1
    (3, 4, 513, 700, 128, 64),
])
def test_attention_vs_oracle(av, orc, B, H, Mq, Nk, L, d):
    q, k, v = _rand_qkv(B * 1000 + Nk, B, H, Mq, Nk, d)
    scale = 1.0 / math.sqrt(d)
    o, lse, A = _run(av, q, k, v, L, scale)
    _compare(orc, q, k, v, L, scale, o, lse, A)
    if L == 0:
        assert np.all(_np(A) == 0)
    if L == Nk:
        np.testing.assert_allclose(_np(A), 1.0, rtol=0, atol=1e-6)


def test_attention_rescale_when_a_later_key_tile_dominates(av, orc):
    """Key tiles 2 and 4 have logits ~6x larger than the rest: the running
    maximum moves twice by more than 2^8, so O and the sums are rescaled in
    tensor memory mid-row; a first tile that dominates never rescales."""
    B, H, Mq, Nk, L, d = 1, 2, 256, 640, 200, 128
    q, k, v = _rand_qkv(7, B, H, Mq, Nk, d)
    kf = _f32(k)
    kf[:, :, 256:384] *= 4.0
    kf[:, :, 512:640] *= 6.0
    k = _bf16(kf)
    scale = 1.0 / math.sqrt(d)
    o, lse, A = _run(av, q, k, v, L, scale)
    _compare(orc, q, k, v, L, scale, o, lse, A)
    kf = _f32(k)
    kf[:, :, 256:] = _f32(_rand_qkv(8, B, H, Mq, Nk, d)[1])[:, :, 256:]
    kf[:, :, :128] *= 6.0
    k = _bf16(kf)
    o, lse, A = _run(av, q, k, v, L, scale)
    _compare(orc, q, k, v, L, scale, o, lse, A)


def test_attention_flux1024_joint_sampled_rows(av, orc):
    """The FLUX-1024 joint attention (24 heads, 512 text + 1024 image tokens,
    d = 128) in the launch the benchmark times: sampled rows against the
    oracle; every row: A in [0,1], lse_txt <= lse_all, O finite; the image
    rows' A equals the spatial-score kernel's A on the same Q_img, K."""
    import torch
    from paper_2608_17995_gb300.workloads import make_transition, make_joint_attention
    tr = make_transition("flux1024")
    q, v = make_joint_attention(tr)
    k = tr.k_all
    o, lse, A = _run(av, q, k, v, tr.L, tr.softmax_scale)
    Mq = q.shape[2]
    rng = np.random.default_rng(3)
    rows = sorted(set(rng.choice(Mq, 48, replace=False).tolist()) | {0, tr.L - 1, tr.L, Mq - 1})
    _compare(orc, q, k, v, tr.L, tr.softmax_scale, o, lse, A, rows=rows)
    Ag, lg = _np(A), _np(lse)
    assert np.all((Ag >= 0) & (Ag <= 1))
    assert np.all(lg[..., 1] <= lg[..., 0] + 1e-6)
    assert torch.isfinite(o.float()).all()
    A_sp = torch.zeros(1, tr.M, dtype=torch.float32, device="cuda")
    av.avits_score_spatial(_dev(tr.q_img), _dev(k), tr.L, tr.softmax_scale, A_sp)
    np.testing.assert_allclose(Ag[:, tr.L:tr.L + tr.M], _np(A_sp), rtol=A_RTOL, atol=1e-6)


def test_attention_many_units_per_cta(av, orc):
    """More units than SMs (B = 2, H = 24, 2048 rows: 384 units), so CTAs
    reload Q, reuse the O staging and wait for the previous unit's epilogue;
    sampled rows of every unit position."""
    B, H, Mq, Nk, L, d = 2, 24, 2048, 2048, 512, 128
    q, k, v = _rand_qkv(11, B, H, Mq, Nk, d)
    scale = 1.0 / math.sqrt(d)
    o, lse, A = _run(av, q, k, v, L, scale)
    rng = np.random.default_rng(5)
    rows = sorted(set(rng.choice(B * Mq, 40, replace=False).tolist()) | {0, Mq - 1, Mq, 2 * Mq - 1})
    _compare(orc, q, k, v, L, scale, o, lse, A, rows=rows)


def test_attention_strided_views_accumulate_and_no_score(av, orc):
    """[B,N,H,d] views (the layout of a model's projections) for q, k, v and
    o; accumulate with a weight; and without A / lse the same O bits."""
    import torch
    B, H, Mq, Nk, L, d = 2, 3, 200, 260, 40, 128
    q, k, v = _rand_qkv(21, B, H, Mq, Nk, d)

    def bnhd(a):
        t = _dev(np.ascontiguousarray(np.transpose(a, (0, 2, 1, 3))))
        return t.permute(0, 2, 1, 3)

    qd, kd, vd = bnhd(q), bnhd(k), bnhd(v)
    assert qd.stride(2) == H * d
    o = torch.zeros(B, Mq, H, d, dtype=torch.bfloat16, device="cuda").permute(0, 2, 1, 3)
    A_in = np.random.default_rng(1).random((B, Mq)).astype(np.float32)
    o, lse, A = _run(av, q, k, v, L, 0.1, qd=qd, kd=kd, vd=vd, o=o, A_in=A_in, weight=0.25)
    _compare(orc, q, k, v, L, 0.1, o.contiguous(), lse, A, A_in=A_in, weight=0.25)
    o2, _, _ = _run(av, q, k, v, L, 0.1, with_score=False)
    assert torch.equal(o2, o.contiguous())
