"""The allocation-free spatial entry point (avits_score_spatial_noalloc).

Callers such as an inference engine's plugin enqueue hook only hold their
input/output pointers and a stream and may not allocate there; this entry
point keeps its scratch in a fixed device array of the library.  These tests
call it through the C ABI and compare it with avits_score_spatial (which
takes a caller workspace) on two calls in a row.  The file is named so that
pytest collects it last: a run that stops at its first failure has then run
every other test already.  The tests do not depend on that order (every call
clears the part of the array it uses), and pass alone in a fresh process.
"""
import ctypes
import math

import numpy as np
import pytest

pytestmark = pytest.mark.gpu

RTOL = 2e-3   # the bf16-input score tolerance used by the other GPU tests


@pytest.fixture(scope="module")
def av():
    import torch
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    import paper_2608_17995_gb300 as av
    av.build()
    av.lib()
    return av


def _inputs(name, **kw):
    from paper_2608_17995_gb300.pipeline import to_device
    from paper_2608_17995_gb300.workloads import make_transition
    tr = make_transition(name, **kw)
    return tr, to_device(tr.q_img, "bf16"), to_device(tr.k_all, "bf16")


@pytest.mark.parametrize("name,kw", [("flux1024", {}), ("batched", {}),
                                     ("flux1024", dict(G=13, L=77, H=3, k=40))])
def test_noalloc_matches_workspace_entry_twice(av, name, kw):
    import torch
    tr, q, k = _inputs(name, **kw)
    ref = torch.full((tr.B, tr.M), float("nan"), device="cuda")
    lse_ref = torch.zeros(tr.B, tr.H, tr.M, 2, device="cuda")
    av.avits_score_spatial(q, k, tr.L, tr.softmax_scale, ref, lse=lse_ref)
    for _ in range(2):   # the shared array keeps the previous call's contents
        out = torch.full((tr.B, tr.M), float("nan"), device="cuda")
        lse = torch.zeros(tr.B, tr.H, tr.M, 2, device="cuda")
        av.avits_score_spatial_noalloc(q, k, tr.L, tr.softmax_scale, out, lse=lse)
        assert av.avits_device_status() == 0
        assert not torch.isnan(out).any()
        np.testing.assert_allclose(out.cpu().numpy(), ref.cpu().numpy(), rtol=RTOL, atol=1e-6)
        np.testing.assert_allclose(lse.cpu().numpy(), lse_ref.cpu().numpy(), rtol=RTOL, atol=1e-5)


def test_noalloc_accumulates_like_workspace_entry(av):
    import torch
    tr, q, k = _inputs("flux1024", G=16, H=4, L=64, k=64)
    base = torch.rand(tr.B, tr.M, device="cuda")
    ref, out = base.clone(), base.clone()
    av.avits_score_spatial(q, k, tr.L, tr.softmax_scale, ref, weight=0.5, accumulate=True)
    av.avits_score_spatial_noalloc(q, k, tr.L, tr.softmax_scale, out, weight=0.5, accumulate=True)
    torch.cuda.synchronize()
    np.testing.assert_allclose(out.cpu().numpy(), ref.cpu().numpy(), rtol=RTOL, atol=1e-6)


def test_noalloc_rejects_shapes_beyond_the_array(av):
    """A shape whose scratch exceeds the fixed array is refused on the host,
    nothing launched, with the sizes in the error text."""
    import torch
    lib = av.lib()
    lib.avits_score_spatial_noalloc_limit.restype = ctypes.c_size_t
    limit = lib.avits_score_spatial_noalloc_limit()
    B, H, M, d, L = 16, 32, 4096, 128, 512
    Nk = L + M
    need = av.avits_score_spatial_workspace(av.BF16, B, H, M, Nk, d)
    assert need > limit
    # tiny real buffers: the call must fail before touching them as [B,H,M,d]
    q = torch.zeros(8, dtype=torch.bfloat16, device="cuda")
    A = torch.zeros(8, device="cuda")
    fn = lib.avits_score_spatial_noalloc
    vp, i32, i64, f32 = ctypes.c_void_p, ctypes.c_int, ctypes.c_int64, ctypes.c_float
    fn.argtypes = [vp, vp, i32, i32, i32, i32, i32, i32, i32, i64, i64, i64, i64, i64, i64,
                   f32, f32, i32, vp, vp, vp]
    fn.restype = ctypes.c_int
    rc = fn(q.data_ptr(), q.data_ptr(), 1, B, H, M, Nk, L, d, H * M * d, M * d, d,
            H * Nk * d, Nk * d, d, 1.0 / math.sqrt(d), 1.0, 0, A.data_ptr(), None, None)
    assert rc == 1
    lib.avits_score_spatial_noalloc_error.restype = ctypes.c_char_p
    assert b"scratch needed" in lib.avits_score_spatial_noalloc_error()
    assert av.avits_device_status() == 0


def test_noalloc_back_to_back_shapes_on_one_stream(av):
    """Calls with different shapes back to back on one stream (large then
    small, small then large) each match avits_score_spatial: what the
    previous call left in the shared array never leaks into the next one."""
    import torch
    shapes = [("batched", {}), ("flux1024", dict(G=13, L=77, H=3, k=40)), ("flux1024", {}),
              ("batched", {})]
    ins = [_inputs(n, **kw) for n, kw in shapes]
    refs = []
    for tr, q, k in ins:
        ref = torch.full((tr.B, tr.M), float("nan"), device="cuda")
        av.avits_score_spatial(q, k, tr.L, tr.softmax_scale, ref)
        refs.append(ref)
    outs = []
    st = torch.cuda.Stream()
    with torch.cuda.stream(st):
        for tr, q, k in ins:
            out = torch.full((tr.B, tr.M), float("nan"), device="cuda")
            av.avits_score_spatial_noalloc(q, k, tr.L, tr.softmax_scale, out, stream=st)
            outs.append(out)
    st.synchronize()
    assert av.avits_device_status() == 0
    for out, ref in zip(outs, refs):
        assert not torch.isnan(out).any()
        np.testing.assert_allclose(out.cpu().numpy(), ref.cpu().numpy(), rtol=RTOL, atol=1e-6)


def test_noalloc_limit_covers_the_configurations(av):
    """On this device (its SM count sets the per-SM scratch) every
    configuration of the transition fits the fixed array."""
    from paper_2608_17995_gb300.workloads import make_transition
    limit = av.avits_score_spatial_noalloc_limit()
    for name in ("flux1024", "flux2048", "edit", "batched"):
        tr = make_transition(name)
        need = av.avits_score_spatial_workspace(av.BF16, tr.B, tr.H, tr.M, tr.Nk, tr.d)
        assert 0 < need <= limit, (name, need, limit)
    B, H, M, d, L = 8, 24, 640, 128, 512   # the batched second transition
    need = av.avits_score_spatial_workspace(av.BF16, B, H, M, L + M, d)
    assert 0 < need <= limit
