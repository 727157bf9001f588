"""Host-side checks of the C ABI (no GPU needed): the library builds for
sm_103a, exports every symbol include/avits.h declares, and rejects bad
arguments on the host without launching anything."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    import paper_2608_17995_gb300 as av
    av.build()
    return av.lib()


def declared_functions():
    text = open(os.path.join(ROOT, "include", "avits.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(avits_[a-z0-9_]+)\s*\(", text)))


def test_exports_every_declared_symbol(lib):
    names = declared_functions()
    assert len(names) >= 12
    for n in names:
        assert hasattr(lib, n), n


def test_static_strings(lib):
    assert lib.avits_version().decode().count(".") == 2
    assert lib.avits_status_string(0) == b"ok"
    assert b"timed out" in lib.avits_status_string(4)


def test_host_validation_rejects_without_launch(lib):
    P = ctypes.c_void_p(16)          # a non-null, 16-byte aligned dummy pointer
    INVALID, UNSUPPORTED = 1, 2
    # k > M
    assert lib.avits_fuse_select(P, P, 1, 10, 0.5, 1e-6, 11, None, P, None, P, None) == INVALID
    # alpha outside [0,1]
    assert lib.avits_fuse_select(P, P, 1, 10, 1.5, 1e-6, 3, None, P, None, P, None) == INVALID
    # M above the single-CTA selection limit
    assert lib.avits_fuse_select(P, P, 1, 40000, 0.5, 1e-6, 3, None, P, None, P, None) == INVALID
    # L > Nk, non-positive scale, row stride shorter than d
    args = [P, P, 1, 1, 2, 64, 96, 97, 64, 0, 0, 64, 0, 0, 64, 0.125, 1.0, 0, P, None, None, 0, None]
    assert lib.avits_score_spatial(*args) == INVALID
    args[7] = 32
    args[15] = 0.0
    assert lib.avits_score_spatial(*args) == INVALID
    args[15] = 0.125
    args[11] = 32
    assert lib.avits_score_spatial(*args) == INVALID
    # temporal: empty token range, too many snapshots
    assert lib.avits_score_temporal(P, P, 1, 1, 0, 64, 1e-6, P, None) == INVALID
    snaps = (ctypes.c_void_p * 17)(*([16] * 17))
    assert lib.avits_score_temporal_var(snaps, 17, 1, 1, 4, 8, P, None) == INVALID
    # upsample: patch size other than 2, grid that does not match M; a mixed
    # input in bilinear mode needs the cell-map workspace and an even frame
    up = [P, 1, 1, 16, 4, 4, 16, 2, None, None, P, P, 4, 0, P, P, P, P, P, None, 0, None]
    up[7] = 3
    assert lib.avits_selective_upsample(*up) == UNSUPPORTED
    up[7] = 2
    up[4] = 5
    assert lib.avits_selective_upsample(*up) == INVALID
    up[4] = 4
    up[8], up[9], up[13] = P, P, 1
    assert lib.avits_selective_upsample(*up) == INVALID          # no workspace
    wsb = lib.avits_selective_upsample_workspace(1, 1, 4, 4)
    assert wsb == 16 + 4 * 16
    assert lib.avits_selective_upsample_workspace(0, 1, 4, 4) == 0
    up[19], up[20] = P, wsb - 4
    assert lib.avits_selective_upsample(*up) == INVALID          # too small
    up[20] = wsb
    up[4], up[5] = 3, 5                                           # odd frame
    assert lib.avits_selective_upsample(*up) == INVALID
    # merge: both modes need a workspace (16-byte aligned, large enough);
    # bilinear an even frame; misaligned output
    mg = [P, 1, 1, 28, P, P, 8, 8, 1, 2, 1, P, None, 0, None]
    assert lib.avits_merge_final(*mg) == INVALID
    mg[10] = 0
    assert lib.avits_merge_final(*mg) == INVALID          # nearest without workspace
    mg[12], mg[13] = P, 100
    assert lib.avits_merge_final(*mg) == INVALID          # too small
    mg[12], mg[13] = ctypes.c_void_p(P.value + 8), 1 << 20
    assert lib.avits_merge_final(*mg) == INVALID          # misaligned workspace
    mg[10] = 1
    mg[12], mg[13] = P, 1 << 20
    mg[6] = 7
    assert lib.avits_merge_final(*mg) == INVALID
    mg[6] = 8
    mg[11] = ctypes.c_void_p(24)
    assert lib.avits_merge_final(*mg) == INVALID


def test_workspace_queries(lib):
    # a 16-byte header and one 32-bit word per output cell, in both modes
    assert lib.avits_merge_final_workspace(0, 1, 64, 64) == 16 + 64 * 64 * 4
    assert lib.avits_merge_final_workspace(1, 2, 64, 64) == 16 + 2 * 64 * 64 * 4
    assert lib.avits_merge_final_workspace(2, 1, 64, 64) == 0
    assert lib.avits_score_spatial_workspace(0, 1, 2, 256, 288, 64) == 0   # fp32: no workspace
    assert lib.avits_score_spatial_workspace(1, 1, 24, 1024, 1536, 128) > 0


def test_product_path_does_not_touch_the_oracle():
    """The package never imports the oracle (only tests, smoke and the bench
    baseline may)."""
    pkg = os.path.join(ROOT, "paper_2608_17995_gb300")
    for dp, _, files in os.walk(pkg):
        for f in files:
            if f.endswith((".py", ".cu", ".cuh", ".h")):
                text = open(os.path.join(dp, f)).read()
                assert "import oracle" not in text and "avits_oracle" not in text, f


def test_host_validation_of_the_extended_entry_points(lib):
    """The perturbed selection, the key-mask spatial score and the fused
    selection + upsample reject bad arguments on the host."""
    P = ctypes.c_void_p(16)
    INVALID, UNSUPPORTED = 1, 2
    # perturbed selection: k > M, alpha outside [0,1] (the perturbation may be NULL)
    assert lib.avits_fuse_select_perturbed(P, P, None, 1, 10, 0.5, 1e-6, 11, None, P, None, P,
                                           None) == INVALID
    assert lib.avits_fuse_select_perturbed(P, P, P, 1, 10, -0.1, 1e-6, 3, None, P, None, P,
                                           None) == INVALID
    # key mask: a NULL mask, Nk < M, non-positive scale
    km = [P, P, 1, 1, 2, 64, 96, 64, 0, 0, 64, 0, 0, 64, None, 0.125, 1.0, 0, P, None, None, 0,
          None]
    assert lib.avits_score_spatial_keymask(*km) == INVALID
    km[14] = P
    km[6] = 32
    assert lib.avits_score_spatial_keymask(*km) == INVALID
    km[6] = 96
    km[15] = 0.0
    assert lib.avits_score_spatial_keymask(*km) == INVALID
    # fused selection + upsample: the mask is required, k > M, patch size
    # other than 2, bilinear on mixed-level input without its workspace
    su = [P, P, None, 1, 16, 0.5, 1e-6, 4, None, P, None, P, P, 1, 4, 4, 16, 2, None, None, 0,
          P, P, P, P, P, None, 0, None]
    assert lib.avits_select_upsample(*su) == INVALID
    su[10] = P
    su[7] = 17
    assert lib.avits_select_upsample(*su) == INVALID
    su[7] = 4
    su[17] = 3
    assert lib.avits_select_upsample(*su) == UNSUPPORTED
    su[17] = 2
    su[18], su[19], su[20] = P, P, 1
    assert lib.avits_select_upsample(*su) == INVALID


def test_host_validation_of_the_wait_selftest(lib):
    """The failure-detection test hook rejects a missing result buffer and
    limits outside 1 us .. 100 ms before launching anything."""
    P = ctypes.c_void_p(16)
    f = lib.avits_selftest_bounded_wait
    assert f(ctypes.c_ulonglong(1000000), None, None) == 1
    assert f(ctypes.c_ulonglong(0), P, None) == 1
    assert f(ctypes.c_ulonglong(999), P, None) == 1
    assert f(ctypes.c_ulonglong(100000001), P, None) == 1


def test_host_validation_of_the_lse_entry(lib):
    """avits_score_spatial_lse: missing lse_all, L = 0 and a bad scale are
    rejected, fp32 has no tensor-core path; nothing is launched."""
    P = ctypes.c_void_p(16)
    f = lib.avits_score_spatial_lse
    args = lambda lse, dt, L, scale: (P, P, dt, 1, 2, 256, L, 64, 2 * 256 * 64, 256 * 64, 64,
                                      2 * 32 * 64, 32 * 64, 64, lse, ctypes.c_float(scale),
                                      ctypes.c_float(1.0), 0, P, None, P, ctypes.c_size_t(1 << 20),
                                      None)
    assert f(*args(None, 1, 32, 0.125)) == 1
    assert f(*args(P, 1, 0, 0.125)) == 1
    assert f(*args(P, 1, 32, 0.0)) == 1
    assert f(*args(P, 0, 32, 0.125)) == 2


def test_host_validation_of_the_attention_forward(lib):
    """avits_attention_forward rejects bad arguments on the host: sizes, L,
    the scale, short row strides and a missing or short workspace when A is
    wanted (INVALID_ARG); fp32 inputs and H > 255 with A (UNSUPPORTED)."""
    P = ctypes.c_void_p(256)
    INVALID, UNSUPPORTED = 1, 2
    f = lib.avits_attention_forward
    ws = lib.avits_attention_forward_workspace(1, 2, 300)
    assert ws == 8 * 512
    assert lib.avits_attention_forward_workspace(0, 2, 300) == 0

    def call(**kw):
        a = dict(q=P, k=P, v=P, dt=1, B=1, H=2, Mq=300, Nk=333, L=77, d=128, qs=None, ks=None,
                 vs=None, os=None, scale=0.088, o=P, lse=None, w=1.0, acc=0, A=P, ws=P, wsb=ws)
        a.update(kw)
        return f(a["q"], a["k"], a["v"], a["dt"], a["B"], a["H"], a["Mq"], a["Nk"], a["L"],
                 a["d"], a["qs"], a["ks"], a["vs"], a["os"], a["scale"], a["o"], a["lse"], a["w"],
                 a["acc"], a["A"], a["ws"], a["wsb"], None)

    assert call(o=None) == INVALID
    assert call(Mq=0) == INVALID
    assert call(L=334) == INVALID
    assert call(L=-1) == INVALID
    assert call(scale=0.0) == INVALID
    assert call(scale=float("nan")) == INVALID
    short = (ctypes.c_int64 * 3)(0, 0, 64)      # row stride < d
    assert call(qs=short) == INVALID
    assert call(ws=None) == INVALID
    assert call(wsb=ws - 8) == INVALID
    assert call(ws=ctypes.c_void_p(260)) == INVALID      # not 8-byte aligned
    assert call(dt=0) == UNSUPPORTED
    assert call(H=256, wsb=1 << 20) == UNSUPPORTED


def test_nvtx_ranges_compile(tmp_path):
    """With AVITS_NVTX the entry points open NVTX ranges (header-only NVTX v3,
    so nothing to link): the entry-point sources compile with it."""
    import subprocess
    from paper_2608_17995_gb300 import _build
    for src in ("api.cu", "no_alloc.cu"):
        out = tmp_path / (src + ".o")
        cmd = [_build.nvcc(), *_build.ARCH, *_build.FLAGS, "-DAVITS_NVTX", "-c",
               os.path.join(_build.CSRC, src), "-o", str(out)]
        r = subprocess.run(cmd, stdout=subprocess.PIPE, stderr=subprocess.STDOUT, text=True)
        assert r.returncode == 0, r.stdout
        nm = subprocess.run(["nm", str(out)], stdout=subprocess.PIPE, text=True).stdout
        assert "nvtx" in nm.lower()
