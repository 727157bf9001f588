"""One resolution transition on the device: buffers plus the calls in order.

Plumbing only: it owns the output tensors and the workspaces and issues
avits_score_spatiotemporal (or avits_score_spatial + avits_score_temporal) ->
avits_select_upsample (or avits_fuse_select + avits_selective_upsample) ->
avits_merge_final on one stream.
"""
from __future__ import annotations

import numpy as np

from . import (BILINEAR, NEAREST, SpatialWorkspace, avits_fuse_select, avits_merge_final,
               avits_merge_final_workspace, avits_score_spatial, avits_score_spatiotemporal,
               avits_score_temporal, avits_select_upsample, avits_selective_upsample,
               avits_selective_upsample_workspace)


def to_device(arr: np.ndarray, dtype: str, device="cuda"):
    """numpy (float32, or bf16 bit patterns in uint16) -> torch device tensor."""
    import torch
    if dtype == "bf16":
        t = torch.from_numpy(np.ascontiguousarray(arr).view(np.int16)).view(torch.bfloat16)
    elif arr.dtype in (np.int32, np.uint8, np.int8):
        t = torch.from_numpy(np.ascontiguousarray(arr))
    else:
        t = torch.from_numpy(np.ascontiguousarray(arr, dtype=np.float32))
    return t.to(device)


def to_numpy(t, dtype: str = None) -> np.ndarray:
    import torch
    t = t.detach().cpu()
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).numpy().view(np.uint16)
    return t.numpy()


class TransitionBuffers:
    """Inputs (device), outputs and workspaces of one transition of fixed shape."""

    def __init__(self, tr, device="cuda", mode=None, inputs=True):
        import torch
        self.tr = tr
        self.mode = BILINEAR if (mode or tr.mode) == "bilinear" else NEAREST
        dt = torch.bfloat16 if tr.dtype == "bf16" else torch.float32
        B, M, k = tr.B, tr.M, tr.k
        NO = M + 3 * k
        self.full_h, self.full_w = 2 * tr.frame_h, 2 * tr.frame_w
        if inputs:
            self.q = to_device(tr.q_img, tr.dtype, device)
            self.k = to_device(tr.k_all, tr.dtype, device)
            self.h_t = to_device(tr.h_t, tr.dtype, device)
            self.h_prev = to_device(tr.h_prev, tr.dtype, device)
            self.latent = to_device(tr.latent, tr.dtype, device)
            self.pos_in = None if tr.pos_in is None else to_device(tr.pos_in, "i32", device)
            self.span_in = None if tr.span_in is None else to_device(tr.span_in, "i32", device)
        z = dict(device=device)
        self.A = torch.empty(B, M, dtype=torch.float32, **z)
        self.V = torch.empty(B, M, dtype=torch.float32, **z)
        self.S = torch.empty(B, M, dtype=torch.float32, **z)
        self.sel_idx = torch.empty(B, max(k, 1), dtype=torch.int32, **z)
        self.sel_mask = torch.empty(B, M, dtype=torch.uint8, **z)
        self.tok_offset = torch.empty(B, M, dtype=torch.int32, **z)
        self.mixed = torch.empty(B, NO, tr.C * 4, dtype=dt, **z)
        self.pos = torch.empty(B, NO, 2, dtype=torch.int32, **z)
        self.span = torch.empty(B, NO, dtype=torch.int32, **z)
        self.src_tok = torch.empty(B, NO, dtype=torch.int32, **z)
        self.src_sub = torch.empty(B, NO, dtype=torch.int8, **z)
        self.full = torch.empty(B, self.full_h * self.full_w, tr.C * 4, dtype=dt, **z)
        self.ws = SpatialWorkspace(device)
        mb = avits_merge_final_workspace(self.mode, B, self.full_h, self.full_w)
        # zero-filled before first use (the nearest merge's claim map and counter)
        self.merge_ws = torch.zeros(max(mb, 16), dtype=torch.uint8, **z) if mb else None
        # a mixed input in bilinear mode: the input frame's cell map
        ub = avits_selective_upsample_workspace(self.mode, B, tr.frame_h, tr.frame_w)
        self.up_ws = torch.empty(ub, dtype=torch.uint8, **z) if ub else None

    def set_inputs(self, q, k, h_t, h_prev, latent, pos_in=None, span_in=None):
        self.q, self.k, self.h_t, self.h_prev, self.latent = q, k, h_t, h_prev, latent
        self.pos_in, self.span_in = pos_in, span_in

    # the five steps, each one launch (the bilinear merge adds a memset + map)
    def spatial(self, stream=None):
        avits_score_spatial(self.q, self.k, self.tr.L, self.tr.softmax_scale, self.A,
                            workspace=self.ws, stream=stream)

    def scores(self, stream=None):
        """Both scores in one call (temporal overlapped with spatial)."""
        avits_score_spatiotemporal(self.q, self.k, self.tr.L, self.tr.softmax_scale, self.A,
                                   self.h_t, self.h_prev, self.V, workspace=self.ws,
                                   stream=stream)

    def temporal(self, stream=None):
        avits_score_temporal(self.h_t, self.h_prev, self.V, stream=stream)

    def select(self, stream=None):
        avits_fuse_select(self.A, self.V, self.tr.alpha, self.tr.k, self.sel_idx, self.tok_offset,
                          S=self.S, sel_mask=self.sel_mask, stream=stream)

    def upsample(self, stream=None):
        avits_selective_upsample(self.latent, self.tr.frame_h, self.tr.frame_w, self.sel_mask,
                                 self.tok_offset, self.tr.k, self.mixed, self.pos, self.span,
                                 self.src_tok, self.src_sub, mode=self.mode, pos_in=self.pos_in,
                                 span_in=self.span_in, workspace=self.up_ws, stream=stream)

    def select_upsample(self, stream=None):
        """Selection and selective upsampling in one launch."""
        avits_select_upsample(self.A, self.V, self.tr.alpha, self.tr.k, self.sel_idx,
                              self.tok_offset, self.sel_mask, self.latent, self.tr.frame_h,
                              self.tr.frame_w, self.mixed, self.pos, self.span, self.src_tok,
                              self.src_sub, S=self.S, mode=self.mode, pos_in=self.pos_in,
                              span_in=self.span_in, workspace=self.up_ws, stream=stream)

    def merge(self, stream=None):
        avits_merge_final(self.mixed, self.pos, self.span, self.full_h, self.full_w, self.full,
                          mode=self.mode, workspace=self.merge_ws, stream=stream)

    def run(self, stream=None, merge=True, fused_scores=True, fused_tail=True):
        """The transition on one stream: both scores (one call, the temporal
        kernel overlapping the spatial one, unless fused_scores=False), then
        selection and selective upsampling (one launch unless
        fused_tail=False) and the final merge."""
        import torch
        main = stream if stream is not None else torch.cuda.current_stream()
        if fused_scores:
            self.scores(main)
        else:
            self.spatial(main)
            self.temporal(main)
        if fused_tail:
            self.select_upsample(main)
        else:
            self.select(main)
            self.upsample(main)
        if merge:
            self.merge(main)
