/*
 * avits.h — C ABI of the AViTS resolution-transition hot path on GB300 (sm_103a).
 *
 * AViTS (Adaptive Spatiotemporal Token Selection, arxiv 2608.17995) runs a
 * diffusion transformer at half resolution, scores every low-resolution image
 * token by how strongly it attends to the text (spatial importance, Sec. 3.3.1,
 * Eq. 3-5) and by how much it moves between denoising steps (temporal
 * importance, Sec. 3.3.2), fuses the two min-max normalised scores (Eq. 8),
 * keeps the top-K tokens (Eq. 9) and upsamples only those (Sec. 3.2, Stage 2).
 * After Stage 2 the remaining tokens are expanded and the sequence is put back
 * in spatial order (Sec. 3.2, Stage 3).  This library computes that transition:
 *
 *   avits_score_spatial       Eq. 3 + Eq. 5   per-token text attention mass
 *     _keymask                  interleaved text keys given by a mask
 *     _lse                      from the model attention's logsumexp
 *     _noalloc                  without a caller workspace
 *   avits_attention_forward   Eq. 4-5 + Eq. 3  the block's joint attention
 *                             O = softmax(QK^T/sqrt d) V, with its logsumexp
 *                             and the spatial score from the same softmax
 *   avits_score_temporal      Sec. 3.3.2      per-token relative step change
 *   avits_score_spatiotemporal  both scores in one call
 *   avits_score_temporal_var  Eq. 6-7         step variance over N_T snapshots
 *   avits_fuse_select         Sec. 3.3.3, Eq. 8 + Eq. 9   min-max, fuse, top-K
 *     _perturbed                with caller-supplied tie-break noise (Eq. 9)
 *   avits_selective_upsample  Sec. 3.2 Stage 2   packed mixed-resolution sequence
 *   avits_select_upsample     selection + upsample in one launch
 *   avits_merge_final         Sec. 3.2 Stage 3   dense full-resolution latent
 *   avits_selftest_bounded_wait  test hook for the device-side failure path
 *
 * Conventions shared by every call
 * --------------------------------
 *  - Every tensor pointer is DEVICE memory owned by the caller.  The library
 *    allocates no device memory at run time; the split-key partial sums of
 *    avits_score_spatial and the cell map of bilinear avits_merge_final live
 *    in a caller workspace whose size a *_workspace() query returns (the one
 *    exception: the static scratch array of avits_score_spatial_noalloc).
 *  - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *    stream).  Every call is asynchronous and stream ordered; none
 *    synchronises the host except avits_device_status().
 *  - Arguments are checked on the host before anything is launched.  A bad
 *    argument returns AVITS_ERR_INVALID_ARG (or AVITS_ERR_UNSUPPORTED for a
 *    combination the kernels do not implement) and launches nothing.
 *  - A failed launch returns AVITS_ERR_CUDA (the CUDA error is cleared and
 *    its text kept for avits_last_error_string()).
 *  - Errors found on the device (a bounded wait that ran out, a NaN score, a
 *    mixed sequence that does not tile the output frame) are OR-ed into a
 *    per-device status word, read and cleared by avits_device_status().
 *  - Dtypes: AVITS_BF16 (bfloat16 inputs, fp32 arithmetic) and AVITS_F32.
 *    Scores are always fp32.
 *  - Latent tokens hold C*p*p values ordered (channel, patch-row, patch-col),
 *    p = 2 (the 2x2 patchification of FLUX-family models).
 *  - Token grids are raster ordered: token i of a gh x gw grid sits at row
 *    i / gw, column i % gw.
 */
#ifndef AVITS_H
#define AVITS_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  AVITS_OK = 0,
  AVITS_ERR_INVALID_ARG = 1,
  AVITS_ERR_UNSUPPORTED = 2,
  AVITS_ERR_CUDA = 3,
  AVITS_ERR_TIMEOUT = 4,   /* device: a bounded wait gave up */
  AVITS_ERR_NAN = 5,       /* device: a NaN reached the fused score */
  AVITS_ERR_COVERAGE = 6   /* device: merge input does not tile the frame */
} avits_status;

typedef enum { AVITS_F32 = 0, AVITS_BF16 = 1 } avits_dtype;

typedef enum { AVITS_UP_NEAREST = 0, AVITS_UP_BILINEAR = 1 } avits_upmode;

/* ------------------------------------------------------------------------
 * Spatial importance, Sec. 3.3.1, Eq. 3 with the joint-attention extraction
 * of Eq. 4-5.  For batch b, head h and image query i:
 *
 *     l_ij  = softmax_scale * <q_bhi, k_bhj>                 j = 0 .. Nk-1
 *     mass  = sum_{j<L} exp(l_ij) / sum_{j<Nk} exp(l_ij)     (text keys first)
 *     A[b,i] = (accumulate ? A[b,i] : 0) + weight * (1/H) * sum_h mass
 *
 * i.e. the softmax over ALL keys (text, image and, for editing models, the
 * reference-image keys) restricted to the L text columns and summed, then
 * averaged over heads (Eq. 3).  The score matrix is never materialised.
 * `accumulate` + `weight` aggregate over the selected blocks and the N_T
 * collection steps (end of Sec. 3.3.1): e.g. weight = 1/(blocks*N_T).
 *
 * q_img : [B,H,M,d] image-query projections after the model's QK norm (and
 *         RoPE if the model applies it before attention).  Element strides
 *         q_sb, q_sh, q_sn; the d axis is contiguous.  May be a strided view
 *         of the joint Q of Eq. 4 (skip the L text rows).
 * k_all : [B,H,Nk,d] joint keys, the L text keys FIRST, then the image keys,
 *         then optional reference keys.  Strides k_sb, k_sh, k_sn; d contiguous.
 * dt    : AVITS_BF16 (tensor-core path, needs d in {64,128}, 16-byte aligned
 *         base and strides) or AVITS_F32 (CUDA-core path, any d <= 256).
 * softmax_scale > 0 (1/sqrt(d) in the paper).  0 <= L <= Nk.
 * A     : [B,M] fp32, written (accumulate = 0) or added to.
 * lse_opt : NULL or [B,H,M,2] fp32 receiving (log sum_j exp l_ij over all
 *         keys, the same over the text keys), natural log; -inf when a sum
 *         underflows.
 * workspace/ws_bytes : at least avits_score_spatial_workspace(...) bytes of
 *         device scratch: per-row partial statistics of the key ranges each
 *         SM handled, ready flags and one 64-bit head-sum word per row.  It
 *         must be ZERO-FILLED before its first use (e.g. cudaMemset); every
 *         call that completes leaves it zero-filled again, so it is reused as
 *         is, also by calls with other sizes.  After a call that reported
 *         AVITS_ERR_TIMEOUT (avits_device_status), zero it again.  One
 *         workspace must not be used by two calls running concurrently.  The
 *         bf16 tensor-core path is one kernel; H <= 255 on that path (more
 *         heads take the CUDA-core path).
 * ---------------------------------------------------------------------- */
avits_status avits_score_spatial(const void* q_img, const void* k_all, avits_dtype dt,
                                 int B, int H, int M, int Nk, int L, int d,
                                 int64_t q_sb, int64_t q_sh, int64_t q_sn,
                                 int64_t k_sb, int64_t k_sh, int64_t k_sn,
                                 float softmax_scale, float weight, int accumulate,
                                 float* A, float* lse_opt,
                                 void* workspace, size_t ws_bytes, void* stream);

/* Workspace bytes avits_score_spatial needs on the CURRENT device for these
 * sizes (0 if it needs none).  Returns 0 as well for invalid sizes. */
size_t avits_score_spatial_workspace(avits_dtype dt, int B, int H, int M, int Nk, int d);

/* ------------------------------------------------------------------------
 * avits_score_spatial without a workspace argument, for callers that may not
 * allocate device memory where they call this (they only hold their input
 * and output pointers and a stream, e.g. inside an inference engine's plugin
 * enqueue or a runtime's custom-op callback, where cudaMalloc would
 * synchronise the device or is not allowed).  The paper has no counterpart:
 * this is a deployment convenience of this library.
 *
 * Same arguments and results as avits_score_spatial (tensor-core path only:
 * bf16, d in {64,128}, 16-byte aligned layout; anything else returns
 * AVITS_ERR_UNSUPPORTED).  The scratch is a fixed array inside the library,
 * avits_score_spatial_noalloc_limit() bytes (8 MiB) per GPU, held by every
 * GPU that loads the library until the process exits.  A call whose shapes
 * need more returns AVITS_ERR_INVALID_ARG before launching anything, with the
 * sizes in avits_score_spatial_noalloc_error().  The call allocates nothing.
 *  - The scratch a shape needs grows with the device's SM count (per-row
 *    statistics are kept per SM and key range): on a 152-SM GB300 the
 *    FLUX-1024 shape needs 1.2 MB and the batched second transition
 *    (B = 8, H = 24, M = 640, Nk = 1152) 4.8 MB, so a shape that fits on one
 *    GPU may be refused on a part with more SMs.
 *  - The first call on each device looks up the array's device address;
 *    make that first call before any stream capture on that device (a
 *    first call during a capture is refused, the reason in
 *    avits_score_spatial_noalloc_error()).
 *  - All calls on a device share the one array: calls that may overlap on
 *    the GPU (other streams, other host threads) race and must be ordered
 *    by the caller.  Each call clears, on its stream, the part of the array
 *    it uses before its kernel runs, so nothing needs clearing by the caller.
 * ---------------------------------------------------------------------- */
avits_status avits_score_spatial_noalloc(const void* q_img, const void* k_all, avits_dtype dt,
                                         int B, int H, int M, int Nk, int L, int d,
                                         int64_t q_sb, int64_t q_sh, int64_t q_sn,
                                         int64_t k_sb, int64_t k_sh, int64_t k_sn,
                                         float softmax_scale, float weight, int accumulate,
                                         float* A, float* lse_opt, void* stream);

/* Bytes of the static scratch array of avits_score_spatial_noalloc. */
size_t avits_score_spatial_noalloc_limit(void);

/* Why the last avits_score_spatial_noalloc call on this thread was refused
 * (its size, or a first call made during a stream capture; "" otherwise). */
const char* avits_score_spatial_noalloc_error(void);

/* ------------------------------------------------------------------------
 * avits_score_spatial when the caller already has the logsumexp over ALL
 * keys, e.g. from the model's own joint-attention forward (fused attention
 * returns it; Sec. 3.3.1 recomputes the attention only because fused
 * kernels do not expose the weights).  Eq. 5's text mass is
 * exp(lse_txt - lse_all), so only the L text keys are scored here: a third
 * of the key work at FLUX-1024 (L = 512 of Nk = 1536).
 * k_txt   : [B,H,L,d] the text keys (e.g. the first L rows of k_all, with
 *           k_all's strides).  q_img, dt, strides, softmax_scale, weight,
 *           accumulate and A as avits_score_spatial.
 * lse_all : [B,H,M] fp32, contiguous: natural-log logsumexp of s*q_i.k_j over
 *           every key of the joint sequence, for the same s and the same
 *           queries.  Each per-head mass is clamped to [0, 1] before the
 *           head mean (inconsistent values would give masses outside it).
 * lse_opt : NULL or [B,H,M,2]: (lse_all as given, lse_txt).
 * workspace : avits_score_spatial_workspace(dt, B, H, M, L, d) bytes,
 *           zero-filled before first use as for avits_score_spatial.
 * Tensor-core path only (bf16, d in {64,128}, 16-byte aligned layout,
 * H <= 255); anything else returns AVITS_ERR_UNSUPPORTED.
 * ---------------------------------------------------------------------- */
avits_status avits_score_spatial_lse(const void* q_img, const void* k_txt, avits_dtype dt,
                                     int B, int H, int M, int L, int d, int64_t q_sb,
                                     int64_t q_sh, int64_t q_sn, int64_t k_sb, int64_t k_sh,
                                     int64_t k_sn, const float* lse_all, float softmax_scale,
                                     float weight, int accumulate, float* A, float* lse_opt,
                                     void* workspace, size_t ws_bytes, void* stream);

/* ------------------------------------------------------------------------
 * avits_score_spatial for sequences whose text and image tokens interleave
 * (the unified sequences of MLLM-conditioned models, Sec. 3.3.1): the text
 * keys are the keys j with text_mask[b*Nk + j] != 0 instead of the first L.
 * text_mask : [B,Nk] uint8 device memory (one byte per key).  Everything else
 * (Eq. 3-5, layouts, workspace, weight / accumulate, lse_opt) as
 * avits_score_spatial; lse_opt[...,1] is the logsumexp over the masked keys.
 * ---------------------------------------------------------------------- */
avits_status avits_score_spatial_keymask(const void* q_img, const void* k_all, avits_dtype dt,
                                         int B, int H, int M, int Nk, int d, int64_t q_sb,
                                         int64_t q_sh, int64_t q_sn, int64_t k_sb, int64_t k_sh,
                                         int64_t k_sn, const uint8_t* text_mask,
                                         float softmax_scale, float weight, int accumulate,
                                         float* A, float* lse_opt, void* workspace,
                                         size_t ws_bytes, void* stream);

/* ------------------------------------------------------------------------
 * Joint-attention forward of a double-stream block (Eq. 4-5, Sec. 3.3.1) that
 * also produces the spatial score of Eq. 3 from the same softmax.  The paper
 * recomputes Q K^T after the block's attention only because fused attention
 * kernels do not expose the weights; this call IS the block's attention and
 * reads the text mass off it.  For batch b, head h and query row i:
 *
 *     l_ij   = softmax_scale * <q_bhi, k_bhj>                j = 0 .. Nk-1
 *     o_bhi  = sum_j exp(l_ij) v_bhj / sum_j exp(l_ij)
 *     mass   = sum_{j<L} exp(l_ij) / sum_{j<Nk} exp(l_ij)    (text keys first)
 *     A[b,i] = (accumulate ? A[b,i] : 0) + weight * (1/H) * sum_h mass
 *
 * q : [B,H,Mq,d] bf16, the joint queries [Q_txt || Q_img] of Eq. 4 (any rows:
 *     text and image rows alike; A and lse are given for every row).
 * k, v : [B,H,Nk,d] bf16, the joint keys / values, the L text keys FIRST.
 * o : [B,H,Mq,d] bf16 output (must not overlap q, k, v).
 * q_str, k_str, v_str, o_str : element strides (batch, head, row) of each
 *     tensor as an array of 3 int64, or NULL for contiguous [B,H,rows,d]; the
 *     d axis is contiguous.  Bases 16-byte aligned, strides multiples of 8
 *     elements ([B,N,H,d] views of a model's projections qualify).
 * d in {64, 128}; 0 <= L <= Nk; softmax_scale > 0 (1/sqrt(d)).
 * lse_opt : NULL or [B,H,Mq,2] fp32: natural-log logsumexp of the row over
 *     all keys and over the text keys (-inf when L = 0).
 * A : NULL (no score; workspace may then be NULL) or [B,Mq] fp32, written
 *     (accumulate = 0) or added to; H <= 255 when A is given.
 * workspace/ws_bytes : when A is given, avits_attention_forward_workspace()
 *     bytes, 8-byte aligned, ZERO-FILLED before first use; every call that
 *     completes leaves it zero, so it is reused as is (re-zero it after
 *     AVITS_ERR_TIMEOUT).  One workspace per concurrently running call.
 * Precision: P = softmax numerators enter the P V product rounded to bf16
 *     (fp32 accumulation, fp32 row sums), O is rounded to bf16 once.
 * Other dtypes or d values return AVITS_ERR_UNSUPPORTED; one kernel launch.
 * ---------------------------------------------------------------------- */
avits_status avits_attention_forward(const void* q, const void* k, const void* v, avits_dtype dt,
                                     int B, int H, int Mq, int Nk, int L, int d,
                                     const int64_t* q_str, const int64_t* k_str,
                                     const int64_t* v_str, const int64_t* o_str,
                                     float softmax_scale, void* o, float* lse_opt, float weight,
                                     int accumulate, float* A, void* workspace, size_t ws_bytes,
                                     void* stream);

/* Workspace bytes of avits_attention_forward with a score output (0 for
 * invalid sizes). */
size_t avits_attention_forward_workspace(int B, int H, int Mq);

/* ------------------------------------------------------------------------
 * Temporal importance.  Sec. 3.3.2 scores a token by how much its feature
 * moves across the collected denoising steps.  This call takes the two most
 * recent snapshots and returns the relative step change
 *
 *     V[b,i] = ||h_t[b,i,:] - h_prev[b,i,:]||_2 / (||h_prev[b,i,:]||_2 + eps)
 *
 * (eps = 1e-6 by default).  The paper's own N_T-snapshot step variance,
 * Eq. 6-7, is avits_score_temporal_var below.
 * h_t, h_prev : [B,N,D] contiguous, bf16 or fp32, 16-byte aligned.
 * V : [B,N] fp32.  Sums of squares are accumulated in fp32.
 * ---------------------------------------------------------------------- */
avits_status avits_score_temporal(const void* h_t, const void* h_prev, avits_dtype dt,
                                  int B, int N, int D, float eps, float* V, void* stream);

/* ------------------------------------------------------------------------
 * Both scores of one transition in one call: avits_score_spatial followed by
 * avits_score_temporal on the same stream, with the same arguments and
 * results as the two calls (h_t / h_prev are [B,M,D]: the M scored tokens).
 * On the tensor-core path the temporal kernel is launched as a programmatic
 * dependent of the spatial kernel and streams the two snapshots from HBM
 * while the spatial kernel is tensor/MUFU-bound, instead of after it.  Its
 * inputs must be complete when the call is made (as for any stream-ordered
 * call); all results are complete for the next call on the stream.
 * ---------------------------------------------------------------------- */
avits_status avits_score_spatiotemporal(const void* q_img, const void* k_all, avits_dtype dt,
                                        int B, int H, int M, int Nk, int L, int d,
                                        int64_t q_sb, int64_t q_sh, int64_t q_sn,
                                        int64_t k_sb, int64_t k_sh, int64_t k_sn,
                                        float softmax_scale, float weight, int accumulate,
                                        float* A, float* lse_opt,
                                        void* workspace, size_t ws_bytes,
                                        const void* h_t, const void* h_prev, int D, float eps,
                                        float* V, void* stream);

/* ------------------------------------------------------------------------
 * Paper-form temporal importance, Sec. 3.3.2 Eq. 6-7: for each token the
 * unbiased sample variance over N_T snapshots of every channel, averaged
 * over the D channels.
 * snaps : N_T pointers (a HOST array of device pointers), each to a [B,N,D]
 *         contiguous snapshot, oldest first.  N_T >= 2.
 * V : [B,N] fp32.  Two-pass (mean, then squared deviations) in fp32.
 * ---------------------------------------------------------------------- */
avits_status avits_score_temporal_var(const void* const* snaps, int n_t, avits_dtype dt,
                                      int B, int N, int D, float* V, void* stream);

/* ------------------------------------------------------------------------
 * Joint score and selection, Sec. 3.3.3, Eq. 8-9.  Per batch element:
 *
 *   A^ = (A - min A) / ((max A - min A) + eps_norm),   V^ likewise
 *   S  = alpha * A^ + (1 - alpha) * V^                   (fp32, this op order)
 *   sel = the k largest S; ties go to the LOWER token index (the paper breaks
 *         ties with ~1e-6 Gaussian noise; this library is deterministic).
 *         NaN ranks below every number; -0 and +0 are equal.
 *
 * A, V : [B,M] fp32.  0 <= k <= M, M <= 65536.
 * S_opt : NULL or [B,M] fp32.
 * sel_idx : [B,k] int32, the selected token indices in ascending order.
 * sel_mask_opt : NULL or [B,M] uint8 (1 = selected).
 * tok_offset : [B,M] int32, where token i starts in the mixed sequence:
 *              i + 3 * (number of selected tokens before i).
 * A NaN in S also sets AVITS_ERR_NAN in the device status word.
 * ---------------------------------------------------------------------- */
avits_status avits_fuse_select(const float* A, const float* V, int B, int M, float alpha,
                               float eps_norm, int k, float* S_opt, int32_t* sel_idx,
                               uint8_t* sel_mask_opt, int32_t* tok_offset, void* stream);

/* ------------------------------------------------------------------------
 * avits_fuse_select with the paper's tie-breaking perturbation, Eq. 9
 * (Sec. 3.3.3: small Gaussian noise added to the joint score before TopK).
 * The noise is SUPPLIED BY THE CALLER (this library draws no random
 * numbers):
 *   S' = S + perturb   (one more rounded fp32 addition, after Eq. 8)
 * and the selection is taken on S' (ties in S' still go to the lower index).
 * perturb : NULL (exactly avits_fuse_select) or [B,M] fp32 device memory,
 *           e.g. 1e-6 * N(0,1) per token as in the paper.
 * S_opt receives S'.  Everything else as avits_fuse_select.
 * ---------------------------------------------------------------------- */
avits_status avits_fuse_select_perturbed(const float* A, const float* V, const float* perturb,
                                         int B, int M, float alpha, float eps_norm, int k,
                                         float* S_opt, int32_t* sel_idx, uint8_t* sel_mask_opt,
                                         int32_t* tok_offset, void* stream);

/* ------------------------------------------------------------------------
 * Selective upsampling, Sec. 3.2 Stage 2: selected tokens are expanded to
 * the next resolution, the others stay as they are, and all of them go into
 * one packed mixed-resolution sequence of N_out = M + 3k tokens.
 *
 * Token i (input frame position (y,x), span s; without pos_in: (i/gw, i%gw),
 * s = 1) is emitted at tok_offset[i]:
 *   selected : 4 children c = 2a+b (a,b in {0,1}) at output positions
 *              (2y + a*s, 2x + b*s), span s, each child = 2x upsample of
 *              parent pixel (a,b): nearest broadcasts it; bilinear uses the
 *              fixed weights 0.75/0.25 of a half-pixel-centred 2x resize with
 *              edge clamping over the input's pixel image at the token's own
 *              resolution: the dense latent, or for a mixed input of spans
 *              1, 2 and 4, level log2(s) of the input frame's pyramid (a
 *              pixel inside one token pixel is that pixel, any other the
 *              ((a + b) + (c + d)) / 4 average of the four pixels below it).
 *   deferred : the token unchanged at (2y, 2x), span 2s.
 * Output positions are in the doubled frame (2gh x 2gw), usable directly as
 * 2D RoPE ids.
 *
 * latent : [B,M,C*4] bf16/fp32.  Without pos_in, M = gh*gw (a dense grid).
 * pos_in_opt/span_in_opt : NULL, or [B,M,2] / [B,M] int32 for a mixed input
 *          (a second transition) on a gh x gw frame.  In bilinear mode the
 *          tokens must tile the frame with spans 1, 2 or 4 at multiples of
 *          their span, gh and gw even (AVITS_ERR_COVERAGE on the device
 *          otherwise).
 * workspace/ws_bytes : bilinear mode with a mixed input only:
 *          avits_selective_upsample_workspace() bytes, 16-byte aligned, any
 *          contents (the call rebuilds the frame's cell map there); otherwise
 *          ignored (may be NULL).
 * sel_mask, tok_offset : from avits_fuse_select.  k = number selected.
 *          A token whose outputs would not lie inside [0, M+3k) (tok_offset
 *          < 0, or above M+3k-4 for a selected / M+3k-1 for a deferred token)
 *          is not written and raises AVITS_ERR_COVERAGE on the device.
 * out_latent : [B,M+3k,C*4] same dtype.  out_pos : [B,M+3k,2] (row, col).
 * out_span : [B,M+3k].  out_src_tok : [B,M+3k] input token index.
 * out_src_sub : [B,M+3k] int8, child number 0..3, or -1 for a deferred token.
 * ---------------------------------------------------------------------- */
avits_status avits_selective_upsample(const void* latent, avits_dtype dt, int B, int M,
                                      int grid_h, int grid_w, int C, int p,
                                      const int32_t* pos_in_opt, const int32_t* span_in_opt,
                                      const uint8_t* sel_mask, const int32_t* tok_offset, int k,
                                      avits_upmode mode, void* out_latent, int32_t* out_pos,
                                      int32_t* out_span, int32_t* out_src_tok,
                                      int8_t* out_src_sub, void* workspace, size_t ws_bytes,
                                      void* stream);

/* Workspace bytes of avits_selective_upsample / avits_select_upsample in
 * bilinear mode (the input frame's cell map, needed with a mixed input only);
 * 0 for nearest mode or invalid sizes. */
size_t avits_selective_upsample_workspace(avits_upmode mode, int B, int grid_h, int grid_w);

/* ------------------------------------------------------------------------
 * avits_fuse_select_perturbed followed by avits_selective_upsample, in ONE
 * launch (the transition of Sec. 3.2 after Eq. 8-9): every output is what
 * the two calls produce, bit for bit.  Each batch element gets several CTAs
 * that all compute its selection, so none waits for another; the first one
 * writes S_opt, sel_idx, sel_mask and tok_offset.  Up to M = 4096 tokens per
 * element it is one kernel; above that the two kernels run back to back.
 * perturb : NULL or [B,M] fp32 (Eq. 9 tie-breaking noise, as
 *           avits_fuse_select_perturbed).
 * sel_mask : REQUIRED here ([B,M] uint8).  The remaining arguments are those
 *            of avits_fuse_select_perturbed and avits_selective_upsample.
 * ---------------------------------------------------------------------- */
avits_status avits_select_upsample(const float* A, const float* V, const float* perturb, int B,
                                   int M, float alpha, float eps_norm, int k, float* S_opt,
                                   int32_t* sel_idx, uint8_t* sel_mask, int32_t* tok_offset,
                                   const void* latent, avits_dtype dt, int grid_h, int grid_w,
                                   int C, int p, const int32_t* pos_in_opt,
                                   const int32_t* span_in_opt, avits_upmode mode,
                                   void* out_latent, int32_t* out_pos, int32_t* out_span,
                                   int32_t* out_src_tok, int8_t* out_src_sub, void* workspace,
                                   size_t ws_bytes, void* stream);

/* ------------------------------------------------------------------------
 * Final merge, Sec. 3.2 Stage 3: expand every remaining token to full
 * resolution and lay the tokens out in spatial (raster) order.
 * A token at (y,x) with span s covers cells [y,y+s) x [x,x+s) of the
 * full_h x full_w frame; the tokens must tile the frame exactly once:
 * a cell covered twice, a cell left uncovered and a token outside the frame
 * each raise AVITS_ERR_COVERAGE on the device, in both modes.
 *   nearest  : full-res pixel (Y,X) takes token pixel ((Y-2y)/s, (X-2x)/s).
 *   bilinear : spans 1, 2 and 4 at multiples of their span, full_h and
 *              full_w even: span-1 tokens are copied; every coarser token is
 *              refined level by level from the frame's pixel pyramid,
 *              coarsest first: inside a span-4 token, level 1 is the
 *              half-pixel-centred 2x bilinear resize of level 2; then every
 *              cell of span 2 or 4 takes the 2x bilinear resize of level 1.
 *              With spans 1 and 2 only: the low-res grid is rebuilt (span-2
 *              tokens as they are, each group of 4 span-1 children 2x2
 *              average pooled) and the span-2 cells take its 2x resize.  Any
 *              other span raises AVITS_ERR_COVERAGE.
 * mixed : [B,N,C*4].  pos [B,N,2], span [B,N] int32.
 * out_full : [B,full_h*full_w,C*4] same dtype.
 * workspace : avits_merge_final_workspace() bytes (both modes), 16-byte
 *             aligned, ZERO-FILLED before its first use; the calls keep it
 *             consistent afterwards (nearest: a claim map tagged per call and
 *             a counter each call clears; bilinear: a cell map it refills).
 * ---------------------------------------------------------------------- */
avits_status avits_merge_final(const void* mixed, avits_dtype dt, int B, int N,
                               const int32_t* pos, const int32_t* span, int full_h, int full_w,
                               int C, int p, avits_upmode mode, void* out_full,
                               void* workspace, size_t ws_bytes, void* stream);

size_t avits_merge_final_workspace(avits_upmode mode, int B, int full_h, int full_w);

/* ------------------------------------------------------------------------
 * Synchronises `stream`, returns the OR of the device-side error codes
 * raised since the last call (as the lowest-numbered set code, or AVITS_OK)
 * and clears the word.  The only call that blocks the host.
 * ---------------------------------------------------------------------- */
avits_status avits_device_status(void* stream);

/* ------------------------------------------------------------------------
 * Test hook for the failure detection of the device-side waits (a library
 * facility; the paper has no counterpart).  Every spin in the kernels is an
 * mbarrier wait bounded by a wall-clock limit: on expiry it records
 * AVITS_ERR_TIMEOUT in the status word and raises its CTA's abort flag, which
 * ends the waits of the other roles, and the kernel returns.  This call runs
 * that code in one CTA on barriers nothing arrives at, so a test can exercise
 * the path on a GPU without faulting it: warp 0 waits with `limit_ns`, warp 1
 * waits on another barrier with 100 x limit_ns and gives up when warp 0
 * raises the abort flag.
 * limit_ns : 1e3 .. 1e8 (1 us .. 100 ms); else AVITS_ERR_INVALID_ARG.
 * result   : device int64[5], written: [0] warp 0 completed (0 expected),
 *            [1] warp 0's wait in ns, [2] warp 1 completed (0 expected),
 *            [3] warp 1's wait in ns, [4] the abort flag (1 expected).
 * The status word then holds AVITS_ERR_TIMEOUT (avits_device_status).
 * ---------------------------------------------------------------------- */
avits_status avits_selftest_bounded_wait(unsigned long long limit_ns, long long* result,
                                         void* stream);

/* Static text of a status code. */
const char* avits_status_string(avits_status s);

/* Text of the last CUDA error seen by this thread's calls ("" if none). */
const char* avits_last_error_string(void);

/* Library version, "MAJOR.MINOR.PATCH". */
const char* avits_version(void);

#ifdef __cplusplus
}
#endif

#endif /* AVITS_H */
