// frame_map.cuh — the cell map of a frame of mixed-span tokens and the pixel
// pyramid that multi-level bilinear resampling reads (Sec. 3.2, Stages 2-3).
//
// A frame of fh x fw cells is tiled by tokens of span s in {1, 2, 4}, each at
// a multiple of s; token pixel (a, b) stands for the s x s full pixels
// (2y + a*s .., 2x + b*s ..).  The map holds, per cell, the covering token's
// index within its element and log2(s).  Level l of the pyramid: a level-l
// pixel inside one token pixel (span >= 2^l) is that pixel; any other is
// ((a + b) + (c + d)) * 0.25 of its four level-(l-1) pixels (a, b the upper
// row).  A selected token of span 2^l is upsampled from level l (Stage 2);
// the merge refines every token coarser than a level from the level above,
// coarsest first (Stage 3).
#pragma once

#include "avits_common.cuh"

namespace avits {

constexpr int kMapLevelShift = 28;
constexpr int32_t kMapTokMask = (1 << kMapLevelShift) - 1;
constexpr int kMaxMapLevel = 2;   // spans 1, 2 and 4

__device__ __forceinline__ int32_t map_entry(int tok, int lvl) {
  return tok | (lvl << kMapLevelShift);
}
__device__ __forceinline__ int map_tok(int32_t e) { return e & kMapTokMask; }
__device__ __forceinline__ int map_lvl(int32_t e) { return (e >> kMapLevelShift) & 3; }

// Pixel (R, Q) of level l, channel ch; tok = the element's tokens [N, T4],
// map = the element's cell map (fw cells per row).  0 for a hole (the map
// kernel reports it).
template <int l, typename T>
__device__ float frame_pixel(const T* __restrict__ tok, int T4, const int32_t* __restrict__ map,
                             int fw, int ch, int R, int Q) {
  const int Y = R << l, X = Q << l;   // the block's first full pixel
  const int32_t e = map[(int64_t)(Y >> 1) * fw + (X >> 1)];
  if (e < 0) return 0.f;
  const int lv = map_lvl(e);
  if constexpr (l > 0) {
    if (lv < l) {
      const float a = frame_pixel<l - 1>(tok, T4, map, fw, ch, 2 * R, 2 * Q);
      const float b = frame_pixel<l - 1>(tok, T4, map, fw, ch, 2 * R, 2 * Q + 1);
      const float c = frame_pixel<l - 1>(tok, T4, map, fw, ch, 2 * R + 1, 2 * Q);
      const float d = frame_pixel<l - 1>(tok, T4, map, fw, ch, 2 * R + 1, 2 * Q + 1);
      return __fmul_rn(__fadd_rn(__fadd_rn(a, b), __fadd_rn(c, d)), 0.25f);
    }
  }
  // the token's first cell is the cell rounded down to its span
  const int s = 1 << lv;
  const int ty = (Y - 2 * ((Y >> 1) & ~(s - 1))) >> lv;
  const int tx = (X - 2 * ((X >> 1) & ~(s - 1))) >> lv;
  return load_elem(tok, (int64_t)map_tok(e) * T4 + ch * 4 + ty * 2 + tx);
}

template <typename T>
__device__ __forceinline__ float frame_pixel_at(int l, const T* __restrict__ tok, int T4,
                                                const int32_t* __restrict__ map, int fw, int ch,
                                                int R, int Q) {
  if (l == 0) return frame_pixel<0>(tok, T4, map, fw, ch, R, Q);
  if (l == 1) return frame_pixel<1>(tok, T4, map, fw, ch, R, Q);
  return frame_pixel<2>(tok, T4, map, fw, ch, R, Q);
}

// Axis weights of a half-pixel-centred 2x bilinear resize: output pixel P of
// a 2n-pixel axis reads source pixels r0, r1 (clamped to [0, n-1]) with
// weights w0, w1: even P = 2m -> (m-1: 1/4, m: 3/4); odd P -> (m: 3/4, m+1: 1/4).
__device__ __forceinline__ void bil_axis(int P, int n, int& r0, int& r1, float& w0, float& w1) {
  const int m = P >> 1;
  if ((P & 1) == 0) { r0 = m - 1; r1 = m; w0 = 0.25f; w1 = 0.75f; }
  else { r0 = m; r1 = m + 1; w0 = 0.75f; w1 = 0.25f; }
  r0 = max(r0, 0);
  r1 = min(r1, n - 1);
}

// wy0*(wx0*p00 + wx1*p01) + wy1*(wx0*p10 + wx1*p11), rounded step by step
__device__ __forceinline__ float bil_combine(float p00, float p01, float p10, float p11,
                                            float wy0, float wy1, float wx0, float wx1) {
  const float top = __fadd_rn(__fmul_rn(wx0, p00), __fmul_rn(wx1, p01));
  const float bot = __fadd_rn(__fmul_rn(wx0, p10), __fmul_rn(wx1, p11));
  return __fadd_rn(__fmul_rn(wy0, top), __fmul_rn(wy1, bot));
}

// Pixel (P, Q) of the 2x bilinear resize of level l ((2fh >> l) x (2fw >> l)
// pixels).
template <typename T>
__device__ __forceinline__ float frame_resize2x(int l, const T* __restrict__ tok, int T4,
                                                const int32_t* __restrict__ map, int fh, int fw,
                                                int ch, int P, int Q) {
  int r0, r1, c0, c1;
  float wy0, wy1, wx0, wx1;
  bil_axis(P, (2 * fh) >> l, r0, r1, wy0, wy1);
  bil_axis(Q, (2 * fw) >> l, c0, c1, wx0, wx1);
  return bil_combine(frame_pixel_at(l, tok, T4, map, fw, ch, r0, c0),
                     frame_pixel_at(l, tok, T4, map, fw, ch, r0, c1),
                     frame_pixel_at(l, tok, T4, map, fw, ch, r1, c0),
                     frame_pixel_at(l, tok, T4, map, fw, ch, r1, c1), wy0, wy1, wx0, wx1);
}

// Builds the cell map of B elements of N tokens (map pre-filled with -1) on
// `s`: a token off the frame, off its alignment, of a span other than 1, 2 or
// 4, or overlapping another raises AVITS_ERR_COVERAGE (holes are found by
// the readers).  Defined in merge.cu.
cudaError_t launch_cell_map(int B, int N, const int32_t* pos, const int32_t* span, int fh, int fw,
                            int32_t* map, unsigned int* status, cudaStream_t s);

}  // namespace avits
