// upsample_token.cuh — one input token of the selective upsample (Sec. 3.2,
// Stage 2), done by one warp; shared by upsample_kernel and the fused
// selection + upsample kernel.
//
// Token i of element b starts at output o (tok_offset):
//   deferred  -> its C*4 values copied, position (2y, 2x), span 2s;
//   selected  -> 4 children (a,b) at (2y + a*s, 2x + b*s), span s; a child is
//                the 2x upsample of the parent's pixel (a,b): nearest
//                broadcasts the pixel; bilinear applies the fixed 0.25 / 0.75
//                weights of a half-pixel-centred 2x resize with edge clamping,
//                reading neighbouring pixels from the dense input latent, or,
//                for a mixed input, from level log2(s) of the input frame's
//                pixel pyramid through its cell map (frame_map.cuh).
// Nearest with 16-byte token rows: each lane writes whole 16-byte chunks
// (coalesced); otherwise lanes split the (child, channel) work, each writing
// the 4 pixels of one channel of one child.  Lanes 0-3 write the position /
// span / source maps.
#pragma once

#include "avits_common.cuh"
#include "frame_map.cuh"

namespace avits {

template <typename T>
struct UpsampleArgs {
  const T* latent;                 // [B,M,C*4]
  int M, gh, gw, C, n_out;
  const int32_t* pos_in;           // [B,M,2] or NULL (raster positions, span 1)
  const int32_t* span_in;          // [B,M]
  T* out;                          // [B,n_out,C*4]
  int32_t* out_pos;                // [B,n_out,2]
  int32_t* out_span;               // [B,n_out]
  int32_t* out_src_tok;            // [B,n_out]
  int8_t* out_src_sub;             // [B,n_out]
  // bilinear with a mixed input: the input frame's cell map [B,gh,gw]
  // (frame_map.cuh); NULL for a dense grid
  const int32_t* map = nullptr;
  unsigned int* status = nullptr;  // device status word (an offset out of range)
};

// Where a token's C*4 source values are read from: element b's rows of the
// input latent in global memory, or a copy of rows [lo, lo + n) in shared
// memory (the fused selection + upsample kernel).
template <typename T>
struct GlobalRows {
  const T* latent;   // [B,M,C*4]
  int M, T4;
  __device__ const T* row(int b, int tok) const {
    return latent + ((int64_t)b * M + tok) * T4;
  }
};
template <typename T>
struct SharedRows {
  const T* rows;     // rows [lo, lo + n) of one element
  int lo, T4;
  __device__ const T* row(int, int tok) const { return rows + (int64_t)(tok - lo) * T4; }
};

// Token i of element b, selected or not, starting at output o; one warp.
// Src::row(b, tok) gives the token's source values (tok's bilinear
// neighbours included).
template <typename T, bool kBilinear, typename Src>
__device__ __forceinline__ void upsample_token(const UpsampleArgs<T>& u, const Src& rows, int b,
                                               int i, int o, bool sel, int lane) {
  using PV = typename Pix4<T>::V;
  const int C = u.C, gw = u.gw, gh = u.gh, M = u.M;
  const int T4 = C * 4;
  const int64_t in_tok = (int64_t)b * M + i;
  int y, x, s;
  if (u.pos_in) {
    y = u.pos_in[in_tok * 2];
    x = u.pos_in[in_tok * 2 + 1];
    s = u.span_in[in_tok];
  } else {
    y = i / gw;
    x = i - y * gw;
    s = 1;
  }
  // the outputs must lie inside the element's sequence: an offset from the
  // caller that does not is reported (AVITS_ERR_COVERAGE) and the token is
  // not written
  if (o < 0 || o > u.n_out - (sel ? 4 : 1)) {
    if (lane == 0) raise_status(u.status, AVITS_ERR_COVERAGE);
    return;
  }
  const T* src = rows.row(b, i);
  const int64_t out_tok0 = (int64_t)b * u.n_out + o;
  const int tb = T4 * (int)sizeof(T);
  if (!kBilinear && (tb & 15) == 0) {
    // 16-byte chunks: a deferred token is copied, a selected one gives each
    // child (a, b) the chunk whose channel pixels all equal the parent's
    // pixel (a, b); one chunk per lane (bf16, 16 channels: 32 lanes, 4 children)
    const int cpc = tb / 16;
    if (!sel) {
      uint4* dst = reinterpret_cast<uint4*>(u.out + out_tok0 * T4);
      for (int q = lane; q < cpc; q += 32) dst[q] = reinterpret_cast<const uint4*>(src)[q];
    } else {
      for (int q = lane; q < 4 * cpc; q += 32) {
        const int child = q / cpc, j = q - child * cpc;
        const int a = child >> 1, bb = child & 1;
        reinterpret_cast<uint4*>(u.out + (out_tok0 + child) * T4)[j] =
            gather_chunk<T>(src, j, a, a, bb, bb);
      }
    }
  } else if (!sel) {
    PV* dst = reinterpret_cast<PV*>(u.out + out_tok0 * T4);
    const PV* sp = reinterpret_cast<const PV*>(src);
    for (int c = lane; c < C; c += 32) dst[c] = sp[c];
  } else {
    // a mixed input token of span 2^l is resized from level l of the input
    // frame's pyramid; an invalid position or span (reported by the map
    // kernel) gives zeros
    const int lv = (s == 1) ? 0 : (s == 2) ? 1 : (s == 4) ? 2 : -1;
    const bool frame_ok = lv >= 0 && y >= 0 && x >= 0 && y + s <= gh && x + s <= gw &&
                          ((y | x) & (s - 1)) == 0;
    for (int task = lane; task < 4 * C; task += 32) {
      const int child = task / C, c = task - child * C;
      const int a = child >> 1, bb = child & 1;
      PV v;
      if (kBilinear && u.map) {
        float r[4] = {0.f, 0.f, 0.f, 0.f};
        if (frame_ok) {
          const T* tokb = u.latent + (int64_t)b * M * T4;
          const int32_t* mapb = u.map + (int64_t)b * gh * gw;
          const int R0 = 2 * ((2 * y) >> lv) + 2 * a, Q0 = 2 * ((2 * x) >> lv) + 2 * bb;
#pragma unroll
          for (int q = 0; q < 4; ++q)
            r[q] = frame_resize2x(lv, tokb, T4, mapb, gh, gw, c, R0 + (q >> 1), Q0 + (q & 1));
        }
        v = Pix4<T>::make(r[0], r[1], r[2], r[3]);
      } else if (!kBilinear) {
        const float p = load_elem(src, c * 4 + a * 2 + bb);
        v = Pix4<T>::make(p, p, p, p);
      } else {
        const int IH = 2 * gh, IW = 2 * gw;
        float r[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const int ph = q >> 1, pw = q & 1;
          int r0, r1, c0, c1;
          float wy0, wy1, wx0, wx1;
          bil_axis(4 * y + 2 * a + ph, IH, r0, r1, wy0, wy1);
          bil_axis(4 * x + 2 * bb + pw, IW, c0, c1, wx0, wx1);
          auto pix = [&](int R, int Q) {
            return load_elem(rows.row(b, (R >> 1) * gw + (Q >> 1)), c * 4 + (R & 1) * 2 + (Q & 1));
          };
          r[q] = bil_combine(pix(r0, c0), pix(r0, c1), pix(r1, c0), pix(r1, c1), wy0, wy1, wx0, wx1);
        }
        v = Pix4<T>::make(r[0], r[1], r[2], r[3]);
      }
      reinterpret_cast<PV*>(u.out + (out_tok0 + child) * T4)[c] = v;
    }
  }
  if (!sel) {
    if (lane == 0) {
      u.out_pos[out_tok0 * 2] = 2 * y;
      u.out_pos[out_tok0 * 2 + 1] = 2 * x;
      u.out_span[out_tok0] = 2 * s;
      u.out_src_tok[out_tok0] = i;
      u.out_src_sub[out_tok0] = -1;
    }
    return;
  }
  if (lane < 4) {
    const int a = lane >> 1, bb = lane & 1;
    const int64_t ot = out_tok0 + lane;
    u.out_pos[ot * 2] = 2 * y + a * s;
    u.out_pos[ot * 2 + 1] = 2 * x + bb * s;
    u.out_span[ot] = s;
    u.out_src_tok[ot] = i;
    u.out_src_sub[ot] = (int8_t)lane;
  }
}

}  // namespace avits
