// upsample.cu — selective upsampling into a packed mixed-resolution sequence
// (Sec. 3.2, Stage 2).
//
// One warp per input token i.  Its outputs start at tok_offset[i] (from the
// selection kernel), so no scan is needed here:
//   deferred  -> the token's C*4 values copied, position (2y,2x), span 2s;
//   selected  -> 4 children (a,b) at (2y + a*s, 2x + b*s), span s.  A child is
//                the 2x upsample of the parent's pixel (a,b): nearest
//                broadcasts the pixel; bilinear applies the fixed 0.25 / 0.75
//                weights of a half-pixel-centred 2x resize with edge clamping,
//                reading neighbouring pixels from the dense input latent.
// Lanes split the (child, channel) work; each writes the 4 pixels of one
// channel of one child (8 B for bf16, 16 B for fp32) and lanes 0-3 write the
// position / span / source maps.  Algorithmic bytes per launch:
// B*M*T*elt (read) + B*M*5 (mask, offset) + B*N_out*(T*elt + 17).
#include "avits_common.cuh"
#include "avits_internal.h"

namespace avits {
namespace {

constexpr int kWarpsPerCta = 8;

template <typename T>
struct Pix4;   // 4 pixels of one channel, stored together

template <>
struct Pix4<float> {
  using V = float4;
  __device__ static V make(float a, float b, float c, float d) { return make_float4(a, b, c, d); }
};
template <>
struct Pix4<__nv_bfloat16> {
  using V = uint2;
  __device__ static V make(float a, float b, float c, float d) {
    const __nv_bfloat162 lo = __floats2bfloat162_rn(a, b);
    const __nv_bfloat162 hi = __floats2bfloat162_rn(c, d);
    return make_uint2(*reinterpret_cast<const uint32_t*>(&lo),
                      *reinterpret_cast<const uint32_t*>(&hi));
  }
};

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

template <typename T, bool kBilinear>
__global__ void __launch_bounds__(kWarpsPerCta * 32)
upsample_kernel(const T* __restrict__ latent, int B, int M, int gh, int gw, int C,
                const int32_t* __restrict__ pos_in, const int32_t* __restrict__ span_in,
                const uint8_t* __restrict__ mask, const int32_t* __restrict__ tok_offset,
                int n_out, T* __restrict__ out, int32_t* __restrict__ out_pos,
                int32_t* __restrict__ out_span, int32_t* __restrict__ out_src_tok,
                int8_t* __restrict__ out_src_sub) {
  using PV = typename Pix4<T>::V;
  pdl_wait_then_trigger();
  const int lane = threadIdx.x & 31;
  const int64_t gwarp = (int64_t)blockIdx.x * kWarpsPerCta + (threadIdx.x >> 5);
  if (gwarp >= (int64_t)B * M) return;
  const int b = (int)(gwarp / M), i = (int)(gwarp % M);
  const int T4 = C * 4;
  const int64_t in_tok = (int64_t)b * M + i;
  const int o = tok_offset[in_tok];
  const bool sel = mask[in_tok] != 0;
  int y, x, s;
  if (pos_in) {
    y = pos_in[in_tok * 2];
    x = pos_in[in_tok * 2 + 1];
    s = span_in[in_tok];
  } else {
    y = i / gw;
    x = i - y * gw;
    s = 1;
  }
  const T* src = latent + in_tok * T4;
  const int64_t out_tok0 = (int64_t)b * n_out + o;
  if (!sel) {
    PV* dst = reinterpret_cast<PV*>(out + out_tok0 * T4);
    const PV* sp = reinterpret_cast<const PV*>(src);
    for (int c = lane; c < C; c += 32) dst[c] = sp[c];
    if (lane == 0) {
      out_pos[out_tok0 * 2] = 2 * y;
      out_pos[out_tok0 * 2 + 1] = 2 * x;
      out_span[out_tok0] = 2 * s;
      out_src_tok[out_tok0] = i;
      out_src_sub[out_tok0] = -1;
    }
    return;
  }
  for (int task = lane; task < 4 * C; task += 32) {
    const int child = task / C, c = task - child * C;
    const int a = child >> 1, bb = child & 1;
    PV v;
    if (!kBilinear) {
      const float p = load_elem(src, c * 4 + a * 2 + bb);
      v = Pix4<T>::make(p, p, p, p);
    } else {
      const int IH = 2 * gh, IW = 2 * gw;
      const T* lb = latent + (int64_t)b * M * T4;
      float r[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const int ph = q >> 1, pw = q & 1;
        int r0, r1, c0, c1;
        float wy0, wy1, wx0, wx1;
        bil_axis(4 * y + 2 * a + ph, IH, r0, r1, wy0, wy1);
        bil_axis(4 * x + 2 * bb + pw, IW, c0, c1, wx0, wx1);
        auto pix = [&](int R, int Q) {
          return load_elem(lb, (int64_t)((R >> 1) * gw + (Q >> 1)) * T4 + c * 4 + (R & 1) * 2 +
                                   (Q & 1));
        };
        r[q] = bil_combine(pix(r0, c0), pix(r0, c1), pix(r1, c0), pix(r1, c1), wy0, wy1, wx0, wx1);
      }
      v = Pix4<T>::make(r[0], r[1], r[2], r[3]);
    }
    reinterpret_cast<PV*>(out + (out_tok0 + child) * T4)[c] = v;
  }
  if (lane < 4) {
    const int a = lane >> 1, bb = lane & 1;
    const int64_t ot = out_tok0 + lane;
    out_pos[ot * 2] = 2 * y + a * s;
    out_pos[ot * 2 + 1] = 2 * x + bb * s;
    out_span[ot] = s;
    out_src_tok[ot] = i;
    out_src_sub[ot] = (int8_t)lane;
  }
}

template <typename T>
cudaError_t launch_t(const void* latent, int B, int M, int gh, int gw, int C,
                     const int32_t* pos_in, const int32_t* span_in, const uint8_t* mask,
                     const int32_t* tok_offset, int k, avits_upmode mode, void* out,
                     int32_t* out_pos, int32_t* out_span, int32_t* out_src_tok,
                     int8_t* out_src_sub, cudaStream_t s) {
  const int64_t warps = (int64_t)B * M;
  const int grid = (int)((warps + kWarpsPerCta - 1) / kWarpsPerCta);
  const int n_out = M + 3 * k;
  cudaError_t e = prefer_max_shared<upsample_kernel<T, true>>();
  if (e == cudaSuccess) e = prefer_max_shared<upsample_kernel<T, false>>();
  if (e != cudaSuccess) return e;
  auto kern = (mode == AVITS_UP_BILINEAR) ? upsample_kernel<T, true> : upsample_kernel<T, false>;
  e = launch_pdl(kern, dim3(grid), dim3(kWarpsPerCta * 32), 0, s,
                             static_cast<const T*>(latent), B, M, gh, gw, C, pos_in, span_in, mask,
                             tok_offset, n_out, static_cast<T*>(out), out_pos, out_span,
                             out_src_tok, out_src_sub);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_upsample(const void* latent, avits_dtype dt, int B, int M, int gh, int gw,
                            int C, const int32_t* pos_in, const int32_t* span_in,
                            const uint8_t* mask, const int32_t* tok_offset, int k,
                            avits_upmode mode, void* out, int32_t* out_pos, int32_t* out_span,
                            int32_t* out_src_tok, int8_t* out_src_sub, cudaStream_t s) {
  if (dt == AVITS_BF16)
    return launch_t<__nv_bfloat16>(latent, B, M, gh, gw, C, pos_in, span_in, mask, tok_offset, k,
                                   mode, out, out_pos, out_span, out_src_tok, out_src_sub, s);
  return launch_t<float>(latent, B, M, gh, gw, C, pos_in, span_in, mask, tok_offset, k, mode, out,
                         out_pos, out_span, out_src_tok, out_src_sub, s);
}

}  // namespace avits
