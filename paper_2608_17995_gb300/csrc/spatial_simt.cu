// spatial_simt.cu — spatial importance (Sec. 3.3.1, Eq. 3 with Eq. 4-5) on
// the CUDA cores, for fp32 inputs (which tensor cores cannot take at the fp32
// score tolerance) and for head widths the tensor-core kernel does not tile.
//
// One warp per image query (b, i), looping over the heads in order so that
// the head mean of Eq. 3 is a fixed-order sum.  Per head, the query row sits
// in shared memory; lanes stride over the keys, each keeping a running
// (max, sum over all keys, sum over text keys) in the log2 domain; the lanes
// are merged with shuffles.  text mass = sum_txt / sum_all.  The text keys
// are the first L, or those a caller's key mask marks (interleaved text and
// image keys).
#include "avits_common.cuh"
#include "avits_internal.h"

namespace avits {
namespace {

constexpr int kWarpsPerCta = 8;
constexpr int kMaxD = 256;

__device__ __forceinline__ float fast_ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

template <typename T>
__global__ void __launch_bounds__(kWarpsPerCta * 32)
spatial_simt_kernel(const T* __restrict__ q, const T* __restrict__ k, int B, int H, int M, int Nk,
                    int L, int d, int64_t q_sb, int64_t q_sh, int64_t q_sn, int64_t k_sb,
                    int64_t k_sh, int64_t k_sn, float c_log2, float weight, int accumulate,
                    float* __restrict__ A, float* __restrict__ lse,
                    const uint8_t* __restrict__ tmask) {
  __shared__ float qs[kWarpsPerCta][kMaxD];
  const int lane = threadIdx.x & 31, wl = threadIdx.x >> 5;
  const int64_t row = (int64_t)blockIdx.x * kWarpsPerCta + wl;
  if (row >= (int64_t)B * M) return;
  const int b = (int)(row / M), i = (int)(row % M);
  const float ln2 = 0.69314718055994530942f;
  float head_sum = 0.f;
  for (int h = 0; h < H; ++h) {
    const T* qr = q + (int64_t)b * q_sb + (int64_t)h * q_sh + (int64_t)i * q_sn;
    for (int c = lane; c < d; c += 32) qs[wl][c] = load_elem(qr, c);
    __syncwarp();
    float m = -INFINITY, la = 0.f, lt = 0.f;
    const T* kb = k + (int64_t)b * k_sb + (int64_t)h * k_sh;
    for (int j = lane; j < Nk; j += 32) {
      const T* kr = kb + (int64_t)j * k_sn;
      float dot = 0.f;
      for (int c = 0; c < d; ++c) dot = fmaf(qs[wl][c], load_elem(kr, c), dot);
      const float x = dot * c_log2;
      if (x > m) {
        const float corr = fast_ex2(m - x);
        la *= corr;
        lt *= corr;
        m = x;
      }
      const float e = fast_ex2(x - m);
      la += e;
      if (tmask ? tmask[(int64_t)b * Nk + j] != 0 : j < L) lt += e;
    }
    // merge the lanes
    float mw = m;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) mw = fmaxf(mw, __shfl_xor_sync(0xffffffffu, mw, o));
    const float f = (m == -INFINITY) ? 0.f : fast_ex2(m - mw);
    la *= f;
    lt *= f;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      la += __shfl_xor_sync(0xffffffffu, la, o);
      lt += __shfl_xor_sync(0xffffffffu, lt, o);
    }
    const float mass = lt / la;
    head_sum += mass;
    if (lse && lane == 0) {
      float* lp = lse + ((((int64_t)b * H + h) * M) + i) * 2;
      lp[0] = (mw + __log2f(la)) * ln2;
      lp[1] = lt > 0.f ? (mw + __log2f(lt)) * ln2 : -INFINITY;
    }
    __syncwarp();
  }
  if (lane == 0) {
    const float a = weight * (head_sum / (float)H);
    A[row] = accumulate ? A[row] + a : a;
  }
}

}  // namespace

cudaError_t launch_spatial_simt(const SpatialArgs& a, cudaStream_t s) {
  const int64_t rows = (int64_t)a.B * a.M;
  const int grid = (int)((rows + kWarpsPerCta - 1) / kWarpsPerCta);
  const float c_log2 = a.scale * 1.4426950408889634f;
  if (a.dt == AVITS_BF16)
    spatial_simt_kernel<__nv_bfloat16><<<grid, kWarpsPerCta * 32, 0, s>>>(
        static_cast<const __nv_bfloat16*>(a.q), static_cast<const __nv_bfloat16*>(a.k), a.B, a.H,
        a.M, a.Nk, a.L, a.d, a.q_sb, a.q_sh, a.q_sn, a.k_sb, a.k_sh, a.k_sn, c_log2, a.weight,
        a.accumulate, a.A, a.lse, a.tmask);
  else
    spatial_simt_kernel<float><<<grid, kWarpsPerCta * 32, 0, s>>>(
        static_cast<const float*>(a.q), static_cast<const float*>(a.k), a.B, a.H, a.M, a.Nk, a.L,
        a.d, a.q_sb, a.q_sh, a.q_sn, a.k_sb, a.k_sh, a.k_sn, c_log2, a.weight, a.accumulate, a.A,
        a.lse, a.tmask);
  return cudaGetLastError();
}

}  // namespace avits
