// temporal.cu — temporal importance (Sec. 3.3.2).
//
// avits_score_temporal: V = ||h_t - h_prev|| / (||h_prev|| + eps) per token.
// HBM-bound: each token row (D values of each snapshot) is read once with
// 16-byte vector loads, a warp per token, all of a lane's loads issued before
// any arithmetic so that each warp keeps ~24 x 16 B in flight; fp32 sums,
// shuffle reduction.  Algorithmic bytes: 2 * B*N*D*elt + 4*B*N.
//
// avits_score_temporal_var: Eq. 6-7, unbiased variance over N_T snapshots
// averaged over channels; two passes over the snapshot values held in
// registers (mean, then squared deviations).
#include "avits_common.cuh"
#include "avits_internal.h"

namespace avits {
namespace {

constexpr int kWarpsPerCta = 8;

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// bf16, D % 8 == 0: chunks of 8 values.
template <int kUnroll>
__global__ void __launch_bounds__(kWarpsPerCta * 32)
temporal_bf16_kernel(const uint4* __restrict__ ht, const uint4* __restrict__ hp, int64_t ntok,
                     int chunks, float eps, float* __restrict__ V) {
  const int lane = threadIdx.x & 31;
  const int64_t warp = (int64_t)blockIdx.x * kWarpsPerCta + (threadIdx.x >> 5);
  const int64_t nwarps = (int64_t)gridDim.x * kWarpsPerCta;
  for (int64_t t = warp; t < ntok; t += nwarps) {
    const uint4* a = ht + t * chunks;
    const uint4* p = hp + t * chunks;
    float dd = 0.f, pp = 0.f;
    for (int c0 = 0; c0 < chunks; c0 += 32 * kUnroll) {
      uint4 ra[kUnroll], rp[kUnroll];
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        const int c = c0 + u * 32 + lane;
        if (c < chunks) {
          ra[u] = __ldcs(a + c);
          rp[u] = __ldcs(p + c);
        } else {
          ra[u] = make_uint4(0, 0, 0, 0);
          rp[u] = make_uint4(0, 0, 0, 0);
        }
      }
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        const uint32_t wa[4] = {ra[u].x, ra[u].y, ra[u].z, ra[u].w};
        const uint32_t wp[4] = {rp[u].x, rp[u].y, rp[u].z, rp[u].w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float a0 = bf16_lo(wa[e]), a1 = bf16_hi(wa[e]);
          const float p0 = bf16_lo(wp[e]), p1 = bf16_hi(wp[e]);
          const float d0 = a0 - p0, d1 = a1 - p1;
          dd = fmaf(d0, d0, dd);
          dd = fmaf(d1, d1, dd);
          pp = fmaf(p0, p0, pp);
          pp = fmaf(p1, p1, pp);
        }
      }
    }
    dd = warp_sum(dd);
    pp = warp_sum(pp);
    if (lane == 0) V[t] = sqrtf(dd) / (sqrtf(pp) + eps);
  }
}

// fp32, D % 4 == 0: chunks of 4 values.
template <int kUnroll>
__global__ void __launch_bounds__(kWarpsPerCta * 32)
temporal_f32_kernel(const float4* __restrict__ ht, const float4* __restrict__ hp, int64_t ntok,
                    int chunks, float eps, float* __restrict__ V) {
  const int lane = threadIdx.x & 31;
  const int64_t warp = (int64_t)blockIdx.x * kWarpsPerCta + (threadIdx.x >> 5);
  const int64_t nwarps = (int64_t)gridDim.x * kWarpsPerCta;
  for (int64_t t = warp; t < ntok; t += nwarps) {
    const float4* a = ht + t * chunks;
    const float4* p = hp + t * chunks;
    float dd = 0.f, pp = 0.f;
    for (int c0 = 0; c0 < chunks; c0 += 32 * kUnroll) {
      float4 ra[kUnroll], rp[kUnroll];
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        const int c = c0 + u * 32 + lane;
        ra[u] = c < chunks ? __ldcs(a + c) : make_float4(0.f, 0.f, 0.f, 0.f);
        rp[u] = c < chunks ? __ldcs(p + c) : make_float4(0.f, 0.f, 0.f, 0.f);
      }
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        const float av[4] = {ra[u].x, ra[u].y, ra[u].z, ra[u].w};
        const float pv[4] = {rp[u].x, rp[u].y, rp[u].z, rp[u].w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float d0 = av[e] - pv[e];
          dd = fmaf(d0, d0, dd);
          pp = fmaf(pv[e], pv[e], pp);
        }
      }
    }
    dd = warp_sum(dd);
    pp = warp_sum(pp);
    if (lane == 0) V[t] = sqrtf(dd) / (sqrtf(pp) + eps);
  }
}

// Any D, any dtype (scalar loads).
template <typename T>
__global__ void __launch_bounds__(kWarpsPerCta * 32)
temporal_scalar_kernel(const T* __restrict__ ht, const T* __restrict__ hp, int64_t ntok, int D,
                       float eps, float* __restrict__ V) {
  const int lane = threadIdx.x & 31;
  const int64_t warp = (int64_t)blockIdx.x * kWarpsPerCta + (threadIdx.x >> 5);
  const int64_t nwarps = (int64_t)gridDim.x * kWarpsPerCta;
  for (int64_t t = warp; t < ntok; t += nwarps) {
    float dd = 0.f, pp = 0.f;
    for (int c = lane; c < D; c += 32) {
      const float a = load_elem(ht, t * D + c), p = load_elem(hp, t * D + c);
      dd = fmaf(a - p, a - p, dd);
      pp = fmaf(p, p, pp);
    }
    dd = warp_sum(dd);
    pp = warp_sum(pp);
    if (lane == 0) V[t] = sqrtf(dd) / (sqrtf(pp) + eps);
  }
}

struct SnapPtrs {
  const void* p[kMaxSnapshots];
};

// Eq. 6-7: per channel mean over snapshots (Eq. 6), unbiased variance, then
// the channel mean (Eq. 7).
template <typename T>
__global__ void __launch_bounds__(kWarpsPerCta * 32)
temporal_var_kernel(SnapPtrs snaps, int n_t, int64_t ntok, int D, float* __restrict__ V) {
  const int lane = threadIdx.x & 31;
  const int64_t warp = (int64_t)blockIdx.x * kWarpsPerCta + (threadIdx.x >> 5);
  const int64_t nwarps = (int64_t)gridDim.x * kWarpsPerCta;
  const float inv_n = 1.0f / (float)n_t;
  const float inv_n1 = 1.0f / (float)(n_t - 1);
  for (int64_t t = warp; t < ntok; t += nwarps) {
    float acc = 0.f;
    for (int c = lane; c < D; c += 32) {
      float z[kMaxSnapshots];
      float mean = 0.f;
#pragma unroll
      for (int s = 0; s < kMaxSnapshots; ++s) {
        if (s < n_t) {
          z[s] = load_elem(static_cast<const T*>(snaps.p[s]), t * D + c);
          mean += z[s];
        }
      }
      mean *= inv_n;
      float ss = 0.f;
#pragma unroll
      for (int s = 0; s < kMaxSnapshots; ++s) {
        if (s < n_t) {
          const float dv = z[s] - mean;
          ss = fmaf(dv, dv, ss);
        }
      }
      acc += ss * inv_n1;
    }
    acc = warp_sum(acc);
    if (lane == 0) V[t] = acc / (float)D;
  }
}

int grid_for(int64_t ntok, int num_sms) {
  const int64_t want = (ntok + kWarpsPerCta - 1) / kWarpsPerCta;
  const int64_t cap = (int64_t)num_sms * 16;
  return (int)(want < cap ? (want > 0 ? want : 1) : cap);
}

}  // namespace

cudaError_t launch_temporal(const void* ht, const void* hp, avits_dtype dt, int B, int N, int D,
                            float eps, float* V, int num_sms, cudaStream_t s) {
  const int64_t ntok = (int64_t)B * N;
  const int grid = grid_for(ntok, num_sms);
  const bool al = ((reinterpret_cast<uintptr_t>(ht) | reinterpret_cast<uintptr_t>(hp)) & 15u) == 0;
  if (dt == AVITS_BF16) {
    if (al && D % 8 == 0) {
      const int chunks = D / 8;
      if (chunks >= 256)
        temporal_bf16_kernel<12><<<grid, kWarpsPerCta * 32, 0, s>>>(
            static_cast<const uint4*>(ht), static_cast<const uint4*>(hp), ntok, chunks, eps, V);
      else
        temporal_bf16_kernel<2><<<grid, kWarpsPerCta * 32, 0, s>>>(
            static_cast<const uint4*>(ht), static_cast<const uint4*>(hp), ntok, chunks, eps, V);
    } else {
      temporal_scalar_kernel<__nv_bfloat16><<<grid, kWarpsPerCta * 32, 0, s>>>(
          static_cast<const __nv_bfloat16*>(ht), static_cast<const __nv_bfloat16*>(hp), ntok, D,
          eps, V);
    }
  } else {
    if (al && D % 4 == 0) {
      const int chunks = D / 4;
      if (chunks >= 256)
        temporal_f32_kernel<8><<<grid, kWarpsPerCta * 32, 0, s>>>(
            static_cast<const float4*>(ht), static_cast<const float4*>(hp), ntok, chunks, eps, V);
      else
        temporal_f32_kernel<1><<<grid, kWarpsPerCta * 32, 0, s>>>(
            static_cast<const float4*>(ht), static_cast<const float4*>(hp), ntok, chunks, eps, V);
    } else {
      temporal_scalar_kernel<float><<<grid, kWarpsPerCta * 32, 0, s>>>(
          static_cast<const float*>(ht), static_cast<const float*>(hp), ntok, D, eps, V);
    }
  }
  return cudaGetLastError();
}

cudaError_t launch_temporal_var(const void* const* snaps, int n_t, avits_dtype dt, int B, int N,
                                int D, float* V, int num_sms, cudaStream_t s) {
  SnapPtrs sp{};
  for (int i = 0; i < n_t; ++i) sp.p[i] = snaps[i];
  const int64_t ntok = (int64_t)B * N;
  const int grid = grid_for(ntok, num_sms);
  if (dt == AVITS_BF16)
    temporal_var_kernel<__nv_bfloat16><<<grid, kWarpsPerCta * 32, 0, s>>>(sp, n_t, ntok, D, V);
  else
    temporal_var_kernel<float><<<grid, kWarpsPerCta * 32, 0, s>>>(sp, n_t, ntok, D, V);
  return cudaGetLastError();
}

}  // namespace avits
