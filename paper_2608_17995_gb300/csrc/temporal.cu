// temporal.cu — temporal importance (Sec. 3.3.2).
//
// avits_score_temporal: V = ||h_t - h_prev|| / (||h_prev|| + eps) per token.
// HBM-bound.  Main path: each CTA stages up to 8 token rows of both
// snapshots in shared memory with bulk copies (cp.async.bulk, one per row,
// completing on one mbarrier), so a whole chunk is in flight with a single
// issuing thread; then one warp per token reduces its two rows from shared
// memory (fp32 sums, shuffle reduction).  Chunks are small (2 tokens) and
// many CTAs fit on an SM, so all of the input is in flight at once and the
// kernel can share SMs with the spatial kernel.  Rows that are not 16-byte
// multiples use a register path.  Algorithmic bytes: 2 * B*N*D*elt + 4*B*N.
//
// avits_score_temporal_var: Eq. 6-7, unbiased variance over N_T snapshots
// averaged over channels; two passes over the snapshot values held in
// registers (mean, then squared deviations).  Main path: one CTA per token,
// 16-byte loads, the N_T vectors of a position all issued before they are
// reduced (HBM-bound: N_T * D * elt bytes per token).
#include "avits_common.cuh"
#include "avits_internal.h"

#include <algorithm>

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

// ------------------------------------------------ bulk-copy staged path --
// 2 tokens (24 KB at D = 3072 bf16) per CTA-chunk: small enough to share an
// SM with the spatial kernel's CTA, so the two can run concurrently.
constexpr int kStageTokens = 2;
constexpr int kStageBytesMax = 32 * 1024;

__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
          smem_u32(dst)),
      "l"(src), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
}

// kOverlapped: launched as a programmatic dependent of a running kernel (the
// spatial score); lets its own dependents be scheduled, and waits for the
// running kernel to finish before exiting so that a dependent of this grid
// also sees that kernel's results.
template <typename T, bool kOverlapped>
__global__ void __launch_bounds__(kWarpsPerCta * 32)
temporal_staged_kernel(const T* __restrict__ ht, const T* __restrict__ hp, int64_t ntok, int D,
                       int tpc, float eps, float* __restrict__ V, unsigned int* status) {
  if (kOverlapped) {
    // beside a running kernel: its inputs were complete before that kernel
    // started; let the dependents of this grid be scheduled
    if (threadIdx.x == 0) asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  } else {
    pdl_wait_then_trigger();
  }
  extern __shared__ __align__(128) uint8_t sm[];
  __shared__ __align__(8) uint64_t bar;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const uint32_t row_bytes = (uint32_t)D * sizeof(T);
  T* s_t = reinterpret_cast<T*>(sm);
  T* s_p = reinterpret_cast<T*>(sm + (size_t)tpc * row_bytes);
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();
  const int64_t nchunks = (ntok + tpc - 1) / tpc;
  uint32_t phase = 0;
  for (int64_t c = blockIdx.x; c < nchunks; c += gridDim.x, phase ^= 1u) {
    const int64_t t0 = c * tpc;
    const int64_t left = ntok - t0;
    const int n = left < (int64_t)tpc ? (int)left : tpc;
    if (threadIdx.x == 0) {
      mbar_arrive_expect_tx(&bar, 2u * (uint32_t)n * row_bytes);
      for (int i = 0; i < n; ++i) {
        bulk_g2s(sm + (size_t)i * row_bytes, ht + (t0 + i) * D, row_bytes, &bar);
        bulk_g2s(sm + (size_t)(tpc + i) * row_bytes, hp + (t0 + i) * D, row_bytes, &bar);
      }
    }
    // every thread waits for the chunk (bounded); a timeout skips the chunk
    const bool ok = mbar_wait_bounded(&bar, phase, nullptr, status);
    if (ok) {
      for (int i = warp; i < n; i += kWarpsPerCta) {
        const T* a = s_t + (size_t)i * D;
        const T* p = s_p + (size_t)i * D;
        float dd = 0.f, pp = 0.f;
        if (sizeof(T) == 2) {
          const uint4* a4 = reinterpret_cast<const uint4*>(a);
          const uint4* p4 = reinterpret_cast<const uint4*>(p);
          for (int k = lane; k < (int)(row_bytes / 16); k += 32) {
            const uint4 ra = a4[k], rp = p4[k];
            const uint32_t wa[4] = {ra.x, ra.y, ra.z, ra.w};
            const uint32_t wp[4] = {rp.x, rp.y, rp.z, rp.w};
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              const float d0 = bf16_lo(wa[e]) - bf16_lo(wp[e]), d1 = bf16_hi(wa[e]) - bf16_hi(wp[e]);
              dd = fmaf(d0, d0, fmaf(d1, d1, dd));
              pp = fmaf(bf16_lo(wp[e]), bf16_lo(wp[e]), fmaf(bf16_hi(wp[e]), bf16_hi(wp[e]), pp));
            }
          }
        } else {
          const float4* a4 = reinterpret_cast<const float4*>(a);
          const float4* p4 = reinterpret_cast<const float4*>(p);
          for (int k = lane; k < (int)(row_bytes / 16); k += 32) {
            const float4 ra = a4[k], rp = p4[k];
            const float av[4] = {ra.x, ra.y, ra.z, ra.w}, pv[4] = {rp.x, rp.y, rp.z, rp.w};
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
        if (lane == 0) V[t0 + i] = sqrtf(dd) / (sqrtf(pp) + eps);
      }
    }
    // the buffer is reused by the next chunk.  After a timeout anywhere in
    // the CTA no further chunk is issued: thread 0 waits once more (bounded)
    // for the copies already armed on the barrier, so that none lands in
    // shared memory after the CTA has exited, and the CTA stops.
    if (!__syncthreads_and(ok)) {
      if (threadIdx.x == 0) mbar_wait_bounded(&bar, phase, nullptr, status);
      __syncthreads();
      break;
    }
  }
  if (kOverlapped) asm volatile("griddepcontrol.wait;" ::: "memory");
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


// Element e of a 16-byte vector, as fp32.
template <typename T>
__device__ __forceinline__ float vec_elem(const uint4& v, int e);
template <>
__device__ __forceinline__ float vec_elem<float>(const uint4& v, int e) {
  const uint32_t w = e == 0 ? v.x : e == 1 ? v.y : e == 2 ? v.z : v.w;
  return __uint_as_float(w);
}
template <>
__device__ __forceinline__ float vec_elem<__nv_bfloat16>(const uint4& v, int e) {
  const int q = e >> 1;
  const uint32_t w = q == 0 ? v.x : q == 1 ? v.y : q == 2 ? v.z : v.w;
  return (e & 1) ? bf16_hi(w) : bf16_lo(w);
}

// 16-byte vectors of kE elements; kNT >= n_t snapshots kept in registers.
constexpr int kVarThreads = 128;

template <typename T, int kNT>
__global__ void __launch_bounds__(kVarThreads)
temporal_var_vec_kernel(SnapPtrs snaps, int n_t, int64_t ntok, int D, float* __restrict__ V) {
  constexpr int kE = 16 / (int)sizeof(T);
  __shared__ float part[kVarThreads / 32];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int nv = D / kE;
  const float inv_n = 1.0f / (float)n_t;
  const float inv_n1 = 1.0f / (float)(n_t - 1);
  for (int64_t t = blockIdx.x; t < ntok; t += gridDim.x) {
    float acc = 0.f;
    for (int v = threadIdx.x; v < nv; v += kVarThreads) {
      uint4 raw[kNT];
#pragma unroll
      for (int s = 0; s < kNT; ++s)
        if (s < n_t)
          raw[s] = __ldcs(reinterpret_cast<const uint4*>(static_cast<const T*>(snaps.p[s]) +
                                                        t * D) + v);
#pragma unroll
      for (int e = 0; e < kE; ++e) {
        float z[kNT];
        float mean = 0.f;
#pragma unroll
        for (int s = 0; s < kNT; ++s) {
          if (s < n_t) {
            z[s] = vec_elem<T>(raw[s], e);
            mean += z[s];
          }
        }
        mean *= inv_n;
        float ss = 0.f;
#pragma unroll
        for (int s = 0; s < kNT; ++s) {
          if (s < n_t) {
            const float dv = z[s] - mean;
            ss = fmaf(dv, dv, ss);
          }
        }
        acc += ss * inv_n1;
      }
    }
    acc = warp_sum(acc);
    if (lane == 0) part[w] = acc;
    __syncthreads();
    if (threadIdx.x == 0) {
      float tot = 0.f;
#pragma unroll
      for (int k = 0; k < kVarThreads / 32; ++k) tot += part[k];
      V[t] = tot / (float)D;
    }
    __syncthreads();   // part[] is reused by the next token
  }
}

}  // namespace

template <typename T, bool kOverlapped = false>
cudaError_t launch_staged(const void* ht, const void* hp, int64_t ntok, int D, float eps, float* V,
                          int num_sms, unsigned int* status, cudaStream_t s) {
  const size_t row = (size_t)D * sizeof(T);
  const int tpc = (int)std::min<size_t>(kStageTokens, kStageBytesMax / (2 * row));
  const size_t smem = 2 * (size_t)tpc * row;
  static int done[64] = {};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (!(dev >= 0 && dev < 64 && __atomic_load_n(&done[dev], __ATOMIC_ACQUIRE))) {
    e = cudaFuncSetAttribute(temporal_staged_kernel<T, false>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize, kStageBytesMax);
    if (e != cudaSuccess) return e;
    e = cudaFuncSetAttribute(temporal_staged_kernel<T, true>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize, kStageBytesMax);
    if (e != cudaSuccess) return e;
    // the same (all shared) carveout as the spatial kernel it runs beside
    e = cudaFuncSetAttribute(temporal_staged_kernel<T, true>,
                             cudaFuncAttributePreferredSharedMemoryCarveout,
                             cudaSharedmemCarveoutMaxShared);
    if (e != cudaSuccess) return e;
    if (dev >= 0 && dev < 64) __atomic_store_n(&done[dev], 1, __ATOMIC_RELEASE);
  }
  const int64_t nchunks = (ntok + tpc - 1) / tpc;
  e = prefer_max_shared<temporal_staged_kernel<T, false>>();
  if (e != cudaSuccess) return e;
  if (!kOverlapped) {
    const int grid = (int)std::min<int64_t>(nchunks, (int64_t)std::max(num_sms, 1) * 16);
    e = launch_pdl(temporal_staged_kernel<T, false>, dim3(grid), dim3(kWarpsPerCta * 32), smem, s,
                   static_cast<const T*>(ht), static_cast<const T*>(hp), ntok, D, tpc, eps, V,
                   status);
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
  }
  // one CTA per SM (it shares the SM with the running kernel's CTA)
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3((unsigned)std::min<int64_t>(nchunks, (int64_t)std::max(num_sms, 1)));
  cfg.blockDim = dim3(kWarpsPerCta * 32);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  e = cudaLaunchKernelEx(&cfg, temporal_staged_kernel<T, true>, static_cast<const T*>(ht),
                         static_cast<const T*>(hp), ntok, D, tpc, eps, V, status);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

cudaError_t launch_temporal(const void* ht, const void* hp, avits_dtype dt, int B, int N, int D,
                            float eps, float* V, int num_sms, unsigned int* status, cudaStream_t s) {
  const int64_t ntok = (int64_t)B * N;
  const int grid = grid_for(ntok, num_sms);
  const bool al = ((reinterpret_cast<uintptr_t>(ht) | reinterpret_cast<uintptr_t>(hp)) & 15u) == 0;
  const size_t row = (size_t)D * (dt == AVITS_BF16 ? 2 : 4);
  if (al && row % 16 == 0 && 2 * row <= (size_t)kStageBytesMax) {
    return dt == AVITS_BF16
               ? launch_staged<__nv_bfloat16>(ht, hp, ntok, D, eps, V, num_sms, status, s)
               : launch_staged<float>(ht, hp, ntok, D, eps, V, num_sms, status, s);
  }
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

cudaError_t launch_temporal_overlapped(const void* ht, const void* hp, avits_dtype dt, int B,
                                       int N, int D, float eps, float* V, int num_sms,
                                       unsigned int* status, cudaStream_t s) {
  const int64_t ntok = (int64_t)B * N;
  const bool al = ((reinterpret_cast<uintptr_t>(ht) | reinterpret_cast<uintptr_t>(hp)) & 15u) == 0;
  const size_t row = (size_t)D * (dt == AVITS_BF16 ? 2 : 4);
  if (!(al && row % 16 == 0 && 2 * row <= (size_t)kStageBytesMax))
    return launch_temporal(ht, hp, dt, B, N, D, eps, V, num_sms, status, s);   // stream order
  return dt == AVITS_BF16
             ? launch_staged<__nv_bfloat16, true>(ht, hp, ntok, D, eps, V, num_sms, status, s)
             : launch_staged<float, true>(ht, hp, ntok, D, eps, V, num_sms, status, s);
}

cudaError_t launch_temporal_var(const void* const* snaps, int n_t, avits_dtype dt, int B, int N,
                                int D, float* V, int num_sms, cudaStream_t s) {
  SnapPtrs sp{};
  for (int i = 0; i < n_t; ++i) sp.p[i] = snaps[i];
  const int64_t ntok = (int64_t)B * N;
  const int elt = (dt == AVITS_BF16) ? 2 : 4;
  bool vec = ((int64_t)D * elt) % 16 == 0;
  for (int i = 0; i < n_t; ++i) vec = vec && (reinterpret_cast<uintptr_t>(snaps[i]) & 15u) == 0;
  if (vec) {
    // one CTA per token (grid-stride beyond 2^31 - 1 tokens).  A plain
    // launch: as a programmatic dependent its waiting CTAs took SM slots from
    // the kernel before it and measured slower.
    const unsigned grid = (unsigned)std::min<int64_t>(ntok, (int64_t)INT32_MAX);
    if (dt == AVITS_BF16) {
      if (n_t <= 4)
        temporal_var_vec_kernel<__nv_bfloat16, 4><<<grid, kVarThreads, 0, s>>>(sp, n_t, ntok, D, V);
      else if (n_t <= 8)
        temporal_var_vec_kernel<__nv_bfloat16, 8><<<grid, kVarThreads, 0, s>>>(sp, n_t, ntok, D, V);
      else
        temporal_var_vec_kernel<__nv_bfloat16, kMaxSnapshots>
            <<<grid, kVarThreads, 0, s>>>(sp, n_t, ntok, D, V);
    } else {
      if (n_t <= 4)
        temporal_var_vec_kernel<float, 4><<<grid, kVarThreads, 0, s>>>(sp, n_t, ntok, D, V);
      else if (n_t <= 8)
        temporal_var_vec_kernel<float, 8><<<grid, kVarThreads, 0, s>>>(sp, n_t, ntok, D, V);
      else
        temporal_var_vec_kernel<float, kMaxSnapshots><<<grid, kVarThreads, 0, s>>>(sp, n_t, ntok, D, V);
    }
    return cudaGetLastError();
  }
  const int grid = grid_for(ntok, num_sms);
  if (dt == AVITS_BF16)
    temporal_var_kernel<__nv_bfloat16><<<grid, kWarpsPerCta * 32, 0, s>>>(sp, n_t, ntok, D, V);
  else
    temporal_var_kernel<float><<<grid, kWarpsPerCta * 32, 0, s>>>(sp, n_t, ntok, D, V);
  return cudaGetLastError();
}

}  // namespace avits
