// spatial_simt.cu — spatial importance (Sec. 3.3.1, Eq. 3 with Eq. 4-5) on
// the CUDA cores, for fp32 inputs (which tensor cores cannot take at the fp32
// score tolerance) and for head widths the tensor-core kernel does not tile.
//
// A CTA takes `rows` (8, 4 or 2) consecutive image queries of one batch
// element, 8 / rows warps per query, and loops over the heads in order so
// that the head mean of Eq. 3 is a fixed-order sum.  Per head the query rows sit in shared memory and the
// keys come through shared memory in chunks of up to 96 KB, loaded by the
// whole CTA with coalesced 16-byte loads (one copy serves all 8 queries;
// each key row padded so that the lanes, which read 32 different keys at the
// same column, do not collide on a bank).  Lane l of a query's warp w takes
// keys 32w + l, 32(w + P) + l, ... of each chunk (P warps per query),
// keeping a running (max, sum over all keys, sum over text keys) in the log2
// domain; the lanes are merged with shuffles, the warps of a query in order
// through shared memory.  text mass
// = sum_txt / sum_all.  The text keys are the first L, or those a caller's
// key mask marks (interleaved text and image keys).
#include "avits_common.cuh"
#include "avits_internal.h"

namespace avits {
namespace {

constexpr int kWarpsPerCta = 8;
constexpr int kMaxD = 256;
constexpr int kChunkFloats = 24576;  // key chunk: at most 96 KB of padded rows

__device__ __forceinline__ float fast_ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Row stride (floats) of a key in shared memory: d + 4 when d is a multiple
// of 4 (16-byte aligned rows, read as float4; eight lanes' rows fall on eight
// different 16-byte bank groups), else d + 1 (32 lanes' rows, 32 banks).
__host__ __device__ __forceinline__ int key_stride(int d) { return (d % 4 == 0) ? d + 4 : d + 1; }

// Keys per chunk for head width d <= 256: a multiple of 32 (64 to 1024) whose
// padded rows fit in 96 KB (with the query rows, two CTAs per SM).
__host__ __device__ __forceinline__ int chunk_keys(int d) {
  return min(1024, (kChunkFloats / key_stride(d)) & ~31);
}

// One chunk of nk key rows (d values each, row stride k_sn elements) into
// ks[r * key_stride(d) + c] as fp32.  kVec: 16-byte loads (4 fp32 / 8 bf16 values;
// d, the strides and the base are multiples of them, checked on the host),
// eight per thread in flight; otherwise one element per load.
template <typename T, bool kVec>
__device__ __forceinline__ void load_chunk(const T* kb, int64_t k_sn, int nk, int d, float* ks) {
  const int ld = key_stride(d);
  if constexpr (kVec) {
    constexpr int V = 16 / (int)sizeof(T);
    const int dv = d / V, total = nk * dv;
    for (int v0 = threadIdx.x; v0 < total; v0 += 8 * kWarpsPerCta * 32) {
      uint4 w[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const int v = v0 + u * kWarpsPerCta * 32;
        w[u] = make_uint4(0u, 0u, 0u, 0u);
        if (v < total) {
          const int r = v / dv, cv = v - r * dv;
          w[u] = *reinterpret_cast<const uint4*>(kb + (int64_t)r * k_sn + cv * V);
        }
      }
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const int v = v0 + u * kWarpsPerCta * 32;
        if (v < total) {
          const int r = v / dv, cv = v - r * dv;
          float* dst = ks + r * ld + cv * V;
          if constexpr (sizeof(T) == 4) {
            dst[0] = __uint_as_float(w[u].x);
            dst[1] = __uint_as_float(w[u].y);
            dst[2] = __uint_as_float(w[u].z);
            dst[3] = __uint_as_float(w[u].w);
          } else {
            const uint32_t ww[4] = {w[u].x, w[u].y, w[u].z, w[u].w};
#pragma unroll
            for (int t = 0; t < 4; ++t) {
              dst[2 * t] = bf16_lo(ww[t]);
              dst[2 * t + 1] = bf16_hi(ww[t]);
            }
          }
        }
      }
    }
  } else {
    for (int e = threadIdx.x; e < nk * d; e += kWarpsPerCta * 32) {
      const int r = e / d, c = e - r * d;
      ks[r * ld + c] = load_elem(kb + (int64_t)r * k_sn, c);
    }
  }
}

template <typename T, bool kVec>
__global__ void __launch_bounds__(kWarpsPerCta * 32)
spatial_simt_kernel(const T* __restrict__ q, const T* __restrict__ k, int B, int H, int M, int Nk,
                    int L, int d, int64_t q_sb, int64_t q_sh, int64_t q_sn, int64_t k_sb,
                    int64_t k_sh, int64_t k_sn, float c_log2, float weight, int accumulate,
                    float* __restrict__ A, float* __restrict__ lse,
                    const uint8_t* __restrict__ tmask, int rows) {
  __shared__ __align__(16) float qs[kWarpsPerCta][kMaxD];
  __shared__ float part[kWarpsPerCta][3];
  extern __shared__ float4 ks4[];   // [kc][key_stride(d)] floats
  float* ks = reinterpret_cast<float*>(ks4);
  const int lane = threadIdx.x & 31, wl = threadIdx.x >> 5;
  // `rows` queries per CTA, P = 8 / rows warps per query, each taking every
  // P-th group of 32 keys of a chunk
  const int P = kWarpsPerCta / rows;
  const int r = wl / P, pw = wl - r * P;
  const int tiles = (M + rows - 1) / rows;
  const int b = (int)(blockIdx.x / tiles);
  const int i = (int)(blockIdx.x % tiles) * rows + r;
  const bool active = i < M;   // every warp takes part in the chunk loads
  const int kc = chunk_keys(d), ld = key_stride(d);
  const float ln2 = 0.69314718055994530942f;
  float head_sum = 0.f;
  for (int h = 0; h < H; ++h) {
    if (active && pw == 0) {
      const T* qr = q + (int64_t)b * q_sb + (int64_t)h * q_sh + (int64_t)i * q_sn;
      for (int c = lane; c < d; c += 32) qs[r][c] = load_elem(qr, c);
    }
    float m = -INFINITY, la = 0.f, lt = 0.f;
    const T* kb = k + (int64_t)b * k_sb + (int64_t)h * k_sh;
    for (int j0 = 0; j0 < Nk; j0 += kc) {
      const int nk = min(kc, Nk - j0);
      __syncthreads();   // the previous chunk has been read (and qs written)
      load_chunk<T, kVec>(kb + (int64_t)j0 * k_sn, k_sn, nk, d, ks);
      __syncthreads();
      if (active) {
        for (int jj = pw * 32 + lane; jj < nk; jj += 32 * P) {
          const float* kr = ks + jj * ld;
          // four partial sums (columns c mod 4) break the FMA chain
          float d0 = 0.f, d1 = 0.f, d2 = 0.f, d3 = 0.f;
          if (d % 4 == 0) {   // 16-byte shared loads (the query row is broadcast)
            const float4* q4 = reinterpret_cast<const float4*>(qs[r]);
            const float4* k4 = reinterpret_cast<const float4*>(kr);
#pragma unroll 4
            for (int c4 = 0; c4 < d / 4; ++c4) {
              const float4 a = q4[c4], kk = k4[c4];
              d0 = fmaf(a.x, kk.x, d0);
              d1 = fmaf(a.y, kk.y, d1);
              d2 = fmaf(a.z, kk.z, d2);
              d3 = fmaf(a.w, kk.w, d3);
            }
          } else {
            int c = 0;
            for (; c + 3 < d; c += 4) {
              d0 = fmaf(qs[r][c], kr[c], d0);
              d1 = fmaf(qs[r][c + 1], kr[c + 1], d1);
              d2 = fmaf(qs[r][c + 2], kr[c + 2], d2);
              d3 = fmaf(qs[r][c + 3], kr[c + 3], d3);
            }
            for (; c < d; ++c) d0 = fmaf(qs[r][c], kr[c], d0);
          }
          const float dot = (d0 + d1) + (d2 + d3);
          const int j = j0 + jj;
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
      }
    }
    // merge the lanes, then the P warps of the query in a fixed order
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
    if (lane == 0) {
      part[wl][0] = mw;
      part[wl][1] = la;
      part[wl][2] = lt;
    }
    __syncthreads();
    if (active && pw == 0) {
      float M_ = part[wl][0], la_ = part[wl][1], lt_ = part[wl][2];
      for (int o = 1; o < P; ++o) {
        const float m2 = part[wl + o][0];
        const float mx = fmaxf(M_, m2);
        if (mx != -INFINITY) {
          const float f1 = fast_ex2(M_ - mx), f2 = fast_ex2(m2 - mx);
          la_ = la_ * f1 + part[wl + o][1] * f2;
          lt_ = lt_ * f1 + part[wl + o][2] * f2;
          M_ = mx;
        }
      }
      head_sum += lt_ / la_;
      if (lse && lane == 0) {
        float* lp = lse + ((((int64_t)b * H + h) * M) + i) * 2;
        lp[0] = (M_ + __log2f(la_)) * ln2;
        lp[1] = lt_ > 0.f ? (M_ + __log2f(lt_)) * ln2 : -INFINITY;
      }
    }
    // qs and part are rewritten for the next head (the chunk loop's first
    // barrier orders the next qs write after this head's last reads)
  }
  if (active && pw == 0 && lane == 0) {
    const int64_t row = (int64_t)b * M + i;
    const float a = weight * (head_sum / (float)H);
    A[row] = accumulate ? A[row] + a : a;
  }
}

template <auto Kernel>
cudaError_t opt_in(size_t smem) {
  return cudaFuncSetAttribute(Kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
}

// The shared-memory opt-in of every instance, once per device (first call,
// outside any stream capture in practice).
cudaError_t simt_smem_once() {
  static int done[64] = {};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev >= 0 && dev < 64 && __atomic_load_n(&done[dev], __ATOMIC_ACQUIRE)) return cudaSuccess;
  const size_t smem = (size_t)kChunkFloats * sizeof(float);
  e = opt_in<spatial_simt_kernel<float, false>>(smem);
  if (e == cudaSuccess) e = opt_in<spatial_simt_kernel<float, true>>(smem);
  if (e == cudaSuccess) e = opt_in<spatial_simt_kernel<__nv_bfloat16, false>>(smem);
  if (e == cudaSuccess) e = opt_in<spatial_simt_kernel<__nv_bfloat16, true>>(smem);
  if (e == cudaSuccess && dev >= 0 && dev < 64) __atomic_store_n(&done[dev], 1, __ATOMIC_RELEASE);
  return e;
}

template <typename T>
cudaError_t launch_typed(const SpatialArgs& a, unsigned grid, int rows, size_t smem, float c_log2,
                         cudaStream_t s) {
  // 16-byte key loads: d, the key strides and the base multiples of a vector
  const int64_t V = 16 / (int64_t)sizeof(T);
  const bool vec = (reinterpret_cast<uintptr_t>(a.k) & 15u) == 0 && a.d % V == 0 &&
                   a.k_sn % V == 0 && (a.H == 1 || a.k_sh % V == 0) &&
                   (a.B == 1 || a.k_sb % V == 0);
  const T* q = static_cast<const T*>(a.q);
  const T* k = static_cast<const T*>(a.k);
  if (vec)
    spatial_simt_kernel<T, true><<<grid, kWarpsPerCta * 32, smem, s>>>(
        q, k, a.B, a.H, a.M, a.Nk, a.L, a.d, a.q_sb, a.q_sh, a.q_sn, a.k_sb, a.k_sh, a.k_sn, c_log2,
        a.weight, a.accumulate, a.A, a.lse, a.tmask, rows);
  else
    spatial_simt_kernel<T, false><<<grid, kWarpsPerCta * 32, smem, s>>>(
        q, k, a.B, a.H, a.M, a.Nk, a.L, a.d, a.q_sb, a.q_sh, a.q_sn, a.k_sb, a.k_sh, a.k_sn, c_log2,
        a.weight, a.accumulate, a.A, a.lse, a.tmask, rows);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_spatial_simt(const SpatialArgs& a, int num_sms, cudaStream_t s) {
  // queries per CTA: 8 (one warp each) when that gives two CTAs per SM;
  // fewer, with the key groups of a query split over 8 / rows warps, when the
  // batch has few queries (every CTA reads the whole key panel once per head)
  const int64_t queries = (int64_t)a.B * a.M;
  int rows = kWarpsPerCta;
  while (rows > 2 && queries / rows < 2 * (int64_t)num_sms) rows >>= 1;
  const int tiles = (a.M + rows - 1) / rows;
  const int64_t grid = (int64_t)a.B * tiles;
  if (grid > 0x7fffffff) return cudaErrorInvalidValue;
  cudaError_t e = simt_smem_once();
  if (e != cudaSuccess) return e;
  const size_t smem = (size_t)chunk_keys(a.d) * key_stride(a.d) * sizeof(float);
  const float c_log2 = a.scale * 1.4426950408889634f;
  return a.dt == AVITS_BF16
             ? launch_typed<__nv_bfloat16>(a, (unsigned)grid, rows, smem, c_log2, s)
             : launch_typed<float>(a, (unsigned)grid, rows, smem, c_log2, s);
}

}  // namespace avits
