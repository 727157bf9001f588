// select.cu — joint score and token selection (Sec. 3.3.3, Eq. 8-9).
//
// One CTA of 1024 threads per batch element; the M scores stay in shared
// memory as order-preserving 32-bit keys.
//   1. min / max of A and V (NaN ignored), block reduction;
//   2. S = (alpha * A^) + ((1 - alpha) * V^) with explicitly rounded fp32
//      operations in that order (no contraction), so that the same A, V give
//      bit-identical S wherever the selection is recomputed;
//   3. the k-th largest key by MSB-first radix select, 4 passes of 8 bits
//      with a 256-bin shared histogram;
//   4. keys above it are selected, and among keys equal to it the lowest
//      indices (a block scan over contiguous per-thread ranges);
//   5. a second block scan yields sel_idx (ascending) and tok_offset.
// Key map: NaN -> 0 (below everything); -0 -> +0; otherwise the IEEE bits
// with the sign bit flipped (positive) or all bits flipped (negative).
#include "avits_common.cuh"
#include "avits_internal.h"

namespace avits {
namespace {

constexpr int kThreads = 1024;
constexpr int kWarps = kThreads / 32;

__device__ __forceinline__ uint32_t order_key(float s) {
  if (s != s) return 0u;
  const float c = (s == 0.0f) ? 0.0f : s;
  const uint32_t u = __float_as_uint(c);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// Exclusive prefix sum over the block (thread order); returns the total.
__device__ __forceinline__ uint32_t block_exclusive_scan(uint32_t v, uint32_t* warp_tot,
                                                         uint32_t* excl) {
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  uint32_t x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) warp_tot[w] = x;
  __syncthreads();
  if (w == 0) {
    uint32_t t = warp_tot[lane];
    uint32_t s = t;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t y = __shfl_up_sync(0xffffffffu, s, o);
      if (lane >= o) s += y;
    }
    warp_tot[lane] = s - t;        // exclusive over warps
    if (lane == 31) warp_tot[32] = s;
  }
  __syncthreads();
  *excl = warp_tot[w] + x - v;
  const uint32_t total = warp_tot[32];
  __syncthreads();
  return total;
}

__global__ void __launch_bounds__(kThreads)
fuse_select_kernel(const float* __restrict__ A, const float* __restrict__ V, int M, float alpha,
                   float eps, int k, float* __restrict__ S_out, int32_t* __restrict__ sel_idx,
                   uint8_t* __restrict__ mask, int32_t* __restrict__ tok_offset,
                   unsigned int* status) {
  extern __shared__ uint32_t keys[];
  __shared__ float red[4][kWarps];
  __shared__ uint32_t hist[256];
  __shared__ uint32_t warp_tot[33];
  __shared__ uint32_t sh_digit, sh_remaining;
  __shared__ int sh_nan;

  const int b = blockIdx.x;
  const int tid = threadIdx.x, lane = tid & 31, w = tid >> 5;
  const float* a = A + (int64_t)b * M;
  const float* v = V + (int64_t)b * M;

  // 1. min / max (fminf / fmaxf skip NaN)
  float amn = __int_as_float(0x7f800000), amx = -amn, vmn = amn, vmx = -amn;
  for (int i = tid; i < M; i += kThreads) {
    const float x = a[i], y = v[i];
    amn = fminf(amn, x); amx = fmaxf(amx, x);
    vmn = fminf(vmn, y); vmx = fmaxf(vmx, y);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    amn = fminf(amn, __shfl_xor_sync(0xffffffffu, amn, o));
    amx = fmaxf(amx, __shfl_xor_sync(0xffffffffu, amx, o));
    vmn = fminf(vmn, __shfl_xor_sync(0xffffffffu, vmn, o));
    vmx = fmaxf(vmx, __shfl_xor_sync(0xffffffffu, vmx, o));
  }
  if (lane == 0) { red[0][w] = amn; red[1][w] = amx; red[2][w] = vmn; red[3][w] = vmx; }
  if (tid == 0) sh_nan = 0;
  __syncthreads();
  amn = red[0][0]; amx = red[1][0]; vmn = red[2][0]; vmx = red[3][0];
  for (int j = 1; j < kWarps; ++j) {
    amn = fminf(amn, red[0][j]); amx = fmaxf(amx, red[1][j]);
    vmn = fminf(vmn, red[2][j]); vmx = fmaxf(vmx, red[3][j]);
  }

  // 2. fused score, fixed rounding order
  const float aden = __fadd_rn(__fsub_rn(amx, amn), eps);
  const float vden = __fadd_rn(__fsub_rn(vmx, vmn), eps);
  const float one_m = __fsub_rn(1.0f, alpha);
  int any_nan = 0;
  for (int i = tid; i < M; i += kThreads) {
    const float an = __fdiv_rn(__fsub_rn(a[i], amn), aden);
    const float vn = __fdiv_rn(__fsub_rn(v[i], vmn), vden);
    const float s = __fadd_rn(__fmul_rn(alpha, an), __fmul_rn(one_m, vn));
    if (S_out) S_out[(int64_t)b * M + i] = s;
    any_nan |= (s != s);
    keys[i] = order_key(s);
  }
  if (any_nan) sh_nan = 1;
  __syncthreads();
  if (tid == 0 && sh_nan) raise_status(status, AVITS_ERR_NAN);

  // 3. radix select of the k-th largest key
  uint32_t prefix = 0u, pmask = 0u;
  uint32_t remaining = (uint32_t)k;
  if (k > 0 && k < M) {
    for (int pass = 0; pass < 4; ++pass) {
      const int shift = 24 - 8 * pass;
      if (tid < 256) hist[tid] = 0u;
      __syncthreads();
      for (int i = tid; i < M; i += kThreads) {
        const uint32_t key = keys[i];
        if ((key & pmask) == prefix) atomicAdd(&hist[(key >> shift) & 255u], 1u);
      }
      __syncthreads();
      if (w == 0) {
        // lane l owns digits 255-8l ... 248-8l (descending order of keys)
        uint32_t cnt[8], tot = 0;
#pragma unroll
        for (int e = 0; e < 8; ++e) { cnt[e] = hist[255 - 8 * lane - e]; tot += cnt[e]; }
        uint32_t inc = tot;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const uint32_t y = __shfl_up_sync(0xffffffffu, inc, o);
          if (lane >= o) inc += y;
        }
        const uint32_t before = inc - tot;     // keys in higher digits
        if (before < remaining && remaining <= inc) {
          uint32_t c = before;
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            if (c < remaining && remaining <= c + cnt[e]) {
              sh_digit = 255u - 8u * lane - e;
              sh_remaining = remaining - c;
            }
            c += cnt[e];
          }
        }
      }
      __syncthreads();
      prefix |= sh_digit << shift;
      pmask |= 255u << shift;
      remaining = sh_remaining;
      __syncthreads();
    }
  }
  const uint32_t T = prefix;

  // 4-5. selection and compaction over contiguous per-thread ranges
  const int per = (M + kThreads - 1) / kThreads;
  const int lo = min(M, tid * per), hi = min(M, lo + per);
  uint32_t gt = 0, eq = 0;
  if (k > 0 && k < M) {
    for (int i = lo; i < hi; ++i) {
      const uint32_t key = keys[i];
      gt += key > T;
      eq += key == T;
    }
  }
  uint32_t eq_before;
  block_exclusive_scan(eq, warp_tot, &eq_before);
  uint32_t nsel;
  if (k == 0) nsel = 0;
  else if (k == M) nsel = (uint32_t)(hi - lo);
  else {
    const uint32_t take = remaining > eq_before ? min(remaining - eq_before, eq) : 0u;
    nsel = gt + take;
  }
  uint32_t sel_before;
  block_exclusive_scan(nsel, warp_tot, &sel_before);
  uint32_t eq_seen = eq_before, c = sel_before;
  for (int i = lo; i < hi; ++i) {
    bool sel;
    if (k == 0) sel = false;
    else if (k == M) sel = true;
    else {
      const uint32_t key = keys[i];
      sel = key > T;
      if (key == T) { sel = eq_seen < remaining; ++eq_seen; }
    }
    tok_offset[(int64_t)b * M + i] = i + 3 * (int)c;
    if (mask) mask[(int64_t)b * M + i] = sel ? 1 : 0;
    if (sel) { sel_idx[(int64_t)b * k + c] = i; ++c; }
  }
}

}  // namespace

cudaError_t launch_fuse_select(const float* A, const float* V, int B, int M, float alpha,
                               float eps, int k, float* S, int32_t* sel_idx, uint8_t* mask,
                               int32_t* tok_offset, unsigned int* status, cudaStream_t s) {
  const size_t smem = (size_t)M * sizeof(uint32_t);
  if (smem > 48 * 1024) {
    // opt in once per device to the largest size any call can ask for
    static int done[64] = {};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (!(dev >= 0 && dev < 64 && __atomic_load_n(&done[dev], __ATOMIC_ACQUIRE))) {
      e = cudaFuncSetAttribute(fuse_select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               (int)(kSelectMaxM * sizeof(uint32_t)));
      if (e != cudaSuccess) return e;
      if (dev >= 0 && dev < 64) __atomic_store_n(&done[dev], 1, __ATOMIC_RELEASE);
    }
  }
  fuse_select_kernel<<<B, kThreads, smem, s>>>(A, V, M, alpha, eps, k, S, sel_idx, mask,
                                               tok_offset, status);
  return cudaGetLastError();
}

}  // namespace avits
