// avits_common.cuh — device helpers shared by the AViTS kernels (sm_103a).
//
// Status word: device-side errors are OR-ed, as bit (1 << code), into one
// 32-bit word per device that avits_device_status() reads and clears.
// Bounded waits: every spin in these kernels gives up after a wall-clock
// limit (globaltimer) or an iteration cap, records AVITS_ERR_TIMEOUT and
// returns false; callers then drain what they issued and exit.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>
#include <cuda_bf16.h>

#include "avits.h"

namespace avits {

// Kernels receive the device address of the per-device status word (owned by
// api.cu) and OR (1 << code) into it.
__device__ __forceinline__ void raise_status(unsigned int* st, avits_status s) {
  if (st) atomicOr(st, 1u << static_cast<unsigned>(s));
}

// Wall-clock limit of a bounded wait and an iteration cap that ends it even
// if the timer stalled.
constexpr unsigned long long kWaitLimitNs = 1000ull * 1000ull * 1000ull;   // 1 s
constexpr unsigned long long kWaitMaxIters = 1ull << 28;

__device__ __forceinline__ unsigned long long globaltimer_ns() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// ---------------------------------------------------------------- mbarrier --
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count));
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Non-blocking test of the same condition (never suspends the thread).
__device__ __forceinline__ bool mbar_test_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Wait for the phase of `bar` with the given parity to complete.  Gives up
// when *abort_flag becomes non-zero (another role timed out; pass nullptr to
// ignore it) or after the time limit (limit_ns, 1 s by default) or the
// iteration cap, in which case it raises AVITS_ERR_TIMEOUT and sets
// *abort_flag.  Returns true on completion.
__device__ __forceinline__ bool mbar_wait_bounded(uint64_t* bar, uint32_t parity,
                                                  volatile int* abort_flag, unsigned int* st,
                                                  unsigned long long limit_ns = kWaitLimitNs) {
  if (mbar_try_wait(bar, parity)) return true;
  const unsigned long long t0 = globaltimer_ns();
  for (unsigned long long it = 1; it < kWaitMaxIters; ++it) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((it & 63ull) == 0) {
      if (abort_flag && *abort_flag) return false;
      if (globaltimer_ns() - t0 > limit_ns) break;
    }
  }
  raise_status(st, AVITS_ERR_TIMEOUT);
  if (abort_flag) *abort_flag = 1;
  return false;
}

// ------------------------------------------- programmatic dependent launch --
// Every kernel of the path waits for the kernel before it on the stream to
// complete (and its writes to be visible) before touching memory, then lets
// the next kernel be scheduled; launched with launch_pdl, a kernel's launch
// and prologue overlap the tail of the one before it.
__device__ __forceinline__ void pdl_wait_then_trigger() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// All kernels of the path prefer the same (all shared) L1/shared carveout:
// two kernels with different carveouts cannot share an SM, which would stop
// a programmatic dependent from starting beside its predecessor.  Set once
// per kernel and device.
template <auto Kernel>
inline cudaError_t prefer_max_shared() {
  static int done[64] = {};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev >= 0 && dev < 64 && __atomic_load_n(&done[dev], __ATOMIC_ACQUIRE)) return cudaSuccess;
  e = cudaFuncSetAttribute(Kernel, cudaFuncAttributePreferredSharedMemoryCarveout,
                           cudaSharedmemCarveoutMaxShared);
  if (e == cudaSuccess && dev >= 0 && dev < 64) __atomic_store_n(&done[dev], 1, __ATOMIC_RELEASE);
  return e;
}

template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                              cudaStream_t s, Args... args) {
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}

// ------------------------------------------------------------- bf16 loads --
__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

__device__ __forceinline__ float load_elem(const float* p, int64_t i) { return p[i]; }
__device__ __forceinline__ float load_elem(const __nv_bfloat16* p, int64_t i) {
  return __bfloat162float(p[i]);
}
__device__ __forceinline__ void store_elem(float* p, int64_t i, float v) { p[i] = v; }
__device__ __forceinline__ void store_elem(__nv_bfloat16* p, int64_t i, float v) {
  p[i] = __float2bfloat16_rn(v);
}

// The 4 pixels of one channel of a latent token, stored together (the
// within-token layout is channel, patch row, patch column).
template <typename T>
struct Pix4;
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

// One 16-byte chunk j of a latent token (channel, patch row, patch column
// layout) whose channel pixels are taken from a source token's pixels
// (r0|r1, c0|c1): pixel (0,0) <- (r0,c0), (0,1) <- (r0,c1), (1,0) <- (r1,c0),
// (1,1) <- (r1,c1).  bf16: a chunk holds two channels; fp32: one.  `src`
// points at the source token (global or shared memory).
template <typename T>
__device__ __forceinline__ uint4 gather_chunk(const void* src, int j, int r0, int r1, int c0,
                                              int c1);
template <>
__device__ __forceinline__ uint4 gather_chunk<__nv_bfloat16>(const void* src, int j, int r0,
                                                             int r1, int c0, int c1) {
  const uint16_t* t = static_cast<const uint16_t*>(src);
  uint32_t w[4];
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const uint16_t* ch = t + (2 * j + h) * 4;
    w[2 * h] = (uint32_t)ch[r0 * 2 + c0] | ((uint32_t)ch[r0 * 2 + c1] << 16);
    w[2 * h + 1] = (uint32_t)ch[r1 * 2 + c0] | ((uint32_t)ch[r1 * 2 + c1] << 16);
  }
  return make_uint4(w[0], w[1], w[2], w[3]);
}
template <>
__device__ __forceinline__ uint4 gather_chunk<float>(const void* src, int j, int r0, int r1,
                                                     int c0, int c1) {
  const uint32_t* ch = static_cast<const uint32_t*>(src) + j * 4;
  return make_uint4(ch[r0 * 2 + c0], ch[r0 * 2 + c1], ch[r1 * 2 + c0], ch[r1 * 2 + c1]);
}

}  // namespace avits
