// tc_common.cuh — sm_103a tensor-core, TMA and tensor-memory helpers shared
// by the tcgen05 kernels (spatial_tc.cu, attention_tc.cu): inline PTX for
// TMA tile copies, shared-memory matrix descriptors, tcgen05.mma / commit /
// ld / st, packed fp32 arithmetic, and the host-side tensor-map encoding.
#pragma once

#include <cuda.h>

#include "avits_common.cuh"

namespace avits {
namespace tc {

// ------------------------------------------------------------------- TMA ---
__device__ __forceinline__ void tma_load_4d(void* dst, const CUtensorMap* map, int c0, int c1,
                                            int c2, int c3, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.4d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3, %4, %5}], [%6];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(c2), "r"(c3),
      "r"(smem_u32(bar))
      : "memory");
}

// Shared -> global tile store (bulk-group completion); elements outside the
// tensor are not written.
__device__ __forceinline__ void tma_store_4d(const CUtensorMap* map, const void* src, int c0,
                                             int c1, int c2, int c3) {
  asm volatile(
      "cp.async.bulk.tensor.4d.global.shared::cta.tile.bulk_group [%0, {%1, %2, %3, %4}], [%5];" ::
          "l"(reinterpret_cast<uint64_t>(map)),
      "r"(c0), "r"(c1), "r"(c2), "r"(c3), "r"(smem_u32(src))
      : "memory");
}
__device__ __forceinline__ void bulk_commit() {
  asm volatile("cp.async.bulk.commit_group;" ::: "memory");
}
// The shared-memory sources of every committed store have been read.
__device__ __forceinline__ void bulk_wait_read() {
  asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
}
// Every committed store has completed.
__device__ __forceinline__ void bulk_wait_all() {
  asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");
}
// Generic-proxy writes to shared memory become visible to the async proxy
// (TMA, tcgen05.mma operands).
__device__ __forceinline__ void fence_async_shared() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// ---------------------------------------------- shared-memory descriptors ---
// K-major operand, 128-byte swizzle, 8-row core-matrix groups 1024 B apart.
__device__ __forceinline__ uint64_t sw128_desc(const void* p) {
  const uint32_t a = smem_u32(p);
  return (uint64_t)((a >> 4) & 0x3FFFu) | ((uint64_t)1 << 16) | ((uint64_t)(1024 >> 4) << 32) |
         ((uint64_t)1 << 46) | ((uint64_t)2 << 61);
}

// The same descriptor as two 32-bit words: the low word holds the start
// address (bits 0-13, in 16-byte units) and the leading-byte offset, the high
// word the stride, version and swizzle fields, which are equal for every tile.
// A K-step moves the start address only (no carry: shared memory < 256 KB), so
// the issuer adds constants to the low word instead of rebuilding descriptors.
__device__ __forceinline__ uint32_t sw128_desc_lo(const void* p) {
  return (uint32_t)sw128_desc(p);
}
__device__ __forceinline__ uint32_t sw128_desc_hi() {
  return (uint32_t)(((uint64_t)(1024 >> 4) << 32 | ((uint64_t)1 << 46) | ((uint64_t)2 << 61)) >> 32);
}

// MN-major operand (rows of the tile run along K, 64 elements of N per
// 128-byte row), 128-byte swizzle: the leading-byte offset is the distance
// between consecutive 64-element blocks of N, the stride 1024 B between
// 8-row groups of K.  Low word only; the high word is sw128_desc_hi().
__device__ __forceinline__ uint32_t sw128_mn_desc_lo(const void* p, uint32_t n_block_bytes) {
  return ((smem_u32(p) >> 4) & 0x3FFFu) | (((n_block_bytes >> 4) & 0x3FFFu) << 16);
}

// Instruction descriptor of tcgen05.mma kind::f16: bf16 A and B, fp32 D,
// M x N, B K-major (b_mn = false) or MN-major (true); A is always K-major.
__host__ __device__ constexpr uint32_t idesc_bf16(int M, int N, bool b_mn) {
  return (1u << 4) | (1u << 7) | (1u << 10) | (b_mn ? (1u << 16) : 0u) |
         ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

// --------------------------------------------------------------- tcgen05 ---
// D (tensor memory) (+)= A (shared) x B (shared); descriptors as low words
// plus the common high word.
__device__ __forceinline__ void mma_ss(uint32_t d_tmem, uint32_t a_lo, uint32_t b_lo, uint32_t hi,
                                       uint32_t idesc, uint32_t acc) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t.reg .b64 ad, bd;\n\t"
      "setp.ne.b32 p, %5, 0;\n\t"
      "mov.b64 ad, {%1, %3};\n\tmov.b64 bd, {%2, %3};\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], ad, bd, %4, p;\n\t}" ::"r"(d_tmem),
      "r"(a_lo), "r"(b_lo), "r"(hi), "r"(idesc), "r"(acc));
}

// D (tensor memory) (+)= A (tensor memory: one row per lane, bf16 pairs along
// the columns, element 2c in the low half of column c) x B (shared).
__device__ __forceinline__ void mma_ts(uint32_t d_tmem, uint32_t a_tmem, uint32_t b_lo,
                                       uint32_t hi, uint32_t idesc, uint32_t acc) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t.reg .b64 bd;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "mov.b64 bd, {%2, %3};\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], bd, %5, p;\n\t}" ::"r"(d_tmem),
      "r"(a_tmem), "r"(b_lo), "r"(hi), "r"(acc), "r"(idesc));
}

// The mbarrier completes once every tcgen05 operation this thread issued
// before has completed.
__device__ __forceinline__ void mma_commit(uint64_t* bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
          smem_u32(bar))
      : "memory");
}

__device__ __forceinline__ void fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

__device__ __forceinline__ void tmem_alloc(uint32_t* dst_smem, uint32_t cols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                   smem_u32(dst_smem)),
               "r"(cols));
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t base, uint32_t cols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(base), "r"(cols));
}

#define AVITS_R8(b) "=r"(r[b]), "=r"(r[b + 1]), "=r"(r[b + 2]), "=r"(r[b + 3]), \
                    "=r"(r[b + 4]), "=r"(r[b + 5]), "=r"(r[b + 6]), "=r"(r[b + 7])
#define AVITS_W8(b) "+r"(r[b]), "+r"(r[b + 1]), "+r"(r[b + 2]), "+r"(r[b + 3]), \
                    "+r"(r[b + 4]), "+r"(r[b + 5]), "+r"(r[b + 6]), "+r"(r[b + 7])
#define AVITS_I8(b) "r"(r[b]), "r"(r[b + 1]), "r"(r[b + 2]), "r"(r[b + 3]), \
                    "r"(r[b + 4]), "r"(r[b + 5]), "r"(r[b + 6]), "r"(r[b + 7])

// 16 / 32 consecutive 32-bit columns of this thread's TMEM lane.
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, "
      "%11, %12, %13, %14, %15}, [%16];"
      : AVITS_R8(0), AVITS_R8(8)
      : "r"(taddr));
}
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, "
      "%11, %12, %13, %14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, "
      "%28, %29, %30, %31}, [%32];"
      : AVITS_R8(0), AVITS_R8(8), AVITS_R8(16), AVITS_R8(24)
      : "r"(taddr));
}

// Completes the thread's outstanding tcgen05.ld; the registers are tied to
// the wait so that no use can be scheduled before it.
__device__ __forceinline__ void tmem_wait(uint32_t (&r)[16]) {
  asm volatile("tcgen05.wait::ld.sync.aligned;" : AVITS_W8(0), AVITS_W8(8) : : "memory");
}
__device__ __forceinline__ void tmem_wait32(uint32_t (&r)[32]) {
  asm volatile("tcgen05.wait::ld.sync.aligned;"
               : AVITS_W8(0), AVITS_W8(8), AVITS_W8(16), AVITS_W8(24)
               :
               : "memory");
}

__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, "
      "%11, %12, %13, %14, %15, %16};" ::"r"(taddr),
      AVITS_I8(0), AVITS_I8(8)
      : "memory");
}
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, "
      "%11, %12, %13, %14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, "
      "%28, %29, %30, %31, %32};" ::"r"(taddr),
      AVITS_I8(0), AVITS_I8(8), AVITS_I8(16), AVITS_I8(24)
      : "memory");
}
// The thread's tcgen05.st have completed.
__device__ __forceinline__ void tmem_wait_st() {
  asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

// ------------------------------------------------------------ arithmetic ---
__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ float max3(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}

// (a0, a1) * b + c on both lanes of a packed pair.
__device__ __forceinline__ void ffma2(float a0, float a1, float b, float c, float& d0, float& d1) {
  asm("{\n\t.reg .b64 ra, rb, rc, rd;\n\t"
      "mov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %4};\n\tmov.b64 rc, {%5, %5};\n\t"
      "fma.rn.f32x2 rd, ra, rb, rc;\n\tmov.b64 {%0, %1}, rd;\n\t}"
      : "=f"(d0), "=f"(d1)
      : "f"(a0), "f"(a1), "f"(b), "f"(c));
}

// (s0, s1) += (e0, e1) on a packed pair.
__device__ __forceinline__ void fadd2(float& s0, float& s1, float e0, float e1) {
  asm("{\n\t.reg .b64 ra, rb;\n\t"
      "mov.b64 ra, {%0, %1};\n\tmov.b64 rb, {%2, %3};\n\t"
      "add.rn.f32x2 ra, ra, rb;\n\tmov.b64 {%0, %1}, ra;\n\t}"
      : "+f"(s0), "+f"(s1)
      : "f"(e0), "f"(e1));
}

// (a0, a1) *= b on a packed pair.
__device__ __forceinline__ void fmul2(float& a0, float& a1, float b) {
  asm("{\n\t.reg .b64 ra, rb;\n\t"
      "mov.b64 ra, {%0, %1};\n\tmov.b64 rb, {%2, %2};\n\t"
      "mul.rn.f32x2 ra, ra, rb;\n\tmov.b64 {%0, %1}, ra;\n\t}"
      : "+f"(a0), "+f"(a1)
      : "f"(b));
}

// Two fp32 -> one bf16x2 word (round to nearest even), lo in the low half.
__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  uint32_t w;
  asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(w) : "f"(hi), "f"(lo));
  return w;
}

__device__ __forceinline__ void bar_sync(int id, int count) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(count) : "memory");
}

// ------------------------------------------------- fixed-point head sum ---
// Eq. 3's mean over heads, independent of the order the heads arrive in:
// word = heads << 56 | NaN masses << 48 | sum of round(mass * 2^40), added
// atomically; H <= 255, so neither count overflows its byte and the sum stays
// below 2^48.  The head that completes the word writes (or adds)
// weight * mean to *a and clears the word for the next call.
__device__ __forceinline__ void head_sum_add(unsigned long long* w, int H, float mass,
                                             float weight, int accumulate, float* a) {
  unsigned long long inc = 1ull << 56;
  if (mass != mass)
    inc |= 1ull << 48;
  else
    inc += __float2ull_rn(fminf(fmaxf(mass, 0.f), 1.f) * 0x1p40f);
  const unsigned long long v = atomicAdd(w, inc) + inc;
  if ((int)(v >> 56) != H) return;
  *w = 0ull;   // every head is in: clear the word for the next call
  float r;
  if ((v >> 48) & 0xFFull) {
    r = __int_as_float(0x7fc00000);
  } else {
    const double mean = (double)(v & ((1ull << 48) - 1ull)) * 0x1p-40 / (double)H;
    r = (float)((double)weight * mean);
  }
  *a = accumulate ? *a + r : r;
}

// ------------------------------------------------------------------ host ---
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

inline EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static bool tried = false;
  if (!tried) {
    tried = true;
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  }
  return fn;
}

// Tensor map of a bf16 [B,H,rows,d] view with element strides (sb, sh, sn),
// d contiguous: boxes of 64 elements of d x 128 rows, 128-byte swizzle.  A
// dimension of extent 1 gets a packed stride (its stride is never used).
inline bool make_map(CUtensorMap* map, const void* base, int B, int H, int rows, int d,
                     int64_t sb, int64_t sh, int64_t sn) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  const int64_t e = 2;
  int64_t s_n = sn * e;
  int64_t s_h = (H > 1) ? sh * e : s_n * rows;
  int64_t s_b = (B > 1) ? sb * e : s_h * H;
  cuuint64_t dims[4] = {(cuuint64_t)d, (cuuint64_t)rows, (cuuint64_t)H, (cuuint64_t)B};
  cuuint64_t strides[3] = {(cuuint64_t)s_n, (cuuint64_t)s_h, (cuuint64_t)s_b};
  cuuint32_t box[4] = {64, 128, 1, 1};
  cuuint32_t estr[4] = {1, 1, 1, 1};
  CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides,
                  box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

// Element strides of a [B,H,rows,d] view that a tensor map can take: 16-byte
// multiples, positive where the dimension has more than one entry.
inline bool strides_ok(int B, int H, int64_t sb, int64_t sh, int64_t sn) {
  if (sn % 8 != 0 || sn <= 0) return false;
  if (H > 1 && (sh % 8 != 0 || sh <= 0)) return false;
  if (B > 1 && (sb % 8 != 0 || sb <= 0)) return false;
  return true;
}

}  // namespace tc
}  // namespace avits
