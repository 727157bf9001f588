// spatial_tc.cu — spatial importance (Sec. 3.3.1, Eq. 3 with the joint-
// attention extraction of Eq. 4-5) on the sm_103a tensor cores.
//
// For every image query i and head h the text mass of the joint softmax is
//   sum_{j<L} exp(l_ij) / sum_{j<Nk} exp(l_ij),  l_ij = scale * q_i . k_j,
// and A_i is its mean over heads.  Only Q K^T is a contraction (there is no
// P V product in the method), so the kernel is a flash-style pass that keeps
// per row a running (max, sum over all keys, sum over text keys) and never
// writes the score matrix.
//
// Work decomposition (persistent, one CTA per SM):
//   unit  = (b, h, 256 query rows = two 128-row tiles)
//   item  = (unit, 128-key tile)
// The B*H*ceil(M/256)*ceil(Nk/128) items are split into equal contiguous
// ranges, one per CTA, so every SM issues the same number of MMA tiles.  A
// unit whose key tiles fall into several CTAs' ranges leaves one piece of
// per-row partial statistics (max, sum over all keys, sum over text keys;
// the two column halves merged in shared memory) per CTA.  The merge is part
// of this kernel:
//   * the CTA holding the unit's first item is its merger.  That piece is the
//     last segment of its range, so the other pieces (the first segments of
//     the following CTAs) are mostly finished long before.  Their holders
//     store each row's statistics as two 64-bit words, (m, l_all) and
//     (l_txt, l_all), each written in one single-copy-atomic store; l_all
//     is never 0 (the row's largest term is 1), so a word is either the
//     zero left by the previous call or this call's value.  The merger
//     polls both words of every row until they are non-zero, clears them,
//     merges the pieces in slot order and forms the text mass of every
//     (row, head) of the unit.  No flag and no fence stand between a piece
//     and its merger: a piece is one store away from it;
//   * the head mean of Eq. 3 is an exact integer sum: each (row, head) mass
//     in [0, 1] is added as a 40-bit fixed-point number to one 64-bit word per
//     row that also counts the heads (top byte) and the NaN masses (next
//     byte).  The atomic add returns the new word, so the head that completes
//     the count writes A and clears the word for the next call.  Integer
//     addition is associative: A does not depend on the order in which CTAs
//     finish.
// The workspace is zero between calls: the caller zeroes it once, and a call
// that completes clears every word it used (head-sum words and pieces), so
// a later call with other sizes, whose row words may lie where these pieces
// were, also finds zeros.
//
// Roles (19 warps):
//   warp 0        TMA producer: Q tile 0, the first K tile, Q tile 1, then the
//                 K tiles through a 4-stage ring (128-byte swizzle, no
//                 multicast); each Q tile has its own barrier so the first MMA
//                 starts after 64 KB rather than 96 KB.
//   warps 1, 18   MMA issuers, one per query tile: S = Q K^T with
//                 tcgen05.mma kind::f16 (bf16 in, fp32 accumulate in tensor
//                 memory), 128x128 per tile, two S buffers per Q tile (all 512
//                 TMEM columns).  A barrier wait in the issuing thread costs
//                 the tensor pipe a bubble; a second issuer fills it.
//   warps 2-17    four softmax warpgroups: query tile t and column half c
//                 (64 of the 128 keys of a tile) per warpgroup, so all 16
//                 warps work on the same item while the MMA fills the other S
//                 buffer; one TMEM lane (= one query row) per thread, 16
//                 columns per tcgen05.ld, ex2 on the MUFU against the running
//                 row maximum with packed f32x2 FMA/add.  The exact chunk
//                 maximum is only computed when a chunk sum would leave
//                 [0, 2^64) (first chunk, a larger logit, NaN).  The text keys
//                 come first, so the text sum is a prefix of the row sum.  At
//                 d = 128 a 128x128 tile costs the tensor pipe and the MUFU
//                 (32 ex2 / clock / SM) the same 512 cycles; evaluating part
//                 of the exponentials on the FMA pipe with a polynomial was
//                 measured slower on this chip (the loop is issue-bound), so
//                 every exponential goes to the MUFU.
// Every wait is bounded (avits_common.cuh); on a timeout all roles stop
// issuing, drain what they issued, release tensor memory and exit.
#include <cuda.h>

#include "avits_common.cuh"
#include "avits_internal.h"
#include "tc_common.cuh"

namespace avits {
namespace {

using namespace tc;

constexpr int kBM = 128;       // query rows per tile (= TMEM lanes)
constexpr int kBN = 128;       // keys per tile
constexpr int kQTiles = 2;     // query tiles per unit
constexpr int kUnitRows = kBM * kQTiles;
constexpr int kSoftmaxWarps = 16;
constexpr int kMmaWarp1 = 2 + kSoftmaxWarps;            // issuer of query tile 1
constexpr int kThreads = 96 + kSoftmaxWarps * 32;
constexpr int kTmemCols = 512;
constexpr uint32_t kIdesc = (1u << 4)                       // D: fp32
                            | (1u << 7) | (1u << 10)        // A, B: bf16
                            | ((uint32_t)(kBN >> 3) << 17)  // N
                            | ((uint32_t)(kBM >> 4) << 24); // M

__device__ __forceinline__ void mma_bf16(uint32_t d_tmem, uint32_t a_lo, uint32_t b_lo,
                                         uint32_t hi, uint32_t acc) {
  mma_ss(d_tmem, a_lo, b_lo, hi, kIdesc, acc);
}

template <int D>
struct Cfg {
  static constexpr int kCB = D / 64;                   // 128-byte column blocks per row
  static constexpr int kTileBytes = kCB * kBM * 128;   // one 128-row bf16 tile
  static constexpr int kStages = (D == 128) ? 4 : 8;
  static constexpr int kQBytes = kQTiles * kTileBytes;
  static constexpr int kKBytes = kStages * kTileBytes;
};

struct Bars {
  uint64_t q_full[kQTiles], q_empty;
  uint64_t k_full[8], k_empty[8];
  uint64_t s_full[kQTiles][2], s_empty[kQTiles][2];
  uint64_t drain[kQTiles];
  uint32_t tmem_base;
  int abort;
};

// The column halves' row statistics meet here at the end of a segment: one
// buffer per segment parity, per query tile, 128 rows x (m, la, lt).
constexpr int kXchBytes = 2 * kQTiles * kBM * 3 * (int)sizeof(float);

template <int D>
constexpr int smem_bytes() {
  return Cfg<D>::kQBytes + Cfg<D>::kKBytes + (int)sizeof(Bars) + kXchBytes + 1024;
}

struct TcParams {
  int B, H, M, Nk, L;
  int n_qp, n_kt, n_units;
  int total, per;          // items in all, items per CTA (total < 2^31 checked on the host)
  int max_parts;
  float c_log2, weight;
  int accumulate;
  float* A;
  float* lse;
  unsigned long long* part;  // [n_units][max_parts][256][2] pieces of the non-merger CTAs
  unsigned long long* acc;   // [B][n_qp * 256] head count | NaN count | fixed-point mass sum
  int rows_pad;     // n_qp * 256
  unsigned int* status;
  const uint8_t* tmask;   // [B,Nk] text-key mask, or NULL (text keys = the first L)
  const float* lse_all;   // [B,H,M] caller's logsumexp over all keys (natural log), or NULL
};

// Running row statistics in the log2 domain: x = c_log2 * (q.k); the sums
// are of 2^(x - m).
struct RowStat {
  float m, la, lt;
};

__device__ __forceinline__ void merge_stat(RowStat& a, float m2, float la2, float lt2) {
  const float m = fmaxf(a.m, m2);
  if (m == -INFINITY) return;
  const float f1 = ex2(a.m - m), f2 = ex2(m2 - m);
  a.la = a.la * f1 + la2 * f2;
  a.lt = a.lt * f1 + lt2 * f2;
  a.m = m;
}

// One chunk of 16 keys that are all valid and all text (kText) or all image
// keys: the common case, kept free of the masking and boundary logic (a
// per-chunk branch on the key kind measured ~15% slower on the whole item).
template <bool kText>
__device__ __forceinline__ void process_chunk_full(const uint32_t (&r)[16], float c, RowStat& st) {
  float v[16];
#pragma unroll
  for (int e = 0; e < 16; ++e) v[e] = __uint_as_float(r[e]);
  const float nm = -st.m;
  float s0 = 0.f, s1 = 0.f, s2 = 0.f, s3 = 0.f;
#pragma unroll
  for (int e = 0; e < 16; e += 4) {
    float x0, x1, x2, x3;
    ffma2(v[e], v[e + 1], c, nm, x0, x1);
    ffma2(v[e + 2], v[e + 3], c, nm, x2, x3);
    fadd2(s0, s1, ex2(x0), ex2(x1));
    fadd2(s2, s3, ex2(x2), ex2(x3));
  }
  fadd2(s0, s1, s2, s3);
  float cs = s0 + s1;
  if (!(cs < 0x1p64f)) {
    // first chunk of a row, a logit 64 log2-units above the running maximum,
    // or a NaN: take the exact chunk maximum and rescale the running sums
    float cm = v[0];
#pragma unroll
    for (int e = 1; e < 16; ++e) cm = fmaxf(cm, v[e]);
    const float mx = fmaxf(st.m, cm * c);
    const float corr = ex2(st.m - mx);
    st.la *= corr;
    st.lt *= corr;
    st.m = mx;
    cs = 0.f;
#pragma unroll
    for (int e = 0; e < 16; ++e) cs += ex2(fmaf(v[e], c, -mx));
  }
  st.la += cs;
  if (kText) st.lt += cs;
}

// One 16-column chunk whose first key is col0 (< Nk), possibly ragged (keys
// beyond Nk) or straddling the text / image boundary.
__device__ __forceinline__ void process_chunk(const uint32_t (&r)[16], int col0, int Nk, int L,
                                              float c, RowStat& st) {
  float v[16];
#pragma unroll
  for (int e = 0; e < 16; ++e) v[e] = __uint_as_float(r[e]);
  const int nvalid = Nk - col0;
  if (nvalid < 16) {
#pragma unroll
    for (int e = 0; e < 16; ++e)
      if (e >= nvalid) v[e] = -INFINITY;
  }
  const float nm = -st.m;
  float x[16];
#pragma unroll
  for (int e = 0; e < 16; e += 2) ffma2(v[e], v[e + 1], c, nm, x[e], x[e + 1]);
  float s0 = 0.f, s1 = 0.f, s2 = 0.f, s3 = 0.f;
#pragma unroll
  for (int e = 0; e < 16; e += 4) {
    fadd2(s0, s1, ex2(x[e]), ex2(x[e + 1]));
    fadd2(s2, s3, ex2(x[e + 2]), ex2(x[e + 3]));
  }
  fadd2(s0, s1, s2, s3);
  float cs = s0 + s1;
  if (!(cs < 0x1p64f)) {
    // first chunk of a row, a logit 64 log2-units above the running maximum,
    // or a NaN: take the exact chunk maximum and rescale the running sums
    const float t0 = max3(v[0], v[1], v[2]), t1 = max3(v[3], v[4], v[5]);
    const float t2 = max3(v[6], v[7], v[8]), t3 = max3(v[9], v[10], v[11]);
    const float t4 = max3(v[12], v[13], v[14]);
    const float mx = fmaxf(st.m, fmaxf(max3(t0, t1, t2), max3(t3, t4, v[15])) * c);
    const float corr = ex2(st.m - mx);
    st.la *= corr;
    st.lt *= corr;
    st.m = mx;
    cs = 0.f;
#pragma unroll
    for (int e = 0; e < 16; ++e) cs += ex2(fmaf(v[e], c, -mx));
  }
  st.la += cs;
  if (col0 + 16 <= L) {
    st.lt += cs;
  } else if (col0 < L) {   // the chunk straddles the text / image boundary
    float ts = 0.f;
#pragma unroll
    for (int e = 0; e < 16; ++e) ts += (col0 + e < L) ? ex2(fmaf(v[e], c, -st.m)) : 0.f;
    st.lt += ts;
  }
}

// ------------------------------------------------ merge across CTAs (gpu) --
__device__ __forceinline__ unsigned long long pack2(float lo, float hi) {
  return (unsigned long long)__float_as_uint(lo) | ((unsigned long long)__float_as_uint(hi) << 32);
}
__device__ __forceinline__ void st_word(unsigned long long* a, unsigned long long v) {
  asm volatile("st.relaxed.gpu.global.b64 [%0], %1;" ::"l"(a), "l"(v) : "memory");
}
__device__ __forceinline__ unsigned long long ld_word(const unsigned long long* a) {
  unsigned long long v;
  asm volatile("ld.relaxed.gpu.global.b64 %0, [%1];" : "=l"(v) : "l"(a) : "memory");
  return v;
}

// Poll a piece's two words until both hold this call's values (non-zero);
// bounded like the mbarrier waits.
__device__ __forceinline__ bool piece_wait(const unsigned long long* w, unsigned long long& w0,
                                           unsigned long long& w1, volatile int* abort_flag,
                                           unsigned int* st) {
  w0 = ld_word(w);
  w1 = ld_word(w + 1);
  if (w0 != 0ull && w1 != 0ull) return true;
  const unsigned long long t0 = globaltimer_ns();
  for (unsigned long long it = 1; it < kWaitMaxIters; ++it) {
    if (w0 == 0ull) w0 = ld_word(w);
    if (w1 == 0ull) w1 = ld_word(w + 1);
    if (w0 != 0ull && w1 != 0ull) return true;
    if ((it & 15ull) == 0) {
      if (abort_flag && *abort_flag) return false;
      if (globaltimer_ns() - t0 > kWaitLimitNs) break;
    }
  }
  raise_status(st, AVITS_ERR_TIMEOUT);
  if (abort_flag) *abort_flag = 1;
  return false;
}

// Eq. 3's head sum of this row (fixed point, order independent).
__device__ __forceinline__ void head_sum_add(const TcParams& p, int b, int row, float mass) {
  tc::head_sum_add(p.acc + (long long)b * p.rows_pad + row, p.H, mass, p.weight, p.accumulate,
                   p.A + (long long)b * p.M + row);
}

// Kinds of the 64 keys a softmax warp reduces per item.
enum ItemKind { kItemImage = 0, kItemText = 1, kItemGeneral = 2, kItemMasked = 3 };

// A chunk whose text keys are given by a mask (bit e = key col0 + e is a text
// key), possibly with invalid keys beyond Nk: the mixed case of a caller's
// key mask.  Same lazy running maximum as process_chunk_full; the text sum
// takes the exponentials of the masked keys.
__device__ __forceinline__ void process_chunk_masked(const uint32_t (&r)[16], int col0, int Nk,
                                                     uint32_t m16, float c, RowStat& st) {
  float v[16];
#pragma unroll
  for (int e = 0; e < 16; ++e) v[e] = __uint_as_float(r[e]);
  if (col0 + 16 > Nk) {
#pragma unroll
    for (int e = 0; e < 16; ++e)
      if (col0 + e >= Nk) v[e] = -INFINITY;
  }
  const float nm = -st.m;
  float ev[16];
  float s0 = 0.f, s1 = 0.f, s2 = 0.f, s3 = 0.f;
#pragma unroll
  for (int e = 0; e < 16; e += 4) {
    float x0, x1, x2, x3;
    ffma2(v[e], v[e + 1], c, nm, x0, x1);
    ffma2(v[e + 2], v[e + 3], c, nm, x2, x3);
    ev[e] = ex2(x0); ev[e + 1] = ex2(x1); ev[e + 2] = ex2(x2); ev[e + 3] = ex2(x3);
    fadd2(s0, s1, ev[e], ev[e + 1]);
    fadd2(s2, s3, ev[e + 2], ev[e + 3]);
  }
  fadd2(s0, s1, s2, s3);
  float cs = s0 + s1;
  if (!(cs < 0x1p64f)) {
    // first chunk of a row, a logit 64 log2-units above the running maximum,
    // or a NaN: the exact chunk maximum, then the exponentials again
    float cm = v[0];
#pragma unroll
    for (int e = 1; e < 16; ++e) cm = fmaxf(cm, v[e]);
    const float mx = fmaxf(st.m, cm * c);
    if (mx == -INFINITY) return;   // no valid key
    const float corr = ex2(st.m - mx);
    st.la *= corr;
    st.lt *= corr;
    st.m = mx;
    cs = 0.f;
#pragma unroll
    for (int e = 0; e < 16; ++e) {
      ev[e] = ex2(fmaf(v[e], c, -mx));
      cs += ev[e];
    }
  }
  float t0 = 0.f, t1 = 0.f;
#pragma unroll
  for (int e = 0; e < 16; e += 2) {
    t0 += ((m16 >> e) & 1u) ? ev[e] : 0.f;
    t1 += ((m16 >> (e + 1)) & 1u) ? ev[e + 1] : 0.f;
  }
  st.la += cs;
  st.lt += t0 + t1;
}

template <int kKind>
__device__ __forceinline__ void softmax_item(uint32_t tb, int c0, int Nk, int L, float c,
                                             RowStat& st, uint64_t* s_empty, int lane,
                                             uint32_t w0 = 0u, uint32_t w1 = 0u) {
  uint32_t ra[16], rb[16];
  const int nch = (kKind >= kItemGeneral) ? max(0, min(4, (Nk - c0 + 15) >> 4)) : 4;
  auto chunk = [&](const uint32_t(&r)[16], int k) {
    if (kKind == kItemGeneral) {
      if (k < nch) process_chunk(r, c0 + 16 * k, Nk, L, c, st);
    } else if (kKind == kItemMasked) {
      const uint32_t m16 = ((k < 2 ? w0 : w1) >> (16 * (k & 1))) & 0xFFFFu;
      if (k < nch) process_chunk_masked(r, c0 + 16 * k, Nk, m16, c, st);
    } else {
      process_chunk_full<kKind == kItemText>(r, c, st);
    }
  };
  tmem_ld16(tb, ra);
  tmem_wait(ra);
  tmem_ld16(tb + 16, rb);
  chunk(ra, 0);
  tmem_wait(rb);
  tmem_ld16(tb + 32, ra);
  chunk(rb, 1);
  tmem_wait(ra);
  tmem_ld16(tb + 48, rb);
  chunk(ra, 2);
  tmem_wait(rb);
  fence_before();
  __syncwarp();
  if (lane == 0) mbar_arrive(s_empty);
  chunk(rb, 3);
}

struct Segment {
  int u, kt0, nk;
};

__device__ __forceinline__ Segment segment_at(int it, int it_end, int n_kt) {
  Segment s;
  s.u = it / n_kt;
  s.kt0 = it - s.u * n_kt;
  s.nk = min(n_kt - s.kt0, it_end - it);
  return s;
}

// Number of CTAs whose item range overlaps unit u, and the first of them.
__device__ __forceinline__ int first_cta(int u, int n_kt, int per) { return (u * n_kt) / per; }
__device__ __forceinline__ int pieces(int u, int n_kt, int per) {
  return ((u + 1) * n_kt - 1) / per - (u * n_kt) / per + 1;
}

// End of a segment, for the thread of row `rowu` of unit u holding the CTA's
// piece st (both column halves merged).  A non-merger stores the piece; the
// merger (slot 0) collects the other pieces, merges all of them in slot
// order, forms the text mass (Eq. 5) and adds it to the row's head sum.
__device__ __forceinline__ void unit_piece_done(const TcParams& p, int u, int rowu, RowStat st,
                                                volatile int* abort_flag) {
  const int slot = (int)blockIdx.x - first_cta(u, p.n_kt, p.per);
  if (slot != 0) {
    unsigned long long* w = p.part + (((long long)u * p.max_parts + slot) * kUnitRows + rowu) * 2;
    st_word(w, pack2(st.m, st.la));
    st_word(w + 1, pack2(st.lt, st.la));
    return;
  }
  const int np = pieces(u, p.n_kt, p.per);
  bool ok = true;
#pragma unroll 1
  for (int s = 1; s < np && ok; ++s) {
    unsigned long long* w = p.part + (((long long)u * p.max_parts + s) * kUnitRows + rowu) * 2;
    unsigned long long w0, w1;
    ok = piece_wait(w, w0, w1, abort_flag, p.status);
    if (!ok) break;
    // consumed: zero, so that a completed call leaves the whole workspace
    // zero whatever layout (shape) the next call gives it
    st_word(w, 0ull);
    st_word(w + 1, 0ull);
    merge_stat(st, __uint_as_float((uint32_t)w0), __uint_as_float((uint32_t)(w0 >> 32)),
               __uint_as_float((uint32_t)w1));
  }
  if (!ok) return;
  const int bh = u / p.n_qp, qp = u - bh * p.n_qp;
  const int b = bh / p.H, h = bh - b * p.H;
  const int row = qp * kUnitRows + rowu;
  if (row >= p.M) return;
  const float ln2 = 0.69314718055994530942f;
  float* lp = p.lse ? p.lse + (((long long)b * p.H + h) * p.M + row) * 2 : nullptr;
  float mass;
  if (p.lse_all) {
    // the keys of this pass are the text keys only: mass = exp(lse_txt -
    // lse_all) against the caller's logsumexp over all keys
    const float la_all = p.lse_all[((long long)b * p.H + h) * p.M + row];
    mass = st.lt > 0.f ? exp2f(st.m + log2f(st.lt) - la_all * 1.4426950408889634f) : 0.f;
    if (lp) {
      lp[0] = la_all;
      lp[1] = st.lt > 0.f ? (st.m + log2f(st.lt)) * ln2 : -INFINITY;
    }
  } else {
    mass = st.lt / st.la;
    if (lp) {
      lp[0] = (st.m + __log2f(st.la)) * ln2;
      lp[1] = st.lt > 0.f ? (st.m + __log2f(st.lt)) * ln2 : -INFINITY;
    }
  }
  head_sum_add(p, b, row, mass);
}

// kMask: the text keys come from the caller's key mask (p.tmask) instead of
// being the first L; a separate instance keeps the plain kernel unchanged.
template <int D, bool kMask>
__global__ void __maxnreg__(88)
spatial_tc_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                  const TcParams p) {
  using C = Cfg<D>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* sQ = smem;
  uint8_t* sK = smem + C::kQBytes;
  Bars* bars = reinterpret_cast<Bars*>(sK + C::kKBytes);
  float* xch = reinterpret_cast<float*>(bars + 1);   // kXchBytes

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int it_begin = (int)blockIdx.x * p.per;
  const int it_end = min(it_begin + p.per, p.total);
  if (it_begin >= it_end) return;   // block-uniform

  // Prologue that touches no global data: it overlaps the tail of the kernel
  // before this one on the stream (programmatic dependent launch).  The
  // tensor maps are kernel parameters; fetching them early takes their
  // latency off the first TMA copy.
  if (threadIdx.x == 0) {
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmQ)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmK)) : "memory");
    for (int t = 0; t < kQTiles; ++t) mbar_init(&bars->q_full[t], 1);
    mbar_init(&bars->q_empty, kQTiles);   // one commit per MMA issuer
    for (int s = 0; s < C::kStages; ++s) {
      mbar_init(&bars->k_full[s], 1);
      mbar_init(&bars->k_empty[s], kQTiles);
    }
    for (int t = 0; t < kQTiles; ++t)
      for (int b = 0; b < 2; ++b) {
        mbar_init(&bars->s_full[t][b], 1);
        mbar_init(&bars->s_empty[t][b], 8);   // 8 softmax warps read each tile
      }
    for (int t = 0; t < kQTiles; ++t) mbar_init(&bars->drain[t], 1);
    bars->abort = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  // Q and K may come from the kernel before this one on the stream; tensor
  // memory is only taken once that kernel has finished
  asm volatile("griddepcontrol.wait;" ::: "memory");
  if (threadIdx.x == 0) {
    // the first segment's Q tiles and first K tile go out before tensor
    // memory is taken (the copies only need the barriers initialised above);
    // the producer loop below skips them
    const Segment seg = segment_at(it_begin, it_end, p.n_kt);
    const int bh = seg.u / p.n_qp, qp = seg.u - bh * p.n_qp;
    const int b = bh / p.H, h = bh - b * p.H;
    mbar_arrive_expect_tx(&bars->q_full[0], C::kTileBytes);
    for (int cb = 0; cb < C::kCB; ++cb)
      tma_load_4d(sQ + cb * (kBM * 128), &tmQ, cb * 64, qp * kUnitRows, h, b, &bars->q_full[0]);
    mbar_arrive_expect_tx(&bars->k_full[0], C::kTileBytes);
    for (int cb = 0; cb < C::kCB; ++cb)
      tma_load_4d(sK + cb * (kBM * 128), &tmK, cb * 64, seg.kt0 * kBN, h, b, &bars->k_full[0]);
    mbar_arrive_expect_tx(&bars->q_full[1], C::kTileBytes);
    for (int cb = 0; cb < C::kCB; ++cb)
      tma_load_4d(sQ + C::kTileBytes + cb * (kBM * 128), &tmQ, cb * 64, qp * kUnitRows + kBM, h,
                  b, &bars->q_full[1]);
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(&bars->tmem_base)),
                 "r"(kTmemCols));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
  }
  fence_before();
  __syncthreads();
  fence_after();
  const uint32_t tmem = bars->tmem_base;
  volatile int* abort_flag = &bars->abort;
  // the next kernel may be scheduled now (it waits for this grid to finish
  // before it reads anything); a softmax thread signals it, keeping the
  // producer free
  if (threadIdx.x == 64) asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

  if (warp == 0) {
    // ------------------------------------------------------ TMA producer --
    if (lane == 0) {
      bool ok = true;
      int li = 0;
      int sg = 0;
      int q_armed = 0;   // Q tiles armed in the latest segment
      for (int it = it_begin; it < it_end && ok;) {
        const Segment seg = segment_at(it, it_end, p.n_kt);
        const int bh = seg.u / p.n_qp, qp = seg.u - bh * p.n_qp;
        const int b = bh / p.H, h = bh - b * p.H;
        // the Q buffer is free at the start; later segments wait for the
        // MMAs of the previous one
        if (sg > 0) ok = mbar_wait_bounded(&bars->q_empty, (uint32_t)((sg & 1) ^ 1), abort_flag, p.status);
        if (!ok) break;
        const bool first = (sg == 0);   // Q tiles and K tile 0 already issued
        ++sg;   // Q of this segment is being issued
        q_armed = first ? kQTiles : 0;
        for (int j = 0; j < seg.nk; ++j, ++li) {
          // Q tile 0 before the first K tile, Q tile 1 right after it
          if (!first && (j == 0 || (j == 1 && kQTiles > 1))) {
            const int t = j;
            ++q_armed;
            mbar_arrive_expect_tx(&bars->q_full[t], C::kTileBytes);
            for (int cb = 0; cb < C::kCB; ++cb)
              tma_load_4d(sQ + t * C::kTileBytes + cb * (kBM * 128), &tmQ, cb * 64,
                          qp * kUnitRows + t * kBM, h, b, &bars->q_full[t]);
          }
          if (li == 1) {
            // cold start: the first K tile lands before the rest of the ring
            // is requested, so the first MMAs do not wait behind every
            // CTA's whole prologue in HBM
            ok = mbar_wait_bounded(&bars->k_full[0], 0, abort_flag, p.status);
            if (!ok) break;
          }
          if (li == 0) continue;   // K tile 0 went out before the set-up
          const int stage = (int)(li % C::kStages);
          const uint32_t ph = (uint32_t)((li / C::kStages) & 1);
          ok = mbar_wait_bounded(&bars->k_empty[stage], ph ^ 1u, abort_flag, p.status);
          if (!ok) break;
          mbar_arrive_expect_tx(&bars->k_full[stage], C::kTileBytes);
          for (int cb = 0; cb < C::kCB; ++cb)
            tma_load_4d(sK + stage * C::kTileBytes + cb * (kBM * 128), &tmK, cb * 64,
                        (seg.kt0 + j) * kBN, h, b, &bars->k_full[stage]);
        }
        if (ok && seg.nk == 1 && !first) {   // a one-tile segment still needs Q tile 1
          ++q_armed;
          mbar_arrive_expect_tx(&bars->q_full[1], C::kTileBytes);
          for (int cb = 0; cb < C::kCB; ++cb)
            tma_load_4d(sQ + C::kTileBytes + cb * (kBM * 128), &tmQ, cb * 64,
                        qp * kUnitRows + kBM, h, b, &bars->q_full[1]);
        }
        it += seg.nk;
      }
      if (!ok) {
        // drain the copies still in flight before the CTA exits: the Q tiles
        // of the last segment started, then every armed K stage
        for (int t = 0; t < q_armed; ++t)
          mbar_wait_bounded(&bars->q_full[t], (uint32_t)((sg - 1) & 1), nullptr, p.status);
        for (int s = 0; s < C::kStages; ++s) {
          const int armed = li - s;   // items issued on stage s: li - s > 0
          if (armed > 0) {
            const int last = (armed - 1) / C::kStages;
            mbar_wait_bounded(&bars->k_full[s], (uint32_t)(last & 1), nullptr, p.status);
          }
        }
      }
    }
  } else if (warp == 1 || warp == kMmaWarp1) {
    // -------------------------------------------------------- MMA issuers --
    // One issuing thread per query tile.  A barrier wait in an issuing thread
    // stalls that thread's queue of MMAs until the tensor pipe has taken it;
    // with two issuers the other queue keeps the pipe busy meanwhile.
    const int t = (warp == 1) ? 0 : 1;
    if (lane == 0) {
      bool ok = true;
      int li = 0;
      int sg = 0;
      // operand descriptors computed once; per MMA only constant offsets are
      // added (the issuing thread shares its sub-partition with four busy
      // softmax warps, so every instruction it needs delays the MMAs)
      const uint32_t a_lo = sw128_desc_lo(sQ + t * C::kTileBytes);
      const uint32_t b_lo0 = sw128_desc_lo(sK);
      const uint32_t d_hi = sw128_desc_hi();
      const uint32_t d_base = tmem + (uint32_t)(t * 2 * kBN);
      for (int it = it_begin; it < it_end && ok;) {
        const Segment seg = segment_at(it, it_end, p.n_kt);
        for (int j = 0; j < seg.nk && ok; ++j, ++li) {
          const int stage = (int)(li % C::kStages);
          const uint32_t ph = (uint32_t)((li / C::kStages) & 1);
          const int sb = (int)(li & 1);
          const uint32_t sph = (uint32_t)((li >> 1) & 1);
          ok = mbar_wait_bounded(&bars->k_full[stage], ph, abort_flag, p.status);
          if (!ok) break;
          if (j == 0) {
            ok = mbar_wait_bounded(&bars->q_full[t], (uint32_t)(sg & 1), abort_flag, p.status);
            if (!ok) break;
          }
          ok = mbar_wait_bounded(&bars->s_empty[t][sb], sph ^ 1u, abort_flag, p.status);
          if (!ok) break;
          fence_after();
          const uint32_t d_tmem = d_base + (uint32_t)(sb * kBN);
          const uint32_t b_lo = b_lo0 + (uint32_t)((stage * C::kTileBytes) >> 4);
#pragma unroll
          for (int kk = 0; kk < D / 16; ++kk) {
            const uint32_t off = (uint32_t)(((kk >> 2) * (kBM * 128) + (kk & 3) * 32) >> 4);
            mma_bf16(d_tmem, a_lo + off, b_lo + off, d_hi, kk > 0 ? 1u : 0u);
          }
          mma_commit(&bars->s_full[t][sb]);
          mma_commit(&bars->k_empty[stage]);
        }
        if (!ok) break;
        mma_commit(&bars->q_empty);
        it += seg.nk;
        ++sg;
      }
      // all issued MMAs complete before tensor memory is released
      mma_commit(&bars->drain[t]);
      mbar_wait_bounded(&bars->drain[t], 0, nullptr, p.status);
    }
  } else {
    // ---------------------------------------------------- softmax-reduce --
    const int g = (warp - 2) >> 2;        // warpgroup: query tile t, column half ch
    const int t = g >> 1, half = g & 1;
    const int quad = warp & 3;            // TMEM lane quadrant this warp may access
    const int rowt = quad * 32 + lane;    // row within the tile
    const int rowu = t * kBM + rowt;      // row within the unit
    const uint32_t tlane = tmem + ((uint32_t)(quad * 32) << 16) + (uint32_t)(t * 2 * kBN + half * 64);
    int li0 = 0, sgi = 0;
    for (int it = it_begin; it < it_end;) {
      const Segment seg = segment_at(it, it_end, p.n_kt);
      RowStat st{-INFINITY, 0.f, 0.f};
      const uint8_t* mrow = kMask ? p.tmask + (long long)((seg.u / p.n_qp) / p.H) * p.Nk : nullptr;
      for (int j = 0; j < seg.nk; ++j) {
        const int li = li0 + j;
        const int sb = li & 1;
        const uint32_t sph = (uint32_t)((li >> 1) & 1);
        // the key mask does not depend on S: its bytes (lane l: keys c0 + l
        // and c0 + 32 + l) are loaded before the wait for the S buffer
        bool mb0 = false, mb1 = false;
        if constexpr (kMask) {
          const int cm0 = (seg.kt0 + j) * kBN + half * 64 + lane;
          mb0 = cm0 < p.Nk && mrow[cm0] != 0;
          mb1 = cm0 + 32 < p.Nk && mrow[cm0 + 32] != 0;
        }
        bool ok = (*abort_flag == 0) && mbar_wait_bounded(&bars->s_full[t][sb], sph, abort_flag, p.status);
        ok = __all_sync(0xffffffffu, ok);   // tcgen05.ld below is warp-collective
        if (ok) {
          fence_after();
          const uint32_t tb = tlane + (uint32_t)(sb * kBN);
          const int c0 = (seg.kt0 + j) * kBN + half * 64;   // first key of this half
          uint64_t* empty = &bars->s_empty[t][sb];
          // the kind is uniform over the warp: one branch per item
          if constexpr (kMask) {
            // the caller's key mask: bit l of w0 / w1 = key c0 + l / c0 + 32 + l
            const uint32_t w0 = __ballot_sync(0xffffffffu, mb0);
            const uint32_t w1 = __ballot_sync(0xffffffffu, mb1);
            const bool full = c0 + 64 <= p.Nk;
            if (full && (w0 & w1) == 0xffffffffu)
              softmax_item<kItemText>(tb, c0, p.Nk, p.L, p.c_log2, st, empty, lane);
            else if (full && (w0 | w1) == 0u)
              softmax_item<kItemImage>(tb, c0, p.Nk, p.L, p.c_log2, st, empty, lane);
            else
              softmax_item<kItemMasked>(tb, c0, p.Nk, p.L, p.c_log2, st, empty, lane, w0, w1);
          } else if (c0 + 64 <= p.Nk && c0 + 64 <= p.L)
            softmax_item<kItemText>(tb, c0, p.Nk, p.L, p.c_log2, st, empty, lane);
          else if (c0 + 64 <= p.Nk && c0 >= p.L)
            softmax_item<kItemImage>(tb, c0, p.Nk, p.L, p.c_log2, st, empty, lane);
          else
            softmax_item<kItemGeneral>(tb, c0, p.Nk, p.L, p.c_log2, st, empty, lane);
        } else {
          __syncwarp();
          if (lane == 0) mbar_arrive(&bars->s_empty[t][sb]);
        }
      }
      // the two column halves of this tile's rows meet in shared memory
      // (a buffer per segment parity, so one barrier per segment suffices);
      // half 0 merges them into the CTA's piece of the unit and takes it
      // through the merge across CTAs
      float* xs = xch + (((sgi & 1) * kQTiles + t) * kBM + rowt) * 3;
      if (half == 1) {
        xs[0] = st.m;
        xs[1] = st.la;
        xs[2] = st.lt;
      }
      if (t == 0)   // the 8 softmax warps of query tile t (constant ids)
        bar_sync(1, 8 * 32);
      else
        bar_sync(2, 8 * 32);
      if (half == 0) {
        merge_stat(st, xs[0], xs[1], xs[2]);
        unit_piece_done(p, seg.u, rowu, st, abort_flag);
      }
      ++sgi;
      li0 += seg.nk;
      it += seg.nk;
    }
  }

  fence_before();
  __syncthreads();
  if (warp == 1) {
    fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                 "r"(kTmemCols));
  }
}

struct Plan {
  int n_qp, n_kt, n_units, max_parts, grid;
  long long total, per;
  size_t acc_bytes, part_bytes, bytes;
};

size_t align256(size_t x) { return (x + 255) & ~static_cast<size_t>(255); }

Plan make_plan(int B, int H, int M, int Nk, int num_sms) {
  Plan pl{};
  pl.n_qp = (M + kUnitRows - 1) / kUnitRows;
  pl.n_kt = (Nk + kBN - 1) / kBN;
  pl.n_units = B * H * pl.n_qp;
  pl.total = (long long)pl.n_units * pl.n_kt;
  const int sms = num_sms > 0 ? num_sms : 1;
  pl.per = (pl.total + sms - 1) / sms;
  if (pl.per < 1) pl.per = 1;
  pl.grid = (int)((pl.total + pl.per - 1) / pl.per);
  pl.max_parts = (int)((pl.n_kt + pl.per - 1) / pl.per) + 1;
  // [head-sum words][pieces: two words per row], all zero between calls
  pl.acc_bytes = align256(sizeof(unsigned long long) * (size_t)B * pl.n_qp * kUnitRows);
  pl.part_bytes = align256(2 * sizeof(unsigned long long) * (size_t)pl.n_units * pl.max_parts * kUnitRows);
  pl.bytes = pl.acc_bytes + pl.part_bytes;
  return pl;
}

// All-shared carveout and the dynamic shared-memory opt-in of one instance.
template <auto Kernel, int D>
cudaError_t smem_attrs() {
  cudaError_t e = cudaFuncSetAttribute(Kernel, cudaFuncAttributePreferredSharedMemoryCarveout,
                                       cudaSharedmemCarveoutMaxShared);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(Kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem_bytes<D>());
  return e;
}

// The dynamic shared-memory opt-in is a per-device function attribute: set it
// once per device (first call, outside any stream capture in practice).
cudaError_t set_smem_once() {
  static int done[64] = {};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev >= 0 && dev < 64 && __atomic_load_n(&done[dev], __ATOMIC_ACQUIRE)) return cudaSuccess;
  // one carveout (all shared) for every kernel of the path, so that kernels
  // launched as programmatic dependents can share an SM with this one
  e = smem_attrs<spatial_tc_kernel<128, false>, 128>();
  if (e == cudaSuccess) e = smem_attrs<spatial_tc_kernel<128, true>, 128>();
  if (e == cudaSuccess) e = smem_attrs<spatial_tc_kernel<64, false>, 64>();
  if (e == cudaSuccess) e = smem_attrs<spatial_tc_kernel<64, true>, 64>();
  if (e == cudaSuccess && dev >= 0 && dev < 64) __atomic_store_n(&done[dev], 1, __ATOMIC_RELEASE);
  return e;
}

}  // namespace

bool spatial_tc_eligible(const SpatialArgs& a) {
  if (a.dt != AVITS_BF16) return false;
  if (a.d != 64 && a.d != 128) return false;
  if ((reinterpret_cast<uintptr_t>(a.q) | reinterpret_cast<uintptr_t>(a.k)) & 15u) return false;
  if (!strides_ok(a.B, a.H, a.q_sb, a.q_sh, a.q_sn)) return false;
  if (!strides_ok(a.B, a.H, a.k_sb, a.k_sh, a.k_sn)) return false;
  if (!(a.scale > 0.f)) return false;
  if (a.H > 255) return false;   // the head count of the fixed-point head sum is one byte
  const long long n_qp = (a.M + kUnitRows - 1) / kUnitRows, n_kt = (a.Nk + kBN - 1) / kBN;
  if ((long long)a.B * a.H * n_qp * (n_kt + 1) >= (1ll << 31)) return false;
  return encode_fn() != nullptr;
}

size_t spatial_tc_workspace(int B, int H, int M, int Nk, int d, int num_sms) {
  (void)d;
  return make_plan(B, H, M, Nk, num_sms).bytes;
}

size_t spatial_tc_zeroed_bytes(int B, int H, int M, int Nk, int d, int num_sms) {
  (void)d;
  return make_plan(B, H, M, Nk, num_sms).bytes;
}

cudaError_t launch_spatial_tc(const SpatialArgs& a, int num_sms, cudaStream_t s,
                              const LaunchHook* between) {
  const Plan pl = make_plan(a.B, a.H, a.M, a.Nk, num_sms);
  if (a.ws_bytes < pl.bytes || a.ws == nullptr) return cudaErrorInvalidValue;
  CUtensorMap mq, mk;
  if (!make_map(&mq, a.q, a.B, a.H, a.M, a.d, a.q_sb, a.q_sh, a.q_sn)) return cudaErrorInvalidValue;
  if (!make_map(&mk, a.k, a.B, a.H, a.Nk, a.d, a.k_sb, a.k_sh, a.k_sn)) return cudaErrorInvalidValue;
  uint8_t* ws = static_cast<uint8_t*>(a.ws);
  TcParams p{};
  p.B = a.B; p.H = a.H; p.M = a.M; p.Nk = a.Nk; p.L = a.L;
  p.n_qp = pl.n_qp; p.n_kt = pl.n_kt; p.n_units = pl.n_units;
  p.total = (int)pl.total; p.per = (int)pl.per; p.max_parts = pl.max_parts;
  p.c_log2 = a.scale * 1.4426950408889634f;
  p.weight = a.weight;
  p.accumulate = a.accumulate;
  p.A = a.A;
  p.lse = a.lse;
  p.acc = reinterpret_cast<unsigned long long*>(ws);
  p.part = reinterpret_cast<unsigned long long*>(ws + pl.acc_bytes);
  p.rows_pad = pl.n_qp * kUnitRows;
  p.status = a.status;
  p.tmask = a.tmask;
  p.lse_all = a.lse_all;
  cudaError_t e = set_smem_once();
  if (e != cudaSuccess) return e;
  const bool masked = p.tmask != nullptr;
  if (a.d == 128)
    e = launch_pdl(masked ? spatial_tc_kernel<128, true> : spatial_tc_kernel<128, false>,
                   dim3(pl.grid), dim3(kThreads), smem_bytes<128>(), s, mq, mk, p);
  else
    e = launch_pdl(masked ? spatial_tc_kernel<64, true> : spatial_tc_kernel<64, false>,
                   dim3(pl.grid), dim3(kThreads), smem_bytes<64>(), s, mq, mk, p);
  if (e != cudaSuccess) return e;
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  if (between) {
    // work that may overlap the main kernel (launched as its programmatic
    // dependent); it must not complete before the main kernel does
    e = (*between)(s);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

}  // namespace avits
