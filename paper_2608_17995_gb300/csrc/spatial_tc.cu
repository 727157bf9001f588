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
// ranges, one per CTA, so every SM gets the same number of MMA tiles.  A unit
// cut between CTAs leaves per-row partial (max, sums) in the workspace; the
// last CTA to finish the unit (atomic ticket) merges them in slot order, and
// the last unit of a (b, row block) to finish sums the head masses in head
// order.  Both tickets are reset by their last arriver, so results do not
// depend on CTA timing and the workspace is left zeroed.
//
// Roles (10 warps):
//   warp 0        TMA producer: Q tile pair once per unit (64 KB for d=128),
//                 K tiles through a 4-stage ring, 128-byte swizzled.
//   warp 1        MMA issuer: S = Q K^T with tcgen05.mma kind::f16 (bf16 in,
//                 fp32 accumulate in tensor memory), 128x128 per tile, two S
//                 buffers per Q tile (4 x 128 of the 512 TMEM columns).
//   warps 2-5     softmax-reduce of Q tile 0, warps 6-9 of Q tile 1: one TMEM
//                 lane (= one query row) per thread, 32 columns per
//                 tcgen05.ld, exp2 on the MUFU with a running max; the text
//                 keys come first, so the text sum is a prefix of the row sum.
// Every wait is bounded (avits_common.cuh); on a timeout all roles stop
// issuing, drain what they issued, release tensor memory and exit.
#include <cuda.h>

#include "avits_common.cuh"
#include "avits_internal.h"

namespace avits {
namespace {

constexpr int kBM = 128;       // query rows per tile (= TMEM lanes)
constexpr int kBN = 128;       // keys per tile
constexpr int kQTiles = 2;     // query tiles per unit
constexpr int kUnitRows = kBM * kQTiles;
constexpr int kThreads = 320;
constexpr int kTmemCols = 512;
constexpr uint32_t kIdesc = (1u << 4)                       // D: fp32
                            | (1u << 7) | (1u << 10)        // A, B: bf16
                            | ((uint32_t)(kBN >> 3) << 17)  // N
                            | ((uint32_t)(kBM >> 4) << 24); // M

template <int D>
struct Cfg {
  static constexpr int kCB = D / 64;                   // 128-byte column blocks per row
  static constexpr int kTileBytes = kCB * kBM * 128;   // one 128-row bf16 tile
  static constexpr int kStages = (D == 128) ? 4 : 8;
  static constexpr int kQBytes = kQTiles * kTileBytes;
  static constexpr int kKBytes = kStages * kTileBytes;
};

struct Bars {
  uint64_t q_full, q_empty;
  uint64_t k_full[8], k_empty[8];
  uint64_t s_full[kQTiles][2], s_empty[kQTiles][2];
  uint64_t drain;
  uint32_t tmem_base;
  int abort;
  int last_unit, last_group;
};

template <int D>
constexpr int smem_bytes() {
  return Cfg<D>::kQBytes + Cfg<D>::kKBytes + (int)sizeof(Bars) + 1024;
}

struct TcParams {
  int B, H, M, Nk, L;
  int n_qp, n_kt, n_units;
  long long total, per;
  int max_parts;
  float c_log2, weight;
  int accumulate;
  float* A;
  float* lse;
  float* part;      // [n_units][max_parts][256][3]
  float* mass;      // [B*H][n_qp*256]
  int* unit_cnt;    // [n_units]
  int* grp_cnt;     // [B*n_qp]
  unsigned int* status;
};

// ------------------------------------------------------------------ PTX ----
__device__ __forceinline__ void tma_load_4d(void* dst, const CUtensorMap* map, int c0, int c1,
                                            int c2, int c3, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.4d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3, %4, %5}], [%6];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(c2), "r"(c3),
      "r"(smem_u32(bar))
      : "memory");
}

// Shared-memory matrix descriptor: K-major operand, 128-byte swizzle, 8-row
// core-matrix groups 1024 B apart.
__device__ __forceinline__ uint64_t sw128_desc(const void* p) {
  const uint32_t a = smem_u32(p);
  return (uint64_t)((a >> 4) & 0x3FFFu) | ((uint64_t)1 << 16) | ((uint64_t)(1024 >> 4) << 32) |
         ((uint64_t)1 << 46) | ((uint64_t)2 << 61);
}

__device__ __forceinline__ void mma_bf16(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t acc) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a), "l"(b), "r"(kIdesc), "r"(acc));
}

__device__ __forceinline__ void mma_commit(uint64_t* bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
          smem_u32(bar))
      : "memory");
}

__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

#define AVITS_R8(b) "=r"(r[b]), "=r"(r[b + 1]), "=r"(r[b + 2]), "=r"(r[b + 3]), \
                    "=r"(r[b + 4]), "=r"(r[b + 5]), "=r"(r[b + 6]), "=r"(r[b + 7])
#define AVITS_W8(b) "+r"(r[b]), "+r"(r[b + 1]), "+r"(r[b + 2]), "+r"(r[b + 3]), \
                    "+r"(r[b + 4]), "+r"(r[b + 5]), "+r"(r[b + 6]), "+r"(r[b + 7])

// 32 consecutive fp32 columns of this thread's TMEM lane.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, "
      "%11, %12, %13, %14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, "
      "%28, %29, %30, %31}, [%32];"
      : AVITS_R8(0), AVITS_R8(8), AVITS_R8(16), AVITS_R8(24)
      : "r"(taddr));
}

// Completes the thread's outstanding tcgen05.ld; the registers are tied to
// the wait so no use can be scheduled before it.
__device__ __forceinline__ void tmem_wait(uint32_t (&r)[32]) {
  asm volatile("tcgen05.wait::ld.sync.aligned;"
               : AVITS_W8(0), AVITS_W8(8), AVITS_W8(16), AVITS_W8(24)
               :
               : "memory");
}

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

__device__ __forceinline__ void softmax_bar() { asm volatile("bar.sync 1, 256;" ::: "memory"); }

// Running row statistics in the log2 domain: x = c_log2 * (q.k).
struct RowStat {
  float m, la, lt;
};

// One 32-column chunk: col0 = index of its first key.
__device__ __forceinline__ void process_chunk(const uint32_t (&r)[32], int col0, int Nk, int L,
                                              float c, RowStat& st) {
  float v[32];
#pragma unroll
  for (int e = 0; e < 32; ++e) v[e] = __uint_as_float(r[e]);
  const int nvalid = Nk - col0;
  if (nvalid < 32) {
#pragma unroll
    for (int e = 0; e < 32; ++e)
      if (e >= nvalid) v[e] = -INFINITY;
  }
  float t[11];
#pragma unroll
  for (int e = 0; e < 10; ++e) t[e] = max3(v[3 * e], v[3 * e + 1], v[3 * e + 2]);
  t[10] = fmaxf(v[30], v[31]);
  const float u0 = max3(t[0], t[1], t[2]), u1 = max3(t[3], t[4], t[5]);
  const float u2 = max3(t[6], t[7], t[8]), u3 = fmaxf(t[9], t[10]);
  const float cmax = fmaxf(fmaxf(u0, u1), fmaxf(u2, u3));
  if (cmax == -INFINITY) return;
  const float mx = cmax * c;
  if (mx > st.m) {
    const float corr = ex2(st.m - mx);
    st.la *= corr;
    st.lt *= corr;
    st.m = mx;
  }
  const float nm = -st.m;
  float s[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
  for (int e = 0; e < 32; ++e) s[e & 3] += ex2(fmaf(v[e], c, nm));
  const float cs = (s[0] + s[1]) + (s[2] + s[3]);
  st.la += cs;
  if (col0 + 32 <= L) {
    st.lt += cs;
  } else if (col0 < L) {
    float ts = 0.f;
#pragma unroll
    for (int e = 0; e < 32; ++e)
      if (col0 + e < L) ts += ex2(fmaf(v[e], c, nm));
    st.lt += ts;
  }
}

struct Segment {
  int u, kt0, nk;
};

__device__ __forceinline__ Segment segment_at(long long it, long long it_end, int n_kt) {
  Segment s;
  s.u = (int)(it / n_kt);
  s.kt0 = (int)(it - (long long)s.u * n_kt);
  const long long left = it_end - it;
  s.nk = (int)((long long)(n_kt - s.kt0) < left ? (n_kt - s.kt0) : left);
  return s;
}

template <int D>
__global__ void __launch_bounds__(kThreads, 1)
spatial_tc_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                  const TcParams p) {
  using C = Cfg<D>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* sQ = smem;
  uint8_t* sK = smem + C::kQBytes;
  Bars* bars = reinterpret_cast<Bars*>(sK + C::kKBytes);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const long long it_begin = (long long)blockIdx.x * p.per;
  long long it_end = it_begin + p.per;
  if (it_end > p.total) it_end = p.total;
  if (it_begin >= it_end) return;   // block-uniform

  if (threadIdx.x == 0) {
    mbar_init(&bars->q_full, 1);
    mbar_init(&bars->q_empty, 1);
    for (int s = 0; s < C::kStages; ++s) {
      mbar_init(&bars->k_full[s], 1);
      mbar_init(&bars->k_empty[s], 1);
    }
    for (int t = 0; t < kQTiles; ++t)
      for (int b = 0; b < 2; ++b) {
        mbar_init(&bars->s_full[t][b], 1);
        mbar_init(&bars->s_empty[t][b], 4);
      }
    mbar_init(&bars->drain, 1);
    bars->abort = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(&bars->tmem_base)),
                 "r"(kTmemCols));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = bars->tmem_base;
  volatile int* abort_flag = &bars->abort;

  if (warp == 0) {
    // ------------------------------------------------------ TMA producer --
    if (lane == 0) {
      asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmQ)) : "memory");
      asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmK)) : "memory");
      bool ok = true;
      long long li = 0;
      int sg = 0;
      for (long long it = it_begin; it < it_end && ok;) {
        const Segment seg = segment_at(it, it_end, p.n_kt);
        const int bh = seg.u / p.n_qp, qp = seg.u - bh * p.n_qp;
        const int b = bh / p.H, h = bh - b * p.H;
        if (sg > 0) ok = mbar_wait_bounded(&bars->q_empty, (sg - 1) & 1, abort_flag, p.status);
        if (!ok) break;
        mbar_arrive_expect_tx(&bars->q_full, C::kQBytes);
        for (int t = 0; t < kQTiles; ++t)
          for (int cb = 0; cb < C::kCB; ++cb)
            tma_load_4d(sQ + t * C::kTileBytes + cb * (kBM * 128), &tmQ, cb * 64,
                        qp * kUnitRows + t * kBM, h, b, &bars->q_full);
        for (int j = 0; j < seg.nk; ++j, ++li) {
          const int stage = (int)(li % C::kStages);
          const uint32_t ph = (uint32_t)((li / C::kStages) & 1);
          ok = mbar_wait_bounded(&bars->k_empty[stage], ph ^ 1u, abort_flag, p.status);
          if (!ok) break;
          mbar_arrive_expect_tx(&bars->k_full[stage], C::kTileBytes);
          for (int cb = 0; cb < C::kCB; ++cb)
            tma_load_4d(sK + stage * C::kTileBytes + cb * (kBM * 128), &tmK, cb * 64,
                        (seg.kt0 + j) * kBN, h, b, &bars->k_full[stage]);
        }
        it += seg.nk;
        ++sg;
      }
      if (!ok) {
        // drain the copies still in flight before the CTA exits
        if (sg > 0) mbar_wait_bounded(&bars->q_full, (sg - 1) & 1, nullptr, p.status);
        for (int s = 0; s < C::kStages; ++s) {
          const long long armed = li - s;   // items issued on stage s: li - s > 0
          if (armed > 0) {
            const long long last = (armed - 1) / C::kStages;
            mbar_wait_bounded(&bars->k_full[s], (uint32_t)(last & 1), nullptr, p.status);
          }
        }
      }
    }
  } else if (warp == 1) {
    // --------------------------------------------------------- MMA issuer --
    if (lane == 0) {
      bool ok = true;
      long long li = 0;
      int sg = 0;
      for (long long it = it_begin; it < it_end && ok;) {
        const Segment seg = segment_at(it, it_end, p.n_kt);
        ok = mbar_wait_bounded(&bars->q_full, sg & 1, abort_flag, p.status);
        if (!ok) break;
        tc_fence_after();
        for (int j = 0; j < seg.nk && ok; ++j, ++li) {
          const int stage = (int)(li % C::kStages);
          const uint32_t ph = (uint32_t)((li / C::kStages) & 1);
          const int sb = (int)(li & 1);
          const uint32_t sph = (uint32_t)((li >> 1) & 1);
          ok = mbar_wait_bounded(&bars->k_full[stage], ph, abort_flag, p.status);
          if (!ok) break;
          tc_fence_after();
          for (int t = 0; t < kQTiles; ++t) {
            ok = mbar_wait_bounded(&bars->s_empty[t][sb], sph ^ 1u, abort_flag, p.status);
            if (!ok) break;
            tc_fence_after();
            const uint32_t d_tmem = tmem + (uint32_t)((t * 2 + sb) * kBN);
            const uint8_t* qa = sQ + t * C::kTileBytes;
            const uint8_t* kb = sK + stage * C::kTileBytes;
#pragma unroll
            for (int kk = 0; kk < D / 16; ++kk) {
              const int off = (kk >> 2) * (kBM * 128) + (kk & 3) * 32;
              mma_bf16(d_tmem, sw128_desc(qa + off), sw128_desc(kb + off), kk > 0 ? 1u : 0u);
            }
            mma_commit(&bars->s_full[t][sb]);
          }
          if (!ok) break;
          mma_commit(&bars->k_empty[stage]);
        }
        if (!ok) break;
        mma_commit(&bars->q_empty);
        it += seg.nk;
        ++sg;
      }
      // all issued MMAs complete before tensor memory is released
      mma_commit(&bars->drain);
      mbar_wait_bounded(&bars->drain, 0, nullptr, p.status);
    }
  } else {
    // ---------------------------------------------------- softmax-reduce --
    const int t = (warp - 2) >> 2;        // query tile of this warpgroup
    const int quad = warp & 3;            // TMEM lane quadrant this warp may access
    const int rowt = quad * 32 + lane;    // row within the tile
    const int rowu = t * kBM + rowt;      // row within the unit
    const int sm_tid = threadIdx.x - 64;  // 0..255
    const float ln2 = 0.69314718055994530942f;
    long long li = 0;
    for (long long it = it_begin; it < it_end;) {
      const Segment seg = segment_at(it, it_end, p.n_kt);
      RowStat st{-INFINITY, 0.f, 0.f};
      for (int j = 0; j < seg.nk; ++j, ++li) {
        const int sb = (int)(li & 1);
        const uint32_t sph = (uint32_t)((li >> 1) & 1);
        bool ok = (*abort_flag == 0) && mbar_wait_bounded(&bars->s_full[t][sb], sph, abort_flag, p.status);
        ok = __all_sync(0xffffffffu, ok);   // tcgen05.ld below is warp-collective
        if (ok) {
          tc_fence_after();
          const int kbase = (seg.kt0 + j) * kBN;
          const uint32_t ta = tmem + ((uint32_t)(quad * 32) << 16) + (uint32_t)((t * 2 + sb) * kBN);
          uint32_t ra[32], rb[32];
          tmem_ld32(ta, ra);
          tmem_wait(ra);
          tmem_ld32(ta + 32, rb);
          process_chunk(ra, kbase, p.Nk, p.L, p.c_log2, st);
          tmem_wait(rb);
          tmem_ld32(ta + 64, ra);
          process_chunk(rb, kbase + 32, p.Nk, p.L, p.c_log2, st);
          tmem_wait(ra);
          tmem_ld32(ta + 96, rb);
          process_chunk(ra, kbase + 64, p.Nk, p.L, p.c_log2, st);
          tmem_wait(rb);
          process_chunk(rb, kbase + 96, p.Nk, p.L, p.c_log2, st);
          tc_fence_before();
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&bars->s_empty[t][sb]);
      }

      // ---- epilogue of this unit segment (all 256 softmax threads) ----
      const int u = seg.u;
      const int bh = u / p.n_qp, qp = u - bh * p.n_qp;
      const int b = bh / p.H;
      const int row = qp * kUnitRows + rowu;
      const long long first = ((long long)u * p.n_kt) / p.per;
      const long long last = ((long long)(u + 1) * p.n_kt - 1) / p.per;
      const int nparts = (int)(last - first + 1);
      bool have = true;
      if (nparts > 1) {
        const int slot = (int)(blockIdx.x - first);
        float* pp = p.part + (((long long)u * p.max_parts + slot) * kUnitRows + rowu) * 3;
        pp[0] = st.m;
        pp[1] = st.la;
        pp[2] = st.lt;
        __threadfence();
        softmax_bar();
        if (sm_tid == 0) {
          const int prev = atomicAdd(&p.unit_cnt[u], 1);
          bars->last_unit = (prev == nparts - 1);
          if (prev == nparts - 1) p.unit_cnt[u] = 0;
        }
        softmax_bar();
        have = bars->last_unit != 0;
        if (have) {
          __threadfence();
          float m = -INFINITY;
          for (int s = 0; s < nparts; ++s) {
            const float* q = p.part + (((long long)u * p.max_parts + s) * kUnitRows + rowu) * 3;
            m = fmaxf(m, __ldcg(q));
          }
          float la = 0.f, lt = 0.f;
          for (int s = 0; s < nparts; ++s) {
            const float* q = p.part + (((long long)u * p.max_parts + s) * kUnitRows + rowu) * 3;
            const float ms = __ldcg(q);
            const float f = (ms == -INFINITY) ? 0.f : ex2(ms - m);
            la += __ldcg(q + 1) * f;
            lt += __ldcg(q + 2) * f;
          }
          st.m = m;
          st.la = la;
          st.lt = lt;
        }
      }
      if (have) {
        const float mass = st.lt / st.la;
        if (p.lse && row < p.M) {
          float* lp = p.lse + ((long long)bh * p.M + row) * 2;
          lp[0] = (st.m + __log2f(st.la)) * ln2;
          lp[1] = st.lt > 0.f ? (st.m + __log2f(st.lt)) * ln2 : -INFINITY;
        }
        if (p.H == 1) {
          if (row < p.M) {
            const float a = p.weight * mass;
            float* ap = p.A + (long long)b * p.M + row;
            *ap = p.accumulate ? *ap + a : a;
          }
        } else {
          p.mass[(long long)bh * (p.n_qp * kUnitRows) + row] = mass;
          __threadfence();
        }
      }
      // head reduction: the last of the H units of (b, qp) to finish sums
      if (p.H > 1) {
        // only CTAs that finalised the unit take part in the group ticket;
        // `have` is uniform over the 256 threads
        if (have) {
          softmax_bar();
          if (sm_tid == 0) {
            int* gc = &p.grp_cnt[b * p.n_qp + qp];
            const int prev = atomicAdd(gc, 1);
            bars->last_group = (prev == p.H - 1);
            if (prev == p.H - 1) *gc = 0;
          }
          softmax_bar();
          if (bars->last_group) {
            __threadfence();
            float sum = 0.f;
            const float* mp = p.mass + (long long)b * p.H * (p.n_qp * kUnitRows) + row;
            for (int hh = 0; hh < p.H; ++hh) sum += __ldcg(mp + (long long)hh * p.n_qp * kUnitRows);
            if (row < p.M) {
              const float a = p.weight * (sum / (float)p.H);
              float* ap = p.A + (long long)b * p.M + row;
              *ap = p.accumulate ? *ap + a : a;
            }
          }
        }
      }
      it += seg.nk;
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                 "r"(kTmemCols));
  }
}

// ------------------------------------------------------------------ host ---
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
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

// Element strides of a [B,H,rows,d] view -> byte strides for the tensor map;
// a dimension of extent 1 gets a packed stride (its stride is never used).
bool make_map(CUtensorMap* map, const void* base, int B, int H, int rows, int d, int64_t sb,
              int64_t sh, int64_t sn) {
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

struct Plan {
  int n_qp, n_kt, n_units, max_parts, grid;
  long long total, per;
  size_t off_unit, off_grp, off_part, off_mass, bytes;
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
  size_t o = 0;
  pl.off_unit = o;
  o = align256(o + sizeof(int) * (size_t)pl.n_units);
  pl.off_grp = o;
  o = align256(o + sizeof(int) * (size_t)B * pl.n_qp);
  pl.off_part = o;
  o = align256(o + sizeof(float) * 3 * (size_t)pl.n_units * pl.max_parts * kUnitRows);
  pl.off_mass = o;
  o = align256(o + sizeof(float) * (size_t)B * H * pl.n_qp * kUnitRows);
  pl.bytes = o;
  return pl;
}

bool strides_ok(int B, int H, int64_t sb, int64_t sh, int64_t sn) {
  if (sn % 8 != 0 || sn <= 0) return false;
  if (H > 1 && (sh % 8 != 0 || sh <= 0)) return false;
  if (B > 1 && (sb % 8 != 0 || sb <= 0)) return false;
  return true;
}

// The dynamic shared-memory opt-in is a per-device function attribute: set it
// once per device (first call, outside any stream capture in practice).
cudaError_t set_smem_once() {
  static int done[64] = {};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev >= 0 && dev < 64 && __atomic_load_n(&done[dev], __ATOMIC_ACQUIRE)) return cudaSuccess;
  e = cudaFuncSetAttribute(spatial_tc_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           smem_bytes<128>());
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(spatial_tc_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             smem_bytes<64>());
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
  return encode_fn() != nullptr;
}

size_t spatial_tc_workspace(int B, int H, int M, int Nk, int d, int num_sms) {
  (void)d;
  return make_plan(B, H, M, Nk, num_sms).bytes;
}

cudaError_t launch_spatial_tc(const SpatialArgs& a, int num_sms, cudaStream_t s) {
  const Plan pl = make_plan(a.B, a.H, a.M, a.Nk, num_sms);
  if (a.ws_bytes < pl.bytes || a.ws == nullptr) return cudaErrorInvalidValue;
  CUtensorMap mq, mk;
  if (!make_map(&mq, a.q, a.B, a.H, a.M, a.d, a.q_sb, a.q_sh, a.q_sn)) return cudaErrorInvalidValue;
  if (!make_map(&mk, a.k, a.B, a.H, a.Nk, a.d, a.k_sb, a.k_sh, a.k_sn)) return cudaErrorInvalidValue;
  uint8_t* ws = static_cast<uint8_t*>(a.ws);
  TcParams p{};
  p.B = a.B; p.H = a.H; p.M = a.M; p.Nk = a.Nk; p.L = a.L;
  p.n_qp = pl.n_qp; p.n_kt = pl.n_kt; p.n_units = pl.n_units;
  p.total = pl.total; p.per = pl.per; p.max_parts = pl.max_parts;
  p.c_log2 = a.scale * 1.4426950408889634f;
  p.weight = a.weight;
  p.accumulate = a.accumulate;
  p.A = a.A;
  p.lse = a.lse;
  p.unit_cnt = reinterpret_cast<int*>(ws + pl.off_unit);
  p.grp_cnt = reinterpret_cast<int*>(ws + pl.off_grp);
  p.part = reinterpret_cast<float*>(ws + pl.off_part);
  p.mass = reinterpret_cast<float*>(ws + pl.off_mass);
  p.status = a.status;
  cudaError_t e = set_smem_once();
  if (e != cudaSuccess) return e;
  if (a.d == 128)
    spatial_tc_kernel<128><<<pl.grid, kThreads, smem_bytes<128>(), s>>>(mq, mk, p);
  else
    spatial_tc_kernel<64><<<pl.grid, kThreads, smem_bytes<64>(), s>>>(mq, mk, p);
  return cudaGetLastError();
}

}  // namespace avits
