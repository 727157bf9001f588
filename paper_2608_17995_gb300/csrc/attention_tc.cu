// attention_tc.cu — the joint-attention forward of a double-stream block
// (Eq. 4-5, Sec. 3.3.1) on the sm_103a tensor cores, with the spatial score
// of Eq. 3 read off the same softmax.
//
// For batch b, head h and query row i of the joint sequence [C; Z]:
//   O_i      = sum_j softmax_j(scale * q_i . k_j) v_j        (all Nk keys)
//   lse_i    = log sum_j exp(scale * q_i . k_j), over all keys and over the
//              text keys (the first L)
//   A_i     (+)= weight * mean_h exp(lse_txt_i - lse_all_i)  (Eq. 5, Eq. 3)
// The text mass Eq. 5 extracts is a by-product of the softmax the block
// computes anyway: the only extra work is one running sum per row.
//
// Work decomposition (persistent, one CTA per SM): unit = (b, h, 256 query
// rows = two 128-row tiles); CTA c takes units c, c + grid, ...  Each unit
// runs over all key tiles (128 keys), so O and the row statistics stay in
// the CTA and no partial results cross CTAs (except Eq. 3's head sum).
//
// Tensor memory (512 columns): one S buffer of 128 columns that the two query
// tiles take in turn (S_0(g), S_1(g), S_0(g+1), ...), P_t as bf16 pairs (64
// columns per tile), O_t (D columns per tile).  S is free as soon as its
// softmax has loaded it, so the other tile's S runs on the tensor pipe while
// this one's exponentials are computed; P never goes through shared memory
// (the PV product reads it from tensor memory), which leaves shared memory
// for Q, a 4-stage K / V ring and the O staging: per key tile and SM the
// operand reads are 128 KB (S) + 64 KB (V), the copies 64 KB.
//
// Roles (12 warps):
//   warp 0       TMA producer: Q tiles, then the K and V tiles through a
//                4-stage ring in the order the MMAs consume them (K_0, K_1,
//                V_0, K_2, V_1, ...), 128-byte swizzle; a stage is refilled
//                two key tiles after its last use.
//   warps 1, 2   MMA issuers of query tile 0 / 1 (warp 1 owns tensor
//                memory): for key tile g, S_t(g) = Q_t K_g^T (from shared
//                memory) once the S before it has been loaded, then O_t +=
//                P_t(g-1) V_(g-1) (A = P_t from tensor memory, the
//                tcgen05.mma TS form; V read in its natural [keys, d] layout
//                as an MN-major shared-memory operand, no transpose copy) once
//                that P has been written.
//   warp 3       no role.
//   warps 4-7    softmax and epilogue of query tile 0, warps 8-11 of tile 1:
//                one row per thread (TMEM lane); the row's 128 S columns are
//                loaded into registers and the S buffer released; the row
//                maximum; the running maximum is raised only when a key
//                tile's maximum exceeds it by more than 2^8 (P <= 256
//                otherwise, no loss in bf16 or the fp32 accumulator), and then
//                l and O are rescaled (O in tensor memory, by the whole warp);
//                the exponentials (packed FMA + MUFU), the fp32 sums over all
//                keys and over the text keys (the only addition the score
//                needs) and the bf16 P row, written to tensor memory once the
//                previous PV product has read P_t.  The epilogue divides O by
//                the row sum and stores it 64 columns at a time through a
//                swizzled staging block with a bulk tensor copy.
// Every wait is bounded (avits_common.cuh); after a timeout every role skips
// its remaining work, drains what it issued and the CTA releases tensor
// memory and exits.
#include <cuda.h>

#include "avits_common.cuh"
#include "avits_internal.h"
#include "tc_common.cuh"

namespace avits {
namespace {

using namespace tc;

constexpr int kBM = 128;            // query rows per tile (= TMEM lanes)
constexpr int kBN = 128;            // keys per tile
constexpr int kQTiles = 2;          // query tiles per unit
constexpr int kUnitRows = kBM * kQTiles;
constexpr int kThreads = 12 * 32;
constexpr int kTmemCols = 512;
constexpr float kTau = 8.f;         // lazy rescale threshold (log2 units)
constexpr uint32_t kIdescS = idesc_bf16(kBM, kBN, false);

template <int D>
struct Cfg {
  static constexpr int kCB = D / 64;                   // 128-byte column blocks per row
  static constexpr int kTileBytes = kCB * kBM * 128;   // one 128-row bf16 tile
  static constexpr int kStages = (D == 128) ? 4 : 8;   // K / V ring
  static constexpr int kQBytes = kQTiles * kTileBytes;
  static constexpr int kKVBytes = kStages * kTileBytes;
  static constexpr uint32_t kIdescPV = idesc_bf16(kBM, D, true);
};
// O staging at a unit's end: per query tile one 128-row x 64-column bf16
// block (128-byte swizzle), stored with a bulk tensor copy per 64 columns
constexpr int kStageTileBytes = kBM * 128;
constexpr int kStageBytes = kQTiles * kStageTileBytes;
constexpr int kMaxStages = 8;
// Tensor memory columns: the S buffer both query tiles share, then P_t (bf16
// pairs, 64 columns per tile), then O_t (D columns per tile).
constexpr int kColS = 0, kColP = kBN, kColO = kBN + kQTiles * (kBN / 2);

struct Bars {
  uint64_t q_full[kQTiles], q_empty[kQTiles];
  uint64_t kv_full[kMaxStages], kv_empty[kMaxStages];
  uint64_t s_full[kQTiles], s_empty[kQTiles], p_full[kQTiles], pv_done[kQTiles];
  uint64_t o_full[kQTiles], o_empty[kQTiles], drain[kQTiles];
  uint32_t tmem_base;
  int abort;
};

template <int D>
constexpr int smem_bytes() {
  return Cfg<D>::kQBytes + Cfg<D>::kKVBytes + kStageBytes + (int)sizeof(Bars) + 1024;
}

struct AttnParams {
  int B, H, Mq, Nk, L;
  int n_qp, n_kt, n_units;
  float c_log2, weight;
  int accumulate;
  float* A;                   // [B,Mq] or NULL
  float* lse;                 // [B,H,Mq,2] or NULL
  unsigned long long* acc;    // [B][n_qp * 256] head-sum words (A != NULL)
  int rows_pad;
  unsigned int* status;
};

// WG-wide AND of v over the `count` threads of named barrier `id`.
__device__ __forceinline__ bool bar_and(int id, int count, bool v) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\t"
      "setp.ne.u32 p, %1, 0;\n\t"
      "bar.red.and.pred q, %2, %3, p;\n\t"
      "selp.u32 %0, 1, 0, q;\n\t}"
      : "=r"(r)
      : "r"((uint32_t)v), "r"(id), "r"(count)
      : "memory");
  return r != 0;
}

// Row maximum of 32 S columns whose first key is col0; keys >= Nk are left
// out (kFull: all 32 are valid).
template <bool kFull>
__device__ __forceinline__ float chunk_max(const uint32_t (&r)[32], int col0, int Nk) {
  float v[32];
#pragma unroll
  for (int e = 0; e < 32; ++e) v[e] = __uint_as_float(r[e]);
  if (!kFull) {
#pragma unroll
    for (int e = 0; e < 32; ++e)
      if (col0 + e >= Nk) v[e] = -INFINITY;
  }
  float t[11];
#pragma unroll
  for (int g = 0; g < 10; ++g) t[g] = max3(v[3 * g], v[3 * g + 1], v[3 * g + 2]);
  t[10] = fmaxf(v[30], v[31]);
  const float u0 = max3(t[0], t[1], t[2]), u1 = max3(t[3], t[4], t[5]);
  const float u2 = max3(t[6], t[7], t[8]);
  return fmaxf(max3(u0, u1, u2), fmaxf(t[9], t[10]));
}

// O_t row *= f (D fp32 columns at tO), 16 columns at a time.
template <int D>
__device__ __forceinline__ void rescale_o(uint32_t tO, float f) {
#pragma unroll 1
  for (int k = 0; k < D / 16; ++k) {
    uint32_t r[16];
    tmem_ld16(tO + 16 * k, r);
    tmem_wait(r);
#pragma unroll
    for (int e = 0; e < 16; e += 2) {
      float a0 = __uint_as_float(r[e]), a1 = __uint_as_float(r[e + 1]);
      fmul2(a0, a1, f);
      r[e] = __float_as_uint(a0);
      r[e + 1] = __float_as_uint(a1);
    }
    tmem_st16(tO + 16 * k, r);
  }
}

// Exponentials of 32 S columns (first key col0) against the running maximum
// m, their fp32 sums over all keys and over the text keys, and the bf16
// numerators packed in place: r[i] (i < 16) = keys 2i, 2i + 1 (the even key in
// the low half), the layout the PV product reads P_t in from tensor memory.
// kKind: 0 = valid image keys, 1 = valid text keys, 2 = general (keys beyond
// Nk give 0, text keys counted one by one).
template <int kKind>
__device__ __forceinline__ void exp_chunk(uint32_t (&r)[32], int col0, int Nk, int L, float c,
                                          float m, float& la, float& lt) {
  const float nm = -m;
  float s0 = 0.f, s1 = 0.f, t0 = 0.f;
#pragma unroll
  for (int e = 0; e < 32; e += 2) {
    float x0, x1;
    ffma2(__uint_as_float(r[e]), __uint_as_float(r[e + 1]), c, nm, x0, x1);
    float e0 = ex2(x0), e1 = ex2(x1);
    if (kKind == 2) {
      if (col0 + e >= Nk) e0 = 0.f;
      if (col0 + e + 1 >= Nk) e1 = 0.f;
      if (col0 + e < L) t0 += e0;
      if (col0 + e + 1 < L) t0 += e1;
    }
    fadd2(s0, s1, e0, e1);
    r[e >> 1] = pack_bf16x2(e0, e1);   // slot e / 2 <= e has been read
  }
  const float cs = s0 + s1;
  la += cs;
  if (kKind == 1) lt += cs;
  if (kKind == 2) lt += t0;
}

template <int kKind>
__device__ __forceinline__ void exp_tile(uint32_t (&r0)[32], uint32_t (&r1)[32],
                                         uint32_t (&r2)[32], uint32_t (&r3)[32], int key0,
                                         int Nk, int L, float c, float m, float& la, float& lt) {
  exp_chunk<kKind>(r0, key0, Nk, L, c, m, la, lt);
  exp_chunk<kKind>(r1, key0 + 32, Nk, L, c, m, la, lt);
  exp_chunk<kKind>(r2, key0 + 64, Nk, L, c, m, la, lt);
  exp_chunk<kKind>(r3, key0 + 96, Nk, L, c, m, la, lt);
}

// The 16 packed words at the front of r (32 keys of P) into 16 tensor-memory
// columns of this thread's lane.
__device__ __forceinline__ void tmem_st_p(uint32_t taddr, const uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, "
      "%11, %12, %13, %14, %15, %16};" ::"r"(taddr),
      AVITS_I8(0), AVITS_I8(8)
      : "memory");
}

struct RowState {
  float m, la, lt;
};

// Indices of a key tile's K and V loads in the ring: the load order is the
// order the MMAs consume them, K_0, K_1, V_0, K_2, V_1, ... (S of the next
// key tile is issued before P V of this one).  The K slot after the last
// key tile is left unused.
__device__ __forceinline__ int k_load(int g) { return g == 0 ? 0 : 2 * g - 1; }
__device__ __forceinline__ int v_load(int g) { return 2 * g + 2; }

template <int D>
__global__ void __launch_bounds__(kThreads, 1)
attention_tc_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                    const __grid_constant__ CUtensorMap tmV, const __grid_constant__ CUtensorMap tmO,
                    const AttnParams p) {
  using C = Cfg<D>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* sQ = smem;
  uint8_t* sKV = sQ + C::kQBytes;
  uint8_t* sStage = sKV + C::kKVBytes;   // O staging, one 64-column block per tile
  Bars* bars = reinterpret_cast<Bars*>(sStage + kStageBytes);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n_my = (p.n_units - (int)blockIdx.x + (int)gridDim.x - 1) / (int)gridDim.x;
  if (n_my <= 0) return;   // block-uniform
  const int G = n_my * p.n_kt;   // key tiles this CTA processes (all its units)

  if (threadIdx.x == 0) {
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmQ)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmK)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmV)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmO)) : "memory");
    for (int t = 0; t < kQTiles; ++t) {
      mbar_init(&bars->q_full[t], 1);
      mbar_init(&bars->q_empty[t], 1);
      mbar_init(&bars->s_full[t], 1);
      mbar_init(&bars->s_empty[t], 4);    // the tile's 4 softmax warps
      mbar_init(&bars->p_full[t], 4);
      mbar_init(&bars->pv_done[t], 1);
      mbar_init(&bars->o_full[t], 1);
      mbar_init(&bars->o_empty[t], 4);
      mbar_init(&bars->drain[t], 1);
    }
    for (int s = 0; s < C::kStages; ++s) {
      mbar_init(&bars->kv_full[s], 1);
      mbar_init(&bars->kv_empty[s], kQTiles);   // one commit per issuer
    }
    bars->abort = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    fence_async_shared();
  }
  // Q, K and V may come from the kernel before this one on the stream
  asm volatile("griddepcontrol.wait;" ::: "memory");
  if (warp == 1) tmem_alloc(&bars->tmem_base, kTmemCols);
  fence_before();
  __syncthreads();
  fence_after();
  const uint32_t tmem = bars->tmem_base;
  volatile int* abort_flag = &bars->abort;
  if (threadIdx.x == 96) asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

  auto unit_coords = [&](int u, int& b, int& h, int& qp) {
    const int bh = u / p.n_qp;
    qp = u - bh * p.n_qp;
    b = bh / p.H;
    h = bh - b * p.H;
  };

  if (warp == 0) {
    // ------------------------------------------------------ TMA producer --
    if (lane == 0) {
      bool ok = true;
      int last[C::kStages];   // the latest load armed on each stage, -1 = none
      for (int s = 0; s < C::kStages; ++s) last[s] = -1;
      int q_armed = 0, q_unit = 0;   // Q tiles armed for unit q_unit
      auto load_q = [&](int ui, int t) {
        int b, h, qp;
        unit_coords((int)blockIdx.x + ui * (int)gridDim.x, b, h, qp);
        if (ui > 0)
          ok = mbar_wait_bounded(&bars->q_empty[t], (uint32_t)((ui - 1) & 1), abort_flag, p.status);
        if (!ok) return;
        if (q_unit != ui) { q_unit = ui; q_armed = 0; }
        mbar_arrive_expect_tx(&bars->q_full[t], C::kTileBytes);
        for (int cb = 0; cb < C::kCB; ++cb)
          tma_load_4d(sQ + t * C::kTileBytes + cb * (kBM * 128), &tmQ, cb * 64,
                      qp * kUnitRows + t * kBM, h, b, &bars->q_full[t]);
        ++q_armed;
      };
      // load number idx of the ring: key tile g's K (is_k) or V
      auto load_kv = [&](int idx, bool is_k, int g) {
        int b, h, qp;
        unit_coords((int)blockIdx.x + (g / p.n_kt) * (int)gridDim.x, b, h, qp);
        const int kt = g - (g / p.n_kt) * p.n_kt;
        const int stage = idx % C::kStages;
        const uint32_t ph = (uint32_t)((idx / C::kStages) & 1);
        ok = mbar_wait_bounded(&bars->kv_empty[stage], ph ^ 1u, abort_flag, p.status);
        if (!ok) return;
        mbar_arrive_expect_tx(&bars->kv_full[stage], C::kTileBytes);
        for (int cb = 0; cb < C::kCB; ++cb)
          tma_load_4d(sKV + stage * C::kTileBytes + cb * (kBM * 128), is_k ? &tmK : &tmV, cb * 64,
                      kt * kBN, h, b, &bars->kv_full[stage]);
        last[stage] = idx;
      };
      load_q(0, 0);
      if (ok) load_kv(k_load(0), true, 0);
      if (ok) load_q(0, 1);
      for (int g = 0; g < G && ok; ++g) {
        const int gn = g + 1;
        if (gn < G) {
          if (gn % p.n_kt == 0) {   // the next unit's Q tiles before its first K tile
            load_q(gn / p.n_kt, 0);
            if (ok) load_q(gn / p.n_kt, 1);
          }
          if (ok) load_kv(k_load(gn), true, gn);
        }
        if (ok) load_kv(v_load(g), false, g);
      }
      if (!ok) {
        // drain the copies still in flight before the CTA exits
        for (int t = 0; t < q_armed; ++t)
          mbar_wait_bounded(&bars->q_full[t], (uint32_t)(q_unit & 1), nullptr, p.status);
        for (int s = 0; s < C::kStages; ++s)
          if (last[s] >= 0)
            mbar_wait_bounded(&bars->kv_full[s], (uint32_t)((last[s] / C::kStages) & 1), nullptr,
                              p.status);
      }
    }
  } else if (warp == 1 || warp == 2) {
    // -------------------------------------------------------- MMA issuers --
    // Key tile g: S_t(g) = Q_t K_g^T into the S buffer both tiles share, as
    // soon as the other tile's softmax has loaded the S before it (S_0(g)
    // after S_1(g-1), S_1(g) after S_0(g)); then O_t += P_t(g-1) V_(g-1) with
    // P_t from tensor memory once the softmax has written it.  The next S so
    // runs on the tensor pipe while the softmax works on this one.
    const int t = warp - 1;
    if (lane == 0) {
      bool ok = true;
      const uint32_t q_lo = sw128_desc_lo(sQ + t * C::kTileBytes);
      const uint32_t kv_lo0 = sw128_desc_lo(sKV);
      const uint32_t v_lo0 = sw128_mn_desc_lo(sKV, kBM * 128);
      const uint32_t d_hi = sw128_desc_hi();
      const uint32_t tS = tmem + (uint32_t)kColS;
      const uint32_t tP = tmem + (uint32_t)(kColP + t * (kBN / 2));
      const uint32_t tO = tmem + (uint32_t)(kColO + t * D);
      for (int gi = 0; gi <= G && ok; ++gi) {
        if (gi < G) {
          const int ui = gi / p.n_kt, j = gi - ui * p.n_kt;
          const int lk = k_load(gi), sk = lk % C::kStages;
          ok = mbar_wait_bounded(&bars->kv_full[sk], (uint32_t)((lk / C::kStages) & 1), abort_flag, p.status);
          if (ok && j == 0)
            ok = mbar_wait_bounded(&bars->q_full[t], (uint32_t)(ui & 1), abort_flag, p.status);
          // the shared S buffer: the previous S in the order S_0(0), S_1(0),
          // S_0(1), ... has been loaded by its softmax
          if (ok && t == 0 && gi > 0)
            ok = mbar_wait_bounded(&bars->s_empty[1], (uint32_t)((gi - 1) & 1), abort_flag, p.status);
          if (ok && t == 1)
            ok = mbar_wait_bounded(&bars->s_empty[0], (uint32_t)(gi & 1), abort_flag, p.status);
          if (!ok) break;
          fence_after();
          const uint32_t k_lo = kv_lo0 + (uint32_t)((sk * C::kTileBytes) >> 4);
#pragma unroll
          for (int kk = 0; kk < D / 16; ++kk) {
            const uint32_t off = (uint32_t)(((kk >> 2) * (kBM * 128) + (kk & 3) * 32) >> 4);
            mma_ss(tS, q_lo + off, k_lo + off, d_hi, kIdescS, kk > 0 ? 1u : 0u);
          }
          mma_commit(&bars->s_full[t]);
          mma_commit(&bars->kv_empty[sk]);
          if (j == p.n_kt - 1) mma_commit(&bars->q_empty[t]);
        }
        if (gi > 0) {
          const int g = gi - 1;
          const int ug = g / p.n_kt, jg = g - ug * p.n_kt;
          const int lv = v_load(g), sv = lv % C::kStages;
          ok = mbar_wait_bounded(&bars->p_full[t], (uint32_t)(g & 1), abort_flag, p.status);
          if (ok)
            ok = mbar_wait_bounded(&bars->kv_full[sv], (uint32_t)((lv / C::kStages) & 1), abort_flag, p.status);
          if (ok && jg == 0 && ug > 0)   // the epilogue has read the previous unit's O_t
            ok = mbar_wait_bounded(&bars->o_empty[t], (uint32_t)((ug - 1) & 1), abort_flag, p.status);
          if (!ok) break;
          fence_after();
          const uint32_t v_lo = v_lo0 + (uint32_t)((sv * C::kTileBytes) >> 4);
#pragma unroll
          for (int kk = 0; kk < kBN / 16; ++kk)   // 16 keys: 8 P columns, 16 V rows
            mma_ts(tO, tP + (uint32_t)(kk * 8), v_lo + (uint32_t)((kk * 16 * 128) >> 4), d_hi,
                   C::kIdescPV, (jg > 0 || kk > 0) ? 1u : 0u);
          mma_commit(&bars->pv_done[t]);
          mma_commit(&bars->kv_empty[sv]);
          if (jg == p.n_kt - 1) mma_commit(&bars->o_full[t]);
        }
      }
      // all issued MMAs complete before tensor memory is released
      mma_commit(&bars->drain[t]);
      mbar_wait_bounded(&bars->drain[t], 0, nullptr, p.status);
    }
  } else if (warp >= 4) {
    // --------------------------------------------- softmax and epilogue --
    const int t = (warp - 4) >> 2;
    const int quad = warp & 3;             // TMEM lane quadrant this warp may access
    const int rowt = quad * 32 + lane;     // row within the tile = TMEM lane
    const bool leader = (quad == 0 && lane == 0);
    // named barrier of the tile's 128 threads: 1 + t (literal ids, so that
    // the kernel reserves only the barriers it uses)
    auto tile_sync = [&]() { if (t == 0) bar_sync(1, 128); else bar_sync(2, 128); };
    auto tile_and = [&](bool v) { return t == 0 ? bar_and(1, 128, v) : bar_and(2, 128, v); };
    const uint32_t lane_off = (uint32_t)(quad * 32) << 16;
    const uint32_t tS = tmem + lane_off + (uint32_t)kColS;
    const uint32_t tP = tmem + lane_off + (uint32_t)(kColP + t * (kBN / 2));
    const uint32_t tO = tmem + lane_off + (uint32_t)(kColO + t * D);
    uint8_t* sSt = sStage + t * kStageTileBytes;
    const float c = p.c_log2;
    bool ok = true;
    int gi = 0;
    for (int ui = 0; ui < n_my; ++ui) {
      int b, h, qp;
      unit_coords((int)blockIdx.x + ui * (int)gridDim.x, b, h, qp);
      RowState st{-INFINITY, 0.f, 0.f};
      for (int j = 0; j < p.n_kt; ++j, ++gi) {
        ok = ok && (*abort_flag == 0) &&
             mbar_wait_bounded(&bars->s_full[t], (uint32_t)(gi & 1), abort_flag, p.status);
        ok = __all_sync(0xffffffffu, ok);   // tcgen05.ld / st are warp-collective
        if (ok) {
          fence_after();
          // the row's 128 S columns into registers; the S buffer is then free
          // for the other tile's S
          uint32_t r0[32], r1[32], r2[32], r3[32];
          tmem_ld32(tS, r0);
          tmem_ld32(tS + 32, r1);
          tmem_ld32(tS + 64, r2);
          tmem_ld32(tS + 96, r3);
          tmem_wait32(r0);
          tmem_wait32(r1);
          tmem_wait32(r2);
          tmem_wait32(r3);
          fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&bars->s_empty[t]);
          const int key0 = j * kBN;
          float mx;
          if (key0 + kBN <= p.Nk)
            mx = fmaxf(fmaxf(chunk_max<true>(r0, 0, 0), chunk_max<true>(r1, 0, 0)),
                       fmaxf(chunk_max<true>(r2, 0, 0), chunk_max<true>(r3, 0, 0)));
          else
            mx = fmaxf(fmaxf(chunk_max<false>(r0, key0, p.Nk), chunk_max<false>(r1, key0 + 32, p.Nk)),
                       fmaxf(chunk_max<false>(r2, key0 + 64, p.Nk),
                             chunk_max<false>(r3, key0 + 96, p.Nk)));
          const float mt = mx * c;
          const bool up = mt > st.m + kTau;   // the row's first tile, or 2^8 above its maximum
          float f = 1.f;
          if (up) {
            f = ex2(st.m - mt);
            st.la *= f;
            st.lt *= f;
            st.m = mt;
          }
          // the numerators (bf16 pairs) while the previous PV product may
          // still be reading P_t; the kind is uniform over the warp
          if (key0 + kBN <= p.Nk && key0 >= p.L)
            exp_tile<0>(r0, r1, r2, r3, key0, p.Nk, p.L, c, st.m, st.la, st.lt);
          else if (key0 + kBN <= p.Nk && key0 + kBN <= p.L)
            exp_tile<1>(r0, r1, r2, r3, key0, p.Nk, p.L, c, st.m, st.la, st.lt);
          else
            exp_tile<2>(r0, r1, r2, r3, key0, p.Nk, p.L, c, st.m, st.la, st.lt);
          // P_t(gi - 1) has been read by its PV product and O_t holds it
          if (gi > 0) {
            bool w = mbar_wait_bounded(&bars->pv_done[t], (uint32_t)((gi - 1) & 1), abort_flag, p.status);
            ok = __all_sync(0xffffffffu, w);
          }
          if (ok) {
            // P_t into tensor memory: column c of the row holds keys 2c, 2c + 1
            tmem_st_p(tP, r0);
            tmem_st_p(tP + 16, r1);
            tmem_st_p(tP + 32, r2);
            tmem_st_p(tP + 48, r3);
            // the warp rescales its O rows together when any of them moved
            // (f = 1 leaves a row unchanged)
            if (j > 0 && __any_sync(0xffffffffu, up)) rescale_o<D>(tO, f);
            tmem_wait_st();
            fence_before();
          }
        }
        __syncwarp();
        if (ok && lane == 0) mbar_arrive(&bars->p_full[t]);
      }
      // ---- epilogue: O / l -> bf16 -> swizzled staging, 64 columns at a
      // time -> TMA store
      ok = ok && (*abort_flag == 0) &&
           mbar_wait_bounded(&bars->o_full[t], (uint32_t)(ui & 1), abort_flag, p.status);
      ok = __all_sync(0xffffffffu, ok);
      const float inv = 1.f / st.la;
      const int row0 = qp * kUnitRows + t * kBM;
#pragma unroll 1
      for (int cb = 0; cb < C::kCB; ++cb) {
        if (ok) {
          fence_after();
#pragma unroll 1
          for (int k = 0; k < 2; ++k) {
            uint32_t r[32];
            tmem_ld32(tO + 64 * cb + 32 * k, r);
            tmem_wait32(r);
            uint32_t w[16];
#pragma unroll
            for (int e = 0; e < 16; ++e)
              w[e] = pack_bf16x2(__uint_as_float(r[2 * e]) * inv, __uint_as_float(r[2 * e + 1]) * inv);
            uint8_t* rowp = sSt + rowt * 128;
#pragma unroll
            for (int q = 0; q < 4; ++q)
              *reinterpret_cast<uint4*>(rowp + (((4 * k + q) ^ (rowt & 7)) << 4)) =
                  make_uint4(w[4 * q], w[4 * q + 1], w[4 * q + 2], w[4 * q + 3]);
          }
          fence_before();
        }
        if (cb == C::kCB - 1) {   // every O column of this unit has been read
          __syncwarp();
          if (ok && lane == 0) mbar_arrive(&bars->o_empty[t]);
        }
        fence_async_shared();
        const bool all_ok = tile_and(ok);
        if (all_ok && leader && row0 < p.Mq) {   // a tile past the end stores nothing
          tma_store_4d(&tmO, sSt, cb * 64, row0, h, b);
          bulk_commit();
          bulk_wait_read();   // the staging is rewritten by the next block
        }
        tile_sync();
      }
      const int row = row0 + rowt;
      if (ok && row < p.Mq) {
        const float ln2 = 0.69314718055994530942f;
        if (p.lse) {
          float* lp = p.lse + (((long long)b * p.H + h) * p.Mq + row) * 2;
          lp[0] = (st.m + log2f(st.la)) * ln2;
          lp[1] = st.lt > 0.f ? (st.m + log2f(st.lt)) * ln2 : -INFINITY;
        }
        if (p.A)
          head_sum_add(p.acc + (long long)b * p.rows_pad + row, p.H, st.lt / st.la, p.weight,
                       p.accumulate, p.A + (long long)b * p.Mq + row);
      }
    }
    if (leader) bulk_wait_all();
  }

  fence_before();
  __syncthreads();
  if (warp == 1) {
    fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

struct Plan {
  int n_qp, n_kt, n_units, grid;
  size_t acc_bytes;
};

Plan make_plan(int B, int H, int Mq, int Nk, int num_sms) {
  Plan pl{};
  pl.n_qp = (Mq + kUnitRows - 1) / kUnitRows;
  pl.n_kt = (Nk + kBN - 1) / kBN;
  pl.n_units = B * H * pl.n_qp;
  const int sms = num_sms > 0 ? num_sms : 1;
  pl.grid = pl.n_units < sms ? pl.n_units : sms;
  pl.acc_bytes = (sizeof(unsigned long long) * (size_t)B * pl.n_qp * kUnitRows + 255) &
                 ~static_cast<size_t>(255);
  return pl;
}

template <auto Kernel, int D>
cudaError_t smem_attrs() {
  cudaError_t e = cudaFuncSetAttribute(Kernel, cudaFuncAttributePreferredSharedMemoryCarveout,
                                       cudaSharedmemCarveoutMaxShared);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(Kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem_bytes<D>());
  return e;
}

cudaError_t set_smem_once() {
  static int done[64] = {};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev >= 0 && dev < 64 && __atomic_load_n(&done[dev], __ATOMIC_ACQUIRE)) return cudaSuccess;
  e = smem_attrs<attention_tc_kernel<128>, 128>();
  if (e == cudaSuccess) e = smem_attrs<attention_tc_kernel<64>, 64>();
  if (e == cudaSuccess && dev >= 0 && dev < 64) __atomic_store_n(&done[dev], 1, __ATOMIC_RELEASE);
  return e;
}

static_assert(smem_bytes<128>() <= 232448, "attention kernel shared memory above the opt-in limit");

}  // namespace

size_t attention_tc_workspace(int B, int H, int Mq) {
  return make_plan(B, H, Mq, 1, 1).acc_bytes;
}

bool attention_tc_layout_ok(const AttnArgs& a) {
  if (a.d != 64 && a.d != 128) return false;
  const void* ptrs[4] = {a.q, a.k, a.v, a.o};
  for (const void* ptr : ptrs)
    if (reinterpret_cast<uintptr_t>(ptr) & 15u) return false;
  for (int i = 0; i < 4; ++i)
    if (!strides_ok(a.B, a.H, a.str[i][0], a.str[i][1], a.str[i][2])) return false;
  return encode_fn() != nullptr;
}

cudaError_t launch_attention_tc(const AttnArgs& a, int num_sms, cudaStream_t s) {
  const Plan pl = make_plan(a.B, a.H, a.Mq, a.Nk, num_sms);
  CUtensorMap mq, mk, mv, mo;
  if (!make_map(&mq, a.q, a.B, a.H, a.Mq, a.d, a.str[0][0], a.str[0][1], a.str[0][2]) ||
      !make_map(&mk, a.k, a.B, a.H, a.Nk, a.d, a.str[1][0], a.str[1][1], a.str[1][2]) ||
      !make_map(&mv, a.v, a.B, a.H, a.Nk, a.d, a.str[2][0], a.str[2][1], a.str[2][2]) ||
      !make_map(&mo, a.o, a.B, a.H, a.Mq, a.d, a.str[3][0], a.str[3][1], a.str[3][2]))
    return cudaErrorInvalidValue;
  AttnParams p{};
  p.B = a.B; p.H = a.H; p.Mq = a.Mq; p.Nk = a.Nk; p.L = a.L;
  p.n_qp = pl.n_qp; p.n_kt = pl.n_kt; p.n_units = pl.n_units;
  p.c_log2 = a.scale * 1.4426950408889634f;
  p.weight = a.weight;
  p.accumulate = a.accumulate;
  p.A = a.A;
  p.lse = a.lse;
  p.acc = static_cast<unsigned long long*>(a.ws);
  p.rows_pad = pl.n_qp * kUnitRows;
  p.status = a.status;
  cudaError_t e = set_smem_once();
  if (e != cudaSuccess) return e;
  if (a.d == 128)
    e = launch_pdl(attention_tc_kernel<128>, dim3(pl.grid), dim3(kThreads), smem_bytes<128>(), s,
                   mq, mk, mv, mo, p);
  else
    e = launch_pdl(attention_tc_kernel<64>, dim3(pl.grid), dim3(kThreads), smem_bytes<64>(), s,
                   mq, mk, mv, mo, p);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace avits
