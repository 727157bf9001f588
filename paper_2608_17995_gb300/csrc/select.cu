// select.cu — joint score and token selection (Sec. 3.3.3, Eq. 8-9).
//
// One CTA per batch element (256 threads up to M = 256, 512 beyond; up to 8
// keys per thread in registers), few barriers:
//   1. min / max of A and V (NaN ignored): warp shuffles, one shared-memory
//      round, every warp finishes the reduction itself;
//   2. S = (alpha * A^) + ((1 - alpha) * V^) with explicitly rounded fp32
//      operations in that order (no contraction), so that the same A, V give
//      bit-identical S wherever the selection is recomputed; with a
//      caller-supplied perturbation (the tie-breaking noise of Eq. 9) one more
//      rounded addition S + perturb follows; each S becomes
//      an order-preserving 32-bit key (NaN -> 0, below everything; -0 -> +0;
//      otherwise the IEEE bits with the sign bit flipped if positive, all
//      bits flipped if negative), kept in registers and in shared memory;
//   3. the k-th largest key.  Keys in registers: first one pass over 256
//      buckets of the score VALUE (floor(256 S) clamped to [0, 255], a non-
//      decreasing function of S, so of the key; scores in [0, 1] spread over
//      the buckets where their top key bits do not), a shared-memory
//      histogram and one block scan give the bucket holding the k-th key;
//      when that bucket holds at most 32 keys one warp ranks them pairwise
//      (key descending, index ascending) and the k-th is found.  Otherwise
//      (clustered or tied scores), and for keys in shared memory: MSB-first
//      radix select with 4-bit digits: each warp counts its keys per digit
//      with ballots (lane j < 16 counts digit j; no shared-memory atomics,
//      which would all hit one bin since the keys share their top bits), the
//      per-warp counts go to a double-buffered table and every warp scans the
//      16 digits itself, so a pass costs one barrier; the passes stop once
//      the k-th key's digit is taken whole;
//   4. the selection: keys above the threshold, and of the keys equal to it
//      the lowest indices first.  Keys in registers: every key's selected-
//      before count from per-warp ballots and one table of warp counts (one
//      barrier), coalesced writes; keys in shared memory: contiguous per-
//      thread index ranges with ONE block scan of (keys above, keys equal),
//      a thread's selected-before count being above_before +
//      min(r, equal_before) for the r equal keys still needed.  Either way
//      it yields sel_idx (ascending), the mask and tok_offset.
#include "avits_common.cuh"
#include "avits_internal.h"
#include "upsample_token.cuh"

namespace avits {
namespace {

constexpr int kMaxThreads = 512;
constexpr int kMaxRegKeys = 8;   // keys per thread kept in registers (M <= 4096)

__device__ __forceinline__ uint32_t order_key(float s) {
  if (s != s) return 0u;
  const float c = (s == 0.0f) ? 0.0f : s;
  const uint32_t u = __float_as_uint(c);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// Per-warp digit counts of the keys matching `prefix` on `pmask`; lane j < 16
// returns the count of digit j at `shift`.
__device__ __forceinline__ uint32_t count_digits(uint32_t key, bool valid, uint32_t prefix,
                                                 uint32_t pmask, int shift, int lane) {
  const bool take = valid && (key & pmask) == prefix;
  const uint32_t d = (key >> shift) & 15u;
  uint32_t m = __ballot_sync(0xffffffffu, take);
  const uint32_t b0 = __ballot_sync(0xffffffffu, take && (d & 1u));
  const uint32_t b1 = __ballot_sync(0xffffffffu, take && (d & 2u));
  const uint32_t b2 = __ballot_sync(0xffffffffu, take && (d & 4u));
  const uint32_t b3 = __ballot_sync(0xffffffffu, take && (d & 8u));
  m &= (lane & 1) ? b0 : ~b0;
  m &= (lane & 2) ? b1 : ~b1;
  m &= (lane & 4) ? b2 : ~b2;
  m &= (lane & 8) ? b3 : ~b3;
  return __popc(m);
}

// Bucket of a fused score for the first selection pass: non-decreasing in S,
// equal scores share a bucket, NaN (the lowest key) goes to bucket 0 and
// scores outside [0, 1] (possible with a perturbation) to the end buckets.
__device__ __forceinline__ int score_bucket(float s) {
  if (s != s) return 0;
  return (int)fminf(fmaxf(s * 256.0f, 0.0f), 255.0f);
}

// Block-wide prefix count of one flag per key, keys in registers (key
// i = threadIdx.x + r * kThreads): before[r] = flagged keys of lower index;
// returns the total.  `tab` holds R * kWarps words of shared memory; one
// barrier, after which every warp scans the table of warp counts itself.
template <int kThreads, int R>
__device__ __forceinline__ uint32_t flag_prefix(const bool (&f)[R], uint32_t (&before)[R],
                                                uint32_t* tab, int lane, int w) {
  constexpr int kWarps = kThreads / 32;
  constexpr int E = R * kWarps;           // table entries in (r, warp) order
  constexpr int PER = (E + 31) / 32;      // entries per lane
  uint32_t bal[R];
#pragma unroll
  for (int r = 0; r < R; ++r) bal[r] = __ballot_sync(0xffffffffu, f[r]);
  if (lane == 0) {
#pragma unroll
    for (int r = 0; r < R; ++r) tab[r * kWarps + w] = __popc(bal[r]);
  }
  __syncthreads();
  uint32_t loc[PER], sum = 0u;
#pragma unroll
  for (int j = 0; j < PER; ++j) {
    const int e = lane * PER + j;
    loc[j] = e < E ? tab[e] : 0u;
    sum += loc[j];
  }
  uint32_t inc = sum;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t y = __shfl_up_sync(0xffffffffu, inc, o);
    if (lane >= o) inc += y;
  }
  const uint32_t excl = inc - sum;
  const uint32_t lt = (1u << lane) - 1u;
#pragma unroll
  for (int r = 0; r < R; ++r) {
    // entry e of this warp's row r lives in lane e / PER, position e % PER
    const int e = r * kWarps + w, src = e / PER, jj = e - src * PER;
    uint32_t pre = excl;
#pragma unroll
    for (int j = 0; j < PER; ++j) pre += (j < jj) ? loc[j] : 0u;
    before[r] = __shfl_sync(0xffffffffu, pre, src) + __popc(bal[r] & lt);
  }
  return __shfl_sync(0xffffffffu, inc, 31);
}

struct SelArgs {
  const float* A;
  const float* V;
  const float* perturb;   // NULL or [B,M]
  int M;
  float alpha, eps;
  int k;
  float* S_out;           // NULL or [B,M]
  int32_t* sel_idx;
  uint8_t* mask;          // NULL or [B,M]
  int32_t* tok_offset;
  unsigned int* status;
};

// The selection of batch element b by one CTA.  kRegKeys keys per thread in
// registers when M <= kRegKeys * kThreads; larger M (kRegKeys = 0) keeps them
// in shared memory only, in `keys` (the CTA's dynamic shared memory, M words).
// write_out: this CTA writes S, sel_idx, the mask and tok_offset.  offs_s /
// sel_s (or NULL): every token's start in the mixed sequence and whether it
// is selected, left in shared memory for the fused upsample.
template <int kThreads, int kRegKeys>
__device__ __forceinline__ void select_body(const SelArgs& g, int b, bool write_out,
                                            uint32_t* keys, int32_t* offs_s, uint8_t* sel_s) {
  constexpr int kWarps = kThreads / 32;
  __shared__ float red[4][kWarps];
  __shared__ uint32_t cnt[2][kWarps][16];
  __shared__ uint32_t scan_tot[kWarps];
  __shared__ int sh_nan;
  __shared__ __align__(16) uint32_t hist[256];       // bucket counts (keys in registers)
  __shared__ __align__(16) uint32_t cand_key[32];   // the k-th key's bucket, when small
  __shared__ __align__(16) int cand_idx[32];
  __shared__ uint32_t rank_part[8][32];  // candidate ranks, partial over 8 groups
  __shared__ uint32_t sh_ncand;
  __shared__ int sh_Tidx;
  __shared__ uint32_t ptab[kRegKeys > 0 ? kRegKeys * kWarps : 1];   // flag_prefix table
  const float* __restrict__ A = g.A;
  const float* __restrict__ V = g.V;
  const float* __restrict__ perturb = g.perturb;
  const int M = g.M, k = g.k;
  const float alpha = g.alpha, eps = g.eps;
  float* __restrict__ S_out = write_out ? g.S_out : nullptr;
  int32_t* __restrict__ sel_idx = g.sel_idx;
  uint8_t* __restrict__ mask = g.mask;
  int32_t* __restrict__ tok_offset = g.tok_offset;

  pdl_wait_then_trigger();
  const int tid = threadIdx.x, lane = tid & 31, w = tid >> 5;
  const float* a = A + (int64_t)b * M;
  const float* v = V + (int64_t)b * M;
  const float* pt = perturb ? perturb + (int64_t)b * M : nullptr;
  constexpr bool in_regs = kRegKeys > 0;
  constexpr int R = kRegKeys > 0 ? kRegKeys : 1;

  // 1. min / max (fminf / fmaxf skip NaN); A and V kept for step 2
  float ra[R], rv[R];
  const float inf = __int_as_float(0x7f800000);
  float amn = inf, amx = -inf, vmn = inf, vmx = -inf;
  if constexpr (in_regs) {
#pragma unroll
    for (int r = 0; r < R; ++r) {
      const int i = tid + r * kThreads;
      ra[r] = (i < M) ? a[i] : __int_as_float(0x7fc00000);
      rv[r] = (i < M) ? v[i] : __int_as_float(0x7fc00000);
    }
#pragma unroll
    for (int r = 0; r < R; ++r) {
      amn = fminf(amn, ra[r]); amx = fmaxf(amx, ra[r]);
      vmn = fminf(vmn, rv[r]); vmx = fmaxf(vmx, rv[r]);
    }
  } else {
    for (int i = tid; i < M; i += kThreads) {
      const float x = a[i], y = v[i];
      amn = fminf(amn, x); amx = fmaxf(amx, x);
      vmn = fminf(vmn, y); vmx = fmaxf(vmx, y);
    }
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
  if constexpr (in_regs) {
    for (int j = tid; j < 256; j += kThreads) hist[j] = 0u;
    if (tid == 0) sh_ncand = 0u;
  }
  __syncthreads();
  {
    const bool in = lane < kWarps;
    amn = in ? red[0][lane] : inf;
    amx = in ? red[1][lane] : -inf;
    vmn = in ? red[2][lane] : inf;
    vmx = in ? red[3][lane] : -inf;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      amn = fminf(amn, __shfl_xor_sync(0xffffffffu, amn, o));
      amx = fmaxf(amx, __shfl_xor_sync(0xffffffffu, amx, o));
      vmn = fminf(vmn, __shfl_xor_sync(0xffffffffu, vmn, o));
      vmx = fmaxf(vmx, __shfl_xor_sync(0xffffffffu, vmx, o));
    }
  }

  // 2. fused score in a fixed rounding order, keys
  const float aden = __fadd_rn(__fsub_rn(amx, amn), eps);
  const float vden = __fadd_rn(__fsub_rn(vmx, vmn), eps);
  const float one_m = __fsub_rn(1.0f, alpha);
  int any_nan = 0;
  uint32_t rk[R];
  int bk[R];
  auto fuse = [&](float x, float y, int i) {
    const float an = __fdiv_rn(__fsub_rn(x, amn), aden);
    const float vn = __fdiv_rn(__fsub_rn(y, vmn), vden);
    const float sc = __fadd_rn(__fmul_rn(alpha, an), __fmul_rn(one_m, vn));
    return pt ? __fadd_rn(sc, pt[i]) : sc;
  };
  if (in_regs) {
#pragma unroll
    for (int r = 0; r < R; ++r) {
      const int i = tid + r * kThreads;
      rk[r] = 0u;
      bk[r] = -1;
      if (i < M) {
        const float s = fuse(ra[r], rv[r], i);
        if (S_out) S_out[(int64_t)b * M + i] = s;
        any_nan |= (s != s);
        rk[r] = order_key(s);
        bk[r] = score_bucket(s);
        atomicAdd(&hist[bk[r]], 1u);
      }
    }
  } else {
    for (int i = tid; i < M; i += kThreads) {
      const float s = fuse(a[i], v[i], i);
      if (S_out) S_out[(int64_t)b * M + i] = s;
      any_nan |= (s != s);
      keys[i] = order_key(s);
    }
  }
  if (any_nan) sh_nan = 1;

  // 3. the k-th largest key: T on the top (32 - shift) key bits, of the keys
  // whose prefix is T the `remaining` lowest indices are selected
  uint32_t prefix = 0u, pmask = 0u, remaining = (uint32_t)k;
  int shift = 32;
  bool radix = k > 0 && k < M;
  uint32_t T = 0u;
  uint32_t last_bin = 0u;   // keys with the k-th key's prefix (radix path)
  int t_idx = 0x7fffffff;   // the last selected index among keys with prefix T
  __syncthreads();   // histogram (keys in registers) or keys[] complete
  if constexpr (in_regs) {
    if (radix) {
      // every warp scans the 256 bucket counts itself (no barrier): lane l
      // holds buckets 255 - 8l - 7 .. 255 - 8l, taken in descending order
      const uint4 h0 = *reinterpret_cast<const uint4*>(hist + 248 - 8 * lane);
      const uint4 h1 = *reinterpret_cast<const uint4*>(hist + 252 - 8 * lane);
      const uint32_t hv[8] = {h0.x, h0.y, h0.z, h0.w, h1.x, h1.y, h1.z, h1.w};
      uint32_t lsum = 0u;
#pragma unroll
      for (int j = 0; j < 8; ++j) lsum += hv[j];
      uint32_t inc = lsum;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const uint32_t y = __shfl_up_sync(0xffffffffu, inc, o);
        if (lane >= o) inc += y;
      }
      uint32_t cum = inc - lsum;
      int my_bucket = -1;
      uint32_t my_nb = 0u, my_above = 0u;
#pragma unroll
      for (int j = 7; j >= 0; --j) {
        if (cum < (uint32_t)k && (uint32_t)k <= cum + hv[j]) {
          my_bucket = 248 - 8 * lane + j;
          my_nb = hv[j];
          my_above = cum;
        }
        cum += hv[j];
      }
      const int src = __ffs(__ballot_sync(0xffffffffu, my_bucket >= 0)) - 1;
      const int bucket = __shfl_sync(0xffffffffu, my_bucket, src);
      const uint32_t nb = __shfl_sync(0xffffffffu, my_nb, src);
      const uint32_t need = (uint32_t)k - __shfl_sync(0xffffffffu, my_above, src);   // 1..nb
      if (nb <= 32u) {
        radix = false;
        // compaction of the bucket's keys: one shared-memory atomic per warp
        bool in[R];
        uint32_t bal[R], wcount = 0u;
#pragma unroll
        for (int r = 0; r < R; ++r) {
          in[r] = bk[r] == bucket;
          bal[r] = __ballot_sync(0xffffffffu, in[r]);
          wcount += (uint32_t)__popc(bal[r]);
        }
        if (wcount != 0u) {
          uint32_t base = 0u;
          if (lane == 0) base = atomicAdd(&sh_ncand, wcount);
          base = __shfl_sync(0xffffffffu, base, 0);
          const uint32_t lt = (1u << lane) - 1u;
#pragma unroll
          for (int r = 0; r < R; ++r) {
            if (in[r]) {
              const uint32_t slot = base + __popc(bal[r] & lt);
              cand_key[slot] = rk[r];
              cand_idx[slot] = tid + r * kThreads;
            }
            base += (uint32_t)__popc(bal[r]);
          }
        }
        __syncthreads();
        // rank of candidate j = candidates above it (keys above, equal keys of
        // lower index), the 32 x 32 comparisons spread over the CTA: thread
        // (j = lane, g = warp < 8) compares candidate j with candidates
        // 4g .. 4g + 3; every warp then sums the 8 partial counts itself
        const bool have = (uint32_t)lane < nb;
        const uint32_t kj = have ? cand_key[lane] : 0u;
        const int ij = have ? cand_idx[lane] : 0;
        if (w < 8) {
          const int g0 = 4 * w;
          uint32_t part = 0u;
          if (have && (uint32_t)g0 < nb) {
            const uint4 kv = *reinterpret_cast<const uint4*>(cand_key + g0);
            const int4 iv = *reinterpret_cast<const int4*>(cand_idx + g0);
            const uint32_t ka[4] = {kv.x, kv.y, kv.z, kv.w};
            const int ia[4] = {iv.x, iv.y, iv.z, iv.w};
#pragma unroll
            for (int e = 0; e < 4; ++e)
              part += ((uint32_t)(g0 + e) < nb && (ka[e] > kj || (ka[e] == kj && ia[e] < ij))) ? 1u : 0u;
          }
          rank_part[w][lane] = part;
        }
        __syncthreads();
        uint32_t rank = 0u;
#pragma unroll
        for (int g = 0; g < 8; ++g) rank += rank_part[g][lane];
        const int kth = __ffs(__ballot_sync(0xffffffffu, have && rank == need - 1u)) - 1;
        T = __shfl_sync(0xffffffffu, kj, kth);
        t_idx = __shfl_sync(0xffffffffu, ij, kth);
        shift = 0;
      }
    }
  }
  if (radix) {
    for (int pass = 0; pass < 8; ++pass) {
      shift -= 4;
      uint32_t c = 0;
      if (in_regs) {
#pragma unroll
        for (int r = 0; r < R; ++r) {
          const int i = tid + r * kThreads;
          c += count_digits(rk[r], i < M, prefix, pmask, shift, lane);
        }
      } else {
        for (int i0 = 0; i0 < M; i0 += kThreads) {
          const int i = i0 + tid;
          c += count_digits(i < M ? keys[i] : 0u, i < M, prefix, pmask, shift, lane);
        }
      }
      if (lane < 16) cnt[pass & 1][w][lane] = c;
      __syncthreads();
      // every warp: lane l holds digit 15 - l (descending order), l < 16
      uint32_t tot = 0;
      if (lane < 16) {
        uint32_t part[kWarps];
#pragma unroll
        for (int ww = 0; ww < kWarps; ++ww) part[ww] = cnt[pass & 1][ww][15 - lane];
#pragma unroll
        for (int ww = 0; ww < kWarps; ++ww) tot += part[ww];
      }
      uint32_t inc = tot;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const uint32_t y = __shfl_up_sync(0xffffffffu, inc, o);
        if (lane >= o) inc += y;
      }
      const uint32_t before = inc - tot;
      const bool hit = lane < 16 && before < remaining && remaining <= inc;
      const uint32_t hmask = __ballot_sync(0xffffffffu, hit);
      const int src = __ffs(hmask) - 1;
      const uint32_t digit = 15u - (uint32_t)src;
      const uint32_t rem = __shfl_sync(0xffffffffu, remaining - before, src);
      const uint32_t bin = __shfl_sync(0xffffffffu, tot, src);
      prefix |= digit << shift;
      pmask |= 15u << shift;
      remaining = rem;
      last_bin = bin;
      if (rem == bin) break;   // the digit is taken whole: no tie left to break
    }
    T = prefix >> shift;
  }
  if (write_out && tid == 0 && sh_nan) raise_status(g.status, AVITS_ERR_NAN);

  if constexpr (in_regs) {
    // 4. keys in registers
    const bool none = k == 0, all = k == M;
    if (radix && remaining < last_bin) {
      // radix path ending in equal keys: the index of the `remaining`-th
      // lowest-index key with prefix T (a prefix count of the equal flags)
      bool f[R];
      uint32_t eb[R];
#pragma unroll
      for (int r = 0; r < R; ++r) f[r] = tid + r * kThreads < M && (rk[r] >> shift) == T;
      flag_prefix<kThreads, R>(f, eb, ptab, lane, w);
#pragma unroll
      for (int r = 0; r < R; ++r)
        if (f[r] && eb[r] == remaining - 1u) sh_Tidx = tid + r * kThreads;
      __syncthreads();
      t_idx = sh_Tidx;
    }
    bool f[R];
    uint32_t before[R];
#pragma unroll
    for (int r = 0; r < R; ++r) {
      const int i = tid + r * kThreads;
      bool sel = false;
      if (i < M && !none) {
        if (all) {
          sel = true;
        } else {
          const uint32_t kp = rk[r] >> shift;
          sel = kp > T || (kp == T && i <= t_idx);
        }
      }
      f[r] = sel;
    }
    flag_prefix<kThreads, R>(f, before, ptab, lane, w);
#pragma unroll
    for (int r = 0; r < R; ++r) {
      const int i = tid + r * kThreads;
      if (i < M) {
        const int c = (int)before[r];
        if (write_out) {
          tok_offset[(int64_t)b * M + i] = i + 3 * c;
          if (mask) mask[(int64_t)b * M + i] = f[r] ? 1 : 0;
          if (f[r]) sel_idx[(int64_t)b * k + c] = i;
        }
        if (offs_s) {
          offs_s[i] = i + 3 * c;
          sel_s[i] = f[r] ? 1 : 0;
        }
      }
    }
  } else {
  // 4. keys in shared memory: one scan of (above, equal) over contiguous
  // per-thread ranges
  const int per = (M + kThreads - 1) / kThreads;
  const int lo = min(M, tid * per), hi = min(M, lo + per);
  uint32_t gt = 0, eq = 0;
  if (k > 0 && k < M) {
    for (int i = lo; i < hi; ++i) {
      const uint32_t kp = keys[i] >> shift;
      gt += kp > T;
      eq += kp == T;
    }
  }
  // packed inclusive scan: high 16 bits above-count, low 16 bits equal-count
  const uint32_t mine = (gt << 16) | eq;
  uint32_t x = mine;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) scan_tot[w] = x;
  __syncthreads();
  uint32_t wbefore = 0;
#pragma unroll
  for (int ww = 0; ww < kWarps; ++ww) wbefore += (ww < w) ? scan_tot[ww] : 0u;
  const uint32_t excl = wbefore + x - mine;
  const uint32_t gt_before = excl >> 16, eq_before = excl & 0xFFFFu;
  uint32_t c;
  if (k == 0) c = 0;
  else if (k == M) c = (uint32_t)lo;
  else c = gt_before + min(remaining, eq_before);
  uint32_t eq_seen = eq_before;
  for (int i = lo; i < hi; ++i) {
    bool sel;
    if (k == 0) sel = false;
    else if (k == M) sel = true;
    else {
      const uint32_t kp = keys[i] >> shift;
      sel = kp > T;
      if (kp == T) { sel = eq_seen < remaining; ++eq_seen; }
    }
    if (write_out) {
      tok_offset[(int64_t)b * M + i] = i + 3 * (int)c;
      if (mask) mask[(int64_t)b * M + i] = sel ? 1 : 0;
      if (sel) sel_idx[(int64_t)b * k + c] = i;
    }
    if (offs_s) {
      offs_s[i] = i + 3 * (int)c;
      sel_s[i] = sel ? 1 : 0;
    }
    if (sel) ++c;
  }
  }
}

template <int kThreads, int kRegKeys>
__global__ void __launch_bounds__(kThreads)
fuse_select_kernel(const SelArgs g) {
  extern __shared__ uint32_t keys[];
  select_body<kThreads, kRegKeys>(g, blockIdx.x, true, keys, nullptr, nullptr);
}

// One-launch selection + selective upsample (Eq. 8-9, then Sec. 3.2 Stage
// 2).  The grid has `parts` CTAs per batch element, CTA `part` owning the
// contiguous tokens [lo, hi).  Every CTA first starts copying the latent
// rows it will read (its tokens, and for bilinear the neighbouring grid rows)
// into shared memory with cp.async, then computes the element's selection
// (latency-bound work, so the redundant copies only occupy otherwise idle
// SMs) while the copy lands; part 0 writes the selection outputs; finally
// each warp upsamples its tokens from shared memory.  No CTA waits for
// another.
template <int kThreads, int kRegKeys, typename T, bool kBilinear>
__global__ void __launch_bounds__(kThreads)
select_upsample_kernel(const SelArgs g, const UpsampleArgs<T> u, int parts, int stage_rows) {
  extern __shared__ uint32_t keys[];
  const int b = blockIdx.x / parts, part = blockIdx.x - b * parts;
  const int M = g.M, T4 = u.C * 4;
  int32_t* offs_s = reinterpret_cast<int32_t*>(keys + M);
  uint8_t* sel_s = reinterpret_cast<uint8_t*>(offs_s + M);
  T* rows_s = reinterpret_cast<T*>(keys + ((9 * M + 15) / 16) * 4);   // 16-byte aligned
  const int chunk = (M + parts - 1) / parts;
  const int lo = min(M, part * chunk), hi = min(M, lo + chunk);
  const int halo = kBilinear ? u.gw + 1 : 0;
  const int s_lo = max(0, lo - halo), s_hi = min(M, hi + halo);
  // the latent is an input of this kernel: read it after the wait on the
  // kernel before (select_body's first step), so issue the copy just after
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const bool staged = stage_rows > 0;
  if (staged) {
    const char* src = reinterpret_cast<const char*>(u.latent + ((int64_t)b * M + s_lo) * T4);
    char* dst = reinterpret_cast<char*>(rows_s);
    const int n16 = (s_hi - s_lo) * T4 * (int)sizeof(T) / 16;
    for (int q = threadIdx.x; q < n16; q += kThreads)
      asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_u32(dst + 16 * q)),
                   "l"(src + 16 * q)
                   : "memory");
    asm volatile("cp.async.commit_group;" ::: "memory");
  }
  select_body<kThreads, kRegKeys>(g, b, part == 0, keys, offs_s, sel_s);
  if (staged) asm volatile("cp.async.wait_all;" ::: "memory");
  __syncthreads();
  constexpr int kWarps = kThreads / 32;
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  if (staged) {
    const SharedRows<T> rows{rows_s, s_lo, T4};
    for (int i = lo + w; i < hi; i += kWarps)
      upsample_token<T, kBilinear>(u, rows, b, i, offs_s[i], sel_s[i] != 0, lane);
  } else {
    const GlobalRows<T> rows{u.latent, M, T4};
    for (int i = lo + w; i < hi; i += kWarps)
      upsample_token<T, kBilinear>(u, rows, b, i, offs_s[i], sel_s[i] != 0, lane);
  }
}

}  // namespace

cudaError_t launch_fuse_select(const float* A, const float* V, const float* perturb, int B, int M,
                               float alpha, float eps, int k, float* S, int32_t* sel_idx,
                               uint8_t* mask, int32_t* tok_offset, unsigned int* status,
                               cudaStream_t s) {
  const size_t smem = (size_t)M * sizeof(uint32_t);
  if (smem > 48 * 1024) {
    // opt in once per device to the largest size any call can ask for
    static int done[64] = {};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (!(dev >= 0 && dev < 64 && __atomic_load_n(&done[dev], __ATOMIC_ACQUIRE))) {
      const int mx = (int)(kSelectMaxM * sizeof(uint32_t));
      e = cudaFuncSetAttribute(fuse_select_kernel<kMaxThreads, 0>,
                               cudaFuncAttributeMaxDynamicSharedMemorySize, mx);
      if (e != cudaSuccess) return e;
      e = cudaFuncSetAttribute(fuse_select_kernel<kMaxThreads, kMaxRegKeys>,
                               cudaFuncAttributeMaxDynamicSharedMemorySize, mx);
      if (e != cudaSuccess) return e;
      if (dev >= 0 && dev < 64) __atomic_store_n(&done[dev], 1, __ATOMIC_RELEASE);
    }
  }
  // 256 threads up to M = 256, 512 beyond (up to 2 keys per thread at
  // FLUX-1024: the per-key work of the fuse step is the longest part, measured
  // 3.50 -> 3.33 us against 256 threads); shared memory only above 4096
  void (*kern)(const SelArgs);
  int threads;
  if (M <= 256) {
    threads = 256;
    kern = fuse_select_kernel<256, 1>;
  } else if (M <= 1024) {
    threads = kMaxThreads;
    kern = M <= kMaxThreads ? fuse_select_kernel<kMaxThreads, 1> : fuse_select_kernel<kMaxThreads, 2>;
  } else {
    threads = kMaxThreads;
    const int per = (M + kMaxThreads - 1) / kMaxThreads;
    kern = per <= 4             ? fuse_select_kernel<kMaxThreads, 4>
           : per <= kMaxRegKeys ? fuse_select_kernel<kMaxThreads, kMaxRegKeys>
                                : fuse_select_kernel<kMaxThreads, 0>;
  }
  cudaError_t ce = prefer_max_shared<fuse_select_kernel<256, 1>>();
  if (ce == cudaSuccess) ce = prefer_max_shared<fuse_select_kernel<kMaxThreads, 1>>();
  if (ce == cudaSuccess) ce = prefer_max_shared<fuse_select_kernel<kMaxThreads, 2>>();
  if (ce == cudaSuccess) ce = prefer_max_shared<fuse_select_kernel<kMaxThreads, 4>>();
  if (ce == cudaSuccess) ce = prefer_max_shared<fuse_select_kernel<kMaxThreads, kMaxRegKeys>>();
  if (ce == cudaSuccess) ce = prefer_max_shared<fuse_select_kernel<kMaxThreads, 0>>();
  if (ce != cudaSuccess) return ce;
  const SelArgs g{A, V, perturb, M, alpha, eps, k, S, sel_idx, mask, tok_offset, status};
  cudaError_t e = launch_pdl(kern, dim3(B), dim3(threads), smem, s, g);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

namespace {

constexpr int kFusedThreads = 512;
constexpr int kFusedCtasTotal = 152;   // CTAs of the fused kernel over all elements
constexpr int kFusedMaxM = kFusedThreads * kMaxRegKeys;   // 4096

template <typename T, bool kBilinear>
cudaError_t launch_fused_t(const SelArgs& g, const UpsampleArgs<T>& u, int B, int M,
                           cudaStream_t s) {
  const int per = (M + kFusedThreads - 1) / kFusedThreads;
  auto kern = per <= 1   ? select_upsample_kernel<kFusedThreads, 1, T, kBilinear>
              : per <= 2 ? select_upsample_kernel<kFusedThreads, 2, T, kBilinear>
              : per <= 4 ? select_upsample_kernel<kFusedThreads, 4, T, kBilinear>
                         : select_upsample_kernel<kFusedThreads, 8, T, kBilinear>;
  cudaError_t e = prefer_max_shared<select_upsample_kernel<kFusedThreads, 1, T, kBilinear>>();
  if (e == cudaSuccess) e = prefer_max_shared<select_upsample_kernel<kFusedThreads, 2, T, kBilinear>>();
  if (e == cudaSuccess) e = prefer_max_shared<select_upsample_kernel<kFusedThreads, 4, T, kBilinear>>();
  if (e == cudaSuccess) e = prefer_max_shared<select_upsample_kernel<kFusedThreads, 8, T, kBilinear>>();
  if (e != cudaSuccess) return e;
  // about 2 tokens per warp, at most one CTA per SM over all elements (every
  // CTA repeats its element's selection)
  const int parts = std::max(1, std::min((M + 15) / 16, std::max(1, kFusedCtasTotal / B)));
  const int chunk = (M + parts - 1) / parts;
  const int halo = kBilinear ? u.gw + 1 : 0;
  const size_t row_bytes = (size_t)u.C * 4 * sizeof(T);
  // rows copied to shared memory: the CTA's tokens and their bilinear
  // neighbours, when rows are whole 16-byte copies and the copy fits
  int stage_rows = std::min(M, chunk + 2 * halo);
  const size_t head = ((9 * (size_t)M + 15) / 16) * 16;
  if (row_bytes % 16 != 0 || (reinterpret_cast<uintptr_t>(u.latent) & 15u) != 0 ||
      head + stage_rows * row_bytes > 96 * 1024)
    stage_rows = 0;
  const size_t smem = head + (size_t)stage_rows * row_bytes;
  if (smem > 48 * 1024) {
    e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, 96 * 1024);
    if (e != cudaSuccess) return e;
  }
  e = launch_pdl(kern, dim3((unsigned)(B * parts)), dim3(kFusedThreads), smem, s, g, u, parts,
                 stage_rows);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

template <typename T>
cudaError_t launch_fused_mode(const SelArgs& g, const void* latent, int B, int M, int gh, int gw,
                              int C, const int32_t* pos_in, const int32_t* span_in,
                              avits_upmode mode, void* out, int32_t* out_pos, int32_t* out_span,
                              int32_t* out_src_tok, int8_t* out_src_sub, cudaStream_t s) {
  const UpsampleArgs<T> u{static_cast<const T*>(latent), M, gh, gw, C, M + 3 * g.k, pos_in,
                          span_in, static_cast<T*>(out), out_pos, out_span, out_src_tok,
                          out_src_sub};
  return mode == AVITS_UP_BILINEAR ? launch_fused_t<T, true>(g, u, B, M, s)
                                   : launch_fused_t<T, false>(g, u, B, M, s);
}

}  // namespace

cudaError_t launch_select_upsample(const float* A, const float* V, const float* perturb, int B,
                                   int M, float alpha, float eps, int k, float* S,
                                   int32_t* sel_idx, uint8_t* mask, int32_t* tok_offset,
                                   unsigned int* status, const void* latent, avits_dtype dt,
                                   int gh, int gw, int C, const int32_t* pos_in,
                                   const int32_t* span_in, avits_upmode mode, void* out,
                                   int32_t* out_pos, int32_t* out_span, int32_t* out_src_tok,
                                   int8_t* out_src_sub, void* ws, cudaStream_t s) {
  if (M > kFusedMaxM || (mode == AVITS_UP_BILINEAR && pos_in)) {
    // beyond one CTA's registers, or a mixed bilinear input (whose cell map
    // is built between the selection and the upsample): the separate
    // launches, same outputs
    cudaError_t e = launch_fuse_select(A, V, perturb, B, M, alpha, eps, k, S, sel_idx, mask,
                                       tok_offset, status, s);
    if (e != cudaSuccess) return e;
    return launch_upsample(latent, dt, B, M, gh, gw, C, pos_in, span_in, mask, tok_offset, k,
                           mode, out, out_pos, out_span, out_src_tok, out_src_sub, ws, status, s);
  }
  const SelArgs g{A, V, perturb, M, alpha, eps, k, S, sel_idx, mask, tok_offset, status};
  if (dt == AVITS_BF16)
    return launch_fused_mode<__nv_bfloat16>(g, latent, B, M, gh, gw, C, pos_in, span_in, mode,
                                             out, out_pos, out_span, out_src_tok, out_src_sub, s);
  return launch_fused_mode<float>(g, latent, B, M, gh, gw, C, pos_in, span_in, mode, out, out_pos,
                                  out_span, out_src_tok, out_src_sub, s);
}

}  // namespace avits
