// merge.cu — final merge to the dense full-resolution latent (Sec. 3.2,
// Stage 3: the remaining tokens are expanded and the sequence is laid out in
// spatial order).
//
// Nearest: one warp per mixed token scatters its s x s cells; full-res pixel
// (Y,X) of a token at (y,x) with span s takes token pixel ((Y-2y)/s, (X-2x)/s).
// Coverage is checked in the same kernel: every cell is claimed by an
// atomicExch of this call's tag into a claim map in the caller's workspace
// (an old value equal to the tag = a cell covered twice), and every CTA adds
// (1 << 40) | cells claimed to one 64-bit word; the CTA whose add completes
// the CTA count compares the claimed total with B * fh * fw (fewer = a hole,
// since no cell was claimed twice), clears the word and advances the tag
// for the next call.  The map needs no clearing between calls.
// Bilinear (spans 1, 2 and 4): a cell map is scattered first (atomicExch into
// a -1-filled workspace, so double cover and holes are detected), then every
// output (cell, channel) gathers: span-1 cells are copied, coarser cells take
// the half-pixel-centred 2x bilinear resize of level 1 of the frame's pixel
// pyramid (frame_map.cuh), refined first from level 2 inside span-4 tokens.
// Algorithmic bytes: B*N*(T*elt + 12) read + B*fh*fw*T*elt written.
#include <algorithm>

#include "avits_common.cuh"
#include "avits_internal.h"
#include "frame_map.cuh"

namespace avits {
namespace {

// Workspace of the merge: a 16-byte header, then one 32-bit word per output
// cell.  Nearest: header = (tag of the last call, unused, 64-bit CTA count |
// claimed cells), words = claim map.  Bilinear: the words are the cell map.
struct MergeHeader {
  uint32_t last_tag;
  uint32_t unused;
  unsigned long long count;   // (CTAs done << 40) | cells claimed
};
constexpr int kMergeHeaderBytes = 16;

// Claim tags have bit 31 set (bilinear cell-map entries, -1 aside, have it
// clear, so a workspace used in both modes never confuses the two) and a
// 31-bit call counter in 1 .. 2^31 - 2 (never 0, the zeroed map).
__device__ __forceinline__ uint32_t next_tag(uint32_t last) {
  const uint32_t g = last & 0x7FFFFFFFu;
  return 0x80000000u | ((g == 0u || g >= 0x7FFFFFFEu) ? 1u : g + 1u);
}

// Batch-1 sized inputs (at most one token per warp of a capped grid): one
// warp per token, one pass.  A token's area is known once its position and
// span are read, so the CTA's count goes out first; the claims, the count's
// atomic and the pixel loads are then in flight together and their results
// are examined last: the check adds no round trip to the copy's two
// (position, then pixels).
template <typename T>
__global__ void __launch_bounds__(8 * 32)
merge_nearest_warp_kernel(const T* __restrict__ mixed, int B, int N,
                          const int32_t* __restrict__ pos, const int32_t* __restrict__ span,
                          int fh, int fw, int C, T* __restrict__ out, MergeHeader* hdr,
                          uint32_t* __restrict__ claim, unsigned int* status) {
  using PV = typename Pix4<T>::V;
  constexpr int kStage = 1024;   // a token of up to 1 KB takes the vector path
  pdl_wait_then_trigger();
  __shared__ __align__(16) uint8_t stage_all[8 * kStage];
  __shared__ unsigned int cta_cells;
  if (threadIdx.x == 0) cta_cells = 0u;
  const uint32_t last = *reinterpret_cast<volatile uint32_t*>(&hdr->last_tag);
  const int lane = threadIdx.x & 31;
  const int64_t t = (int64_t)blockIdx.x * 8 + (threadIdx.x >> 5);
  int b = 0, y = 0, x = 0, sp = 0;
  bool valid = false;
  if (t < (int64_t)B * N) {
    b = (int)(t / N);
    y = pos[t * 2];
    x = pos[t * 2 + 1];
    sp = span[t];
    valid = !(sp <= 0 || y < 0 || x < 0 || y + sp > fh || x + sp > fw);
    if (!valid && lane == 0) raise_status(status, AVITS_ERR_COVERAGE);
  }
  __syncthreads();   // cta_cells is initialised
  if (valid && lane == 0) atomicAdd(&cta_cells, (unsigned int)(sp * sp));
  __syncthreads();
  unsigned long long v = 0ull;
  if (threadIdx.x == 0)
    v = atomicAdd(&hdr->count, (1ull << 40) | (unsigned long long)cta_cells) +
        ((1ull << 40) | (unsigned long long)cta_cells);
  const uint32_t tag = next_tag(last);
  uint32_t old0 = 0u, old1 = 0u;   // claims of cells lane and lane + 32
  bool twice = false;
  if (valid) {
    const int64_t base = (int64_t)b * fh * fw;
    const int area = sp * sp;
    const int T4 = C * 4;
    const T* src = mixed + t * T4;
    const int tb = T4 * (int)sizeof(T);
    const bool vec = (tb & 15) == 0 && tb <= kStage;
    uint8_t* stage = stage_all + (threadIdx.x >> 5) * kStage;
    if (vec)
      for (int q = lane; q < tb / 16; q += 32)
        reinterpret_cast<uint4*>(stage)[q] = __ldg(reinterpret_cast<const uint4*>(src) + q);
    if (lane < area)
      old0 = atomicExch(&claim[base + (int64_t)(y + lane / sp) * fw + (x + lane % sp)], tag);
    if (lane + 32 < area)
      old1 = atomicExch(&claim[base + (int64_t)(y + (lane + 32) / sp) * fw + (x + (lane + 32) % sp)],
                        tag);
    for (int cell = lane + 64; cell < area; cell += 32)   // spans above 8
      twice |= atomicExch(&claim[base + (int64_t)(y + cell / sp) * fw + (x + cell % sp)], tag) == tag;
    if (vec) {
      __syncwarp();
      const int cpc = tb / 16;
      for (int q = lane; q < area * cpc; q += 32) {
        const int cell = q / cpc, j = q - cell * cpc;
        const int u = cell / sp, w = cell - u * sp;
        const int r0 = (2 * u) / sp, r1 = (2 * u + 1) / sp;
        const int c0 = (2 * w) / sp, c1 = (2 * w + 1) / sp;
        const uint4 chunk = (sp == 1) ? reinterpret_cast<const uint4*>(stage)[j]
                                      : gather_chunk<T>(stage, j, r0, r1, c0, c1);
        const int64_t ocell = base + (int64_t)(y + u) * fw + (x + w);
        reinterpret_cast<uint4*>(out + ocell * T4)[j] = chunk;
      }
    } else {
      for (int task = lane; task < area * C; task += 32) {
        const int cell = task / C, c = task - cell * C;
        const int u = cell / sp, w = cell - u * sp;
        const int r0 = (2 * u) / sp, r1 = (2 * u + 1) / sp;
        const int c0 = (2 * w) / sp, c1 = (2 * w + 1) / sp;
        const T* sc = src + c * 4;
        const float p00 = load_elem(sc, r0 * 2 + c0), p01 = load_elem(sc, r0 * 2 + c1);
        const float p10 = load_elem(sc, r1 * 2 + c0), p11 = load_elem(sc, r1 * 2 + c1);
        const int64_t ocell = base + (int64_t)(y + u) * fw + (x + w);
        reinterpret_cast<PV*>(out + ocell * T4)[c] = Pix4<T>::make(p00, p01, p10, p11);
      }
    }
  }
  if (threadIdx.x == 0 && (v >> 40) == (unsigned long long)gridDim.x) {
    // every CTA has counted its cells: no cell is claimed twice unless that
    // is reported, so fewer claimed cells than cells means a hole
    if ((v & ((1ull << 40) - 1ull)) != (unsigned long long)B * fh * fw)
      raise_status(status, AVITS_ERR_COVERAGE);
    hdr->count = 0ull;
    hdr->last_tag = tag;
  }
  if (twice || old0 == tag || old1 == tag) raise_status(status, AVITS_ERR_COVERAGE);
}

// Large batches: kLanesPerTok (8) lanes per token (8 x 16 bytes = a
// 16-channel bf16 token), four tokens in flight per warp; kNearestWarps warps
// per CTA, at most
// kNearestCtasPerSm CTAs per SM looping over the tokens (every CTA adds to
// the one count word, and same-address atomics are serialised: one CTA per
// 8 tokens of a batch of 64 made the count the bound).  A token's area is
// known once its position and span are read, so pass 1 sums the CTA's
// areas and its count goes out before pass 2 copies; the claims, the
// count's atomic and the pixel loads are then in flight together and their
// results are examined last.  The first token of each lane group keeps its
// position in registers between the passes (at batch 1 that is its only
// token).
constexpr int kNearestWarps = 8;
constexpr int kNearestCtasPerSm = 4;
constexpr int kStageBytes = 512;   // per token slot: a token of up to 512 B takes the vector path

template <typename T, int kLanesPerTok>
__global__ void __launch_bounds__(kNearestWarps * 32)
merge_nearest_kernel(const T* __restrict__ mixed, int B, int N, const int32_t* __restrict__ pos,
                     const int32_t* __restrict__ span, int fh, int fw, int C, T* __restrict__ out,
                     MergeHeader* hdr, uint32_t* __restrict__ claim, unsigned int* status) {
  using PV = typename Pix4<T>::V;
  constexpr int kToksPerWarp = 32 / kLanesPerTok;
  pdl_wait_then_trigger();
  __shared__ __align__(16) uint8_t stage_all[kNearestWarps * kToksPerWarp * kStageBytes];
  __shared__ unsigned int cta_cells;
  if (threadIdx.x == 0) cta_cells = 0u;
  const uint32_t last = *reinterpret_cast<volatile uint32_t*>(&hdr->last_tag);
  const int lane = threadIdx.x & 31, grp = lane / kLanesPerTok, gl = lane % kLanesPerTok;
  const int warp = threadIdx.x >> 5;
  const int64_t ntok = (int64_t)B * N;
  const int64_t tstride = (int64_t)gridDim.x * kNearestWarps * kToksPerWarp;
  const int64_t t0 = ((int64_t)blockIdx.x * kNearestWarps + warp) * kToksPerWarp + grp;
  // pass 1: validate the tokens and sum their areas
  unsigned int cells = 0u;
  int y0 = 0, x0 = 0, s0 = 0;
  for (int64_t t = t0; t < ntok; t += tstride) {
    const int y = pos[t * 2], x = pos[t * 2 + 1], sp = span[t];
    if (t == t0) { y0 = y; x0 = x; s0 = sp; }
    if (sp <= 0 || y < 0 || x < 0 || y + sp > fh || x + sp > fw) {
      if (gl == 0) raise_status(status, AVITS_ERR_COVERAGE);
    } else if (gl == 0) {
      cells += (unsigned int)(sp * sp);
    }
  }
  __syncthreads();   // cta_cells is initialised
  if (cells) atomicAdd(&cta_cells, cells);
  __syncthreads();
  unsigned long long v = 0ull;
  if (threadIdx.x == 0)
    v = atomicAdd(&hdr->count, (1ull << 40) | (unsigned long long)cta_cells) +
        ((1ull << 40) | (unsigned long long)cta_cells);
  const uint32_t tag = next_tag(last);
  bool twice = false;
  uint8_t* stage = stage_all + (warp * kToksPerWarp + grp) * kStageBytes;
  const int T4 = C * 4;
  const int tb = T4 * (int)sizeof(T);
  const bool vec = (tb & 15) == 0 && tb <= kStageBytes;
  // pass 2: claim the cells and copy (all lanes of the warp run the same
  // number of iterations, so the warp-wide syncs below are safe)
  const int64_t iters = (ntok - (t0 - grp) + tstride - 1) / tstride;
  for (int64_t it = 0; it < iters; ++it) {
    const int64_t t = t0 + it * tstride;
    const bool have = t < ntok;
    int y = 0, x = 0, sp = 0;
    if (have) {
      if (it == 0) { y = y0; x = x0; sp = s0; }
      else { y = pos[t * 2]; x = pos[t * 2 + 1]; sp = span[t]; }
    }
    const bool ok = have && !(sp <= 0 || y < 0 || x < 0 || y + sp > fh || x + sp > fw);
    const T* src = mixed + (have ? t : 0) * T4;
    if (vec) {
      __syncwarp();   // the slot's previous token is read
      if (ok)
        for (int q = gl; q < tb / 16; q += kLanesPerTok)
          reinterpret_cast<uint4*>(stage)[q] = __ldg(reinterpret_cast<const uint4*>(src) + q);
      __syncwarp();
    }
    if (!ok) continue;
    const int b = (int)(t / N);
    const int64_t base = (int64_t)b * fh * fw;
    const int area = sp * sp;
    // claims of cells gl and gl + kLanesPerTok are examined after the copy,
    // so their round trip overlaps it
    uint32_t old0 = 0u, old1 = 0u;
    if (gl < area)
      old0 = atomicExch(&claim[base + (int64_t)(y + gl / sp) * fw + (x + gl % sp)], tag);
    if (gl + kLanesPerTok < area) {
      const int c1 = gl + kLanesPerTok;
      old1 = atomicExch(&claim[base + (int64_t)(y + c1 / sp) * fw + (x + c1 % sp)], tag);
    }
    for (int cell = gl + 2 * kLanesPerTok; cell < area; cell += kLanesPerTok)
      twice |= atomicExch(&claim[base + (int64_t)(y + cell / sp) * fw + (x + cell % sp)], tag) == tag;
    if (vec) {
      // 16-byte output chunks: cell (u, w) of the token's s x s block takes,
      // for channel c, the token's pixels (r0|r1, c0|c1); chunks of one cell
      // are consecutive, so the stores are coalesced
      const int cpc = tb / 16;
      for (int q = gl; q < area * cpc; q += kLanesPerTok) {
        const int cell = q / cpc, j = q - cell * cpc;
        const int u = cell / sp, w = cell - u * sp;
        const int r0 = (2 * u) / sp, r1 = (2 * u + 1) / sp;
        const int c0 = (2 * w) / sp, c1 = (2 * w + 1) / sp;
        const uint4 chunk = (sp == 1) ? reinterpret_cast<const uint4*>(stage)[j]
                                      : gather_chunk<T>(stage, j, r0, r1, c0, c1);
        const int64_t ocell = base + (int64_t)(y + u) * fw + (x + w);
        reinterpret_cast<uint4*>(out + ocell * T4)[j] = chunk;
      }
    } else {
      for (int task = gl; task < area * C; task += kLanesPerTok) {
        const int cell = task / C, c = task - cell * C;
        const int u = cell / sp, w = cell - u * sp;
        const int r0 = (2 * u) / sp, r1 = (2 * u + 1) / sp;
        const int c0 = (2 * w) / sp, c1 = (2 * w + 1) / sp;
        const T* sc = src + c * 4;
        const float p00 = load_elem(sc, r0 * 2 + c0), p01 = load_elem(sc, r0 * 2 + c1);
        const float p10 = load_elem(sc, r1 * 2 + c0), p11 = load_elem(sc, r1 * 2 + c1);
        const int64_t ocell = base + (int64_t)(y + u) * fw + (x + w);
        reinterpret_cast<PV*>(out + ocell * T4)[c] = Pix4<T>::make(p00, p01, p10, p11);
      }
    }
    twice |= old0 == tag || old1 == tag;
  }
  if (threadIdx.x == 0 && (v >> 40) == (unsigned long long)gridDim.x) {
    // every CTA has counted its cells: no cell is claimed twice unless that
    // is reported, so fewer claimed cells than cells means a hole
    if ((v & ((1ull << 40) - 1ull)) != (unsigned long long)B * fh * fw)
      raise_status(status, AVITS_ERR_COVERAGE);
    hdr->count = 0ull;
    hdr->last_tag = tag;
  }
  if (twice) raise_status(status, AVITS_ERR_COVERAGE);   // a cell claimed twice
}

// The cell map starts as -1 everywhere (a hole until a token claims it).
__global__ void merge_fill_kernel(int32_t* __restrict__ map, int64_t n) {
  pdl_wait_then_trigger();
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x)
    map[i] = -1;
}

// One thread per token: its s x s cells get map_entry(token, log2 s).
__global__ void merge_map_kernel(int B, int N, const int32_t* __restrict__ pos,
                                 const int32_t* __restrict__ span, int fh, int fw,
                                 int32_t* __restrict__ map, unsigned int* status) {
  pdl_wait_then_trigger();
  const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= (int64_t)B * N) return;
  const int b = (int)(t / N), ti = (int)(t % N);
  const int y = pos[t * 2], x = pos[t * 2 + 1], s = span[t];
  const int lvl = (s == 1) ? 0 : (s == 2) ? 1 : (s == 4) ? 2 : -1;
  if (lvl < 0 || y < 0 || x < 0 || y + s > fh || x + s > fw || ((y | x) & (s - 1))) {
    raise_status(status, AVITS_ERR_COVERAGE);
    return;
  }
  const int32_t entry = map_entry(ti, lvl);
  for (int u = 0; u < s; ++u)
    for (int v = 0; v < s; ++v) {
      const int old = atomicExch(&map[(int64_t)b * fh * fw + (int64_t)(y + u) * fw + x + v], entry);
      if (old != -1) raise_status(status, AVITS_ERR_COVERAGE);
    }
}

// One thread per (output cell, channel).  A span-1 cell is copied.  A coarser
// cell's four pixels are the 2x bilinear resize of level 1 around it (a 3 x 3
// neighbourhood of level-1 pixels, clamped to the frame), where level 1 is the
// frame's own pyramid level, or, inside a span-4 token, the 2x bilinear
// resize of level 2 (the coarse-to-fine cascade; spans are at most 4).
template <typename T>
__global__ void merge_bilinear_kernel(const T* __restrict__ mixed, int B, int N, int fh, int fw,
                                      int C, const int32_t* __restrict__ map, T* __restrict__ out,
                                      unsigned int* status) {
  using PV = typename Pix4<T>::V;
  pdl_wait_then_trigger();
  const int64_t g = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t cells = (int64_t)fh * fw;
  if (g >= (int64_t)B * cells * C) return;
  const int c = (int)(g % C);
  const int64_t bc = g / C;
  const int b = (int)(bc / cells);
  const int cell = (int)(bc % cells);
  const int Y = cell / fw, X = cell - Y * fw;
  const int T4 = C * 4;
  const int32_t* mapb = map + (int64_t)b * cells;
  const T* mb = mixed + (int64_t)b * N * T4;
  const int32_t e = mapb[cell];
  PV* dst = reinterpret_cast<PV*>(out + bc * T4) + c;
  if (e < 0) {
    raise_status(status, AVITS_ERR_COVERAGE);
    *dst = Pix4<T>::make(0.f, 0.f, 0.f, 0.f);
    return;
  }
  if (map_lvl(e) == 0) {
    *dst = reinterpret_cast<const PV*>(mb + (int64_t)map_tok(e) * T4)[c];
    return;
  }
  // level-1 pixels (rows Y-1..Y+1, columns X-1..X+1, clamped): the frame's
  // own, or inside a span-4 token the resize of level 2
  int rr[3], cc[3];
#pragma unroll
  for (int k = 0; k < 3; ++k) {
    rr[k] = min(max(Y - 1 + k, 0), fh - 1);
    cc[k] = min(max(X - 1 + k, 0), fw - 1);
  }
  float lv[3][3];
#pragma unroll
  for (int i = 0; i < 3; ++i)
#pragma unroll
    for (int j = 0; j < 3; ++j) {
      const int32_t en = mapb[(int64_t)rr[i] * fw + cc[j]];
      lv[i][j] = (en >= 0 && map_lvl(en) >= 2)
                     ? frame_resize2x(2, mb, T4, mapb, fh, fw, c, rr[i], cc[j])
                     : frame_pixel<1>(mb, T4, mapb, fw, c, rr[i], cc[j]);
    }
  float r[4];
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    // output pixel row 2Y + a draws on level-1 rows (Y - 1, Y) for a = 0 and
    // (Y, Y + 1) for a = 1 with weights (1/4, 3/4) / (3/4, 1/4), clamped at
    // the frame edge: neighbourhood rows a and a + 1; columns likewise
    const int a = q >> 1, bq = q & 1;
    const float wy0 = a ? 0.75f : 0.25f, wy1 = a ? 0.25f : 0.75f;
    const float wx0 = bq ? 0.75f : 0.25f, wx1 = bq ? 0.25f : 0.75f;
    r[q] = bil_combine(lv[a][bq], lv[a][bq + 1], lv[a + 1][bq], lv[a + 1][bq + 1], wy0, wy1, wx0,
                       wx1);
  }
  *dst = Pix4<T>::make(r[0], r[1], r[2], r[3]);
}

template <typename T>
cudaError_t launch_t(const void* mixed, int B, int N, const int32_t* pos, const int32_t* span,
                     int fh, int fw, int C, avits_upmode mode, void* out, void* ws,
                     unsigned int* status, cudaStream_t s) {
  MergeHeader* hdr = static_cast<MergeHeader*>(ws);
  uint32_t* words = reinterpret_cast<uint32_t*>(static_cast<uint8_t*>(ws) + kMergeHeaderBytes);
  if (mode == AVITS_UP_NEAREST) {
    const int64_t ntok = (int64_t)B * N;
    int dev = 0, sms = 0;
    cudaError_t e0 = cudaGetDevice(&dev);
    if (e0 == cudaSuccess) e0 = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e0 != cudaSuccess) return e0;
    const int64_t cap = (int64_t)std::max(1, sms) * kNearestCtasPerSm;
    cudaError_t e = prefer_max_shared<merge_nearest_warp_kernel<T>>();
    if (e == cudaSuccess) e = prefer_max_shared<merge_nearest_kernel<T, 8>>();
    if (e != cudaSuccess) return e;
    if (ntok <= cap * kNearestWarps) {
      // one warp per token, one pass (latency-bound sizes)
      e = launch_pdl(merge_nearest_warp_kernel<T>, dim3((unsigned)((ntok + 7) / 8)),
                     dim3(8 * 32), 0, s, static_cast<const T*>(mixed), B, N, pos, span, fh, fw,
                     C, static_cast<T*>(out), hdr, words, status);
      if (e != cudaSuccess) return e;
      return cudaGetLastError();
    }
    const int64_t per_cta = (int64_t)kNearestWarps * 4;
    const int grid = (int)std::min<int64_t>((ntok + per_cta - 1) / per_cta, cap);
    e = launch_pdl(merge_nearest_kernel<T, 8>, dim3(grid), dim3(kNearestWarps * 32), 0, s,
                               static_cast<const T*>(mixed), B, N, pos, span, fh, fw, C,
                               static_cast<T*>(out), hdr, words, status);
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
  }
  // three kernels (fill, scatter of the cell map, gather), each a
  // programmatic dependent of the one before: their launches overlap, every
  // kernel waits for its predecessor before touching memory
  int32_t* map = reinterpret_cast<int32_t*>(words);
  cudaError_t e = launch_cell_map(B, N, pos, span, fh, fw, map, status, s);
  if (e == cudaSuccess) e = prefer_max_shared<merge_bilinear_kernel<T>>();
  if (e != cudaSuccess) return e;
  const int64_t work = (int64_t)B * fh * fw * C;
  e = launch_pdl(merge_bilinear_kernel<T>, dim3((unsigned)((work + 255) / 256)), dim3(256), 0, s,
                 static_cast<const T*>(mixed), B, N, fh, fw, C,
                 static_cast<const int32_t*>(map), static_cast<T*>(out), status);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_cell_map(int B, int N, const int32_t* pos, const int32_t* span, int fh, int fw,
                            int32_t* map, unsigned int* status, cudaStream_t s) {
  const int64_t ncell = (int64_t)B * fh * fw;
  cudaError_t e = prefer_max_shared<merge_fill_kernel>();
  if (e == cudaSuccess) e = prefer_max_shared<merge_map_kernel>();
  if (e != cudaSuccess) return e;
  const int fill_grid = (int)std::min<int64_t>((ncell + 255) / 256, 1024);
  e = launch_pdl(merge_fill_kernel, dim3(fill_grid), dim3(256), 0, s, map, ncell);
  if (e != cudaSuccess) return e;
  const int64_t nt = (int64_t)B * N;
  e = launch_pdl(merge_map_kernel, dim3((unsigned)((nt + 255) / 256)), dim3(256), 0, s, B, N, pos,
                 span, fh, fw, map, status);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

size_t merge_workspace_bytes(int B, int fh, int fw) {
  return kMergeHeaderBytes + sizeof(uint32_t) * (size_t)B * fh * fw;
}

cudaError_t launch_merge(const void* mixed, avits_dtype dt, int B, int N, const int32_t* pos,
                         const int32_t* span, int fh, int fw, int C, avits_upmode mode,
                         void* out, void* ws, unsigned int* status, cudaStream_t s) {
  if (dt == AVITS_BF16)
    return launch_t<__nv_bfloat16>(mixed, B, N, pos, span, fh, fw, C, mode, out, ws, status, s);
  return launch_t<float>(mixed, B, N, pos, span, fh, fw, C, mode, out, ws, status, s);
}

}  // namespace avits
