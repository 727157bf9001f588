// avits_internal.h — launchers behind the C ABI (host side, not exported).
#pragma once

#include <cstddef>
#include <cstdint>
#include <functional>
#include <cuda_runtime.h>

#include "avits.h"

// NVTX ranges around the C entry points, for timeline tools: compiled in
// with -DAVITS_NVTX (build with AVITS_NVTX=1 in the environment), nothing
// otherwise.  NVTX v3 is header-only; without a tool attached a range costs a
// null check.
#ifdef AVITS_NVTX
#include <nvtx3/nvToolsExt.h>
namespace avits {
struct NvtxRange {
  explicit NvtxRange(const char* name) { nvtxRangePushA(name); }
  ~NvtxRange() { nvtxRangePop(); }
  NvtxRange(const NvtxRange&) = delete;
  NvtxRange& operator=(const NvtxRange&) = delete;
};
}  // namespace avits
#define AVITS_RANGE() ::avits::NvtxRange avits_nvtx_range_(__func__)
#else
#define AVITS_RANGE() ((void)0)
#endif

namespace avits {

// Device address of the status word of the current device (api.cu).
unsigned int* status_word();

// ---- spatial (Eq. 3-5) ------------------------------------------------------
struct SpatialArgs {
  const void* q;
  const void* k;
  avits_dtype dt;
  int B, H, M, Nk, L, d;
  int64_t q_sb, q_sh, q_sn, k_sb, k_sh, k_sn;   // element strides
  float scale, weight;
  int accumulate;
  float* A;
  float* lse;
  void* ws;
  size_t ws_bytes;
  unsigned int* status;
  const uint8_t* tmask = nullptr;   // [B,Nk], nonzero = text key; NULL: keys j < L
  // [B,H,M] natural-log logsumexp over ALL keys, computed by the caller (the
  // model's attention forward); then the keys given are the text keys only
  // and the mass is exp(lse_txt - lse_all).  NULL: the keys are all keys.
  const float* lse_all = nullptr;
};

// tcgen05 / TMA path (bf16, d in {64,128}); returns false if the shape or
// layout is not eligible (the caller then uses the CUDA-core path).
bool spatial_tc_eligible(const SpatialArgs& a);
size_t spatial_tc_workspace(int B, int H, int M, int Nk, int d, int num_sms);
// Leading bytes of that workspace that must be zero before a call (the row
// words and ready flags of the in-kernel merge); a completed call leaves them
// zero again.
size_t spatial_tc_zeroed_bytes(int B, int H, int M, int Nk, int d, int num_sms);
// Launches issued right after the spatial kernel, as its programmatic
// dependents (they must not complete before it does).
using LaunchHook = std::function<cudaError_t(cudaStream_t)>;
cudaError_t launch_spatial_tc(const SpatialArgs& a, int num_sms, cudaStream_t s,
                              const LaunchHook* between = nullptr);

// CUDA-core path (fp32 or bf16, any d <= 256): up to 8 query rows per CTA.
cudaError_t launch_spatial_simt(const SpatialArgs& a, int num_sms, cudaStream_t s);

// ---- joint-attention forward (Eq. 4-5) with the spatial score (Eq. 3) -------
struct AttnArgs {
  const void* q;     // [B,H,Mq,d] bf16
  const void* k;     // [B,H,Nk,d] bf16, the L text keys first
  const void* v;     // [B,H,Nk,d] bf16
  void* o;           // [B,H,Mq,d] bf16
  int B, H, Mq, Nk, L, d;
  int64_t str[4][3];   // element strides (batch, head, row) of q, k, v, o
  float scale, weight;
  int accumulate;
  float* A;          // [B,Mq] or NULL
  float* lse;        // [B,H,Mq,2] or NULL
  void* ws;          // head-sum words (A != NULL), zero between calls
  unsigned int* status;
};
// Layout the tensor-core forward takes: d in {64,128}, 16-byte aligned bases
// and strides.
bool attention_tc_layout_ok(const AttnArgs& a);
size_t attention_tc_workspace(int B, int H, int Mq);
cudaError_t launch_attention_tc(const AttnArgs& a, int num_sms, cudaStream_t s);

// ---- temporal ---------------------------------------------------------------
// Failure-detection test hook (selftest.cu): bounded waits that cannot complete.
cudaError_t launch_wait_selftest(unsigned long long limit_ns, long long* result,
                                 unsigned int* status, cudaStream_t s);

cudaError_t launch_temporal(const void* ht, const void* hp, avits_dtype dt, int B, int N, int D,
                            float eps, float* V, int num_sms, unsigned int* status, cudaStream_t s);
// The temporal score as a programmatic dependent of the kernel just launched
// on `s`: one CTA per SM running beside it, waiting for it before exiting.
cudaError_t launch_temporal_overlapped(const void* ht, const void* hp, avits_dtype dt, int B,
                                       int N, int D, float eps, float* V, int num_sms,
                                       unsigned int* status, cudaStream_t s);
constexpr int kMaxSnapshots = 16;
cudaError_t launch_temporal_var(const void* const* snaps, int n_t, avits_dtype dt, int B, int N,
                                int D, float* V, int num_sms, cudaStream_t s);

// ---- fuse + select (Eq. 8-9) ------------------------------------------------
constexpr int kSelectMaxM = 32768;
cudaError_t launch_fuse_select(const float* A, const float* V, const float* perturb, int B, int M,
                               float alpha, float eps, int k, float* S, int32_t* sel_idx,
                               uint8_t* mask, int32_t* tok_offset, unsigned int* status,
                               cudaStream_t s);

// ---- selective upsample (Stage 2) -------------------------------------------
// Selection + selective upsample in one launch (two above 2048 tokens).
cudaError_t launch_select_upsample(const float* A, const float* V, const float* perturb, int B,
                                   int M, float alpha, float eps, int k, float* S,
                                   int32_t* sel_idx, uint8_t* mask, int32_t* tok_offset,
                                   unsigned int* status, const void* latent, avits_dtype dt,
                                   int gh, int gw, int C, const int32_t* pos_in,
                                   const int32_t* span_in, avits_upmode mode, void* out,
                                   int32_t* out_pos, int32_t* out_span, int32_t* out_src_tok,
                                   int8_t* out_src_sub, void* ws, cudaStream_t s);
// ws: merge_workspace_bytes(B, gh, gw) bytes, 16-byte aligned, used (for the
// input frame's cell map) only in bilinear mode with a mixed input.
cudaError_t launch_upsample(const void* latent, avits_dtype dt, int B, int M, int gh, int gw,
                            int C, const int32_t* pos_in, const int32_t* span_in,
                            const uint8_t* mask, const int32_t* tok_offset, int k,
                            avits_upmode mode, void* out, int32_t* out_pos, int32_t* out_span,
                            int32_t* out_src_tok, int8_t* out_src_sub, void* ws,
                            unsigned int* status, cudaStream_t s);

// ---- final merge (Stage 3) --------------------------------------------------
// Workspace of either mode (and of a mixed bilinear upsample): a 16-byte
// header and one 32-bit word per cell.
size_t merge_workspace_bytes(int B, int fh, int fw);
cudaError_t launch_merge(const void* mixed, avits_dtype dt, int B, int N, const int32_t* pos,
                         const int32_t* span, int fh, int fw, int C, avits_upmode mode,
                         void* out, void* ws, unsigned int* status, cudaStream_t s);

}  // namespace avits
