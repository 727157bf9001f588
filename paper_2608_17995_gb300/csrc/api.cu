// api.cu — the C ABI of libavits (see include/avits.h): host-side argument
// checks, workspace sizing and dispatch to the kernels.  Nothing here
// allocates device memory or synchronises, except avits_device_status().
#include <cstdio>
#include <cstring>
#include <string>

#include "avits_common.cuh"
#include "avits_internal.h"

namespace avits {

__device__ unsigned int g_status = 0u;

namespace {

thread_local std::string t_last_error;

constexpr int kMaxDevices = 64;
unsigned int* g_status_ptr[kMaxDevices] = {};

int num_sms_current() {
  int dev = 0, n = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
  return n;
}

avits_status cuda_status(cudaError_t e) {
  if (e == cudaSuccess) return AVITS_OK;
  t_last_error = cudaGetErrorString(e);
  cudaGetLastError();   // clear a non-sticky error
  return AVITS_ERR_CUDA;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
bool valid_dtype(avits_dtype dt) { return dt == AVITS_F32 || dt == AVITS_BF16; }

// A mixed input in bilinear mode needs the cell map of its frame: an even
// frame, token indices that fit the map entry, and the workspace.
bool mixed_bilinear_ok(avits_upmode mode, const int32_t* pos_in, int B, int M, int gh, int gw,
                       const void* ws, size_t ws_bytes) {
  if (mode != AVITS_UP_BILINEAR || !pos_in) return true;
  if ((gh & 1) || (gw & 1) || M > (1 << 28) - 1) return false;
  return ws && aligned16(ws) && ws_bytes >= merge_workspace_bytes(B, gh, gw);
}

}  // namespace

// The device address of g_status on the current device, looked up once per
// device.  Concurrent first calls store the same value.
unsigned int* status_word() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
  unsigned int* p = __atomic_load_n(&g_status_ptr[dev], __ATOMIC_ACQUIRE);
  if (!p) {
    void* q = nullptr;
    if (cudaGetSymbolAddress(&q, g_status) != cudaSuccess) {
      cudaGetLastError();
      return nullptr;
    }
    p = static_cast<unsigned int*>(q);
    __atomic_store_n(&g_status_ptr[dev], p, __ATOMIC_RELEASE);
  }
  return p;
}

}  // namespace avits

using namespace avits;

extern "C" {

const char* avits_version(void) { return "0.1.0"; }

const char* avits_status_string(avits_status s) {
  switch (s) {
    case AVITS_OK: return "ok";
    case AVITS_ERR_INVALID_ARG: return "invalid argument";
    case AVITS_ERR_UNSUPPORTED: return "unsupported combination";
    case AVITS_ERR_CUDA: return "CUDA error";
    case AVITS_ERR_TIMEOUT: return "device wait timed out";
    case AVITS_ERR_NAN: return "NaN in fused score";
    case AVITS_ERR_COVERAGE: return "mixed sequence does not tile the frame";
  }
  return "unknown status";
}

const char* avits_last_error_string(void) { return t_last_error.c_str(); }

size_t avits_score_spatial_workspace(avits_dtype dt, int B, int H, int M, int Nk, int d) {
  if (B <= 0 || H <= 0 || M <= 0 || Nk <= 0 || d <= 0) return 0;
  if (dt != AVITS_BF16 || (d != 64 && d != 128)) return 0;
  return spatial_tc_workspace(B, H, M, Nk, d, num_sms_current());
}

avits_status avits_score_spatial(const void* q_img, const void* k_all, avits_dtype dt, int B,
                                 int H, int M, int Nk, int L, int d, int64_t q_sb, int64_t q_sh,
                                 int64_t q_sn, int64_t k_sb, int64_t k_sh, int64_t k_sn,
                                 float softmax_scale, float weight, int accumulate, float* A,
                                 float* lse_opt, void* workspace, size_t ws_bytes, void* stream) {
  AVITS_RANGE();
  if (!q_img || !k_all || !A || !valid_dtype(dt)) return AVITS_ERR_INVALID_ARG;
  if (B <= 0 || H <= 0 || M <= 0 || Nk <= 0 || d <= 0 || L < 0 || L > Nk || Nk < M)
    return AVITS_ERR_INVALID_ARG;
  if (!(softmax_scale > 0.f) || !(softmax_scale < 3.0e38f)) return AVITS_ERR_INVALID_ARG;
  if (q_sn < d || k_sn < d || q_sh < 0 || k_sh < 0 || q_sb < 0 || k_sb < 0)
    return AVITS_ERR_INVALID_ARG;
  SpatialArgs a{q_img, k_all, dt, B, H, M, Nk, L, d, q_sb, q_sh, q_sn, k_sb, k_sh, k_sn,
                softmax_scale, weight, accumulate ? 1 : 0, A, lse_opt, workspace, ws_bytes,
                status_word()};
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (spatial_tc_eligible(a)) {
    const int sms = num_sms_current();
    if (ws_bytes < spatial_tc_workspace(B, H, M, Nk, d, sms) || !workspace)
      return AVITS_ERR_INVALID_ARG;
    return cuda_status(launch_spatial_tc(a, sms, s));
  }
  if (d > 256) return AVITS_ERR_UNSUPPORTED;
  return cuda_status(launch_spatial_simt(a, num_sms_current(), s));
}

avits_status avits_score_spatial_lse(const void* q_img, const void* k_txt, avits_dtype dt, int B,
                                     int H, int M, int L, int d, int64_t q_sb, int64_t q_sh,
                                     int64_t q_sn, int64_t k_sb, int64_t k_sh, int64_t k_sn,
                                     const float* lse_all, float softmax_scale, float weight,
                                     int accumulate, float* A, float* lse_opt, void* workspace,
                                     size_t ws_bytes, void* stream) {
  AVITS_RANGE();
  if (!q_img || !k_txt || !lse_all || !A || !valid_dtype(dt)) return AVITS_ERR_INVALID_ARG;
  if (B <= 0 || H <= 0 || M <= 0 || L <= 0 || d <= 0) return AVITS_ERR_INVALID_ARG;
  if (!(softmax_scale > 0.f) || !(softmax_scale < 3.0e38f)) return AVITS_ERR_INVALID_ARG;
  if (q_sn < d || k_sn < d || q_sh < 0 || k_sh < 0 || q_sb < 0 || k_sb < 0)
    return AVITS_ERR_INVALID_ARG;
  SpatialArgs a{q_img, k_txt, dt, B, H, M, L, L, d, q_sb, q_sh, q_sn, k_sb, k_sh, k_sn,
                softmax_scale, weight, accumulate ? 1 : 0, A, lse_opt, workspace, ws_bytes,
                status_word()};
  a.lse_all = lse_all;
  if (!spatial_tc_eligible(a)) return AVITS_ERR_UNSUPPORTED;
  const int sms = num_sms_current();
  if (ws_bytes < spatial_tc_workspace(B, H, M, L, d, sms) || !workspace)
    return AVITS_ERR_INVALID_ARG;
  return cuda_status(launch_spatial_tc(a, sms, static_cast<cudaStream_t>(stream)));
}

avits_status avits_score_spatial_keymask(const void* q_img, const void* k_all, avits_dtype dt,
                                         int B, int H, int M, int Nk, int d, int64_t q_sb,
                                         int64_t q_sh, int64_t q_sn, int64_t k_sb, int64_t k_sh,
                                         int64_t k_sn, const uint8_t* text_mask,
                                         float softmax_scale, float weight, int accumulate,
                                         float* A, float* lse_opt, void* workspace,
                                         size_t ws_bytes, void* stream) {
  AVITS_RANGE();
  if (!q_img || !k_all || !A || !text_mask || !valid_dtype(dt)) return AVITS_ERR_INVALID_ARG;
  if (B <= 0 || H <= 0 || M <= 0 || Nk <= 0 || d <= 0 || Nk < M) return AVITS_ERR_INVALID_ARG;
  if (!(softmax_scale > 0.f) || !(softmax_scale < 3.0e38f)) return AVITS_ERR_INVALID_ARG;
  if (q_sn < d || k_sn < d || q_sh < 0 || k_sh < 0 || q_sb < 0 || k_sb < 0)
    return AVITS_ERR_INVALID_ARG;
  SpatialArgs a{q_img, k_all, dt, B, H, M, Nk, 0, d, q_sb, q_sh, q_sn, k_sb, k_sh, k_sn,
                softmax_scale, weight, accumulate ? 1 : 0, A, lse_opt, workspace, ws_bytes,
                status_word(), text_mask};
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (spatial_tc_eligible(a)) {
    const int sms = num_sms_current();
    if (ws_bytes < spatial_tc_workspace(B, H, M, Nk, d, sms) || !workspace)
      return AVITS_ERR_INVALID_ARG;
    return cuda_status(launch_spatial_tc(a, sms, s));
  }
  if (d > 256) return AVITS_ERR_UNSUPPORTED;
  return cuda_status(launch_spatial_simt(a, num_sms_current(), s));
}

size_t avits_attention_forward_workspace(int B, int H, int Mq) {
  if (B <= 0 || H <= 0 || Mq <= 0) return 0;
  return attention_tc_workspace(B, H, Mq);
}

avits_status avits_attention_forward(const void* q, const void* k, const void* v, avits_dtype dt,
                                     int B, int H, int Mq, int Nk, int L, int d,
                                     const int64_t* q_str, const int64_t* k_str,
                                     const int64_t* v_str, const int64_t* o_str,
                                     float softmax_scale, void* o, float* lse_opt, float weight,
                                     int accumulate, float* A, void* workspace, size_t ws_bytes,
                                     void* stream) {
  AVITS_RANGE();
  if (!q || !k || !v || !o || !valid_dtype(dt)) return AVITS_ERR_INVALID_ARG;
  if (B <= 0 || H <= 0 || Mq <= 0 || Nk <= 0 || d <= 0 || L < 0 || L > Nk)
    return AVITS_ERR_INVALID_ARG;
  if (!(softmax_scale > 0.f) || !(softmax_scale < 3.0e38f)) return AVITS_ERR_INVALID_ARG;
  AttnArgs a{};
  a.q = q; a.k = k; a.v = v; a.o = o;
  a.B = B; a.H = H; a.Mq = Mq; a.Nk = Nk; a.L = L; a.d = d;
  const int64_t* given[4] = {q_str, k_str, v_str, o_str};
  for (int i = 0; i < 4; ++i) {
    const int64_t rows = (i == 1 || i == 2) ? Nk : Mq;
    if (given[i]) {
      for (int j = 0; j < 3; ++j) a.str[i][j] = given[i][j];
      if (a.str[i][2] < d || a.str[i][1] < 0 || a.str[i][0] < 0) return AVITS_ERR_INVALID_ARG;
    } else {
      a.str[i][2] = d;
      a.str[i][1] = rows * d;
      a.str[i][0] = (int64_t)H * rows * d;
    }
  }
  a.scale = softmax_scale;
  a.weight = weight;
  a.accumulate = accumulate ? 1 : 0;
  a.A = A;
  a.lse = lse_opt;
  a.ws = workspace;
  a.status = status_word();
  if (A && (!workspace || (reinterpret_cast<uintptr_t>(workspace) & 7u) ||
            ws_bytes < attention_tc_workspace(B, H, Mq)))
    return AVITS_ERR_INVALID_ARG;
  if (dt != AVITS_BF16) return AVITS_ERR_UNSUPPORTED;
  if (A && H > 255) return AVITS_ERR_UNSUPPORTED;   // the head count of the fixed-point sum
  if ((long long)B * H * ((Mq + 255) / 256) >= (1ll << 31)) return AVITS_ERR_UNSUPPORTED;
  if (!attention_tc_layout_ok(a)) return AVITS_ERR_UNSUPPORTED;
  return cuda_status(launch_attention_tc(a, num_sms_current(), static_cast<cudaStream_t>(stream)));
}

avits_status avits_score_temporal(const void* h_t, const void* h_prev, avits_dtype dt, int B,
                                  int N, int D, float eps, float* V, void* stream) {
  AVITS_RANGE();
  if (!h_t || !h_prev || !V || !valid_dtype(dt)) return AVITS_ERR_INVALID_ARG;
  if (B <= 0 || N <= 0 || D <= 0 || !(eps >= 0.f)) return AVITS_ERR_INVALID_ARG;
  return cuda_status(launch_temporal(h_t, h_prev, dt, B, N, D, eps, V, num_sms_current(),
                                     status_word(), static_cast<cudaStream_t>(stream)));
}

avits_status avits_score_spatiotemporal(const void* q_img, const void* k_all, avits_dtype dt,
                                        int B, int H, int M, int Nk, int L, int d, int64_t q_sb,
                                        int64_t q_sh, int64_t q_sn, int64_t k_sb, int64_t k_sh,
                                        int64_t k_sn, float softmax_scale, float weight,
                                        int accumulate, float* A, float* lse_opt, void* workspace,
                                        size_t ws_bytes, const void* h_t, const void* h_prev,
                                        int D, float eps, float* V, void* stream) {
  AVITS_RANGE();
  if (!q_img || !k_all || !A || !h_t || !h_prev || !V || !valid_dtype(dt))
    return AVITS_ERR_INVALID_ARG;
  if (B <= 0 || H <= 0 || M <= 0 || Nk <= 0 || d <= 0 || L < 0 || L > Nk || Nk < M || D <= 0)
    return AVITS_ERR_INVALID_ARG;
  if (!(softmax_scale > 0.f) || !(softmax_scale < 3.0e38f) || !(eps >= 0.f))
    return AVITS_ERR_INVALID_ARG;
  if (q_sn < d || k_sn < d || q_sh < 0 || k_sh < 0 || q_sb < 0 || k_sb < 0)
    return AVITS_ERR_INVALID_ARG;
  SpatialArgs a{q_img, k_all, dt, B, H, M, Nk, L, d, q_sb, q_sh, q_sn, k_sb, k_sh, k_sn,
                softmax_scale, weight, accumulate ? 1 : 0, A, lse_opt, workspace, ws_bytes,
                status_word()};
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const int sms = num_sms_current();
  if (spatial_tc_eligible(a)) {
    if (ws_bytes < spatial_tc_workspace(B, H, M, Nk, d, sms) || !workspace)
      return AVITS_ERR_INVALID_ARG;
    unsigned int* st = a.status;
    const LaunchHook temporal = [=](cudaStream_t ss) {
      return launch_temporal_overlapped(h_t, h_prev, dt, B, M, D, eps, V, sms, st, ss);
    };
    return cuda_status(launch_spatial_tc(a, sms, s, &temporal));
  }
  if (d > 256) return AVITS_ERR_UNSUPPORTED;
  cudaError_t e = launch_spatial_simt(a, num_sms_current(), s);
  if (e == cudaSuccess) e = launch_temporal(h_t, h_prev, dt, B, M, D, eps, V, sms, a.status, s);
  return cuda_status(e);
}

avits_status avits_score_temporal_var(const void* const* snaps, int n_t, avits_dtype dt, int B,
                                      int N, int D, float* V, void* stream) {
  AVITS_RANGE();
  if (!snaps || !V || !valid_dtype(dt)) return AVITS_ERR_INVALID_ARG;
  if (n_t < 2 || n_t > kMaxSnapshots || B <= 0 || N <= 0 || D <= 0) return AVITS_ERR_INVALID_ARG;
  for (int i = 0; i < n_t; ++i)
    if (!snaps[i]) return AVITS_ERR_INVALID_ARG;
  return cuda_status(launch_temporal_var(snaps, n_t, dt, B, N, D, V, num_sms_current(),
                                         static_cast<cudaStream_t>(stream)));
}

avits_status avits_fuse_select(const float* A, const float* V, int B, int M, float alpha,
                               float eps_norm, int k, float* S_opt, int32_t* sel_idx,
                               uint8_t* sel_mask_opt, int32_t* tok_offset, void* stream) {
  AVITS_RANGE();
  return avits_fuse_select_perturbed(A, V, nullptr, B, M, alpha, eps_norm, k, S_opt, sel_idx,
                                     sel_mask_opt, tok_offset, stream);
}

avits_status avits_fuse_select_perturbed(const float* A, const float* V, const float* perturb,
                                         int B, int M, float alpha, float eps_norm, int k,
                                         float* S_opt, int32_t* sel_idx, uint8_t* sel_mask_opt,
                                         int32_t* tok_offset, void* stream) {
  AVITS_RANGE();
  if (!A || !V || !tok_offset || (k > 0 && !sel_idx)) return AVITS_ERR_INVALID_ARG;
  if (B <= 0 || M <= 0 || M > kSelectMaxM || k < 0 || k > M) return AVITS_ERR_INVALID_ARG;
  if (!(alpha >= 0.f && alpha <= 1.f) || !(eps_norm >= 0.f)) return AVITS_ERR_INVALID_ARG;
  return cuda_status(launch_fuse_select(A, V, perturb, B, M, alpha, eps_norm, k, S_opt, sel_idx,
                                        sel_mask_opt, tok_offset, status_word(),
                                        static_cast<cudaStream_t>(stream)));
}

avits_status avits_selective_upsample(const void* latent, avits_dtype dt, int B, int M,
                                      int grid_h, int grid_w, int C, int p,
                                      const int32_t* pos_in_opt, const int32_t* span_in_opt,
                                      const uint8_t* sel_mask, const int32_t* tok_offset, int k,
                                      avits_upmode mode, void* out_latent, int32_t* out_pos,
                                      int32_t* out_span, int32_t* out_src_tok,
                                      int8_t* out_src_sub, void* workspace, size_t ws_bytes,
                                      void* stream) {
  AVITS_RANGE();
  if (!latent || !sel_mask || !tok_offset || !out_latent || !out_pos || !out_span ||
      !out_src_tok || !out_src_sub || !valid_dtype(dt))
    return AVITS_ERR_INVALID_ARG;
  if (B <= 0 || M <= 0 || grid_h <= 0 || grid_w <= 0 || C <= 0 || k < 0 || k > M)
    return AVITS_ERR_INVALID_ARG;
  if (p != 2) return AVITS_ERR_UNSUPPORTED;
  if ((pos_in_opt == nullptr) != (span_in_opt == nullptr)) return AVITS_ERR_INVALID_ARG;
  if (!pos_in_opt && (int64_t)grid_h * grid_w != M) return AVITS_ERR_INVALID_ARG;
  if (mode != AVITS_UP_NEAREST && mode != AVITS_UP_BILINEAR) return AVITS_ERR_INVALID_ARG;
  if (!aligned16(latent) || !aligned16(out_latent)) return AVITS_ERR_INVALID_ARG;
  if (!mixed_bilinear_ok(mode, pos_in_opt, B, M, grid_h, grid_w, workspace, ws_bytes))
    return AVITS_ERR_INVALID_ARG;
  return cuda_status(launch_upsample(latent, dt, B, M, grid_h, grid_w, C, pos_in_opt, span_in_opt,
                                     sel_mask, tok_offset, k, mode, out_latent, out_pos, out_span,
                                     out_src_tok, out_src_sub, workspace, status_word(),
                                     static_cast<cudaStream_t>(stream)));
}

size_t avits_selective_upsample_workspace(avits_upmode mode, int B, int grid_h, int grid_w) {
  if (mode != AVITS_UP_BILINEAR || B <= 0 || grid_h <= 0 || grid_w <= 0) return 0;
  return merge_workspace_bytes(B, grid_h, grid_w);
}

avits_status avits_select_upsample(const float* A, const float* V, const float* perturb, int B,
                                   int M, float alpha, float eps_norm, int k, float* S_opt,
                                   int32_t* sel_idx, uint8_t* sel_mask, int32_t* tok_offset,
                                   const void* latent, avits_dtype dt, int grid_h, int grid_w,
                                   int C, int p, const int32_t* pos_in_opt,
                                   const int32_t* span_in_opt, avits_upmode mode,
                                   void* out_latent, int32_t* out_pos, int32_t* out_span,
                                   int32_t* out_src_tok, int8_t* out_src_sub, void* workspace,
                                   size_t ws_bytes, void* stream) {
  AVITS_RANGE();
  if (!A || !V || !tok_offset || !sel_mask || (k > 0 && !sel_idx)) return AVITS_ERR_INVALID_ARG;
  if (B <= 0 || M <= 0 || M > kSelectMaxM || k < 0 || k > M) return AVITS_ERR_INVALID_ARG;
  if (!(alpha >= 0.f && alpha <= 1.f) || !(eps_norm >= 0.f)) return AVITS_ERR_INVALID_ARG;
  if (!latent || !out_latent || !out_pos || !out_span || !out_src_tok || !out_src_sub ||
      !valid_dtype(dt))
    return AVITS_ERR_INVALID_ARG;
  if (grid_h <= 0 || grid_w <= 0 || C <= 0) return AVITS_ERR_INVALID_ARG;
  if (p != 2) return AVITS_ERR_UNSUPPORTED;
  if ((pos_in_opt == nullptr) != (span_in_opt == nullptr)) return AVITS_ERR_INVALID_ARG;
  if (!pos_in_opt && (int64_t)grid_h * grid_w != M) return AVITS_ERR_INVALID_ARG;
  if (mode != AVITS_UP_NEAREST && mode != AVITS_UP_BILINEAR) return AVITS_ERR_INVALID_ARG;
  if (!aligned16(latent) || !aligned16(out_latent)) return AVITS_ERR_INVALID_ARG;
  if (!mixed_bilinear_ok(mode, pos_in_opt, B, M, grid_h, grid_w, workspace, ws_bytes))
    return AVITS_ERR_INVALID_ARG;
  return cuda_status(launch_select_upsample(
      A, V, perturb, B, M, alpha, eps_norm, k, S_opt, sel_idx, sel_mask, tok_offset,
      status_word(), latent, dt, grid_h, grid_w, C, pos_in_opt, span_in_opt, mode, out_latent,
      out_pos, out_span, out_src_tok, out_src_sub, workspace, static_cast<cudaStream_t>(stream)));
}

size_t avits_merge_final_workspace(avits_upmode mode, int B, int full_h, int full_w) {
  if ((mode != AVITS_UP_NEAREST && mode != AVITS_UP_BILINEAR) || B <= 0 || full_h <= 0 ||
      full_w <= 0)
    return 0;
  return merge_workspace_bytes(B, full_h, full_w);
}

avits_status avits_merge_final(const void* mixed, avits_dtype dt, int B, int N, const int32_t* pos,
                               const int32_t* span, int full_h, int full_w, int C, int p,
                               avits_upmode mode, void* out_full, void* workspace,
                               size_t ws_bytes, void* stream) {
  AVITS_RANGE();
  if (!mixed || !pos || !span || !out_full || !valid_dtype(dt)) return AVITS_ERR_INVALID_ARG;
  if (B <= 0 || N <= 0 || full_h <= 0 || full_w <= 0 || C <= 0) return AVITS_ERR_INVALID_ARG;
  if (p != 2) return AVITS_ERR_UNSUPPORTED;
  if (mode != AVITS_UP_NEAREST && mode != AVITS_UP_BILINEAR) return AVITS_ERR_INVALID_ARG;
  if (!aligned16(mixed) || !aligned16(out_full)) return AVITS_ERR_INVALID_ARG;
  if (mode == AVITS_UP_BILINEAR && ((full_h & 1) || (full_w & 1) || N > (1 << 28) - 1))
    return AVITS_ERR_INVALID_ARG;
  if (!workspace || !aligned16(workspace) ||
      ws_bytes < avits_merge_final_workspace(mode, B, full_h, full_w))
    return AVITS_ERR_INVALID_ARG;
  return cuda_status(launch_merge(mixed, dt, B, N, pos, span, full_h, full_w, C, mode, out_full,
                                  workspace, status_word(), static_cast<cudaStream_t>(stream)));
}

avits_status avits_selftest_bounded_wait(unsigned long long limit_ns, long long* result,
                                         void* stream) {
  AVITS_RANGE();
  if (!result || limit_ns < 1000ull || limit_ns > 100ull * 1000ull * 1000ull)
    return AVITS_ERR_INVALID_ARG;
  return cuda_status(launch_wait_selftest(limit_ns, result, status_word(),
                                          static_cast<cudaStream_t>(stream)));
}

avits_status avits_device_status(void* stream) {
  AVITS_RANGE();
  cudaError_t e = cudaStreamSynchronize(static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_status(e);
  unsigned int w = 0, zero = 0;
  e = cudaMemcpyFromSymbol(&w, g_status, sizeof(w));
  if (e != cudaSuccess) return cuda_status(e);
  if (w) {
    e = cudaMemcpyToSymbol(g_status, &zero, sizeof(zero));
    if (e != cudaSuccess) return cuda_status(e);
  }
  for (int c = 1; c < 32; ++c)
    if (w & (1u << c)) return static_cast<avits_status>(c);
  return AVITS_OK;
}

}  // extern "C"
