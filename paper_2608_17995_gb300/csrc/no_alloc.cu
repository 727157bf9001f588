// no_alloc.cu — avits_score_spatial_noalloc: the spatial score for callers
// that cannot allocate device memory.
//
// Some callers only ever receive input/output device pointers and a stream
// (an inference engine's plugin "enqueue" hook, a custom-op callback inside
// a serving runtime, code running between pre-planned memory passes): they
// have no allocator they may call there, and cudaMalloc would either
// synchronise the device or be illegal in the context they run in.  This
// entry point gives them the tensor-core spatial score with its scratch in a
// fixed device array of this library instead of a caller workspace.
//
// The array is a file-scope __device__ variable: every GPU that loads the
// library holds kStaticScratchBytes of it until the process exits.  The host
// only knows the array by a stand-in symbol, so its device address is looked
// up once per device (cudaGetSymbolAddress, with that device current) on the
// first call made on that device, and that address is what the kernels get.
#include <cstdio>
#include <cstring>

#include "avits_common.cuh"
#include "avits_internal.h"

namespace avits {
namespace {

// Upper bound of the scratch one call may use (per-row partial statistics
// of every (SM, key range) piece, the ready flags and the per-row head-sum
// words).  Covers the 1024^2 and 2048^2 FLUX-shaped
// transitions, the editing shape and a batch of 8 second transitions.
constexpr size_t kStaticScratchBytes = 8u << 20;

static __device__ __align__(256) unsigned char g_spatial_scratch[kStaticScratchBytes];

constexpr int kMaxDevices = 64;
void* g_scratch_ptr[kMaxDevices] = {};

thread_local char t_noalloc_error[160] = "";

// Device address of g_spatial_scratch on the current device (looked up on
// the first call per device; concurrent first calls store the same value).
cudaError_t scratch_address(void** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  void* p = __atomic_load_n(&g_scratch_ptr[dev], __ATOMIC_ACQUIRE);
  if (!p) {
    e = cudaGetSymbolAddress(&p, g_spatial_scratch);
    if (e != cudaSuccess) return e;
    __atomic_store_n(&g_scratch_ptr[dev], p, __ATOMIC_RELEASE);
  }
  *out = p;
  return cudaSuccess;
}

}  // namespace
}  // namespace avits

using namespace avits;

extern "C" {

avits_status avits_score_spatial_noalloc(const void* q_img, const void* k_all, avits_dtype dt,
                                         int B, int H, int M, int Nk, int L, int d, int64_t q_sb,
                                         int64_t q_sh, int64_t q_sn, int64_t k_sb, int64_t k_sh,
                                         int64_t k_sn, float softmax_scale, float weight,
                                         int accumulate, float* A, float* lse_opt, void* stream) {
  AVITS_RANGE();
  t_noalloc_error[0] = '\0';
  if (!q_img || !k_all || !A || dt != AVITS_BF16) return AVITS_ERR_INVALID_ARG;
  if (B <= 0 || H <= 0 || M <= 0 || Nk <= 0 || d <= 0 || L < 0 || L > Nk || Nk < M)
    return AVITS_ERR_INVALID_ARG;
  if (!(softmax_scale > 0.f) || !(softmax_scale < 3.0e38f)) return AVITS_ERR_INVALID_ARG;
  if (q_sn < d || k_sn < d || q_sh < 0 || k_sh < 0 || q_sb < 0 || k_sb < 0)
    return AVITS_ERR_INVALID_ARG;
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) {
    cudaGetLastError();
    return AVITS_ERR_CUDA;
  }
  void* scratch = nullptr;
  SpatialArgs a{q_img, k_all, dt, B, H, M, Nk, L, d, q_sb, q_sh, q_sn, k_sb, k_sh, k_sn,
                softmax_scale, weight, accumulate ? 1 : 0, A, lse_opt, nullptr,
                kStaticScratchBytes, status_word()};
  if (!spatial_tc_eligible(a)) return AVITS_ERR_UNSUPPORTED;   // d in {64,128}, 16-B layout
  const size_t need = spatial_tc_workspace(B, H, M, Nk, d, sms);
  if (need > kStaticScratchBytes) {
    snprintf(t_noalloc_error, sizeof(t_noalloc_error),
             "avits_score_spatial_noalloc: %zu bytes of scratch needed, the static array "
             "holds %zu", need, kStaticScratchBytes);
    return AVITS_ERR_INVALID_ARG;
  }
  cudaError_t e = scratch_address(&scratch);
  if (e != cudaSuccess) {
    cudaGetLastError();
    cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
    if (cudaStreamIsCapturing(static_cast<cudaStream_t>(stream), &cap) == cudaSuccess &&
        cap != cudaStreamCaptureStatusNone)
      snprintf(t_noalloc_error, sizeof(t_noalloc_error),
               "avits_score_spatial_noalloc: the first call on a device looks up the scratch "
               "address and must come before stream capture (%s)", cudaGetErrorString(e));
    else
      snprintf(t_noalloc_error, sizeof(t_noalloc_error),
               "avits_score_spatial_noalloc: scratch address lookup failed (%s)",
               cudaGetErrorString(e));
    cudaGetLastError();
    return AVITS_ERR_CUDA;
  }
  a.ws = scratch;
  // the row words and ready flags of the in-kernel merge start at zero; a
  // call that stopped on a timeout may have left some set, so every call
  // clears them (a memset on the stream: no allocation)
  e = cudaMemsetAsync(scratch, 0, spatial_tc_zeroed_bytes(B, H, M, Nk, d, sms),
                      static_cast<cudaStream_t>(stream));
  if (e == cudaSuccess) e = launch_spatial_tc(a, sms, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) {
    cudaGetLastError();
    return AVITS_ERR_CUDA;
  }
  return AVITS_OK;
}

size_t avits_score_spatial_noalloc_limit(void) { return kStaticScratchBytes; }

const char* avits_score_spatial_noalloc_error(void) { return t_noalloc_error; }

}  // extern "C"
