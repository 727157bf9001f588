// upsample.cu — selective upsampling into a packed mixed-resolution sequence
// (Sec. 3.2, Stage 2).
//
// One warp per input token i (upsample_token in upsample_token.cuh); its
// outputs start at tok_offset[i] (from the selection kernel), so no scan is
// needed here.  Algorithmic bytes per launch:
// B*M*T*elt (read) + B*M*5 (mask, offset) + B*N_out*(T*elt + 17).
#include "avits_common.cuh"
#include "avits_internal.h"
#include "frame_map.cuh"
#include "upsample_token.cuh"

namespace avits {
namespace {

constexpr int kWarpsPerCta = 8;

template <typename T, bool kBilinear>
__global__ void __launch_bounds__(kWarpsPerCta * 32)
upsample_kernel(const T* __restrict__ latent, int B, int M, int gh, int gw, int C,
                const int32_t* __restrict__ pos_in, const int32_t* __restrict__ span_in,
                const uint8_t* __restrict__ mask, const int32_t* __restrict__ tok_offset,
                int n_out, T* __restrict__ out, int32_t* __restrict__ out_pos,
                int32_t* __restrict__ out_span, int32_t* __restrict__ out_src_tok,
                int8_t* __restrict__ out_src_sub, const int32_t* __restrict__ map,
                unsigned int* status) {
  pdl_wait_then_trigger();
  const int lane = threadIdx.x & 31;
  const int64_t gwarp = (int64_t)blockIdx.x * kWarpsPerCta + (threadIdx.x >> 5);
  if (gwarp >= (int64_t)B * M) return;
  const int b = (int)(gwarp / M), i = (int)(gwarp % M);
  const int64_t in_tok = (int64_t)b * M + i;
  const UpsampleArgs<T> u{latent, M, gh, gw, C, n_out, pos_in, span_in, out,
                          out_pos, out_span, out_src_tok, out_src_sub, map, status};
  const GlobalRows<T> rows{latent, M, C * 4};
  upsample_token<T, kBilinear>(u, rows, b, i, tok_offset[in_tok], mask[in_tok] != 0, lane);
}

template <typename T>
cudaError_t launch_t(const void* latent, int B, int M, int gh, int gw, int C,
                     const int32_t* pos_in, const int32_t* span_in, const uint8_t* mask,
                     const int32_t* tok_offset, int k, avits_upmode mode, void* out,
                     int32_t* out_pos, int32_t* out_span, int32_t* out_src_tok,
                     int8_t* out_src_sub, void* ws, unsigned int* status, cudaStream_t s) {
  const int64_t warps = (int64_t)B * M;
  const int grid = (int)((warps + kWarpsPerCta - 1) / kWarpsPerCta);
  const int n_out = M + 3 * k;
  cudaError_t e = prefer_max_shared<upsample_kernel<T, true>>();
  if (e == cudaSuccess) e = prefer_max_shared<upsample_kernel<T, false>>();
  if (e != cudaSuccess) return e;
  // bilinear with a mixed input: the input frame's cell map first
  int32_t* map = nullptr;
  if (mode == AVITS_UP_BILINEAR && pos_in) {
    map = reinterpret_cast<int32_t*>(static_cast<uint8_t*>(ws) + 16);
    e = launch_cell_map(B, M, pos_in, span_in, gh, gw, map, status, s);
    if (e != cudaSuccess) return e;
  }
  auto kern = (mode == AVITS_UP_BILINEAR) ? upsample_kernel<T, true> : upsample_kernel<T, false>;
  e = launch_pdl(kern, dim3(grid), dim3(kWarpsPerCta * 32), 0, s,
                 static_cast<const T*>(latent), B, M, gh, gw, C, pos_in, span_in, mask,
                 tok_offset, n_out, static_cast<T*>(out), out_pos, out_span, out_src_tok,
                 out_src_sub, static_cast<const int32_t*>(map), status);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_upsample(const void* latent, avits_dtype dt, int B, int M, int gh, int gw,
                            int C, const int32_t* pos_in, const int32_t* span_in,
                            const uint8_t* mask, const int32_t* tok_offset, int k,
                            avits_upmode mode, void* out, int32_t* out_pos, int32_t* out_span,
                            int32_t* out_src_tok, int8_t* out_src_sub, void* ws,
                            unsigned int* status, cudaStream_t s) {
  if (dt == AVITS_BF16)
    return launch_t<__nv_bfloat16>(latent, B, M, gh, gw, C, pos_in, span_in, mask, tok_offset, k,
                                   mode, out, out_pos, out_span, out_src_tok, out_src_sub, ws,
                                   status, s);
  return launch_t<float>(latent, B, M, gh, gw, C, pos_in, span_in, mask, tok_offset, k, mode, out,
                         out_pos, out_span, out_src_tok, out_src_sub, ws, status, s);
}

}  // namespace avits
