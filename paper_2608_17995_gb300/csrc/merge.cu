// merge.cu — final merge to the dense full-resolution latent (Sec. 3.2,
// Stage 3: the remaining tokens are expanded and the sequence is laid out in
// spatial order).
//
// Nearest: one warp per mixed token scatters its s x s cells; full-res pixel
// (Y,X) of a token at (y,x) with span s takes token pixel ((Y-2y)/s, (X-2x)/s).
// Bilinear (spans 1 and 2): a cell map is scattered first (atomicExch into a
// -1-filled workspace, so double cover and holes are detected), then every
// output (cell, channel) gathers: span-1 cells are copied, span-2 cells take
// the half-pixel-centred 2x bilinear resize of the rebuilt low-res grid, in
// which each 2x2 block of span-1 tokens contributes its 2x2 average pools.
// Algorithmic bytes: B*N*(T*elt + 12) read + B*fh*fw*T*elt written.
#include "avits_common.cuh"
#include "avits_internal.h"

namespace avits {
namespace {

constexpr int kWarpsPerCta = 8;

template <typename T>
struct Pix4;
template <>
struct Pix4<float> {
  using V = float4;
  __device__ static V make(float a, float b, float c, float d) { return make_float4(a, b, c, d); }
};
template <>
struct Pix4<__nv_bfloat16> {
  using V = uint2;
  __device__ static V make(float a, float b, float c, float d) {
    const __nv_bfloat162 lo = __floats2bfloat162_rn(a, b);
    const __nv_bfloat162 hi = __floats2bfloat162_rn(c, d);
    return make_uint2(*reinterpret_cast<const uint32_t*>(&lo),
                      *reinterpret_cast<const uint32_t*>(&hi));
  }
};

template <typename T>
__global__ void __launch_bounds__(kWarpsPerCta * 32)
merge_nearest_kernel(const T* __restrict__ mixed, int B, int N, const int32_t* __restrict__ pos,
                     const int32_t* __restrict__ span, int fh, int fw, int C, T* __restrict__ out,
                     unsigned int* status) {
  using PV = typename Pix4<T>::V;
  pdl_wait_then_trigger();
  const int lane = threadIdx.x & 31;
  const int64_t gwarp = (int64_t)blockIdx.x * kWarpsPerCta + (threadIdx.x >> 5);
  if (gwarp >= (int64_t)B * N) return;
  const int b = (int)(gwarp / N);
  const int y = pos[gwarp * 2], x = pos[gwarp * 2 + 1], s = span[gwarp];
  if (s <= 0 || y < 0 || x < 0 || y + s > fh || x + s > fw) {
    if (lane == 0) raise_status(status, AVITS_ERR_COVERAGE);
    return;
  }
  const int T4 = C * 4;
  const T* src = mixed + gwarp * T4;
  const int tasks = s * s * C;
  for (int task = lane; task < tasks; task += 32) {
    const int cell = task / C, c = task - cell * C;
    const int u = cell / s, v = cell - u * s;
    const int r0 = (2 * u) / s, r1 = (2 * u + 1) / s;
    const int c0 = (2 * v) / s, c1 = (2 * v + 1) / s;
    const T* sc = src + c * 4;
    const float p00 = load_elem(sc, r0 * 2 + c0), p01 = load_elem(sc, r0 * 2 + c1);
    const float p10 = load_elem(sc, r1 * 2 + c0), p11 = load_elem(sc, r1 * 2 + c1);
    const int64_t ocell = (int64_t)b * fh * fw + (int64_t)(y + u) * fw + (x + v);
    reinterpret_cast<PV*>(out + ocell * T4)[c] = Pix4<T>::make(p00, p01, p10, p11);
  }
}

__global__ void merge_map_kernel(int B, int N, const int32_t* __restrict__ pos,
                                 const int32_t* __restrict__ span, int fh, int fw,
                                 int32_t* __restrict__ map, unsigned int* status) {
  const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= (int64_t)B * N) return;
  const int b = (int)(t / N), ti = (int)(t % N);
  const int y = pos[t * 2], x = pos[t * 2 + 1], s = span[t];
  if ((s != 1 && s != 2) || y < 0 || x < 0 || y + s > fh || x + s > fw ||
      (s == 2 && ((y | x) & 1))) {
    raise_status(status, AVITS_ERR_COVERAGE);
    return;
  }
  for (int u = 0; u < s; ++u)
    for (int v = 0; v < s; ++v) {
      const int old = atomicExch(&map[(int64_t)b * fh * fw + (int64_t)(y + u) * fw + x + v], ti);
      if (old != -1) raise_status(status, AVITS_ERR_COVERAGE);
    }
}

template <typename T>
__device__ __forceinline__ float low_pixel(const T* __restrict__ mb, const int32_t* __restrict__ mapb,
                                           const int32_t* __restrict__ spanb, int fw, int T4, int ch,
                                           int r, int c) {
  const int t0 = mapb[(r & ~1) * fw + (c & ~1)];
  if (t0 < 0) return 0.f;
  if (spanb[t0] == 2) return load_elem(mb, (int64_t)t0 * T4 + ch * 4 + (r & 1) * 2 + (c & 1));
  const int t1 = mapb[r * fw + c];
  if (t1 < 0) return 0.f;
  const T* p = mb + (int64_t)t1 * T4 + ch * 4;
  const float top = __fadd_rn(load_elem(p, 0), load_elem(p, 1));
  const float bot = __fadd_rn(load_elem(p, 2), load_elem(p, 3));
  return __fmul_rn(__fadd_rn(top, bot), 0.25f);
}

__device__ __forceinline__ void bil_axis(int P, int n, int& r0, int& r1, float& w0, float& w1) {
  const int m = P >> 1;
  if ((P & 1) == 0) { r0 = m - 1; r1 = m; w0 = 0.25f; w1 = 0.75f; }
  else { r0 = m; r1 = m + 1; w0 = 0.75f; w1 = 0.25f; }
  r0 = max(r0, 0);
  r1 = min(r1, n - 1);
}

template <typename T>
__global__ void merge_bilinear_kernel(const T* __restrict__ mixed, int B, int N,
                                      const int32_t* __restrict__ span, int fh, int fw, int C,
                                      const int32_t* __restrict__ map, T* __restrict__ out,
                                      unsigned int* status) {
  using PV = typename Pix4<T>::V;
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
  const int32_t* spanb = span + (int64_t)b * N;
  const T* mb = mixed + (int64_t)b * N * T4;
  const int t = mapb[cell];
  PV* dst = reinterpret_cast<PV*>(out + bc * T4) + c;
  if (t < 0) {
    raise_status(status, AVITS_ERR_COVERAGE);
    *dst = Pix4<T>::make(0.f, 0.f, 0.f, 0.f);
    return;
  }
  if (spanb[t] == 1) {
    *dst = reinterpret_cast<const PV*>(mb + (int64_t)t * T4)[c];
    return;
  }
  float r[4];
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    int r0, r1, c0, c1;
    float wy0, wy1, wx0, wx1;
    bil_axis(2 * Y + (q >> 1), fh, r0, r1, wy0, wy1);
    bil_axis(2 * X + (q & 1), fw, c0, c1, wx0, wx1);
    const float p00 = low_pixel(mb, mapb, spanb, fw, T4, c, r0, c0);
    const float p01 = low_pixel(mb, mapb, spanb, fw, T4, c, r0, c1);
    const float p10 = low_pixel(mb, mapb, spanb, fw, T4, c, r1, c0);
    const float p11 = low_pixel(mb, mapb, spanb, fw, T4, c, r1, c1);
    const float top = __fadd_rn(__fmul_rn(wx0, p00), __fmul_rn(wx1, p01));
    const float bot = __fadd_rn(__fmul_rn(wx0, p10), __fmul_rn(wx1, p11));
    r[q] = __fadd_rn(__fmul_rn(wy0, top), __fmul_rn(wy1, bot));
  }
  *dst = Pix4<T>::make(r[0], r[1], r[2], r[3]);
}

template <typename T>
cudaError_t launch_t(const void* mixed, int B, int N, const int32_t* pos, const int32_t* span,
                     int fh, int fw, int C, avits_upmode mode, void* out, void* ws,
                     unsigned int* status, cudaStream_t s) {
  if (mode == AVITS_UP_NEAREST) {
    const int64_t warps = (int64_t)B * N;
    const int grid = (int)((warps + kWarpsPerCta - 1) / kWarpsPerCta);
    cudaError_t e = prefer_max_shared<merge_nearest_kernel<T>>();
    if (e != cudaSuccess) return e;
    e = launch_pdl(merge_nearest_kernel<T>, dim3(grid), dim3(kWarpsPerCta * 32), 0, s,
                               static_cast<const T*>(mixed), B, N, pos, span, fh, fw, C,
                               static_cast<T*>(out), status);
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
  }
  int32_t* map = static_cast<int32_t*>(ws);
  cudaError_t e = cudaMemsetAsync(map, 0xFF, sizeof(int32_t) * (size_t)B * fh * fw, s);
  if (e != cudaSuccess) return e;
  const int64_t nt = (int64_t)B * N;
  merge_map_kernel<<<(int)((nt + 255) / 256), 256, 0, s>>>(B, N, pos, span, fh, fw, map, status);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const int64_t work = (int64_t)B * fh * fw * C;
  merge_bilinear_kernel<T><<<(int)((work + 255) / 256), 256, 0, s>>>(
      static_cast<const T*>(mixed), B, N, span, fh, fw, C, map, static_cast<T*>(out), status);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_merge(const void* mixed, avits_dtype dt, int B, int N, const int32_t* pos,
                         const int32_t* span, int fh, int fw, int C, avits_upmode mode,
                         void* out, void* ws, unsigned int* status, cudaStream_t s) {
  if (dt == AVITS_BF16)
    return launch_t<__nv_bfloat16>(mixed, B, N, pos, span, fh, fw, C, mode, out, ws, status, s);
  return launch_t<float>(mixed, B, N, pos, span, fh, fw, C, mode, out, ws, status, s);
}

}  // namespace avits
