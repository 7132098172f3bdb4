// Momentum and error kept as sketches (the linear-sketch variant named in Sec. II): the
// per-index pieces a step needs besides the insert, merge, accumulate and query kernels.
//   k_query_at     the median estimate of a table at k given coordinates
//   k_add_sparse   table += scale * S(v) for a sparse vector v (k values at k coordinates):
//                  with scale = -1 the extracted mass leaves the sketch
//   k_take         out[t] = src[idx[t]]
#include "gs_common.cuh"

namespace gs {

namespace {

__global__ void __launch_bounds__(kBlock) k_query_at(const float* __restrict__ T, const __grid_constant__ HashCoeffs h,
                                                     int r, uint32_t c, const int64_t* __restrict__ idx, int64_t k,
                                                     float* __restrict__ out) {
  grid_begin();
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < k; t += stride) {
    const int64_t i = idx[t];
    if (i < 0 || i >= (1ll << 31)) {
      out[t] = __int_as_float(0x7FC00000);
      continue;
    }
    float v[GS_MAX_ROWS];
    for (int j = 0; j < r; ++j) {
      const uint64_t x = affine61(h.a[j], h.b[j], (uint32_t)i);
      const uint64_t y = affine61(h.a2[j], h.b2[j], (uint32_t)i);
      v[j] = apply_sign(T[(size_t)j * c + bucket_of<false>(x, c, c - 1)], signbit_of(y));
    }
    for (int a = 1; a < r; ++a) {  // insertion sort
      const float tv = v[a];
      int b = a - 1;
      while (b >= 0 && v[b] > tv) {
        v[b + 1] = v[b];
        --b;
      }
      v[b + 1] = tv;
    }
    out[t] = (r & 1) ? v[r / 2] : 0.5f * (v[r / 2 - 1] + v[r / 2]);
  }
}

__global__ void __launch_bounds__(kBlock) k_add_sparse(float* __restrict__ T, const __grid_constant__ HashCoeffs h,
                                                       int r, uint32_t c, const int64_t* __restrict__ idx,
                                                       const float* __restrict__ vals, int64_t k, float scale) {
  grid_begin();
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < k; t += stride) {
    const int64_t i = idx[t];
    if (i < 0 || i >= (1ll << 31)) continue;
    const float v = __fmul_rn(scale, vals[t]);
    for (int j = 0; j < r; ++j) {
      const uint64_t x = affine61(h.a[j], h.b[j], (uint32_t)i);
      const uint64_t y = affine61(h.a2[j], h.b2[j], (uint32_t)i);
      red_add_f32(T + (size_t)j * c + bucket_of<false>(x, c, c - 1), apply_sign(v, signbit_of(y)));
    }
  }
}

__global__ void __launch_bounds__(kBlock) k_take(const float* __restrict__ src, int64_t n, const int64_t* __restrict__ idx,
                                                 int64_t k, float* __restrict__ out) {
  grid_begin();
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < k; t += stride) {
    const int64_t i = idx[t];
    out[t] = (i >= 0 && i < n) ? src[i] : __int_as_float(0x7FC00000);
  }
}

template <typename K>
int small_grid(K kernel, int64_t k) {
  const int64_t need = (k + kBlock - 1) / kBlock;
  const int64_t cap = (int64_t)device_info().sms * blocks_per_sm((const void*)kernel, kBlock);
  return (int)(need < 1 ? 1 : (need < cap ? need : cap));
}

}  // namespace

cudaError_t launch_query_at(const float* T, const HashCoeffs& h, int r, uint32_t c, const int64_t* idx, int64_t k,
                            float* out, cudaStream_t s) {
  launch(k_query_at, small_grid(k_query_at, k), kBlock, s, T, h, r, c, idx, k, out);
  return cudaGetLastError();
}

cudaError_t launch_add_sparse(float* T, const HashCoeffs& h, int r, uint32_t c, const int64_t* idx, const float* vals,
                              int64_t k, float scale, cudaStream_t s) {
  launch(k_add_sparse, small_grid(k_add_sparse, k), kBlock, s, T, h, r, c, idx, vals, k, scale);
  return cudaGetLastError();
}

cudaError_t launch_take(const float* src, int64_t n, const int64_t* idx, int64_t k, float* out, cudaStream_t s) {
  launch(k_take, small_grid(k_take, k), kBlock, s, src, n, idx, k, out);
  return cudaGetLastError();
}

}  // namespace gs
