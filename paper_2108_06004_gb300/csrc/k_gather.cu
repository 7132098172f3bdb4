// Step 6: the second round of Alg. 2 -- the exact values of the selected coordinates --
// and step 7, the weight update of Alg. 1 (w <- w - lr * G~, G~ = the gathered values at the
// selected indices and zero elsewhere), which the gather can apply on the fly.
//
// On a cluster the workers exchange their accumulated values at the k selected indices;
// here every worker's error vector is on the device, so one thread per selected index
// reads the P values, sums them in worker order (fp32), writes the sum, and zeroes that
// coordinate of every worker's momentum and error (the selected mass has been applied,
// so it leaves the accumulators).  Indices outside [0, d) touch no memory; their value is
// NaN.
#include "gs_common.cuh"

namespace gs {

namespace {

__global__ void __launch_bounds__(kBlock) k_gather_and_zero(const __grid_constant__ GatherParams prm) {
  grid_begin();
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < prm.k; t += stride) {
    const int64_t i = prm.idx[t];
    if (i < 0 || i >= prm.d) {
      prm.vals[t] = __int_as_float(0x7FC00000);
      continue;
    }
    float v = 0.f;
    for (int p = 0; p < prm.P; ++p) v = __fadd_rn(v, prm.e[p][i]);
    prm.vals[t] = v;
    if (prm.w) prm.w[i] = __fsub_rn(prm.w[i], __fmul_rn(prm.lr, v));
    for (int p = 0; p < prm.P; ++p) {
      prm.u[p][i] = 0.f;
      prm.e[p][i] = 0.f;
    }
  }
}

// w[idx[t]] <- fl(w[idx[t]] - fl(lr * vals[t])); indices outside [0, d) are skipped.
__global__ void __launch_bounds__(kBlock) k_apply_update(float* __restrict__ w, int64_t d,
                                                         const int64_t* __restrict__ idx,
                                                         const float* __restrict__ vals, int64_t k, float lr) {
  grid_begin();
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < k; t += stride) {
    const int64_t i = idx[t];
    if (i >= 0 && i < d) w[i] = __fsub_rn(w[i], __fmul_rn(lr, vals[t]));
  }
}

}  // namespace

cudaError_t launch_apply_update(float* w, int64_t d, const int64_t* idx, const float* vals, int64_t k, float lr,
                                cudaStream_t s) {
  const int64_t need = (k + kBlock - 1) / kBlock;
  const int64_t cap = (int64_t)device_info().sms * blocks_per_sm((const void*)k_apply_update, kBlock);
  const int grid = (int)(need < 1 ? 1 : (need < cap ? need : cap));
  launch(k_apply_update, grid, kBlock, s, w, d, idx, vals, k, lr);
  return cudaGetLastError();
}

cudaError_t launch_gather_and_zero(const GatherParams& p, cudaStream_t s) {
  const int64_t need = (p.k + kBlock - 1) / kBlock;
  const int64_t cap = (int64_t)device_info().sms * blocks_per_sm((const void*)k_gather_and_zero, kBlock);
  const int grid = (int)(need < 1 ? 1 : (need < cap ? need : cap));
  launch(k_gather_and_zero, grid, kBlock, s, p);
  return cudaGetLastError();
}

}  // namespace gs
