// Step 6: the second round of Alg. 2 -- the exact values of the selected coordinates --
// and step 7, the weight update of Alg. 1 (w <- w - lr * G~, G~ = the gathered values at the
// selected indices and zero elsewhere), which the gather can apply on the fly.
//
// On a cluster the workers exchange their accumulated values at the k selected indices;
// here every worker's error vector is on the device.  A group of G lanes (a power of two,
// G >= P up to 32) serves one selected index: lane l loads the values of workers l, l + G,
// ... in parallel; the values are then added in worker order (fp32, p = 0, 1, ..., P - 1:
// the order and rounding of one thread summing alone) by shuffling them past every lane of
// the group; the group's first lane writes the sum, and every lane zeroes its workers'
// momentum and error at that coordinate (the selected mass has been applied, so it leaves
// the accumulators).  Indices outside [0, d) touch no memory; their value is NaN.
#include "gs_common.cuh"

namespace gs {

namespace {

template <int G>
__global__ void __launch_bounds__(kBlock) k_gather_and_zero(const __grid_constant__ GatherParams prm) {
  grid_begin();
  // workers per lane: one while G >= P (G < 32), else up to GS_MAX_WORKERS / 32
  constexpr int kPer = (G == 32) ? (GS_MAX_WORKERS + 31) / 32 : 1;
  const int lane = threadIdx.x & 31;
  const int sub = lane & (G - 1);
  // the lanes of this group: every shuffle below stays inside it, and all of them share t
  const uint32_t gmask = (G == 32) ? 0xFFFFFFFFu : (((1u << G) - 1u) << (lane & ~(G - 1)));
  const int64_t ngroups = (int64_t)gridDim.x * (blockDim.x / G);
  for (int64_t t = (int64_t)blockIdx.x * (blockDim.x / G) + threadIdx.x / G; t < prm.k; t += ngroups) {
    const int64_t i = prm.idx[t];
    const bool ok = i >= 0 && i < prm.d;
    float v[kPer];
#pragma unroll
    for (int q = 0; q < kPer; ++q) {
      const int p = sub + q * G;
      v[q] = (ok && p < prm.P) ? prm.e[p][i] : 0.f;
    }
    float sum = 0.f;
    for (int p = 0; p < prm.P; ++p) {
      float x = 0.f;
#pragma unroll
      for (int q = 0; q < kPer; ++q)
        if (p / G == q) x = v[q];
      sum = __fadd_rn(sum, __shfl_sync(gmask, x, p % G, G));
    }
    if (!ok) {
      if (sub == 0) prm.vals[t] = __int_as_float(0x7FC00000);
      continue;
    }
#pragma unroll
    for (int q = 0; q < kPer; ++q) {
      const int p = sub + q * G;
      if (p < prm.P) {
        prm.u[p][i] = 0.f;
        prm.e[p][i] = 0.f;
      }
    }
    if (sub == 0) {
      prm.vals[t] = sum;
      if (prm.w) prm.w[i] = __fsub_rn(prm.w[i], __fmul_rn(prm.lr, sum));
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

template <int G>
cudaError_t launch_gather_g(const GatherParams& p, cudaStream_t s) {
  const int64_t need = (p.k * G + kBlock - 1) / kBlock;
  const int64_t cap = (int64_t)device_info().sms * blocks_per_sm((const void*)k_gather_and_zero<G>, kBlock);
  const int grid = (int)(need < 1 ? 1 : (need < cap ? need : cap));
  launch(k_gather_and_zero<G>, grid, kBlock, s, p);
  return cudaGetLastError();
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
  if (p.P <= 1) return launch_gather_g<1>(p, s);
  if (p.P <= 2) return launch_gather_g<2>(p, s);
  if (p.P <= 4) return launch_gather_g<4>(p, s);
  if (p.P <= 8) return launch_gather_g<8>(p, s);
  if (p.P <= 16) return launch_gather_g<16>(p, s);
  return launch_gather_g<32>(p, s);
}

}  // namespace gs
