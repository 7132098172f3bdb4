// Step 3: the tree merge of the P workers' sketches (Alg. 1 steps 8-23).
//
// On a cluster each round moves whole sketches between workers; with all P tables on one
// GPU the same reduction tree is applied cell by cell in registers.  A thread loads cell q
// of every worker once (the W interleaved lanes of a group are adjacent, so four of them
// arrive in one 16-byte load), runs the rounds -- round l adds worker a + 2^l into worker a
// for every a that is a multiple of 2^(l+1) with a + 2^l < P, which is the recursive-halving
// schedule including the rule that the largest participant of an odd round sits it out --
// and writes the root value.  Each cell therefore sees exactly the fp32 additions of the
// paper's tree, in the same order, and the tables are read once and written once.
#include "gs_common.cuh"

namespace gs {

namespace {

template <int W>
__device__ __forceinline__ void load_group(const float* __restrict__ src, float* v, int lanes) {
  if (W == 16) {
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const float4 a = __ldcs(reinterpret_cast<const float4*>(src + 4 * q));
      v[4 * q] = a.x; v[4 * q + 1] = a.y; v[4 * q + 2] = a.z; v[4 * q + 3] = a.w;
    }
  } else if (W == 8) {
    const float4 a = __ldcs(reinterpret_cast<const float4*>(src));
    const float4 b = __ldcs(reinterpret_cast<const float4*>(src + 4));
    v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
    v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
  } else if (W == 4) {
    const float4 a = __ldcs(reinterpret_cast<const float4*>(src));
    v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
  } else if (W == 2) {
    const float2 a = __ldcs(reinterpret_cast<const float2*>(src));
    v[0] = a.x; v[1] = a.y;
  } else {
    v[0] = __ldcs(src);
  }
  (void)lanes;
}

// PMAX: compile-time bound on P (a power of two >= P and >= W) so the values stay in
// registers; the rounds test a + s < P at run time.
template <int W, int PMAX>
__global__ void __launch_bounds__(kBlock) k_merge(const __grid_constant__ MergeParams prm) {
  grid_begin();
  static_assert(PMAX % W == 0, "PMAX must be a multiple of W");
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const int P = prm.P;
  const int groups = (P + W - 1) / W;
  for (int64_t q = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; q < prm.cells; q += stride) {
    float v[PMAX];
#pragma unroll
    for (int g = 0; g < PMAX / W; ++g) {
      if (g < groups) {
        load_group<W>(prm.tables + g * prm.group_stride + q * W, v + g * W, W);
      } else {
#pragma unroll
        for (int l = 0; l < W; ++l) v[g * W + l] = 0.f;
      }
    }
#pragma unroll
    for (int s = 1; s < PMAX; s *= 2) {
#pragma unroll
      for (int a = 0; a + s < PMAX; a += 2 * s) {
        if (a + s < P) v[a] = __fadd_rn(v[a + s], v[a]);  // sends = recvs + sends
      }
    }
    prm.merged[q] = v[0];
  }
}

// The same tree over P separately allocated tables: cell q of input i is
// tables[i][q * lane_stride[i]] (worker 0 of a sketch whose tables interleave lane_stride
// workers).
template <int PMAX>
__global__ void __launch_bounds__(kBlock) k_merge_list(const __grid_constant__ MergeListParams prm) {
  grid_begin();
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const int P = prm.P;
  for (int64_t q = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; q < prm.cells; q += stride) {
    float v[PMAX];
#pragma unroll
    for (int i = 0; i < PMAX; ++i) v[i] = i < P ? __ldcs(prm.tables[i] + q * prm.lane_stride[i]) : 0.f;
#pragma unroll
    for (int s = 1; s < PMAX; s *= 2) {
#pragma unroll
      for (int a = 0; a + s < PMAX; a += 2 * s) {
        if (a + s < P) v[a] = __fadd_rn(v[a + s], v[a]);  // sends = recvs + sends
      }
    }
    prm.merged[q] = v[0];
  }
}

template <int PMAX>
cudaError_t launch_list_t(const MergeListParams& p, cudaStream_t s) {
  auto kern = k_merge_list<PMAX>;
  const int64_t need = (p.cells + kBlock - 1) / kBlock;
  const int64_t cap = (int64_t)device_info().sms * blocks_per_sm((const void*)kern, kBlock);
  const int grid = (int)(need < 1 ? 1 : (need < cap ? need : cap));
  launch(kern, grid, kBlock, s, p);
  return cudaGetLastError();
}

template <int W, int PMAX>
cudaError_t launch_t(const MergeParams& p, cudaStream_t s) {
  auto kern = k_merge<W, PMAX>;
  const int64_t need = (p.cells + kBlock - 1) / kBlock;
  const int64_t cap = (int64_t)device_info().sms * blocks_per_sm((const void*)kern, kBlock);
  const int grid = (int)(need < 1 ? 1 : (need < cap ? need : cap));
  launch(kern, grid, kBlock, s, p);
  return cudaGetLastError();
}

template <int W>
cudaError_t launch_w(const MergeParams& p, cudaStream_t s) {
  const int P = p.P;
  if (P <= W && W >= 1) return launch_t<W, W>(p, s);
  if (P <= 8 && W <= 8) return launch_t<W, (W > 8 ? W : 8)>(p, s);
  if (P <= 16) return launch_t<W, 16>(p, s);
  if (P <= 32) return launch_t<W, 32>(p, s);
  return launch_t<W, 64>(p, s);
}

}  // namespace

cudaError_t launch_merge_list(const MergeListParams& p, cudaStream_t s) {
  if (p.P <= 1) return launch_list_t<1>(p, s);
  if (p.P <= 2) return launch_list_t<2>(p, s);
  if (p.P <= 4) return launch_list_t<4>(p, s);
  if (p.P <= 8) return launch_list_t<8>(p, s);
  if (p.P <= 16) return launch_list_t<16>(p, s);
  if (p.P <= 32) return launch_list_t<32>(p, s);
  return launch_list_t<64>(p, s);
}

cudaError_t launch_merge(const MergeParams& p, int W, cudaStream_t s) {
  switch (W) {
    case 1: return launch_w<1>(p, s);
    case 2: return launch_w<2>(p, s);
    case 4: return launch_w<4>(p, s);
    case 8: return launch_w<8>(p, s);
    case 16: return launch_w<16>(p, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace gs
