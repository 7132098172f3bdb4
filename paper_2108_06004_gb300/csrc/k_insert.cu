// Step 1 (accumulate) and step 2 (Count Sketch insert) of the gs-SGD compression step, and
// the fused pass that does both while streaming each worker's vectors once.
//
// Layout: a group of W simulated workers shares one interleaved table [r][c][W] (fp32), so
// the W workers' contributions to cell (j, b) are adjacent.  All workers share the hash
// functions (Sec. III-A: sketches only merge by addition when they do), so the 2r hash
// values of a coordinate serve every worker of the group; a thread evaluates them for
// four consecutive coordinates, the later three in the incremental form x(i+1) = x(i) + a.
//
// L2 reductions are the bound of this pass (random reductions run at a fixed rate of
// requests, whatever their width up to 16 bytes, and the load-store unit merges the
// requests of one warp instruction that fall in the same sector).  So for W >= 4 a group of
// G = W/4 adjacent lanes shares one coordinate quad, each lane owns four workers, and one
// warp instruction writes whole W*4-byte cells with 16-byte vector reductions
// (red.global.add.v4.f32).  For tables larger than the L2 budget the rows are inserted in
// passes over row ranges: the first pass accumulates, later passes only re-read e.  The
// streams carry an evict_first and the reductions an evict_last L2 policy, so that the table
// slice of a pass stays in L2 while the vectors flow past it.
#include "gs_common.cuh"

namespace gs {

namespace {

__device__ __forceinline__ void acc1(float rho, float& u, float& e, float g) {
  u = __fadd_rn(__fmul_rn(rho, u), g);  // fl(fl(rho*u) + g), never contracted to an FMA
  e = __fadd_rn(e, u);
}

__global__ void __launch_bounds__(kBlock) k_accumulate(float* __restrict__ u,
                                                       float* __restrict__ e,
                                                       const float* __restrict__ g, int64_t d,
                                                       float rho, int vec) {
  grid_begin();
  const int64_t nq = (d + 3) / 4;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t q = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; q < nq; q += stride) {
    const int64_t i0 = q * 4;
    if (vec && i0 + 4 <= d) {
      float4 g4 = __ldcs(reinterpret_cast<const float4*>(g + i0));
      float4 u4 = __ldcs(reinterpret_cast<const float4*>(u + i0));
      float4 e4 = __ldcs(reinterpret_cast<const float4*>(e + i0));
      acc1(rho, u4.x, e4.x, g4.x);
      acc1(rho, u4.y, e4.y, g4.y);
      acc1(rho, u4.z, e4.z, g4.z);
      acc1(rho, u4.w, e4.w, g4.w);
      __stcs(reinterpret_cast<float4*>(u + i0), u4);
      __stcs(reinterpret_cast<float4*>(e + i0), e4);
    } else {
      for (int t = 0; t < 4 && i0 + t < d; ++t) {
        float uu = u[i0 + t], ee = e[i0 + t];
        acc1(rho, uu, ee, g[i0 + t]);
        u[i0 + t] = uu;
        e[i0 + t] = ee;
      }
    }
  }
}

// Load (and with ACC, update and store) four consecutive coordinates of lane w.  WIN (the
// request-ceiling probe only) folds the vector offset into a window of prm.winmask + 1 floats.
template <bool ACC, bool VEC, bool WIN = false>
__device__ __forceinline__ void load_lane(const InsertParams& prm, int w, int64_t i0,
                                          int64_t d, float (&ev)[4]) {
  if (VEC && i0 + 4 <= d) {
    const int64_t ia = WIN ? (i0 & prm.winmask) : i0;
    float4 e4 = __ldcs(reinterpret_cast<const float4*>(prm.e[w] + ia));
    if (ACC) {
      float4 g4 = __ldcs(reinterpret_cast<const float4*>(prm.g[w] + ia));
      float4 u4 = __ldcs(reinterpret_cast<const float4*>(prm.u[w] + ia));
      acc1(prm.rho, u4.x, e4.x, g4.x);
      acc1(prm.rho, u4.y, e4.y, g4.y);
      acc1(prm.rho, u4.z, e4.z, g4.z);
      acc1(prm.rho, u4.w, e4.w, g4.w);
      __stcs(reinterpret_cast<float4*>(prm.u[w] + ia), u4);
      __stcs(reinterpret_cast<float4*>(prm.e[w] + ia), e4);
    }
    ev[0] = e4.x;
    ev[1] = e4.y;
    ev[2] = e4.z;
    ev[3] = e4.w;
  } else if (WIN) {
#pragma unroll
    for (int t = 0; t < 4; ++t) ev[t] = 0.f;  // the probe's ragged tail carries no requests
  } else {
#pragma unroll
    for (int t = 0; t < 4; ++t) {
      ev[t] = 0.f;
      if (i0 + t < d) {
        float ee = prm.e[w][i0 + t];
        if (ACC) {
          float uu = prm.u[w][i0 + t];
          acc1(prm.rho, uu, ee, prm.g[w][i0 + t]);
          prm.u[w][i0 + t] = uu;
          prm.e[w][i0 + t] = ee;
        }
        ev[t] = ee;
      }
    }
  }
}

// load_lane with L2 eviction priorities on the vector streams (the coop kernel's form).
template <bool ACC, bool VEC, bool WIN>
__device__ __forceinline__ void load_lane_hinted(const InsertParams& prm, int w, int64_t i0, int64_t d,
                                                 float (&ev)[4], uint64_t pol) {
  if (VEC && i0 + 4 <= d) {
    const int64_t ia = WIN ? (i0 & prm.winmask) : i0;
    float4 e4 = ld_stream(prm.e[w] + ia, pol);
    if (ACC) {
      const float4 g4 = ld_stream(prm.g[w] + ia, pol);
      float4 u4 = ld_stream(prm.u[w] + ia, pol);
      acc1(prm.rho, u4.x, e4.x, g4.x);
      acc1(prm.rho, u4.y, e4.y, g4.y);
      acc1(prm.rho, u4.z, e4.z, g4.z);
      acc1(prm.rho, u4.w, e4.w, g4.w);
      st_stream(prm.u[w] + ia, u4, pol);
      st_stream(prm.e[w] + ia, e4, pol);
    }
    ev[0] = e4.x;
    ev[1] = e4.y;
    ev[2] = e4.z;
    ev[3] = e4.w;
  } else {
    load_lane<ACC, VEC, WIN>(prm, w, i0, d, ev);
  }
}

// W <= 2: one thread = four consecutive coordinates of every worker in the group.
//   ACC: accumulate (u, e update) before inserting e; otherwise insert e as given.
//   VEC: all vectors 16-byte aligned (float4 path for full quads).
//   POW2: c is a power of two (bucket = x & (c - 1)).
template <int W, bool ACC, bool VEC, bool POW2>
__global__ void __launch_bounds__(kBlock) k_accumulate_insert(const __grid_constant__ InsertParams prm) {
  grid_begin();
  const int64_t d = prm.d;
  const int64_t nq = (d + 3) / 4;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t q = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; q < nq; q += stride) {
    const int64_t i0 = q * 4;
    float ev[W][4];
#pragma unroll
    for (int w = 0; w < W; ++w) {
      if (w < prm.nw) {
        load_lane<ACC, VEC>(prm, w, i0, d, ev[w]);
      } else {
#pragma unroll
        for (int t = 0; t < 4; ++t) ev[w][t] = 0.f;
      }
    }
    const int tmax = (d - i0 < 4) ? (int)(d - i0) : 4;
#pragma unroll 1
    for (int j = prm.j0; j < prm.j1; ++j) {
      const uint64_t a = prm.h.a[j], a2 = prm.h.a2[j];
      uint64_t x = affine61(a, prm.h.b[j], (uint32_t)i0);
      uint64_t y = affine61(a2, prm.h.b2[j], (uint32_t)i0);
      float* row = prm.table + (size_t)j * prm.c * W;
#pragma unroll
      for (int t = 0; t < 4; ++t) {
        if (t < tmax) {
          const uint32_t bk = bucket_of<POW2>(x, prm.c, prm.cmask);
          const uint32_t sb = signbit_of(y);
          float* cell = row + (size_t)bk * W;
          if (W == 1) {
            red_add_f32(cell, apply_sign(ev[0][t], sb));
          } else {
            red_add_v2(cell, apply_sign(ev[0][t], sb), apply_sign(ev[W > 1 ? 1 : 0][t], sb));
          }
          x = step61(x, a);
          y = step61(y, a2);
        }
      }
    }
  }
}

// W >= 4: G = W/4 adjacent lanes share one quad of coordinates; lane `sub` of the group
// owns workers 4*sub .. 4*sub+3 and, per row and coordinate, issues one 16-byte reduction
// at offset 4*sub of the cell, so the G lanes of the group cover the whole cell in the same
// instruction.  The hash is evaluated by every lane of the group (issue slots are not the
// bound here).
template <int W, bool ACC, bool VEC, bool POW2, bool WIN = false>
__global__ void __launch_bounds__(kBlock) k_accumulate_insert_coop(const __grid_constant__ InsertParams prm) {
  grid_begin();
  constexpr int G = W / 4;
  const int sub = threadIdx.x % G;
  const int64_t d = prm.d;
  const int64_t nq = (d + 3) / 4;
  const int64_t qstride = (int64_t)gridDim.x * (blockDim.x / G);
  const uint64_t pol_stream = policy_evict_first(), pol_table = policy_evict_last();
  for (int64_t q = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) / G; q < nq; q += qstride) {
    const int64_t i0 = q * 4;
    float ev[4][4];
#pragma unroll
    for (int w4 = 0; w4 < 4; ++w4) {
      const int w = sub * 4 + w4;
      if (w < prm.nw) {
        load_lane_hinted<ACC, VEC, WIN>(prm, w, i0, d, ev[w4], pol_stream);
      } else {
#pragma unroll
        for (int t = 0; t < 4; ++t) ev[w4][t] = 0.f;
      }
    }
    const int tmax = (d - i0 < 4) ? (int)(d - i0) : 4;
#pragma unroll 1
    for (int j = prm.j0; j < prm.j1; ++j) {
      const uint64_t a = prm.h.a[j], a2 = prm.h.a2[j];
      uint64_t x = affine61(a, prm.h.b[j], (uint32_t)i0);
      uint64_t y = affine61(a2, prm.h.b2[j], (uint32_t)i0);
      float* row = prm.table + (size_t)j * prm.c * W + sub * 4;
#pragma unroll
      for (int t = 0; t < 4; ++t) {
        if (t < tmax) {
          const uint32_t bk = bucket_of<POW2>(x, prm.c, prm.cmask);
          const uint32_t sb = signbit_of(y);
          red_add_v4_keep(row + (size_t)bk * W, apply_sign(ev[0][t], sb), apply_sign(ev[1][t], sb),
                          apply_sign(ev[2][t], sb), apply_sign(ev[3][t], sb), pol_table);
          x = step61(x, a);
          y = step61(y, a2);
        }
      }
    }
  }
}

// Insert one vector (prm.e[0]) into lane prm.lane of a W-wide group table.
template <bool POW2>
__global__ void __launch_bounds__(kBlock) k_insert_lane(const __grid_constant__ InsertParams prm, int W) {
  grid_begin();
  const int64_t d = prm.d;
  const int64_t nq = (d + 3) / 4;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const float* v = prm.e[0];
  for (int64_t q = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; q < nq; q += stride) {
    const int64_t i0 = q * 4;
    const int tmax = (d - i0 < 4) ? (int)(d - i0) : 4;
    float ev[4];
#pragma unroll
    for (int t = 0; t < 4; ++t) ev[t] = (t < tmax) ? v[i0 + t] : 0.f;
#pragma unroll 1
    for (int j = prm.j0; j < prm.j1; ++j) {
      const uint64_t a = prm.h.a[j], a2 = prm.h.a2[j];
      uint64_t x = affine61(a, prm.h.b[j], (uint32_t)i0);
      uint64_t y = affine61(a2, prm.h.b2[j], (uint32_t)i0);
      float* row = prm.table + (size_t)j * prm.c * W + prm.lane;
#pragma unroll
      for (int t = 0; t < 4; ++t) {
        if (t < tmax) {
          const uint32_t bk = bucket_of<POW2>(x, prm.c, prm.cmask);
          red_add_f32(row + (size_t)bk * W, apply_sign(ev[t], signbit_of(y)));
          x = step61(x, a);
          y = step61(y, a2);
        }
      }
    }
  }
}

// Shared-memory-staged insert (the alternative to k_accumulate_insert_coop's direct cell
// reductions; the error vectors are already accumulated).  blockIdx.y is the row j and
// blockIdx.z a tile of WT adjacent workers of the group; blockIdx.x a contiguous chunk of the
// coordinates.  The CTA keeps row j of its WT workers' tables in shared memory ([c][WT] fp32),
// adds its chunk into it with shared-memory atomics, then flushes the tile into the group
// table with one WT-wide vector reduction per bucket (buckets the chunk never touched are
// skipped).  Only for tables whose tile fits: c * WT * 4 bytes of dynamic shared memory.
template <int WT, bool POW2>
__global__ void __launch_bounds__(kBlock) k_insert_staged(const __grid_constant__ InsertParams prm, int W,
                                                         int64_t chunk) {
  grid_begin();
  extern __shared__ float tile[];
  const int j = blockIdx.y;
  const int w0 = blockIdx.z * WT;
  const uint32_t c = prm.c;
  for (uint32_t b = threadIdx.x; b < c * WT; b += blockDim.x) tile[b] = 0.f;
  __syncthreads();
  const int64_t d = prm.d;
  const int64_t a0 = (int64_t)blockIdx.x * chunk;
  const int64_t a1 = a0 + chunk < d ? a0 + chunk : d;
  const uint64_t a = prm.h.a[j], a2 = prm.h.a2[j];
  for (int64_t i0 = a0 + 4 * (int64_t)threadIdx.x; i0 < a1; i0 += 4 * (int64_t)blockDim.x) {
    const int tmax = (a1 - i0 < 4) ? (int)(a1 - i0) : 4;
    float ev[WT][4];
#pragma unroll
    for (int w = 0; w < WT; ++w) {
#pragma unroll
      for (int t = 0; t < 4; ++t) ev[w][t] = (w0 + w < prm.nw && t < tmax) ? prm.e[w0 + w][i0 + t] : 0.f;
    }
    uint64_t x = affine61(a, prm.h.b[j], (uint32_t)i0);
    uint64_t y = affine61(a2, prm.h.b2[j], (uint32_t)i0);
#pragma unroll
    for (int t = 0; t < 4; ++t) {
      if (t < tmax) {
        const uint32_t bk = bucket_of<POW2>(x, c, prm.cmask);
        const uint32_t sb = signbit_of(y);
#pragma unroll
        for (int w = 0; w < WT; ++w) atomicAdd(&tile[bk * WT + w], apply_sign(ev[w][t], sb));
        x = step61(x, a);
        y = step61(y, a2);
      }
    }
  }
  __syncthreads();
  float* row = prm.table + (size_t)j * c * W + w0;
  for (uint32_t b = threadIdx.x; b < c; b += blockDim.x) {
    float v[WT];
    bool any = false;
#pragma unroll
    for (int w = 0; w < WT; ++w) {
      v[w] = tile[b * WT + w];
      any = any || v[w] != 0.f;
    }
    if (!any) continue;
    float* cell = row + (size_t)b * W;
    if (WT == 4) red_add_v4(cell, v[0], v[WT > 1 ? 1 : 0], v[WT > 2 ? 2 : 0], v[WT > 3 ? 3 : 0]);
    else if (WT == 2) red_add_v2(cell, v[0], v[WT > 1 ? 1 : 0]);
    else red_add_f32(cell, v[0]);
  }
}

__global__ void k_hash_eval(const __grid_constant__ HashCoeffs h, int r, uint32_t c,
                            const int64_t* __restrict__ coords, int64_t n,
                            int32_t* __restrict__ bucket_out, int8_t* __restrict__ sign_out) {
  grid_begin();
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < n; t += stride) {
    const int64_t i = coords[t];
    const bool ok = (i >= 0 && i < (1ll << 31));
    for (int j = 0; j < r; ++j) {
      if (ok) {
        const uint64_t x = affine61(h.a[j], h.b[j], (uint32_t)i);
        const uint64_t y = affine61(h.a2[j], h.b2[j], (uint32_t)i);
        bucket_out[(int64_t)j * n + t] = (int32_t)(x % (uint64_t)c);
        sign_out[(int64_t)j * n + t] = (y & 1u) ? (int8_t)-1 : (int8_t)1;
      } else {
        bucket_out[(int64_t)j * n + t] = -1;
        sign_out[(int64_t)j * n + t] = 0;
      }
    }
  }
}

template <typename K>
int grid_for(K kernel, int64_t work_items, int block) {
  const int64_t need = (work_items + block - 1) / block;
  const int64_t cap = (int64_t)device_info().sms * blocks_per_sm((const void*)kernel, block);
  return (int)(need < 1 ? 1 : (need < cap ? need : cap));
}

template <int W, bool ACC, bool VEC, bool POW2>
cudaError_t launch_ai_t(const InsertParams& p, cudaStream_t s) {
  if constexpr (W >= 4) {
    auto kern = k_accumulate_insert_coop<W, ACC, VEC, POW2>;
    const int grid = grid_for(kern, (p.d + 3) / 4 * (W / 4), kBlock);
    launch(kern, grid, kBlock, s, p);
  } else {
    auto kern = k_accumulate_insert<W, ACC, VEC, POW2>;
    const int grid = grid_for(kern, (p.d + 3) / 4, kBlock);
    launch(kern, grid, kBlock, s, p);
  }
  return cudaGetLastError();
}

template <int W, bool ACC>
cudaError_t launch_ai_w(const InsertParams& p, bool vec, cudaStream_t s) {
  const bool pow2 = is_pow2(p.c);
  if (vec) return pow2 ? launch_ai_t<W, ACC, true, true>(p, s) : launch_ai_t<W, ACC, true, false>(p, s);
  return pow2 ? launch_ai_t<W, ACC, false, true>(p, s) : launch_ai_t<W, ACC, false, false>(p, s);
}

template <int W>
cudaError_t launch_ai_acc(const InsertParams& p, bool acc, bool vec, cudaStream_t s) {
  return acc ? launch_ai_w<W, true>(p, vec, s) : launch_ai_w<W, false>(p, vec, s);
}

}  // namespace

cudaError_t launch_accumulate(float* u, float* e, const float* g, int64_t d, float rho,
                              cudaStream_t s) {
  const bool vec = ((reinterpret_cast<uintptr_t>(u) | reinterpret_cast<uintptr_t>(e) |
                     reinterpret_cast<uintptr_t>(g)) & 15u) == 0;
  const int grid = grid_for(k_accumulate, (d + 3) / 4, kBlock);
  launch(k_accumulate, grid, kBlock, s, u, e, g, d, rho, vec ? 1 : 0);
  return cudaGetLastError();
}

cudaError_t launch_accumulate_insert(const InsertParams& p, int W, bool acc, bool vec, cudaStream_t s) {
  switch (W) {
    case 1: return launch_ai_acc<1>(p, acc, vec, s);
    case 2: return launch_ai_acc<2>(p, acc, vec, s);
    case 4: return launch_ai_acc<4>(p, acc, vec, s);
    case 8: return launch_ai_acc<8>(p, acc, vec, s);
    case 16: return launch_ai_acc<16>(p, acc, vec, s);
    default: return cudaErrorInvalidValue;
  }
}

template <int W>
cudaError_t launch_ceiling_w(const InsertParams& p, bool acc, cudaStream_t s) {
  auto kern = acc ? k_accumulate_insert_coop<W, true, true, true, true> : k_accumulate_insert_coop<W, false, true, true, true>;
  // the same grid as the insert it stands for
  auto real = acc ? k_accumulate_insert_coop<W, true, true, true> : k_accumulate_insert_coop<W, false, true, true>;
  const int grid = grid_for(real, (p.d + 3) / 4 * (W / 4), kBlock);
  launch(kern, grid, kBlock, s, p);
  return cudaGetLastError();
}

cudaError_t launch_insert_ceiling_probe(const InsertParams& p, int W, bool acc, cudaStream_t s) {
  if (!is_pow2(p.c)) return cudaErrorInvalidValue;
  switch (W) {
    case 4: return launch_ceiling_w<4>(p, acc, s);
    case 8: return launch_ceiling_w<8>(p, acc, s);
    case 16: return launch_ceiling_w<16>(p, acc, s);
    default: return cudaErrorInvalidValue;
  }
}

int staged_tile_width(uint32_t c, int W) {
  int wt = W < 4 ? W : 4;
  while (wt > 1 && (size_t)c * wt * sizeof(float) > kStagedSmemBytes) wt /= 2;
  return (size_t)c * wt * sizeof(float) <= kStagedSmemBytes ? wt : 0;
}

template <int WT, bool POW2>
cudaError_t launch_staged_t(const InsertParams& p, int W, cudaStream_t s) {
  auto kern = k_insert_staged<WT, POW2>;
  const size_t smem = (size_t)p.c * WT * sizeof(float);
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  // about two CTAs per SM over all (row, worker tile) pairs, at least one chunk
  const int tiles = (p.j1 - p.j0) * (W / WT);
  int64_t nchunk = (2 * (int64_t)device_info().sms + tiles - 1) / tiles;
  int64_t chunk = (p.d + nchunk - 1) / nchunk;
  chunk = (chunk + 3) / 4 * 4;
  nchunk = (p.d + chunk - 1) / chunk;
  InsertParams q = p;
  q.table = p.table + (size_t)p.j0 * p.c * W;  // blockIdx.y counts rows from j0
  for (int j = p.j0; j < p.j1; ++j) {  // coefficients re-based so that row blockIdx.y is row j
    q.h.a[j - p.j0] = p.h.a[j];
    q.h.b[j - p.j0] = p.h.b[j];
    q.h.a2[j - p.j0] = p.h.a2[j];
    q.h.b2[j - p.j0] = p.h.b2[j];
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)nchunk, (unsigned)(p.j1 - p.j0), (unsigned)(W / WT));
  cfg.blockDim = dim3(kBlock);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  e = cudaLaunchKernelEx(&cfg, kern, q, W, chunk);
  return e != cudaSuccess ? e : cudaGetLastError();
}

cudaError_t launch_insert_staged(const InsertParams& p, int W, cudaStream_t s) {
  const int wt = staged_tile_width(p.c, W);
  const bool pow2 = is_pow2(p.c);
  switch (wt) {
    case 4: return pow2 ? launch_staged_t<4, true>(p, W, s) : launch_staged_t<4, false>(p, W, s);
    case 2: return pow2 ? launch_staged_t<2, true>(p, W, s) : launch_staged_t<2, false>(p, W, s);
    case 1: return pow2 ? launch_staged_t<1, true>(p, W, s) : launch_staged_t<1, false>(p, W, s);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t launch_insert_lane(const InsertParams& p, int W, cudaStream_t s) {
  if (is_pow2(p.c)) {
    const int grid = grid_for(k_insert_lane<true>, (p.d + 3) / 4, kBlock);
    launch(k_insert_lane<true>, grid, kBlock, s, p, W);
  } else {
    const int grid = grid_for(k_insert_lane<false>, (p.d + 3) / 4, kBlock);
    launch(k_insert_lane<false>, grid, kBlock, s, p, W);
  }
  return cudaGetLastError();
}

cudaError_t launch_hash_eval(const HashCoeffs& h, int r, uint32_t c, const int64_t* coords,
                             int64_t n, int32_t* bucket_out, int8_t* sign_out, cudaStream_t s) {
  const int grid = grid_for(k_hash_eval, n, kBlock);
  launch(k_hash_eval, grid, kBlock, s, h, r, c, coords, n, bucket_out, sign_out);
  return cudaGetLastError();
}

}  // namespace gs
