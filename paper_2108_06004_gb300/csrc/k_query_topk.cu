// Steps 4 and 5: median-of-r query of the merged sketch and top-k selection
// (Alg. 2 steps 1-3, read as a deterministic top-k by |est| with ties to the smaller index).
//
// Pipeline (all on one stream, no host round trip):
//   k_query     est_i = median_j s_j(i) T[j][h_j(i)] for every i, written as fp32, and a
//               2048-bin histogram of key bits 30..20, key = bits of |est_i| (for
//               non-negative floats the bit pattern orders like the value).
//   k_pick      one CTA finds the bin that holds the k-th largest key and how many keys of
//               that bin are still to be taken.
//   k_hist      histogram of the next key bits among keys in the chosen bin (bits 19..9,
//               then bits 8..0); k_pick again after each.  After three levels the k-th
//               largest key tau is exact, and need_eq = k - #{key > tau} keys equal to tau
//               are taken, those of smallest index.
//   k_count     per segment of 16384 coordinates: #{key > tau}, #{key == tau}
//   k_scan      one CTA: exclusive prefix sums over the segments
//   k_write     every segment writes its selected indices at their final positions, so the
//               output is in ascending index order without a sort.
#include <mutex>

#include "gs_common.cuh"

namespace gs {

namespace {

constexpr int kBins = 2048;
constexpr int kSeg = 16384;       // coordinates per CTA in k_count / k_write
constexpr int kPerThread = 16;    // consecutive coordinates per thread in k_write
constexpr int kScanThreads = 1024;
constexpr uint32_t kNone = 0xFFFFFFFFu;

struct SelectState {
  uint32_t prefix;   // key bits fixed so far
  uint32_t k_rem;    // keys still to take inside the prefix
  uint32_t tau;      // the k-th largest key
  uint32_t need_eq;  // keys equal to tau to take
  uint32_t found;    // bit l set when level l found its bin
};

struct Workspace {
  float* est;
  uint32_t* hist;     // 3 * kBins
  SelectState* st;
  uint32_t* blk_gt;   // nblk each
  uint32_t* blk_eq;
  uint32_t* blk_base;
  uint32_t* blk_eqx;
  int64_t nblk;
};

inline size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

Workspace carve(void* base, int64_t d) {
  Workspace w;
  char* p = static_cast<char*>(base);
  const int64_t nblk = (d + kSeg - 1) / kSeg;
  w.est = reinterpret_cast<float*>(p);
  p += align256((size_t)d * sizeof(float));
  w.hist = reinterpret_cast<uint32_t*>(p);
  p += align256(3 * kBins * sizeof(uint32_t));
  w.st = reinterpret_cast<SelectState*>(p);
  p += align256(sizeof(SelectState));
  w.blk_gt = reinterpret_cast<uint32_t*>(p);
  w.blk_eq = w.blk_gt + nblk;
  w.blk_base = w.blk_eq + nblk;
  w.blk_eqx = w.blk_base + nblk;
  w.nblk = nblk;
  return w;
}

__device__ __forceinline__ uint32_t key_of(float v) { return __float_as_uint(v) & 0x7FFFFFFFu; }

// Warp-aggregated shared-memory histogram update; every lane of the warp must call it.
__device__ __forceinline__ void hist_add(uint32_t* sh, uint32_t bin) {
  const uint32_t peers = __match_any_sync(0xFFFFFFFFu, bin);
  const int leader = __ffs(peers) - 1;
  if (bin != kNone && (int)(threadIdx.x & 31) == leader) atomicAdd(&sh[bin], (uint32_t)__popc(peers));
}

__device__ __forceinline__ void hist_flush(const uint32_t* sh, uint32_t* hist, int nbins) {
  __syncthreads();
  for (int b = threadIdx.x; b < nbins; b += blockDim.x) {
    const uint32_t n = sh[b];
    if (n) atomicAdd(&hist[b], n);
  }
}

// Exclusive scan of one uint32 per thread across the block; *total gets the block sum.
__device__ __forceinline__ uint32_t block_excl_scan(uint32_t v, uint32_t* total) {
  __shared__ uint32_t warp_sums[32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int nwarps = (blockDim.x + 31) >> 5;
  uint32_t x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t y = __shfl_up_sync(0xFFFFFFFFu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) warp_sums[warp] = x;
  __syncthreads();
  if (warp == 0) {
    uint32_t w = lane < nwarps ? warp_sums[lane] : 0u;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t y = __shfl_up_sync(0xFFFFFFFFu, w, o);
      if (lane >= o) w += y;
    }
    warp_sums[lane] = w;
  }
  __syncthreads();
  const uint32_t off = warp ? warp_sums[warp - 1] : 0u;
  *total = warp_sums[nwarps - 1];
  __syncthreads();
  return off + x - v;
}

template <int R>
__device__ __forceinline__ float median_of(float (&v)[R]) {
#pragma unroll
  for (int i = 0; i < R; ++i) {
#pragma unroll
    for (int j = 0; j + 1 < R - i; ++j) {
      const float lo = fminf(v[j], v[j + 1]), hi = fmaxf(v[j], v[j + 1]);
      v[j] = lo;
      v[j + 1] = hi;
    }
  }
  if (R & 1) return v[R / 2];
  return 0.5f * (v[R / 2 - 1] + v[R / 2]);
}

struct QueryParams {
  const float* T;     // merged table [r][c]
  float* est;         // [d]
  uint32_t* hist;     // level-1 histogram
  int64_t d;
  int32_t r;
  uint32_t c, cmask;
  int32_t vec;        // est 16-byte aligned
  HashCoeffs h;
};

__device__ __forceinline__ void store_est(const QueryParams& prm, int64_t i0, int tmax,
                                          const float (&m)[4]) {
  if (prm.vec && tmax == 4) {
    *reinterpret_cast<float4*>(prm.est + i0) = make_float4(m[0], m[1], m[2], m[3]);
  } else {
    for (int t = 0; t < tmax; ++t) prm.est[i0 + t] = m[t];
  }
}

// Fast path: R rows known at compile time, c a power of two.
template <int R>
__global__ void __launch_bounds__(kBlock) k_query(const __grid_constant__ QueryParams prm) {
  __shared__ uint32_t sh[kBins];
  for (int b = threadIdx.x; b < kBins; b += blockDim.x) sh[b] = 0;
  __syncthreads();
  const int64_t d = prm.d, nq = (d + 3) / 4;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const int lane = threadIdx.x & 31;
  for (int64_t q0 = (int64_t)blockIdx.x * blockDim.x + (threadIdx.x & ~31); q0 < nq; q0 += stride) {
    const int64_t q = q0 + lane;
    const int64_t i0 = q * 4;
    const int tmax = q < nq ? (d - i0 < 4 ? (int)(d - i0) : 4) : 0;
    float m[4] = {0.f, 0.f, 0.f, 0.f};
    if (tmax > 0) {
      float v[4][R];
#pragma unroll
      for (int j = 0; j < R; ++j) {
        uint64_t x = affine61(prm.h.a[j], prm.h.b[j], (uint32_t)i0);
        uint64_t y = affine61(prm.h.a2[j], prm.h.b2[j], (uint32_t)i0);
        const float* row = prm.T + (size_t)j * prm.c;
#pragma unroll
        for (int t = 0; t < 4; ++t) {
          v[t][j] = 0.f;
          if (t < tmax) {
            v[t][j] = apply_sign(__ldg(row + ((uint32_t)x & prm.cmask)), signbit_of(y));
            x = step61(x, prm.h.a[j]);
            y = step61(y, prm.h.a2[j]);
          }
        }
      }
#pragma unroll
      for (int t = 0; t < 4; ++t) m[t] = median_of<R>(v[t]);
      store_est(prm, i0, tmax, m);
    }
#pragma unroll
    for (int t = 0; t < 4; ++t) hist_add(sh, t < tmax ? (key_of(m[t]) >> 20) : kNone);
  }
  hist_flush(sh, prm.hist, kBins);
}

// General path: any r <= 16 and any c (bucket by 64-bit remainder).
__global__ void __launch_bounds__(kBlock) k_query_generic(const __grid_constant__ QueryParams prm) {
  __shared__ uint32_t sh[kBins];
  for (int b = threadIdx.x; b < kBins; b += blockDim.x) sh[b] = 0;
  __syncthreads();
  const int64_t d = prm.d;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const int lane = threadIdx.x & 31;
  const int r = prm.r;
  for (int64_t i0 = (int64_t)blockIdx.x * blockDim.x + (threadIdx.x & ~31); i0 < d; i0 += stride) {
    const int64_t i = i0 + lane;
    uint32_t bin = kNone;
    if (i < d) {
      float v[GS_MAX_ROWS];
      for (int j = 0; j < r; ++j) {
        const uint64_t x = affine61(prm.h.a[j], prm.h.b[j], (uint32_t)i);
        const uint64_t y = affine61(prm.h.a2[j], prm.h.b2[j], (uint32_t)i);
        v[j] = apply_sign(__ldg(prm.T + (size_t)j * prm.c + bucket_of<false>(x, prm.c, prm.cmask)),
                          signbit_of(y));
      }
      for (int a = 1; a < r; ++a) {  // insertion sort
        const float t = v[a];
        int b = a - 1;
        while (b >= 0 && v[b] > t) {
          v[b + 1] = v[b];
          --b;
        }
        v[b + 1] = t;
      }
      const float m = (r & 1) ? v[r / 2] : 0.5f * (v[r / 2 - 1] + v[r / 2]);
      prm.est[i] = m;
      bin = key_of(m) >> 20;
    }
    hist_add(sh, bin);
  }
  hist_flush(sh, prm.hist, kBins);
}

// Histogram of key bits [shift, shift + nbits) among keys whose bits above are `prefix`.
__global__ void __launch_bounds__(kBlock) k_hist(const float* __restrict__ est, int64_t d, int vec,
                                                 const SelectState* __restrict__ st, uint32_t* hist,
                                                 int shift, int nbits) {
  __shared__ uint32_t sh[kBins];
  const int nbins = 1 << nbits;
  for (int b = threadIdx.x; b < nbins; b += blockDim.x) sh[b] = 0;
  __syncthreads();
  const uint32_t prefix = st->prefix;
  const int match_shift = shift + nbits;
  const int64_t nq = (d + 3) / 4;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const int lane = threadIdx.x & 31;
  for (int64_t q0 = (int64_t)blockIdx.x * blockDim.x + (threadIdx.x & ~31); q0 < nq; q0 += stride) {
    const int64_t q = q0 + lane;
    const int64_t i0 = q * 4;
    const int tmax = q < nq ? (d - i0 < 4 ? (int)(d - i0) : 4) : 0;
    float v[4] = {0.f, 0.f, 0.f, 0.f};
    if (vec && tmax == 4) {
      const float4 f = __ldcs(reinterpret_cast<const float4*>(est + i0));
      v[0] = f.x; v[1] = f.y; v[2] = f.z; v[3] = f.w;
    } else {
      for (int t = 0; t < tmax; ++t) v[t] = est[i0 + t];
    }
#pragma unroll
    for (int t = 0; t < 4; ++t) {
      const uint32_t key = key_of(v[t]);
      const bool hit = t < tmax && (key >> match_shift) == prefix;
      hist_add(sh, hit ? ((key >> shift) & (uint32_t)(nbins - 1)) : kNone);
    }
  }
  hist_flush(sh, hist, nbins);
}

// Find the bin holding the k_rem-th largest key (scanning bins from the top).
__global__ void __launch_bounds__(kScanThreads) k_pick(const uint32_t* __restrict__ hist, int nbits,
                                                       SelectState* st, int level, uint32_t k_init) {
  const int nbins = 1 << nbits;
  const uint32_t k_rem = level == 0 ? k_init : st->k_rem;
  const uint32_t prefix = level == 0 ? 0u : st->prefix;
  const int per = (nbins + blockDim.x - 1) / blockDim.x;
  const int r0 = threadIdx.x * per;  // positions counted from the top bin
  uint32_t local = 0;
  for (int t = 0; t < per; ++t) {
    const int rp = r0 + t;
    if (rp < nbins) local += hist[nbins - 1 - rp];
  }
  uint32_t total;
  uint32_t cum = block_excl_scan(local, &total);
  for (int t = 0; t < per; ++t) {
    const int rp = r0 + t;
    if (rp >= nbins) break;
    const int bin = nbins - 1 - rp;
    const uint32_t cnt = hist[bin];
    if (cum < k_rem && cum + cnt >= k_rem) {
      const uint32_t p = (prefix << nbits) | (uint32_t)bin;
      st->prefix = p;
      st->k_rem = k_rem - cum;
      st->found = (level == 0 ? 0u : st->found) | (1u << level);
      if (level == 2) {
        st->tau = p;
        st->need_eq = k_rem - cum;
      }
    }
    cum += cnt;
  }
}

template <bool VEC>
__device__ __forceinline__ void load16(const float* __restrict__ est, int64_t i0, int64_t d, float (&v)[kPerThread]) {
#pragma unroll
  for (int t4 = 0; t4 < kPerThread; t4 += 4) {
    if (VEC && i0 + t4 + 4 <= d) {
      const float4 f = __ldcs(reinterpret_cast<const float4*>(est + i0 + t4));
      v[t4] = f.x; v[t4 + 1] = f.y; v[t4 + 2] = f.z; v[t4 + 3] = f.w;
    } else {
#pragma unroll
      for (int t = 0; t < 4; ++t) v[t4 + t] = (i0 + t4 + t < d) ? est[i0 + t4 + t] : 0.f;
    }
  }
}

template <bool VEC>
__global__ void __launch_bounds__(kBlock) k_count(const float* __restrict__ est, int64_t d,
                                                  const SelectState* __restrict__ st,
                                                  uint32_t* blk_gt, uint32_t* blk_eq) {
  const uint32_t tau = st->tau;
  const int64_t s0 = (int64_t)blockIdx.x * kSeg;
  const int64_t s1 = s0 + kSeg < d ? s0 + kSeg : d;
  uint32_t gt = 0, eq = 0;
  for (int64_t i0 = s0 + (int64_t)threadIdx.x * kPerThread; i0 < s1; i0 += (int64_t)blockDim.x * kPerThread) {
    float v[kPerThread];
    load16<VEC>(est, i0, s1, v);
#pragma unroll
    for (int t = 0; t < kPerThread; ++t) {
      if (i0 + t < s1) {
        const uint32_t key = key_of(v[t]);
        gt += key > tau;
        eq += key == tau;
      }
    }
  }
  uint32_t tgt, teq;
  block_excl_scan(gt, &tgt);
  block_excl_scan(eq, &teq);
  if (threadIdx.x == 0) {
    blk_gt[blockIdx.x] = tgt;
    blk_eq[blockIdx.x] = teq;
  }
}

__global__ void __launch_bounds__(kScanThreads) k_scan(const uint32_t* __restrict__ blk_gt,
                                                       const uint32_t* __restrict__ blk_eq, int64_t nblk,
                                                       const SelectState* __restrict__ st,
                                                       uint32_t* blk_base, uint32_t* blk_eqx) {
  const uint32_t need_eq = st->need_eq;
  uint32_t carry_gt = 0, carry_eq = 0;
  for (int64_t c0 = 0; c0 < nblk; c0 += blockDim.x) {
    const int64_t b = c0 + threadIdx.x;
    const uint32_t g = b < nblk ? blk_gt[b] : 0u;
    const uint32_t e = b < nblk ? blk_eq[b] : 0u;
    uint32_t tg, te;
    const uint32_t xg = block_excl_scan(g, &tg) + carry_gt;
    const uint32_t xe = block_excl_scan(e, &te) + carry_eq;
    if (b < nblk) {
      blk_base[b] = xg + (xe < need_eq ? xe : need_eq);
      blk_eqx[b] = xe;
    }
    carry_gt += tg;
    carry_eq += te;
  }
}

template <bool VEC>
__global__ void __launch_bounds__(kBlock) k_write(const float* __restrict__ est, int64_t d,
                                                  const SelectState* __restrict__ st,
                                                  const uint32_t* __restrict__ blk_base,
                                                  const uint32_t* __restrict__ blk_eqx,
                                                  int64_t* __restrict__ idx_out, int64_t k) {
  const uint32_t tau = st->tau, need_eq = st->need_eq;
  const int64_t s0 = (int64_t)blockIdx.x * kSeg;
  const int64_t s1 = s0 + kSeg < d ? s0 + kSeg : d;
  const uint32_t base = blk_base[blockIdx.x];
  const uint32_t eqx = blk_eqx[blockIdx.x];
  uint32_t seg_gt = 0, seg_eq = 0;
  for (int64_t c0 = s0; c0 < s1; c0 += (int64_t)blockDim.x * kPerThread) {
    const int64_t i0 = c0 + (int64_t)threadIdx.x * kPerThread;
    float v[kPerThread];
    load16<VEC>(est, i0, s1, v);
    uint32_t gt = 0, eq = 0;
#pragma unroll
    for (int t = 0; t < kPerThread; ++t) {
      if (i0 + t < s1) {
        const uint32_t key = key_of(v[t]);
        gt += key > tau;
        eq += key == tau;
      }
    }
    uint32_t tot;
    const uint32_t pre = block_excl_scan((eq << 16) | gt, &tot);  // both fields < 2^16
    const uint32_t gt_b = seg_gt + (pre & 0xFFFFu);
    const uint32_t eq_b = seg_eq + (pre >> 16);
    const uint32_t eq_sel_before = need_eq > eqx ? min(need_eq - eqx, eq_b) : 0u;
    uint32_t pos = base + gt_b + eq_sel_before;
    uint32_t eq_rank = eqx + eq_b;
#pragma unroll
    for (int t = 0; t < kPerThread; ++t) {
      if (i0 + t < s1) {
        const uint32_t key = key_of(v[t]);
        bool take = key > tau;
        if (key == tau) {
          take = eq_rank < need_eq;
          ++eq_rank;
        }
        if (take) {
          if ((int64_t)pos < k) idx_out[pos] = i0 + t;
          ++pos;
        }
      }
    }
    seg_gt += tot & 0xFFFFu;
    seg_eq += tot >> 16;
  }
}

template <int R>
cudaError_t launch_query_r(const QueryParams& p, cudaStream_t s) {
  auto kern = k_query<R>;
  const int64_t need = ((p.d + 3) / 4 + kBlock - 1) / kBlock;
  const int64_t cap = (int64_t)device_info().sms * blocks_per_sm((const void*)kern, kBlock);
  const int grid = (int)(need < 1 ? 1 : (need < cap ? need : cap));
  kern<<<grid, kBlock, 0, s>>>(p);
  return cudaGetLastError();
}

typedef cudaError_t (*QueryLauncher)(const QueryParams&, cudaStream_t);

template <int... Rs>
struct QueryTable {
  static constexpr QueryLauncher table[sizeof...(Rs)] = {&launch_query_r<Rs>...};
};
template <int... Rs>
constexpr QueryLauncher QueryTable<Rs...>::table[sizeof...(Rs)];

cudaError_t launch_query(const QueryParams& p, cudaStream_t s) {
  using T = QueryTable<1, 2, 3, 4, 5, 6, 7, 8, 9, 10, 11, 12, 13, 14, 15, 16>;
  if (is_pow2(p.c) && p.r >= 1 && p.r <= GS_MAX_ROWS) return T::table[p.r - 1](p, s);
  const int64_t need = (p.d + kBlock - 1) / kBlock;
  const int64_t cap = (int64_t)device_info().sms * blocks_per_sm((const void*)k_query_generic, kBlock);
  const int grid = (int)(need < 1 ? 1 : (need < cap ? need : cap));
  k_query_generic<<<grid, kBlock, 0, s>>>(p);
  return cudaGetLastError();
}

}  // namespace

size_t query_topk_workspace_bytes(int64_t d, int64_t k) {
  (void)k;
  const int64_t nblk = (d + kSeg - 1) / kSeg;
  return align256((size_t)d * sizeof(float)) + align256(3 * kBins * sizeof(uint32_t)) +
         align256(sizeof(SelectState)) + align256((size_t)nblk * 4 * sizeof(uint32_t));
}

cudaError_t launch_query_topk(const float* merged, const HashCoeffs& h, int r, uint32_t c,
                              int64_t d, int64_t k, int64_t* idx_out, float* est_out,
                              void* workspace, cudaStream_t s) {
  Workspace w = carve(workspace, d);
  float* est = est_out ? est_out : w.est;
  const bool vec = (reinterpret_cast<uintptr_t>(est) & 15u) == 0;
  cudaError_t err = cudaMemsetAsync(w.hist, 0, 3 * kBins * sizeof(uint32_t), s);
  if (err != cudaSuccess) return err;
  err = cudaMemsetAsync(w.st, 0, sizeof(SelectState), s);
  if (err != cudaSuccess) return err;

  QueryParams qp;
  qp.T = merged;
  qp.est = est;
  qp.hist = w.hist;
  qp.d = d;
  qp.r = r;
  qp.c = c;
  qp.cmask = c - 1;
  qp.vec = vec ? 1 : 0;
  qp.h = h;
  if ((err = launch_query(qp, s)) != cudaSuccess) return err;

  k_pick<<<1, kScanThreads, 0, s>>>(w.hist, 11, w.st, 0, (uint32_t)k);
  const int64_t nq = (d + 3) / 4;
  const int64_t need = (nq + kBlock - 1) / kBlock;
  const int64_t cap = (int64_t)device_info().sms * blocks_per_sm((const void*)k_hist, kBlock);
  const int hgrid = (int)(need < 1 ? 1 : (need < cap ? need : cap));
  k_hist<<<hgrid, kBlock, 0, s>>>(est, d, vec ? 1 : 0, w.st, w.hist + kBins, 9, 11);
  k_pick<<<1, kScanThreads, 0, s>>>(w.hist + kBins, 11, w.st, 1, 0);
  k_hist<<<hgrid, kBlock, 0, s>>>(est, d, vec ? 1 : 0, w.st, w.hist + 2 * kBins, 0, 9);
  k_pick<<<1, kScanThreads, 0, s>>>(w.hist + 2 * kBins, 9, w.st, 2, 0);

  const int nblk = (int)w.nblk;
  if (vec) k_count<true><<<nblk, kBlock, 0, s>>>(est, d, w.st, w.blk_gt, w.blk_eq);
  else k_count<false><<<nblk, kBlock, 0, s>>>(est, d, w.st, w.blk_gt, w.blk_eq);
  k_scan<<<1, kScanThreads, 0, s>>>(w.blk_gt, w.blk_eq, w.nblk, w.st, w.blk_base, w.blk_eqx);
  if (vec) k_write<true><<<nblk, kBlock, 0, s>>>(est, d, w.st, w.blk_base, w.blk_eqx, idx_out, k);
  else k_write<false><<<nblk, kBlock, 0, s>>>(est, d, w.st, w.blk_base, w.blk_eqx, idx_out, k);
  return cudaGetLastError();
}

// ---- scratch without allocation ---------------------------------------------------------
// For callers that cannot allocate: the selection scratch of the query (three histograms,
// the state, and four counters per segment of kSeg coordinates, enough for d up to
// GS_NOALLOC_MAX_DIM) lives in one array of the library's device memory.
namespace {

constexpr int64_t kNoallocMaxSegs = (GS_NOALLOC_MAX_DIM + kSeg - 1) / kSeg;
constexpr size_t kNoallocHistBytes = 3 * kBins * sizeof(uint32_t);   // multiple of 256
constexpr size_t kNoallocStateBytes = 256;
constexpr size_t kNoallocScratchBytes =
    kNoallocHistBytes + kNoallocStateBytes + (size_t)kNoallocMaxSegs * 4 * sizeof(uint32_t);

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoallocScratchBytes];

// Device address of g_noalloc_scratch on the current device, looked up once per device.
cudaError_t noalloc_scratch(void** out) {
  static std::mutex mu;
  static void* addr[64] = {};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(mu);
  if (!addr[dev]) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess) return e;
    addr[dev] = p;
  }
  *out = addr[dev];
  return cudaSuccess;
}

}  // namespace

cudaError_t launch_query_topk_noalloc(const float* merged, const HashCoeffs& h, int r, uint32_t c,
                                      int64_t d, int64_t k, int64_t* idx_out, float* est_out,
                                      cudaStream_t s) {
  if (d > GS_NOALLOC_MAX_DIM || est_out == nullptr) return cudaErrorInvalidValue;
  void* base = nullptr;
  cudaError_t err = noalloc_scratch(&base);
  if (err != cudaSuccess) return err;
  char* p = static_cast<char*>(base);
  uint32_t* hist = reinterpret_cast<uint32_t*>(p);
  SelectState* st = reinterpret_cast<SelectState*>(p + kNoallocHistBytes);
  const int64_t nblk = (d + kSeg - 1) / kSeg;
  uint32_t* blk_gt = reinterpret_cast<uint32_t*>(p + kNoallocHistBytes + kNoallocStateBytes);
  uint32_t* blk_eq = blk_gt + nblk;
  uint32_t* blk_base = blk_eq + nblk;
  uint32_t* blk_eqx = blk_base + nblk;
  float* est = est_out;
  const bool vec = (reinterpret_cast<uintptr_t>(est) & 15u) == 0;
  // the histograms and the state must start at zero; the counters are fully overwritten
  if ((err = cudaMemsetAsync(hist, 0, kNoallocHistBytes, s)) != cudaSuccess) return err;
  if ((err = cudaMemsetAsync(st, 0, sizeof(SelectState), s)) != cudaSuccess) return err;

  QueryParams qp;
  qp.T = merged;
  qp.est = est;
  qp.hist = hist;
  qp.d = d;
  qp.r = r;
  qp.c = c;
  qp.cmask = c - 1;
  qp.vec = vec ? 1 : 0;
  qp.h = h;
  if ((err = launch_query(qp, s)) != cudaSuccess) return err;

  k_pick<<<1, kScanThreads, 0, s>>>(hist, 11, st, 0, (uint32_t)k);
  const int64_t nq = (d + 3) / 4;
  const int64_t need = (nq + kBlock - 1) / kBlock;
  const int64_t cap = (int64_t)device_info().sms * blocks_per_sm((const void*)k_hist, kBlock);
  const int hgrid = (int)(need < 1 ? 1 : (need < cap ? need : cap));
  k_hist<<<hgrid, kBlock, 0, s>>>(est, d, vec ? 1 : 0, st, hist + kBins, 9, 11);
  k_pick<<<1, kScanThreads, 0, s>>>(hist + kBins, 11, st, 1, 0);
  k_hist<<<hgrid, kBlock, 0, s>>>(est, d, vec ? 1 : 0, st, hist + 2 * kBins, 0, 9);
  k_pick<<<1, kScanThreads, 0, s>>>(hist + 2 * kBins, 9, st, 2, 0);

  const int nb = (int)nblk;
  if (vec) k_count<true><<<nb, kBlock, 0, s>>>(est, d, st, blk_gt, blk_eq);
  else k_count<false><<<nb, kBlock, 0, s>>>(est, d, st, blk_gt, blk_eq);
  k_scan<<<1, kScanThreads, 0, s>>>(blk_gt, blk_eq, nblk, st, blk_base, blk_eqx);
  if (vec) k_write<true><<<nb, kBlock, 0, s>>>(est, d, st, blk_base, blk_eqx, idx_out, k);
  else k_write<false><<<nb, kBlock, 0, s>>>(est, d, st, blk_base, blk_eqx, idx_out, k);
  return cudaGetLastError();
}

}  // namespace gs
