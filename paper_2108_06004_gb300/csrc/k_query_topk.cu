// Steps 4 and 5: median-of-r query of the merged sketch and top-k selection
// (Alg. 2 steps 1-3, read as a deterministic top-k by |est| with ties to the smaller index).
//
// Pipeline (all on one stream, no host round trip):
//   k_query     est_i = median_j s_j(i) T[j][h_j(i)] for every i, written as fp32, and a
//               2048-bin histogram of key bits 30..20, key = bits of |est_i| (for
//               non-negative floats the bit pattern orders like the value).
//   k_hist      histogram of the next key bits among keys in the chosen bin (bits 19..9,
//               then bits 8..0).
//               Each of these kernels ends with a pick: the last CTA to finish (found with a
//               counter after a memory fence, so no CTA waits for another) finds the bin that
//               holds the k-th largest key and how many keys of that bin are still to be
//               taken.  After three levels the k-th largest key tau is exact, and
//               need_eq = k - #{key > tau} keys equal to tau are taken, those of smallest index.
//   k_count     per segment of 16384 coordinates: #{key > tau}, #{key == tau}
//   k_scan      one CTA: exclusive prefix sums over the segments
//   k_write     every segment writes its selected indices at their final positions, so the
//               output is in ascending index order without a sort.
#include <mutex>

#include "gs_common.cuh"

namespace gs {

namespace {

constexpr int kBins = 2048;
constexpr int kSegThreads = 256;
constexpr int kPerThread = 64;                      // consecutive coordinates per thread
constexpr int kSeg = kSegThreads * kPerThread;      // 16384 coordinates per segment
constexpr int kScanThreads = 1024;
constexpr uint32_t kNone = 0xFFFFFFFFu;

struct SelectState {
  uint32_t prefix;   // key bits fixed so far
  uint32_t k_rem;    // keys still to take inside the prefix
  uint32_t tau;      // the k-th largest key
  uint32_t need_eq;  // keys equal to tau to take
  uint32_t found;    // bit l set when level l found its bin
  uint32_t fail;     // pruned query: the threshold fell below the hint (result not usable)
  uint32_t done[3];  // CTAs finished per level (for the last-CTA pick)
};

struct Workspace {
  float* est;
  uint32_t* hist;     // 6 * kBins: three levels for the first pass, three for the exact re-run
  SelectState* st;    // two states: first pass, exact re-run
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
  p += align256(6 * kBins * sizeof(uint32_t));
  w.st = reinterpret_cast<SelectState*>(p);
  p += 2 * align256(sizeof(SelectState));
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

// The whole block finds the bin holding the k_rem-th largest key, scanning from the top bin.
// Histogram values are read past L1 (they were completed by other CTAs' atomics).
// At the last level, with a hint slot: `check` records whether the threshold reached the hint
// the pruned query used (else its result is not usable), and the slot gets the hint for the
// next query, 0.8 times this threshold.
__device__ void pick_bins(const uint32_t* hist, int nbits, SelectState* st, int level, uint32_t k_init,
                          uint32_t* hint, int check) {
  const int nbins = 1 << nbits;
  const uint32_t k_rem = level == 0 ? k_init : __ldcg(&st->k_rem);
  const uint32_t prefix = level == 0 ? 0u : __ldcg(&st->prefix);
  const uint32_t found = level == 0 ? 0u : __ldcg(&st->found);
  const int per = (nbins + blockDim.x - 1) / blockDim.x;
  const int r0 = threadIdx.x * per;  // positions counted from the top bin
  uint32_t local = 0;
  for (int t = 0; t < per; ++t) {
    const int rp = r0 + t;
    if (rp < nbins) local += __ldcg(&hist[nbins - 1 - rp]);
  }
  uint32_t total;
  uint32_t cum = block_excl_scan(local, &total);
  for (int t = 0; t < per; ++t) {
    const int rp = r0 + t;
    if (rp >= nbins) break;
    const int bin = nbins - 1 - rp;
    const uint32_t cnt = __ldcg(&hist[bin]);
    if (cum < k_rem && cum + cnt >= k_rem) {
      const uint32_t p = (prefix << nbits) | (uint32_t)bin;
      st->prefix = p;
      st->k_rem = k_rem - cum;
      st->found = found | (1u << level);
      if (level == 2) {
        st->tau = p;
        st->need_eq = k_rem - cum;
        if (hint) {
          const uint32_t used = __ldcg(hint);
          if (check) st->fail = (p < used) ? 1u : 0u;
          *hint = key_of(0.8f * __uint_as_float(p));
        }
      }
    }
    cum += cnt;
  }
}

// Called by every CTA after its histogram atomics: the last CTA to arrive does the pick.
__device__ __forceinline__ void last_block_pick(const uint32_t* hist, int nbits, SelectState* st, int level,
                                                uint32_t k_init, uint32_t* hint = nullptr, int check = 0) {
  __shared__ uint32_t am_last;
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) am_last = (atomicAdd(&st->done[level], 1u) == gridDim.x - 1) ? 1u : 0u;
  __syncthreads();
  if (am_last) {
    __threadfence();
    pick_bins(hist, nbits, st, level, k_init, hint, check);
  }
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
  SelectState* st;
  int64_t d;
  uint32_t k;
  int32_t r;
  uint32_t c, cmask;
  int32_t vec;        // est 16-byte aligned
  const uint32_t* gate;  // exact re-run: run only if *gate (the first pass's fail flag) is set
  const uint32_t* hint;  // pruned query: hint key (read once)
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
// PRUNE: read the first M = R/2 + 1 rows; the median of all R values lies between the least
// and the largest of any M of them, so |est| <= max_j<M |v_j|.  When that bound is below the
// hint key the coordinate cannot reach the threshold the hint stands for; its remaining rows
// are skipped and 0 is stored (the last pick checks that the threshold did reach the hint).
template <int R, bool PRUNE>
__global__ void __launch_bounds__(kBlock) k_query(const __grid_constant__ QueryParams prm) {
  if (prm.gate && __ldcg(prm.gate) == 0u) return;  // uniform: the exact re-run is not needed
  constexpr int M = PRUNE ? R / 2 + 1 : R;
  __shared__ uint32_t sh[kBins];
  for (int b = threadIdx.x; b < kBins; b += blockDim.x) sh[b] = 0;
  __syncthreads();
  const uint32_t hk = PRUNE ? __ldcg(prm.hint) : 0u;
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
      for (int j = 0; j < M; ++j) {
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
      bool need[4];
#pragma unroll
      for (int t = 0; t < 4; ++t) {
        float ub = 0.f;
#pragma unroll
        for (int j = 0; j < M; ++j) ub = fmaxf(ub, fabsf(v[t][j]));
        need[t] = t < tmax && (!PRUNE || key_of(ub) >= hk);
      }
      if (PRUNE && (need[0] || need[1] || need[2] || need[3])) {
#pragma unroll
        for (int j = M; j < R; ++j) {
          uint64_t x = affine61(prm.h.a[j], prm.h.b[j], (uint32_t)i0);
          uint64_t y = affine61(prm.h.a2[j], prm.h.b2[j], (uint32_t)i0);
          const float* row = prm.T + (size_t)j * prm.c;
#pragma unroll
          for (int t = 0; t < 4; ++t) {
            v[t][j] = 0.f;
            if (t < tmax) {
              if (need[t]) v[t][j] = apply_sign(__ldg(row + ((uint32_t)x & prm.cmask)), signbit_of(y));
              x = step61(x, prm.h.a[j]);
              y = step61(y, prm.h.a2[j]);
            }
          }
        }
      }
#pragma unroll
      for (int t = 0; t < 4; ++t) m[t] = need[t] ? median_of<R>(v[t]) : 0.f;
      store_est(prm, i0, tmax, m);
    }
#pragma unroll
    for (int t = 0; t < 4; ++t) hist_add(sh, t < tmax ? (key_of(m[t]) >> 20) : kNone);
  }
  hist_flush(sh, prm.hist, kBins);
  last_block_pick(prm.hist, 11, prm.st, 0, prm.k);
}

// General path: any r <= 16 and any c (bucket by 64-bit remainder).
__global__ void __launch_bounds__(kBlock) k_query_generic(const __grid_constant__ QueryParams prm) {
  if (prm.gate && __ldcg(prm.gate) == 0u) return;
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
  last_block_pick(prm.hist, 11, prm.st, 0, prm.k);
}

// Histogram of key bits [shift, shift + nbits) among keys whose bits above are the prefix
// picked at the previous level; ends with the pick of this level.  Each thread loads four
// float4 before it processes them, to keep enough L2 reads in flight.
__global__ void __launch_bounds__(kBlock) k_hist(const float* __restrict__ est, int64_t d, int vec,
                                                 SelectState* st, uint32_t* hist, int shift, int nbits,
                                                 int level, const uint32_t* gate, uint32_t* hint, int check) {
  if (gate && __ldcg(gate) == 0u) return;  // uniform: the exact re-run is not needed
  constexpr int U = 4;
  __shared__ uint32_t sh[kBins];
  const int nbins = 1 << nbits;
  for (int b = threadIdx.x; b < nbins; b += blockDim.x) sh[b] = 0;
  __syncthreads();
  const uint32_t prefix = __ldcg(&st->prefix);
  const int match_shift = shift + nbits;
  const int64_t nq = (d + 3) / 4;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const int lane = threadIdx.x & 31;
  for (int64_t q0 = (int64_t)blockIdx.x * blockDim.x + (threadIdx.x & ~31); q0 < nq; q0 += U * stride) {
    float v[U][4];
    int tm[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int64_t q = q0 + u * stride + lane;
      const int64_t i0 = q * 4;
      tm[u] = q < nq ? (d - i0 < 4 ? (int)(d - i0) : 4) : 0;
      if (vec && tm[u] == 4) {
        const float4 f = __ldcs(reinterpret_cast<const float4*>(est + i0));
        v[u][0] = f.x; v[u][1] = f.y; v[u][2] = f.z; v[u][3] = f.w;
      } else {
#pragma unroll
        for (int t = 0; t < 4; ++t) v[u][t] = t < tm[u] ? est[i0 + t] : 0.f;
      }
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      uint32_t bins[4];
      bool any = false;
#pragma unroll
      for (int t = 0; t < 4; ++t) {
        const uint32_t key = key_of(v[u][t]);
        const bool hit = t < tm[u] && (key >> match_shift) == prefix;
        bins[t] = hit ? ((key >> shift) & (uint32_t)(nbins - 1)) : kNone;
        any = any || hit;
      }
      if (__any_sync(0xFFFFFFFFu, any)) {  // most warps hold no key of the chosen bin
#pragma unroll
        for (int t = 0; t < 4; ++t) hist_add(sh, bins[t]);
      }
    }
  }
  hist_flush(sh, hist, nbins);
  last_block_pick(hist, nbits, st, level, 0, hint, check);
}

// Segments of kSeg coordinates; a warp owns kWarpRun consecutive coordinates and reads them as
// kRows rows of 128 (lane l holds coordinates 4l .. 4l+3 of each row), so every load is a
// coalesced float4 and the ascending order of a warp's run is (row, lane, component).
constexpr int kSegWarps = kSegThreads / 32;
constexpr int kWarpRun = kSeg / kSegWarps;   // 2048
constexpr int kRows = kWarpRun / 128;        // 16

template <bool VEC>
__device__ __forceinline__ void load_row(const float* __restrict__ est, int64_t i0, int64_t s1, float (&v)[4]) {
  if (VEC && i0 + 4 <= s1) {
    const float4 f = __ldcg(reinterpret_cast<const float4*>(est + i0));
    v[0] = f.x; v[1] = f.y; v[2] = f.z; v[3] = f.w;
  } else {
#pragma unroll
    for (int t = 0; t < 4; ++t) v[t] = (i0 + t < s1) ? est[i0 + t] : 0.f;
  }
}

// Packed (eq << 16 | gt) counts of one segment; every field stays below 2^16.
__device__ __forceinline__ uint32_t count_key(uint32_t key, uint32_t tau) {
  return (key > tau ? 1u : 0u) | (key == tau ? (1u << 16) : 0u);
}

// The state whose threshold is valid: the exact re-run's when the first pass failed.
__device__ __forceinline__ const SelectState* valid_state(const SelectState* st, const SelectState* st2) {
  return (st2 && __ldcg(&st->fail)) ? st2 : st;
}

template <bool VEC>
__global__ void __launch_bounds__(kSegThreads) k_count(const float* __restrict__ est, int64_t d,
                                                       const SelectState* st0, const SelectState* st2,
                                                       uint32_t* blk_gt, uint32_t* blk_eq) {
  const SelectState* st = valid_state(st0, st2);
  const uint32_t tau = __ldcg(&st->tau);
  const int64_t s0 = (int64_t)blockIdx.x * kSeg;
  const int64_t s1 = s0 + kSeg < d ? s0 + kSeg : d;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t w0 = s0 + (int64_t)warp * kWarpRun;
  uint32_t cnt = 0;
  float v[kRows][4];
#pragma unroll
  for (int j = 0; j < kRows; ++j) load_row<VEC>(est, w0 + j * 128 + lane * 4, s1, v[j]);
#pragma unroll
  for (int j = 0; j < kRows; ++j) {
#pragma unroll
    for (int t = 0; t < 4; ++t) {
      if (w0 + j * 128 + lane * 4 + t < s1) cnt += count_key(key_of(v[j][t]), tau);
    }
  }
  uint32_t tot;
  block_excl_scan(cnt, &tot);
  if (threadIdx.x == 0) {
    blk_gt[blockIdx.x] = tot & 0xFFFFu;
    blk_eq[blockIdx.x] = tot >> 16;
  }
}

__global__ void __launch_bounds__(kScanThreads) k_scan(const uint32_t* __restrict__ blk_gt,
                                                       const uint32_t* __restrict__ blk_eq, int64_t nblk,
                                                       const SelectState* st0, const SelectState* st2,
                                                       uint32_t* blk_base, uint32_t* blk_eqx) {
  const SelectState* st = valid_state(st0, st2);
  const uint32_t need_eq = __ldcg(&st->need_eq);
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

// Warp-inclusive scan of a packed count.
__device__ __forceinline__ uint32_t warp_incl_scan(uint32_t x) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t y = __shfl_up_sync(0xFFFFFFFFu, x, o);
    if (lane >= o) x += y;
  }
  return x;
}

template <bool VEC>
__device__ __forceinline__ void load_row_l1(const float* __restrict__ est, int64_t i0, int64_t s1, float (&v)[4]) {
  if (VEC && i0 + 4 <= s1) {
    const float4 f = __ldg(reinterpret_cast<const float4*>(est + i0));
    v[0] = f.x; v[1] = f.y; v[2] = f.z; v[3] = f.w;
  } else {
#pragma unroll
    for (int t = 0; t < 4; ++t) v[t] = (i0 + t < s1) ? est[i0 + t] : 0.f;
  }
}

// Counts first (all rows in flight), then each row again from L1 to place its keys.
template <bool VEC>
__global__ void __launch_bounds__(kSegThreads) k_write(const float* __restrict__ est, int64_t d,
                                                       const SelectState* st0, const SelectState* st2,
                                                       const uint32_t* __restrict__ blk_base,
                                                       const uint32_t* __restrict__ blk_eqx,
                                                       int64_t* __restrict__ idx_out, int64_t k) {
  __shared__ uint32_t warp_tot[kSegWarps];
  const SelectState* st = valid_state(st0, st2);
  const uint32_t tau = __ldcg(&st->tau), need_eq = __ldcg(&st->need_eq);
  const int64_t s0 = (int64_t)blockIdx.x * kSeg;
  const int64_t s1 = s0 + kSeg < d ? s0 + kSeg : d;
  const uint32_t base = blk_base[blockIdx.x];
  const uint32_t eqx = blk_eqx[blockIdx.x];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t w0 = s0 + (int64_t)warp * kWarpRun;
  uint32_t cnt = 0;
  {
    float v[kRows][4];
#pragma unroll
    for (int j = 0; j < kRows; ++j) load_row_l1<VEC>(est, w0 + j * 128 + lane * 4, s1, v[j]);
#pragma unroll
    for (int j = 0; j < kRows; ++j) {
#pragma unroll
      for (int t = 0; t < 4; ++t) {
        if (w0 + j * 128 + lane * 4 + t < s1) cnt += count_key(key_of(v[j][t]), tau);
      }
    }
  }
  // warp totals -> each warp's prefix inside the segment
  const uint32_t wsum = __shfl_sync(0xFFFFFFFFu, warp_incl_scan(cnt), 31);
  if (lane == 0) warp_tot[warp] = wsum;
  __syncthreads();
  uint32_t wpre = 0;
  for (int w = 0; w < warp; ++w) wpre += warp_tot[w];
  if (wsum == 0) return;
  uint32_t run = wpre;  // packed counts before the current row of this warp, within the segment
  const uint32_t eq_quota = need_eq > eqx ? need_eq - eqx : 0u;  // eq keys of this segment still taken
#pragma unroll 1
  for (int j = 0; j < kRows; ++j) {
    const int64_t i0 = w0 + j * 128 + lane * 4;
    float v[4];
    load_row_l1<VEC>(est, i0, s1, v);
    uint32_t key[4];
    uint32_t c = 0;
#pragma unroll
    for (int t = 0; t < 4; ++t) {
      key[t] = key_of(v[t]);
      if (i0 + t < s1) c += count_key(key[t], tau);
    }
    const uint32_t incl = warp_incl_scan(c);
    const uint32_t row_tot = __shfl_sync(0xFFFFFFFFu, incl, 31);
    if (c) {
      const uint32_t before = run + incl - c;
      const uint32_t gt_before = before & 0xFFFFu, eq_before = before >> 16;
      uint32_t pos = base + gt_before + (eq_before < eq_quota ? eq_before : eq_quota);
      uint32_t eq_rank = eq_before;  // rank among this segment's eq keys
#pragma unroll
      for (int t = 0; t < 4; ++t) {
        if (i0 + t < s1) {
          bool take = key[t] > tau;
          if (key[t] == tau) {
            take = eq_rank < eq_quota;
            ++eq_rank;
          }
          if (take) {
            if ((int64_t)pos < k) idx_out[pos] = i0 + t;
            ++pos;
          }
        }
      }
    }
    run += row_tot;
  }
}

template <int R, bool PRUNE>
cudaError_t launch_query_r(const QueryParams& p, cudaStream_t s) {
  auto kern = k_query<R, PRUNE>;
  const int64_t need = ((p.d + 3) / 4 + kBlock - 1) / kBlock;
  const int64_t cap = (int64_t)device_info().sms * blocks_per_sm((const void*)kern, kBlock);
  const int grid = (int)(need < 1 ? 1 : (need < cap ? need : cap));
  kern<<<grid, kBlock, 0, s>>>(p);
  return cudaGetLastError();
}

typedef cudaError_t (*QueryLauncher)(const QueryParams&, cudaStream_t);

template <bool PRUNE, int... Rs>
struct QueryTable {
  static constexpr QueryLauncher table[sizeof...(Rs)] = {&launch_query_r<Rs, PRUNE>...};
};
template <bool PRUNE, int... Rs>
constexpr QueryLauncher QueryTable<PRUNE, Rs...>::table[sizeof...(Rs)];

cudaError_t launch_query(const QueryParams& p, bool prune, cudaStream_t s) {
  using T = QueryTable<false, 1, 2, 3, 4, 5, 6, 7, 8, 9, 10, 11, 12, 13, 14, 15, 16>;
  using TP = QueryTable<true, 1, 2, 3, 4, 5, 6, 7, 8, 9, 10, 11, 12, 13, 14, 15, 16>;
  if (is_pow2(p.c) && p.r >= 1 && p.r <= GS_MAX_ROWS) return (prune ? TP::table : T::table)[p.r - 1](p, s);
  const int64_t need = (p.d + kBlock - 1) / kBlock;
  const int64_t cap = (int64_t)device_info().sms * blocks_per_sm((const void*)k_query_generic, kBlock);
  const int grid = (int)(need < 1 ? 1 : (need < cap ? need : cap));
  k_query_generic<<<grid, kBlock, 0, s>>>(p);
  return cudaGetLastError();
}

// The query and selection kernels over scratch laid out by the caller.  With `hint`
// (requires hist of 6 * kBins and two states) the first pass prunes against the hint and
// an exact re-run follows, gated on the first pass's fail flag; k_count, k_scan and k_write
// then use whichever state is valid.
cudaError_t run_query_select(const float* merged, const HashCoeffs& h, int r, uint32_t c, int64_t d,
                             int64_t k, int64_t* idx_out, float* est, uint32_t* hist, SelectState* st,
                             SelectState* st2, uint32_t* hint, uint32_t* blk_gt, uint32_t* blk_eq,
                             uint32_t* blk_base, uint32_t* blk_eqx, cudaStream_t s) {
  const bool vec = (reinterpret_cast<uintptr_t>(est) & 15u) == 0;
  const bool prune = hint != nullptr && st2 != nullptr && is_pow2(c);
  cudaError_t err = cudaMemsetAsync(hist, 0, (prune ? 6 : 3) * kBins * sizeof(uint32_t), s);
  if (err != cudaSuccess) return err;
  if ((err = cudaMemsetAsync(st, 0, sizeof(SelectState), s)) != cudaSuccess) return err;
  if (prune && (err = cudaMemsetAsync(st2, 0, sizeof(SelectState), s)) != cudaSuccess) return err;

  QueryParams qp;
  qp.T = merged;
  qp.est = est;
  qp.hist = hist;
  qp.st = st;
  qp.d = d;
  qp.k = (uint32_t)k;
  qp.r = r;
  qp.c = c;
  qp.cmask = c - 1;
  qp.vec = vec ? 1 : 0;
  qp.gate = nullptr;
  qp.hint = hint;
  qp.h = h;
  if ((err = launch_query(qp, prune, s)) != cudaSuccess) return err;

  const int64_t nq = (d + 3) / 4;
  const int64_t need = (nq + kBlock - 1) / kBlock;
  const int64_t cap = (int64_t)device_info().sms * blocks_per_sm((const void*)k_hist, kBlock);
  const int hgrid = (int)(need < 1 ? 1 : (need < cap ? need : cap));
  k_hist<<<hgrid, kBlock, 0, s>>>(est, d, vec ? 1 : 0, st, hist + kBins, 9, 11, 1, nullptr, nullptr, 0);
  k_hist<<<hgrid, kBlock, 0, s>>>(est, d, vec ? 1 : 0, st, hist + 2 * kBins, 0, 9, 2, nullptr,
                                  prune ? hint : nullptr, 1);
  if (prune) {  // exact re-run, a no-op unless the first pass failed
    QueryParams q2 = qp;
    q2.hist = hist + 3 * kBins;
    q2.st = st2;
    q2.gate = &st->fail;
    q2.hint = nullptr;
    if ((err = launch_query(q2, false, s)) != cudaSuccess) return err;
    k_hist<<<hgrid, kBlock, 0, s>>>(est, d, vec ? 1 : 0, st2, hist + 4 * kBins, 9, 11, 1, &st->fail, nullptr, 0);
    k_hist<<<hgrid, kBlock, 0, s>>>(est, d, vec ? 1 : 0, st2, hist + 5 * kBins, 0, 9, 2, &st->fail, hint, 0);
  }
  SelectState* s2 = prune ? st2 : nullptr;

  const int64_t nblk = (d + kSeg - 1) / kSeg;
  const int nb = (int)nblk;
  if (vec) k_count<true><<<nb, kSegThreads, 0, s>>>(est, d, st, s2, blk_gt, blk_eq);
  else k_count<false><<<nb, kSegThreads, 0, s>>>(est, d, st, s2, blk_gt, blk_eq);
  k_scan<<<1, kScanThreads, 0, s>>>(blk_gt, blk_eq, nblk, st, s2, blk_base, blk_eqx);
  if (vec) k_write<true><<<nb, kSegThreads, 0, s>>>(est, d, st, s2, blk_base, blk_eqx, idx_out, k);
  else k_write<false><<<nb, kSegThreads, 0, s>>>(est, d, st, s2, blk_base, blk_eqx, idx_out, k);
  return cudaGetLastError();
}

}  // namespace

size_t query_topk_workspace_bytes(int64_t d, int64_t k) {
  (void)k;
  const int64_t nblk = (d + kSeg - 1) / kSeg;
  return align256((size_t)d * sizeof(float)) + align256(6 * kBins * sizeof(uint32_t)) +
         2 * align256(sizeof(SelectState)) + align256((size_t)nblk * 4 * sizeof(uint32_t));
}

cudaError_t launch_query_topk(const float* merged, const HashCoeffs& h, int r, uint32_t c,
                              int64_t d, int64_t k, int64_t* idx_out, float* est_out,
                              void* workspace, uint32_t* hint, cudaStream_t s) {
  Workspace w = carve(workspace, d);
  float* est = est_out ? est_out : w.est;
  // pruning only when est is internal: a caller asking for est gets every median exactly
  uint32_t* h2 = est_out ? nullptr : hint;
  SelectState* st2 = reinterpret_cast<SelectState*>(reinterpret_cast<char*>(w.st) + align256(sizeof(SelectState)));
  return run_query_select(merged, h, r, c, d, k, idx_out, est, w.hist, w.st, st2, h2, w.blk_gt, w.blk_eq,
                          w.blk_base, w.blk_eqx, s);
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
static_assert(sizeof(SelectState) <= kNoallocStateBytes, "state slot too small");

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
  // the histograms and the state are cleared at the start of the sequence; the segment
  // counters are fully overwritten
  return run_query_select(merged, h, r, c, d, k, idx_out, est_out, hist, st, nullptr, nullptr, blk_gt, blk_eq,
                          blk_base, blk_eqx, s);
}

}  // namespace gs
