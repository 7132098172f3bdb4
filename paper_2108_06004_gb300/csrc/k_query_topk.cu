// Steps 4 and 5: median-of-r query of the merged sketch and top-k selection
// (Alg. 2 steps 1-3, read as a deterministic top-k by |est| with ties to the smaller index).
//
// The selection is a radix select on a 32-bit key in three levels: bits 31..21, 20..10 and
// 9..0.  For the top-k by |est| the key is the bit pattern of |est| (for non-negative floats
// it orders like the value); HEAVYMIX selects on a composite key (see heavy_key).  Each
// histogram kernel ends with a pick: the last CTA to finish (found with a counter after a
// memory fence, so no CTA waits for another) finds the bin that holds the k-th largest key
// and how many keys of that bin are still to be taken.  After three levels the k-th largest
// key tau is exact, and need_eq = k - #{key > tau} keys equal to tau are taken, those of
// smallest index.  Output indices are ascending.
//
// With a caller workspace (gs_query_topk):
//   k_qsample     (only where rows are pruned) the full estimate of a fixed strided sample of
//                 coordinates, its level-1 histogram, and a prune key from it: a lower bound
//                 on the k-th largest |est| of this query, rounded down to a bin edge
//   k_query       est_i for every i (fp32) + level-1 histogram + pick; when the estimate stays
//                 in the workspace, a coordinate whose rows read so far bound its |est| below
//                 the prune key skips its other rows and stores a marker (see below)
//   k_repair      runs only if the level-1 pick fell below the prune key: recomputes every
//                 marked estimate in full, rebuilds the level-1 histogram and picks again
//   k_cand        one pass over est: keys above the picked level-1 bin are selected for
//                 certain and set their bit in a d-bit bitmap; keys inside the bin become
//                 candidates (index, key) and feed the level-2 histogram + pick
//   k_cand_hist3  level-3 histogram of the candidates + pick
//   k_cand_mark   candidates above tau into the bitmap, candidates equal to tau into a second
//   k_bm_count    per block of 65536 coordinates: bits set in each bitmap
//   k_scan        one CTA: exclusive prefix sums over the blocks
//   k_bm_write    every block writes its selected indices at their final positions
// With the fixed scratch (gs_query_topk_noalloc), which cannot hold candidate lists, the
// levels 2 and 3 and the final selection read est in full passes (k_hist, k_count, k_write).
#include <cmath>
#include <mutex>

#include <cuda.h>

#include "gs_common.cuh"

namespace gs {

namespace {

constexpr int kBins = 2048;
constexpr int kL1Shift = 21;  // level 1: key bits 31..21 (11 bits)
constexpr int kL2Shift = 10;  // level 2: key bits 20..10 (11 bits)
constexpr int kL3Bits = 10;   // level 3: key bits 9..0
constexpr int kScanThreads = 1024;
constexpr uint32_t kNone = 0xFFFFFFFFu;
constexpr uint32_t kFull = 0xFFFFFFFFu;

struct SelectState {
  uint32_t prefix;   // key bits fixed so far
  uint32_t k_rem;    // keys still to take inside the prefix
  uint32_t tau;      // the k-th largest key
  uint32_t need_eq;  // keys equal to tau to take
  uint32_t found;    // bit l set when level l found its bin
  uint32_t ncand;    // candidates appended by k_cand
  uint32_t done[3];  // CTAs finished per level (for the last-CTA pick)
  uint32_t prune_key;  // the key below which k_query skips rows (0: none); written once per
                       // query, before k_query, by k_qsample or k_heavy_theta
  uint32_t done_r;     // CTAs finished in k_repair
  uint32_t done_s;     // CTAs finished in k_qsample
};

inline size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

__device__ __forceinline__ uint32_t key_of(float v) { return __float_as_uint(v) & 0x7FFFFFFFu; }

// The query's hash arithmetic, without compares (the query is bound by its integer work).
// For s < 2^62 - 1, s mod p is s - p when s >= p and s otherwise; s >= p exactly when bit 61
// of s + 1 is set, and then s - p = (s + 1) - 2^61 = (s + 1) & p.  So for s < 2p:
//   s mod p = (s + ((s + 1) >> 61)) & p.
__device__ __forceinline__ uint64_t reduce61(uint64_t s) { return (s + ((s + 1) >> 61)) & kP61; }

// x + a mod p for x, a < p (the incremental form of the hash): the same value as step61.
__device__ __forceinline__ uint64_t step61_nb(uint64_t x, uint64_t a) { return reduce61(x + a); }

// (a*i + b) mod p for a, b < p and i < 2^32: the same value as affine61.  The sum of the
// partial products is below 3 * 2^61; one fold leaves it at most p + 2, then reduce61.
__device__ __forceinline__ uint64_t affine61_nb(uint64_t a, uint64_t b, uint32_t i) {
  const uint64_t p0 = (uint64_t)(uint32_t)a * i;
  const uint64_t p1 = (uint64_t)(uint32_t)(a >> 32) * i;
  const uint64_t s = (p1 >> 29) + ((p1 & ((1ull << 29) - 1)) << 32) + fold61(p0) + b;
  return reduce61(fold61(s));
}

// Warp-aggregated shared-memory histogram update; every lane of the warp must call it.
__device__ __forceinline__ void hist_add(uint32_t* sh, uint32_t bin) {
  const uint32_t peers = __match_any_sync(kFull, bin);
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
    const uint32_t y = __shfl_up_sync(kFull, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) warp_sums[warp] = x;
  __syncthreads();
  if (warp == 0) {
    uint32_t w = lane < nwarps ? warp_sums[lane] : 0u;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t y = __shfl_up_sync(kFull, w, o);
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

__device__ __forceinline__ uint32_t warp_incl_scan(uint32_t x) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t y = __shfl_up_sync(kFull, x, o);
    if (lane >= o) x += y;
  }
  return x;
}

// The whole block finds the bin holding the k_rem-th largest key, scanning from the top bin.
// Histogram values are read past L1 (they were completed by other CTAs' atomics).
__device__ void pick_bins(const uint32_t* hist, int nbits, SelectState* st, int level, uint32_t k_init) {
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
      }
    }
    cum += cnt;
  }
}

// Called by every CTA after its histogram atomics: the last CTA to arrive does the pick.
__device__ __forceinline__ void last_block_pick(const uint32_t* hist, int nbits, SelectState* st, int level,
                                                uint32_t k_init, uint32_t* counter = nullptr) {
  __shared__ uint32_t am_last;
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0)
    am_last = (atomicAdd(counter ? counter : &st->done[level], 1u) == gridDim.x - 1) ? 1u : 0u;
  __syncthreads();
  if (am_last) {
    __threadfence();
    pick_bins(hist, nbits, st, level, k_init);
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

// The i-th output (i = 0, 1, ...) of the splitmix64 stream seeded with `seed`: the state after
// i + 1 increments of the golden-ratio constant, mixed (Steele, Lea and Flood, 2014).
__device__ __forceinline__ uint64_t splitmix64_at(uint64_t seed, uint64_t i) {
  uint64_t z = seed + (i + 1) * 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

// Composite key of HEAVYMIX.  Members of H = {i : est_i^2 >= theta} get 0x80000000 | bits(|est_i|):
// all of H ranks above all of NH, and inside H by |est|.  Members of NH get 0x7FFFFFFF - xi_i,
// xi_i = the top 31 bits of splitmix64_at(fill_seed, i): the largest NH keys are the NH
// coordinates with the smallest xi, a uniformly random subset (rand_l(NH)).  The top-k of these
// keys (ties to the smaller index) is H plus k - |H| random coordinates of NH when |H| < k, and
// the k largest |est| of H otherwise.
__device__ __forceinline__ uint32_t heavy_key(float e, double theta, uint64_t fill_seed, uint64_t i) {
  const double e2 = (double)e * (double)e;  // exact
  return e2 >= theta ? (0x80000000u | key_of(e)) : 0x7FFFFFFFu - (uint32_t)(splitmix64_at(fill_seed, i) >> 33);
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
  int32_t hist_on;    // build the level-1 histogram of |est| keys and pick
  int32_t prune;      // skip rows below st->prune_key (estimate internal to the workspace)
  uint32_t* keys;     // HEAVYMIX: also store each coordinate's composite key here, and build the
                      // level-1 histogram (and pick) on those keys instead of |est|
  const double* theta;  // HEAVYMIX: the threshold l2sq / k of H
  uint64_t fill_seed;   // HEAVYMIX: the seed of the random fill
  HashCoeffs h;
};

// Row pruning.  With f = r/2 + 1: if at least f of a coordinate's r signed cells are < t and
// at least f are > -t, then -t < est < t.  For odd r the median is the f-th smallest and the
// f-th largest value; for even r the two middle values are the f-th smallest and the f-th
// largest, and the fp32 mean of two values in (-t, t) stays inside (rounding is monotone and
// twice an fp32 value is exact).  So a coordinate can stop reading rows as soon as both counts
// reach f: its |est| < t, and it cannot be among the top k when t is at most the k-th largest
// |est|.  Rows are read in order; the first f always, each later one only while the coordinate
// is undecided.  A cell with |v| < t counts on both sides, so f of those settle it after the
// first f rows; one cell outside (-t, t) among them costs one more row, not all of them.
// The prune key t is computed by this query itself before k_query runs (k_qsample: from the
// full estimate of a strided sample of coordinates; HEAVYMIX: from its threshold) and kept in
// the query's own selection state, so every CTA of k_query and k_repair reads the same value.
// It is a level-1 bin edge: whether it was safe is then exactly whether the level-1 pick
// lands in its bin or above, which k_repair checks.
// A coordinate that stopped early stores the marker -((32 g + n) * 2^-149): n = the rows whose
// cells it examined (f <= n < r), g = how many of those cells it read from the table (g = n
// when every examined cell is read).  It is a key in level-1 bin 0 that k_repair recognises
// and the measurement can count.
constexpr uint32_t kPrunedBits = 0x80000000u;  // sign bit; the low bits hold n and g

__device__ __forceinline__ uint32_t pruned_marker(int examined, int gathered) {
  return kPrunedBits | ((uint32_t)gathered << 5) | (uint32_t)examined;
}

__device__ __forceinline__ bool is_pruned(uint32_t bits) { return bits - (kPrunedBits + 1u) < 0x3FFu; }

// Counts of a coordinate's cells below t (lt) and above -t (gt), on keys: |v| < t is
// key_of(v) < pk; a NaN counts on neither side.
__device__ __forceinline__ void tally(float v, uint32_t pk, int& lt, int& gt) {
  const uint32_t b = __float_as_uint(v), key = b & 0x7FFFFFFFu;
  const bool inside = key < pk;
  const bool number = key <= 0x7F800000u;
  lt += (inside || (number && (b >> 31))) ? 1 : 0;
  gt += (inside || (number && !(b >> 31))) ? 1 : 0;
}

__device__ __forceinline__ uint32_t prune_key_of(const QueryParams& prm) {
  return prm.prune ? __ldcg(&prm.st->prune_key) : 0u;
}

__device__ __forceinline__ void store_est(const QueryParams& prm, int64_t i0, int tmax,
                                          const float (&m)[4]) {
  if (prm.vec && tmax == 4) {
    *reinterpret_cast<float4*>(prm.est + i0) = make_float4(m[0], m[1], m[2], m[3]);
  } else {
    for (int t = 0; t < tmax; ++t) prm.est[i0 + t] = m[t];
  }
}

// ---- the query ----------------------------------------------------------------------------

// Fast path: R rows known at compile time, c a power of two.  A thread takes four consecutive
// coordinates; their hash values after the first come from the incremental form.
// HM: HEAVYMIX mode (prm.keys set): each coordinate's composite key is stored and histogrammed.
// Up to 7 rows the register budget keeps four CTAs per SM (no spills at 64 registers).
template <int R, bool HM = false>
__global__ void __launch_bounds__(kBlock, R <= 7 ? 4 : 1) k_query(const __grid_constant__ QueryParams prm) {
  grid_begin();
  __shared__ uint32_t sh[kBins];
  for (int b = threadIdx.x; b < kBins; b += blockDim.x) sh[b] = 0;
  __syncthreads();
  const int64_t d = prm.d, nq = (d + 3) / 4;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const int lane = threadIdx.x & 31;
  const uint32_t pk = prune_key_of(prm);
  const double theta = HM ? __ldcg(prm.theta) : 0.0;
  constexpr int kF = R / 2 + 1;  // rows that bound the median
  for (int64_t q0 = (int64_t)blockIdx.x * blockDim.x + (threadIdx.x & ~31); q0 < nq; q0 += stride) {
    const int64_t q = q0 + lane;
    const int64_t i0 = q * 4;
    const int tmax = q < nq ? (d - i0 < 4 ? (int)(d - i0) : 4) : 0;
    float m[4] = {0.f, 0.f, 0.f, 0.f};
    uint32_t hk[4] = {0u, 0u, 0u, 0u};
    if (tmax > 0) {
      float v[4][R];
#pragma unroll
      for (int j = 0; j < kF; ++j) {
        uint64_t x = affine61_nb(prm.h.a[j], prm.h.b[j], (uint32_t)i0);
        uint64_t y = affine61_nb(prm.h.a2[j], prm.h.b2[j], (uint32_t)i0);
        const float* row = prm.T + (size_t)j * prm.c;
#pragma unroll
        for (int t = 0; t < 4; ++t) {
          v[t][j] = 0.f;
          if (t < tmax) {
            v[t][j] = apply_sign(__ldg(row + ((uint32_t)x & prm.cmask)), signbit_of(y));
            x = step61_nb(x, prm.h.a[j]);
            y = step61_nb(y, prm.h.a2[j]);
          }
        }
      }
      // the later rows, each only while the coordinate is undecided
      int lt[4], gt[4], rows[4];
      bool done[4];
#pragma unroll
      for (int t = 0; t < 4; ++t) {
        lt[t] = 0;
        gt[t] = 0;
#pragma unroll
        for (int j = 0; j < kF; ++j) tally(v[t][j], pk, lt[t], gt[t]);
        rows[t] = kF;
        done[t] = pk != 0u && lt[t] >= kF && gt[t] >= kF;
      }
#pragma unroll
      for (int j = kF; j < R; ++j) {
        uint64_t x = affine61_nb(prm.h.a[j], prm.h.b[j], (uint32_t)i0);
        uint64_t y = affine61_nb(prm.h.a2[j], prm.h.b2[j], (uint32_t)i0);
        const float* row = prm.T + (size_t)j * prm.c;
#pragma unroll
        for (int t = 0; t < 4; ++t) {
          v[t][j] = 0.f;
          if (t < tmax) {
            if (!done[t]) {
              v[t][j] = apply_sign(__ldg(row + ((uint32_t)x & prm.cmask)), signbit_of(y));
              tally(v[t][j], pk, lt[t], gt[t]);
              ++rows[t];
            }
            x = step61_nb(x, prm.h.a[j]);
            y = step61_nb(y, prm.h.a2[j]);
          }
        }
        if (j + 1 < R) {
#pragma unroll
          for (int t = 0; t < 4; ++t) done[t] = done[t] || (pk != 0u && lt[t] >= kF && gt[t] >= kF);
        }
      }
#pragma unroll
      for (int t = 0; t < 4; ++t)
        m[t] = done[t] ? __uint_as_float(pruned_marker(rows[t], rows[t])) : median_of<R>(v[t]);
      store_est(prm, i0, tmax, m);
      if (HM) {
#pragma unroll
        for (int t = 0; t < 4; ++t)
          hk[t] = heavy_key(done[t] ? 0.f : m[t], theta, prm.fill_seed, (uint64_t)(i0 + t));
        if (tmax == 4) {
          *reinterpret_cast<uint4*>(prm.keys + i0) = make_uint4(hk[0], hk[1], hk[2], hk[3]);
        } else {
          for (int t = 0; t < tmax; ++t) prm.keys[i0 + t] = hk[t];
        }
      }
    }
    if (prm.hist_on) {
#pragma unroll
      for (int t = 0; t < 4; ++t)
        hist_add(sh, t < tmax ? ((HM ? hk[t] : key_of(m[t])) >> kL1Shift) : kNone);
    }
  }
  if (prm.hist_on) {
    hist_flush(sh, prm.hist, kBins);
    last_block_pick(prm.hist, 11, prm.st, 0, prm.k);
  }
}

// ---- the pruning query with the first rows classified in shared memory ---------------------
// The settle rule needs, for each of the first f = r/2 + 1 cells of a coordinate, only which side
// of the prune key t its value lies on.  For a row that is a class per table cell, two bits:
// whether T counts below t and whether it counts above -t (3 for |T| < t, 1 for T >= t, 2 for
// T <= -t, 0 for NaN); the sign hash of the coordinate swaps the two bits.
// Where the classes of the first f rows fit in shared memory (2 bits per cell), k_pbits writes
// them once per query and k_query_bits looks them up instead of reading those cells from L2.  A
// coordinate that settles within the first f rows then reads no cell at all; one that examines
// later rows reads those cells as k_query does; one that does not settle reads every cell for
// its full median.  The rows examined, the stops and the estimates are the same as k_query's.
constexpr uint32_t kBitsBytes = 192u << 10;   // dynamic shared memory for the classes

constexpr int kBitsBlock = 1024;              // one CTA of 32 warps per SM

// The class as two bits: bit 1 set when the cell counts below t (T < t), bit 0 when it counts
// above -t (T > -t): 3 for |T| < t, 1 for T >= t, 2 for T <= -t, 0 for NaN.
__device__ __forceinline__ uint32_t cell_class(float v, uint32_t pk) {
  const uint32_t b = __float_as_uint(v), key = b & 0x7FFFFFFFu;
  if (key > 0x7F800000u) return 0u;
  if (key < pk) return 3u;
  return (b >> 31) ? 2u : 1u;
}

// Word w holds the classes of cells 16 w .. 16 w + 15 of the first rows of the row-major merged
// table, cell 16 w + u at bits 2u, 2u + 1.  nwords = f * c / 16.
__global__ void __launch_bounds__(kBlock) k_pbits(const float* __restrict__ T, int64_t nwords,
                                                  const SelectState* st, uint32_t* __restrict__ words) {
  grid_begin();
  const uint32_t pk = __ldcg(&st->prune_key);
  for (int64_t w = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; w < nwords; w += (int64_t)gridDim.x * blockDim.x) {
    const float4* src = reinterpret_cast<const float4*>(T) + 4 * w;
    uint32_t out = 0;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const float4 v = __ldg(src + q);
      out |= (cell_class(v.x, pk) | cell_class(v.y, pk) << 2 | cell_class(v.z, pk) << 4 | cell_class(v.w, pk) << 6)
             << (8 * q);
    }
    words[w] = out;
  }
}

template <int R>
__global__ void __launch_bounds__(kBitsBlock, 1) k_query_bits(const __grid_constant__ QueryParams prm,
                                                              const uint32_t* __restrict__ words) {
  grid_begin();
  extern __shared__ uint4 sbits4[];
  const uint32_t* sbits = reinterpret_cast<const uint32_t*>(sbits4);
  __shared__ uint32_t sh[kBins];
  constexpr int kF = R / 2 + 1;
  {
    const int64_t n4 = (int64_t)kF * (prm.c / 16) / 4;
    const uint4* src = reinterpret_cast<const uint4*>(words);
    for (int64_t w = threadIdx.x; w < n4; w += blockDim.x) sbits4[w] = __ldcg(src + w);
  }
  for (int b = threadIdx.x; b < kBins; b += blockDim.x) sh[b] = 0;
  __syncthreads();
  const int64_t d = prm.d, nq = (d + 3) / 4;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const int lane = threadIdx.x & 31;
  const uint32_t pk = prune_key_of(prm);
  for (int64_t q0 = (int64_t)blockIdx.x * blockDim.x + (threadIdx.x & ~31); q0 < nq; q0 += stride) {
    const int64_t q = q0 + lane;
    const int64_t i0 = q * 4;
    const int tmax = q < nq ? (d - i0 < 4 ? (int)(d - i0) : 4) : 0;
    float m[4] = {0.f, 0.f, 0.f, 0.f};
    if (tmax > 0) {
      float v[4][R];
      uint32_t cell[4][kF];  // bucket of each of the first kF rows, sign bit of the cell in bit 31
      int lt[4], gt[4], rows[4];
      bool done[4];
      uint32_t count[4] = {0u, 0u, 0u, 0u};
      // the first kF rows: classes from shared memory, no table reads
#pragma unroll
      for (int j = 0; j < kF; ++j) {
        uint64_t x = affine61_nb(prm.h.a[j], prm.h.b[j], (uint32_t)i0);
        uint64_t y = affine61_nb(prm.h.a2[j], prm.h.b2[j], (uint32_t)i0);
#pragma unroll
        for (int t = 0; t < 4; ++t) {
          cell[t][j] = 0u;
          if (t < tmax) {
            const uint32_t b = (uint32_t)x & prm.cmask;
            const uint32_t g = (uint32_t)j * prm.c + b;
            const uint32_t cls = (sbits[g >> 4] >> ((g & 15u) * 2u)) & 3u;
            // a negative sign swaps the two bits; count[t] holds below-t in bits 0-7 and
            // above-(-t) in bits 8-15: (cls * 0x201) >> 1 puts bit 1 at 0 and bit 0 at 8,
            // cls * 0x81 puts bit 0 at 0 and bit 1 at 8
            const uint32_t s = (uint32_t)y & 1u;
            count[t] += ((cls * (s ? 0x81u : 0x201u)) >> (1u - s)) & 0x101u;
            cell[t][j] = b | signbit_of(y);
            x = step61_nb(x, prm.h.a[j]);
            y = step61_nb(y, prm.h.a2[j]);
          }
        }
      }
#pragma unroll
      for (int t = 0; t < 4; ++t) {
        lt[t] = (int)(count[t] & 0xFFu);
        gt[t] = (int)(count[t] >> 8);
        rows[t] = kF;
        done[t] = pk != 0u && lt[t] >= kF && gt[t] >= kF;
      }
      // the later rows, each only while the coordinate is undecided (read from the table)
#pragma unroll
      for (int j = kF; j < R; ++j) {
        uint64_t x = affine61_nb(prm.h.a[j], prm.h.b[j], (uint32_t)i0);
        uint64_t y = affine61_nb(prm.h.a2[j], prm.h.b2[j], (uint32_t)i0);
        const float* row = prm.T + (size_t)j * prm.c;
#pragma unroll
        for (int t = 0; t < 4; ++t) {
          v[t][j] = 0.f;
          if (t < tmax) {
            if (!done[t]) {
              v[t][j] = apply_sign(__ldg(row + ((uint32_t)x & prm.cmask)), signbit_of(y));
              tally(v[t][j], pk, lt[t], gt[t]);
              ++rows[t];
            }
            x = step61_nb(x, prm.h.a[j]);
            y = step61_nb(y, prm.h.a2[j]);
          }
        }
        if (j + 1 < R) {
#pragma unroll
          for (int t = 0; t < 4; ++t) done[t] = done[t] || (pk != 0u && lt[t] >= kF && gt[t] >= kF);
        }
      }
      // a coordinate that did not settle needs its full median: read its first kF cells now
#pragma unroll
      for (int j = 0; j < kF; ++j) {
#pragma unroll
        for (int t = 0; t < 4; ++t) {
          v[t][j] = 0.f;
          if (t < tmax && !done[t])
            v[t][j] = apply_sign(__ldg(prm.T + (size_t)j * prm.c + (cell[t][j] & 0x7FFFFFFFu)),
                                 cell[t][j] & 0x80000000u);
        }
      }
#pragma unroll
      for (int t = 0; t < 4; ++t)
        m[t] = done[t] ? __uint_as_float(pruned_marker(rows[t], rows[t] - kF)) : median_of<R>(v[t]);
      store_est(prm, i0, tmax, m);
    }
#pragma unroll
    for (int t = 0; t < 4; ++t) hist_add(sh, t < tmax ? (key_of(m[t]) >> kL1Shift) : kNone);
  }
  hist_flush(sh, prm.hist, kBins);
  last_block_pick(prm.hist, 11, prm.st, 0, prm.k);
}

// Runs after k_query.  If the level-1 pick landed in the prune key's bin or above, the k-th
// largest |est| is at least the prune key and pruning changed nothing the selection sees: the
// kernel returns at once.  Otherwise every stored marker (each pruned coordinate, and any
// genuine estimate with the same bits, which recomputes to itself) gets its full median, the
// level-1 histogram is rebuilt from all estimates into hist_r, and the level-1 pick is made
// again.
template <int R>
__global__ void __launch_bounds__(kBlock) k_repair(const __grid_constant__ QueryParams prm, uint32_t* hist_r) {
  grid_begin();
  const uint32_t pk = __ldcg(&prm.st->prune_key);
  if (pk == 0u || __ldcg(&prm.st->prefix) >= (pk >> kL1Shift)) return;  // uniform over the grid
  __shared__ uint32_t sh[kBins];
  for (int b = threadIdx.x; b < kBins; b += blockDim.x) sh[b] = 0;
  __syncthreads();
  const int64_t d = prm.d;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const int lane = threadIdx.x & 31;
  for (int64_t base = (int64_t)blockIdx.x * blockDim.x + (threadIdx.x & ~31); base < d; base += stride) {
    const int64_t i = base + lane;
    uint32_t bin = kNone;
    if (i < d) {
      float e = prm.est[i];
      if (is_pruned(__float_as_uint(e))) {
        float v[R];
#pragma unroll
        for (int j = 0; j < R; ++j) {
          const uint64_t x = affine61(prm.h.a[j], prm.h.b[j], (uint32_t)i);
          const uint64_t y = affine61(prm.h.a2[j], prm.h.b2[j], (uint32_t)i);
          v[j] = apply_sign(__ldg(prm.T + (size_t)j * prm.c + ((uint32_t)x & prm.cmask)), signbit_of(y));
        }
        e = median_of<R>(v);
        prm.est[i] = e;
      }
      bin = key_of(e) >> kL1Shift;
    }
    hist_add(sh, bin);
  }
  hist_flush(sh, hist_r, kBins);
  last_block_pick(hist_r, 11, prm.st, 0, prm.k, &prm.st->done_r);
}

// The prune key of this query, from a fixed strided sample: the first four coordinates of
// every kSampleQuads * 4 (all rows, full median).  The last CTA finds the level-1 bin holding
// the j_target-th largest sampled key and stores its lower edge as st->prune_key (0, i.e. no
// pruning, when that is bin 0 or the sample holds fewer keys).  j_target is set on the host
// well above the sample's expected share of the top k, so that the key lies below the k-th
// largest |est| of the whole estimate except with negligible probability; k_repair makes the
// result exact in that case as well.
constexpr int64_t kSampleQuads = 64;

template <int R>
__global__ void __launch_bounds__(kBlock) k_qsample(const __grid_constant__ QueryParams prm, uint32_t* hist_s,
                                                    uint32_t j_target) {
  grid_begin();
  __shared__ uint32_t sh[kBins];
  __shared__ uint32_t am_last;
  for (int b = threadIdx.x; b < kBins; b += blockDim.x) sh[b] = 0;
  __syncthreads();
  const int64_t d = prm.d, nq = (d + 3) / 4, ns = (nq + kSampleQuads - 1) / kSampleQuads;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const int lane = threadIdx.x & 31;
  for (int64_t s0 = (int64_t)blockIdx.x * blockDim.x + (threadIdx.x & ~31); s0 < ns; s0 += stride) {
    const int64_t sq = s0 + lane;
    const int64_t i0 = sq * kSampleQuads * 4;
    const int tmax = sq < ns ? (d - i0 < 4 ? (int)(d - i0) : 4) : 0;
    float m[4] = {0.f, 0.f, 0.f, 0.f};
    if (tmax > 0) {
      float v[4][R];
#pragma unroll
      for (int j = 0; j < R; ++j) {
        uint64_t x = affine61_nb(prm.h.a[j], prm.h.b[j], (uint32_t)i0);
        uint64_t y = affine61_nb(prm.h.a2[j], prm.h.b2[j], (uint32_t)i0);
        const float* row = prm.T + (size_t)j * prm.c;
#pragma unroll
        for (int t = 0; t < 4; ++t) {
          v[t][j] = 0.f;
          if (t < tmax) {
            v[t][j] = apply_sign(__ldg(row + ((uint32_t)x & prm.cmask)), signbit_of(y));
            x = step61_nb(x, prm.h.a[j]);
            y = step61_nb(y, prm.h.a2[j]);
          }
        }
      }
#pragma unroll
      for (int t = 0; t < 4; ++t) m[t] = median_of<R>(v[t]);
    }
#pragma unroll
    for (int t = 0; t < 4; ++t) hist_add(sh, t < tmax ? (key_of(m[t]) >> kL1Shift) : kNone);
  }
  hist_flush(sh, hist_s, kBins);
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) am_last = (atomicAdd(&prm.st->done_s, 1u) == gridDim.x - 1) ? 1u : 0u;
  __syncthreads();
  if (!am_last) return;
  __threadfence();
  const int per = (kBins + blockDim.x - 1) / blockDim.x;
  const int r0 = threadIdx.x * per;  // positions counted from the top bin
  uint32_t local = 0;
  for (int t = 0; t < per; ++t) {
    if (r0 + t < kBins) local += __ldcg(&hist_s[kBins - 1 - (r0 + t)]);
  }
  uint32_t total;
  uint32_t cum = block_excl_scan(local, &total);
  for (int t = 0; t < per; ++t) {
    const int rp = r0 + t;
    if (rp >= kBins) break;
    const int bin = kBins - 1 - rp;
    const uint32_t cnt = __ldcg(&hist_s[bin]);
    if (cum < j_target && cum + cnt >= j_target) prm.st->prune_key = bin > 0 ? (uint32_t)bin << kL1Shift : 0u;
    cum += cnt;
  }
}

// Request-ceiling probe of the query (measurement aid): the loads of k_query with every row
// read (the same grid, hash buckets and incremental form), without the median, the estimate
// store or the histogram.  Each CTA writes the sum of what it read to out[blockIdx.x], so that
// the loads cannot be dropped.
template <int R>
__global__ void __launch_bounds__(kBlock) k_gather_probe(const __grid_constant__ QueryParams prm, float* out) {
  grid_begin();
  __shared__ float warp_sum[kBlock / 32];
  const int64_t d = prm.d, nq = (d + 3) / 4;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  float acc = 0.f;
  for (int64_t q = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; q < nq; q += stride) {
    const int64_t i0 = q * 4;
    const int tmax = d - i0 < 4 ? (int)(d - i0) : 4;
#pragma unroll
    for (int j = 0; j < R; ++j) {
      uint64_t x = affine61(prm.h.a[j], prm.h.b[j], (uint32_t)i0);
      const float* row = prm.T + (size_t)j * prm.c;
#pragma unroll
      for (int t = 0; t < 4; ++t) {
        if (t < tmax) {
          acc += __ldg(row + ((uint32_t)x & prm.cmask));
          x = step61(x, prm.h.a[j]);
        }
      }
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) acc += __shfl_down_sync(kFull, acc, o);
  if ((threadIdx.x & 31) == 0) warp_sum[threadIdx.x >> 5] = acc;
  __syncthreads();
  if (threadIdx.x == 0) {
    float t = 0.f;
    for (int w = 0; w < kBlock / 32; ++w) t += warp_sum[w];
    out[blockIdx.x] = t;
  }
}

// General path: any r <= 16 and any c (bucket by 64-bit remainder).
__global__ void __launch_bounds__(kBlock) k_query_generic(const __grid_constant__ QueryParams prm) {
  grid_begin();
  __shared__ uint32_t sh[kBins];
  for (int b = threadIdx.x; b < kBins; b += blockDim.x) sh[b] = 0;
  __syncthreads();
  const int64_t d = prm.d;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const int lane = threadIdx.x & 31;
  const int r = prm.r;
  const double theta = prm.keys ? __ldcg(prm.theta) : 0.0;
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
      uint32_t key = key_of(m);
      if (prm.keys) {
        key = heavy_key(m, theta, prm.fill_seed, (uint64_t)i);
        prm.keys[i] = key;
      }
      bin = key >> kL1Shift;
    }
    if (prm.hist_on) hist_add(sh, bin);
  }
  if (prm.hist_on) {
    hist_flush(sh, prm.hist, kBins);
    last_block_pick(prm.hist, 11, prm.st, 0, prm.k);
  }
}

// Four float4 of est per thread in flight (kU strides of the grid-stride loop).
constexpr int kU = 4;

__device__ __forceinline__ void load_quads(const float* __restrict__ est, int64_t d, int vec, int64_t q0,
                                           int64_t stride, float (&v)[kU][4], int (&tm)[kU]) {
  const int64_t nq = (d + 3) / 4;
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int u = 0; u < kU; ++u) {
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
}

// ---- selection with candidate lists --------------------------------------------------------

// One pass over est after the level-1 pick.  Keys above the level-1 bin are selected for
// certain: their bit goes into gt_bm.  Keys inside the bin are candidates (index, key): they
// feed the level-2 histogram and are appended to `cand`; the level-2 pick follows.  Both are
// rare (fewer than k keys lie above the bin, and the bin is a narrow band of keys), so the
// common path per key is a mask, a shift and a compare.  Candidates collect in a block-local
// buffer (slots taken with a warp-aggregated shared atomic) that is copied out with one
// global reservation per block; a block whose buffer fills up appends the rest directly
// (warp-aggregated global atomics), which only happens for inputs with many equal keys.
// `src` holds the keys as 32-bit words: the bits of est (kmask drops the sign) or a key array.
constexpr int kCandBuf = 2048;

__device__ __forceinline__ void cand_append(uint32_t i, uint32_t key, uint32_t* sh_n, uint2* sh_cand,
                                            SelectState* st, uint2* __restrict__ cand) {
  const int lane = threadIdx.x & 31;
  uint32_t am = __activemask();
  int leader = __ffs(am) - 1;
  uint32_t base = 0;
  if (lane == leader) base = atomicAdd(sh_n, (uint32_t)__popc(am));
  base = __shfl_sync(am, base, leader);
  const uint32_t slot = base + __popc(am & ((1u << lane) - 1u));
  if (slot < (uint32_t)kCandBuf) {
    sh_cand[slot] = make_uint2(i, key);
    return;
  }
  am = __activemask();
  leader = __ffs(am) - 1;
  uint32_t gbase = 0;
  if (lane == leader) gbase = atomicAdd(&st->ncand, (uint32_t)__popc(am));
  gbase = __shfl_sync(am, gbase, leader);
  cand[gbase + __popc(am & ((1u << lane) - 1u))] = make_uint2(i, key);
}

__global__ void __launch_bounds__(kBlock) k_cand(const float* __restrict__ src, int64_t d, int vec, uint32_t kmask,
                                                 SelectState* st, uint32_t* hist2, uint2* __restrict__ cand,
                                                 uint32_t* gt_bm) {
  grid_begin();
  __shared__ uint32_t sh[kBins];
  __shared__ uint2 sh_cand[kCandBuf];
  __shared__ uint32_t sh_n, sh_base;
  for (int b = threadIdx.x; b < kBins; b += blockDim.x) sh[b] = 0;
  if (threadIdx.x == 0) sh_n = 0;
  __syncthreads();
  const uint32_t b1 = __ldcg(&st->prefix);
  const int64_t nq = (d + 3) / 4;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const int lane = threadIdx.x & 31;
  for (int64_t q0 = (int64_t)blockIdx.x * blockDim.x + (threadIdx.x & ~31); q0 < nq; q0 += kU * stride) {
    float v[kU][4];
    int tm[kU];
    load_quads(src, d, vec, q0, stride, v, tm);
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      const uint32_t i0 = (uint32_t)((q0 + u * stride + lane) * 4);
#pragma unroll
      for (int t = 0; t < 4; ++t) {
        const uint32_t key = __float_as_uint(v[u][t]) & kmask;
        if (t < tm[u] && (key >> kL1Shift) >= b1) {
          const uint32_t i = i0 + t;
          if ((key >> kL1Shift) > b1) {
            atomicOr(&gt_bm[i >> 5], 1u << (i & 31));
          } else {
            atomicAdd(&sh[(key >> kL2Shift) & (kBins - 1)], 1u);
            cand_append(i, key, &sh_n, sh_cand, st, cand);
          }
        }
      }
    }
  }
  __syncthreads();
  const uint32_t n = sh_n < (uint32_t)kCandBuf ? sh_n : (uint32_t)kCandBuf;
  if (threadIdx.x == 0) sh_base = n ? atomicAdd(&st->ncand, n) : 0u;
  __syncthreads();
  for (uint32_t t = threadIdx.x; t < n; t += blockDim.x) cand[sh_base + t] = sh_cand[t];
  hist_flush(sh, hist2, kBins);
  last_block_pick(hist2, 11, st, 1, 0);
}

// Level-3 histogram of the candidates that match the 22-bit prefix; the last pick gives tau.
__global__ void __launch_bounds__(kBlock) k_cand_hist3(const uint2* __restrict__ cand, SelectState* st,
                                                       uint32_t* hist3) {
  grid_begin();
  constexpr int kN3 = 1 << kL3Bits;
  __shared__ uint32_t sh[kN3];
  for (int b = threadIdx.x; b < kN3; b += blockDim.x) sh[b] = 0;
  __syncthreads();
  const uint32_t n = __ldcg(&st->ncand);
  const uint32_t p22 = __ldcg(&st->prefix);
  const uint32_t stride = gridDim.x * blockDim.x;
  const int lane = threadIdx.x & 31;
  for (uint32_t t0 = blockIdx.x * blockDim.x + (threadIdx.x & ~31u); t0 < n; t0 += stride) {
    const uint32_t t = t0 + lane;
    uint32_t bin = kNone;
    if (t < n) {
      const uint32_t key = cand[t].y;
      if ((key >> kL2Shift) == p22) bin = key & (uint32_t)(kN3 - 1);
    }
    if (__any_sync(kFull, bin != kNone)) hist_add(sh, bin);
  }
  hist_flush(sh, hist3, kN3);
  last_block_pick(hist3, kL3Bits, st, 2, 0);
}

// Candidates above tau into gt_bm, candidates equal to tau into eq_bm.
__global__ void __launch_bounds__(kBlock) k_cand_mark(const uint2* __restrict__ cand, const SelectState* st,
                                                      uint32_t* gt_bm, uint32_t* eq_bm) {
  grid_begin();
  const uint32_t n = __ldcg(&st->ncand);
  const uint32_t tau = __ldcg(&st->tau);
  for (uint32_t t = blockIdx.x * blockDim.x + threadIdx.x; t < n; t += gridDim.x * blockDim.x) {
    const uint2 c = cand[t];
    if (c.y > tau) atomicOr(&gt_bm[c.x >> 5], 1u << (c.x & 31));
    else if (c.y == tau) atomicOr(&eq_bm[c.x >> 5], 1u << (c.x & 31));
  }
}

constexpr int kBmThreads = 256;
constexpr int kBmWordsPerThread = 8;
constexpr int kBmWords = kBmThreads * kBmWordsPerThread;  // 2048 words = 65536 coordinates per block

__global__ void __launch_bounds__(kBmThreads) k_bm_count(const uint32_t* __restrict__ gt_bm,
                                                         const uint32_t* __restrict__ eq_bm, int64_t nbw,
                                                         uint32_t* blk_gt, uint32_t* blk_eq) {
  grid_begin();
  const int64_t w0 = (int64_t)blockIdx.x * kBmWords + (int64_t)threadIdx.x * kBmWordsPerThread;
  uint32_t gt = 0, eq = 0;
#pragma unroll
  for (int j = 0; j < kBmWordsPerThread; ++j) {
    if (w0 + j < nbw) {
      gt += __popc(__ldcg(&gt_bm[w0 + j]));
      eq += __popc(__ldcg(&eq_bm[w0 + j]));
    }
  }
  uint32_t tg, te;
  block_excl_scan(gt, &tg);
  block_excl_scan(eq, &te);
  if (threadIdx.x == 0) {
    blk_gt[blockIdx.x] = tg;
    blk_eq[blockIdx.x] = te;
  }
}

__global__ void __launch_bounds__(kScanThreads) k_scan(const uint32_t* __restrict__ blk_gt,
                                                       const uint32_t* __restrict__ blk_eq, int64_t nblk,
                                                       const SelectState* st, uint32_t* blk_base,
                                                       uint32_t* blk_eqx) {
  grid_begin();
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

// Walks the set bits of each thread's words in index order: bits of gt_bm are taken, bits of
// eq_bm are taken while their rank among the keys equal to tau is below need_eq.
__global__ void __launch_bounds__(kBmThreads) k_bm_write(const uint32_t* __restrict__ gt_bm,
                                                         const uint32_t* __restrict__ eq_bm, int64_t nbw,
                                                         const SelectState* st, const uint32_t* __restrict__ blk_base,
                                                         const uint32_t* __restrict__ blk_eqx,
                                                         int64_t* __restrict__ idx_out, int64_t k) {
  grid_begin();
  const uint32_t need_eq = __ldcg(&st->need_eq);
  const uint32_t base = blk_base[blockIdx.x];
  const uint32_t eqx = blk_eqx[blockIdx.x];
  const int64_t w0 = (int64_t)blockIdx.x * kBmWords + (int64_t)threadIdx.x * kBmWordsPerThread;
  uint32_t g[kBmWordsPerThread], e[kBmWordsPerThread];
  uint32_t gt = 0, eq = 0;
#pragma unroll
  for (int j = 0; j < kBmWordsPerThread; ++j) {
    const bool in = w0 + j < nbw;
    g[j] = in ? __ldcg(&gt_bm[w0 + j]) : 0u;
    e[j] = in ? __ldcg(&eq_bm[w0 + j]) : 0u;
    gt += __popc(g[j]);
    eq += __popc(e[j]);
  }
  uint32_t tg, te;
  const uint32_t pre_gt = block_excl_scan(gt, &tg);
  const uint32_t pre_eq = block_excl_scan(eq, &te);
  if (gt + eq == 0) return;
  const uint32_t eq_quota = need_eq > eqx ? need_eq - eqx : 0u;  // this block's share of ties
  uint32_t pos = base + pre_gt + (pre_eq < eq_quota ? pre_eq : eq_quota);
  uint32_t eq_rank = pre_eq;
#pragma unroll
  for (int j = 0; j < kBmWordsPerThread; ++j) {
    uint32_t bits = g[j] | e[j];
    while (bits) {
      const int b = __ffs(bits) - 1;
      bits &= bits - 1u;
      bool take = (g[j] >> b) & 1u;
      if (!take) {
        take = eq_rank < eq_quota;
        ++eq_rank;
      }
      if (take) {
        if ((int64_t)pos < k) idx_out[pos] = (w0 + j) * 32 + b;
        ++pos;
      }
    }
  }
}

// ---- selection by full passes over est (fixed-scratch variant) -----------------------------

// Histogram of key bits [shift, shift + nbits) among keys whose bits above are the prefix
// picked at the previous level; ends with the pick of this level.
__global__ void __launch_bounds__(kBlock) k_hist(const float* __restrict__ est, int64_t d, int vec,
                                                 SelectState* st, uint32_t* hist, int shift, int nbits,
                                                 int level) {
  grid_begin();
  __shared__ uint32_t sh[kBins];
  const int nbins = 1 << nbits;
  for (int b = threadIdx.x; b < nbins; b += blockDim.x) sh[b] = 0;
  __syncthreads();
  const uint32_t prefix = __ldcg(&st->prefix);
  const int match_shift = shift + nbits;
  const int64_t nq = (d + 3) / 4;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t q0 = (int64_t)blockIdx.x * blockDim.x + (threadIdx.x & ~31); q0 < nq; q0 += kU * stride) {
    float v[kU][4];
    int tm[kU];
    load_quads(est, d, vec, q0, stride, v, tm);
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      uint32_t bins[4];
      bool any = false;
#pragma unroll
      for (int t = 0; t < 4; ++t) {
        const uint32_t key = key_of(v[u][t]);
        const bool hit = t < tm[u] && (key >> match_shift) == prefix;
        bins[t] = hit ? ((key >> shift) & (uint32_t)(nbins - 1)) : kNone;
        any = any || hit;
      }
      if (__any_sync(kFull, any)) {  // most warps hold no key of the chosen bin
#pragma unroll
        for (int t = 0; t < 4; ++t) hist_add(sh, bins[t]);
      }
    }
  }
  hist_flush(sh, hist, nbins);
  last_block_pick(hist, nbits, st, level, 0);
}

// Segments of kSeg coordinates; a warp owns kWarpRun consecutive coordinates and reads them as
// kRows rows of 128 (lane l holds coordinates 4l .. 4l+3 of each row), so every load is a
// coalesced float4 and the ascending order of a warp's run is (row, lane, component).
constexpr int kSegThreads = 256;
constexpr int kSeg = 16384;
constexpr int kSegWarps = kSegThreads / 32;
constexpr int kWarpRun = kSeg / kSegWarps;   // 2048
constexpr int kRows = kWarpRun / 128;        // 16

template <bool VEC>
__device__ __forceinline__ void load_row(const float* __restrict__ est, int64_t i0, int64_t s1, float (&v)[4]) {
  if (VEC && i0 + 4 <= s1) {
    const float4 f = __ldg(reinterpret_cast<const float4*>(est + i0));
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

template <bool VEC>
__global__ void __launch_bounds__(kSegThreads) k_count(const float* __restrict__ est, int64_t d,
                                                       const SelectState* st, uint32_t* blk_gt,
                                                       uint32_t* blk_eq) {
  grid_begin();
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

// Counts first (all rows in flight), then each row again from L1 to place its keys.
template <bool VEC>
__global__ void __launch_bounds__(kSegThreads) k_write(const float* __restrict__ est, int64_t d,
                                                       const SelectState* st, const uint32_t* __restrict__ blk_base,
                                                       const uint32_t* __restrict__ blk_eqx,
                                                       int64_t* __restrict__ idx_out, int64_t k) {
  grid_begin();
  __shared__ uint32_t warp_tot[kSegWarps];
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
    for (int j = 0; j < kRows; ++j) load_row<VEC>(est, w0 + j * 128 + lane * 4, s1, v[j]);
#pragma unroll
    for (int j = 0; j < kRows; ++j) {
#pragma unroll
      for (int t = 0; t < 4; ++t) {
        if (w0 + j * 128 + lane * 4 + t < s1) cnt += count_key(key_of(v[j][t]), tau);
      }
    }
  }
  // warp totals -> each warp's prefix inside the segment
  const uint32_t wsum = __shfl_sync(kFull, warp_incl_scan(cnt), 31);
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
    load_row<VEC>(est, i0, s1, v);
    uint32_t key[4];
    uint32_t c = 0;
#pragma unroll
    for (int t = 0; t < 4; ++t) {
      key[t] = key_of(v[t]);
      if (i0 + t < s1) c += count_key(key[t], tau);
    }
    const uint32_t incl = warp_incl_scan(c);
    const uint32_t row_tot = __shfl_sync(kFull, incl, 31);
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

// ---- HEAVYMIX (Alg. 2 as printed) ----------------------------------------------------------

// Sum of squares of each row of the merged table in fp64; blockIdx.y is the row.
__global__ void __launch_bounds__(kBlock) k_row_sumsq(const float* __restrict__ T, uint32_t c, double* sumsq) {
  grid_begin();
  __shared__ double warp_acc[kBlock / 32];
  const int j = blockIdx.y;
  const float* row = T + (size_t)j * c;
  double acc = 0.0;
  for (uint32_t b = blockIdx.x * blockDim.x + threadIdx.x; b < c; b += gridDim.x * blockDim.x) {
    const double v = (double)row[b];
    acc += v * v;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) acc += __shfl_down_sync(kFull, acc, o);
  if ((threadIdx.x & 31) == 0) warp_acc[threadIdx.x >> 5] = acc;
  __syncthreads();
  if (threadIdx.x < 32) {
    double v = threadIdx.x < kBlock / 32 ? warp_acc[threadIdx.x] : 0.0;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_down_sync(kFull, v, o);
    if (threadIdx.x == 0) atomicAdd(&sumsq[j], v);
  }
}

// l2sq = median over rows of the row sums of squares (the sketch's estimate of ||g||^2);
// theta = l2sq / k, the threshold of H.
// With `prune`, also the prune key of the query that follows: a coordinate with |est| < f,
// f^2 <= theta, lies outside H, and only its index enters the selection (through the random
// fill), so no repair is ever needed.
__global__ void k_heavy_theta(const double* __restrict__ sumsq, int r, int64_t k, double* theta,
                              double* l2sq_out, SelectState* st, int prune) {
  grid_begin();
  if (blockIdx.x != 0 || threadIdx.x != 0) return;
  double v[GS_MAX_ROWS];
  for (int j = 0; j < r; ++j) v[j] = __ldcg(&sumsq[j]);
  for (int a = 1; a < r; ++a) {
    const double t = v[a];
    int b = a - 1;
    while (b >= 0 && v[b] > t) {
      v[b + 1] = v[b];
      --b;
    }
    v[b + 1] = t;
  }
  const double m = (r & 1) ? v[r / 2] : 0.5 * (v[r / 2 - 1] + v[r / 2]);
  const double th = m / (double)k;
  theta[0] = th;
  if (l2sq_out) l2sq_out[0] = m;
  if (prune && th > 0.0 && th <= 1e300) {
    float f = __double2float_rd(sqrt(th));
    if ((double)f * (double)f > th) f = nextafterf(f, 0.f);  // the product is exact in double
    st->prune_key = key_of(f) & ~((1u << kL1Shift) - 1u);
  }
}

// ---- launchers -----------------------------------------------------------------------------

template <typename K>
int persistent_grid(K kernel, int64_t work_items, int block) {
  const int64_t need = (work_items + block - 1) / block;
  const int64_t cap = (int64_t)device_info().sms * blocks_per_sm((const void*)kernel, block);
  return (int)(need < 1 ? 1 : (need < cap ? need : cap));
}

template <int R>
cudaError_t launch_query_r(const QueryParams& p, cudaStream_t s) {
  auto kern = p.keys ? k_query<R, true> : k_query<R, false>;
  launch(kern, persistent_grid(kern, (p.d + 3) / 4, kBlock), kBlock, s, p);
  return cudaGetLastError();
}

typedef cudaError_t (*QueryLauncher)(const QueryParams&, cudaStream_t);

template <int... Rs>
struct QueryTable {
  static constexpr QueryLauncher table[sizeof...(Rs)] = {&launch_query_r<Rs>...};
};
template <int... Rs>
constexpr QueryLauncher QueryTable<Rs...>::table[sizeof...(Rs)];

// k_query_bits<R> for a pruning query whose first rows' classes fit kBitsBytes: the classes are
// written into `words` (f * c / 4 bytes of scratch) first.
template <int R>
cudaError_t launch_query_bits_r(const QueryParams& p, uint32_t* words, cudaStream_t s) {
  constexpr int kF = R / 2 + 1;
  const int64_t nwords = (int64_t)kF * (p.c / 16);
  const int gw = (int)((nwords + kBlock - 1) / kBlock);
  launch(k_pbits, gw, kBlock, s, p.T, nwords, p.st, words);
  auto kern = k_query_bits<R>;
  const size_t smem = (size_t)nwords * sizeof(uint32_t);
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  const int64_t need = ((p.d + 3) / 4 + kBitsBlock - 1) / kBitsBlock;
  const int grid = (int)(need < device_info().sms ? (need < 1 ? 1 : need) : device_info().sms);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)grid);
  cfg.blockDim = dim3(kBitsBlock);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  e = cudaLaunchKernelEx(&cfg, kern, p, (const uint32_t*)words);
  return e != cudaSuccess ? e : cudaGetLastError();
}

typedef cudaError_t (*BitsLauncher)(const QueryParams&, uint32_t*, cudaStream_t);

template <int... Rs>
struct BitsTable {
  static constexpr BitsLauncher table[sizeof...(Rs)] = {&launch_query_bits_r<Rs>...};
};
template <int... Rs>
constexpr BitsLauncher BitsTable<Rs...>::table[sizeof...(Rs)];

// Whether a pruning query of r rows and c (a power of two) columns classifies its first rows in
// shared memory.
bool query_uses_bits(int r, uint32_t c) {
  const uint64_t bytes = (uint64_t)(r / 2 + 1) * c / 4;
  return r >= 3 && r <= GS_MAX_ROWS && is_pow2(c) && c >= 64 && bytes <= kBitsBytes;
}

template <int R>
cudaError_t launch_repair_r(const QueryParams& p, uint32_t* hist_r, cudaStream_t s) {
  auto kern = k_repair<R>;
  // one CTA per SM: the kernel almost always returns at once, and a repair is rare
  launch(kern, device_info().sms, kBlock, s, p, hist_r);
  return cudaGetLastError();
}

typedef cudaError_t (*RepairLauncher)(const QueryParams&, uint32_t*, cudaStream_t);

template <int... Rs>
struct RepairTable {
  static constexpr RepairLauncher table[sizeof...(Rs)] = {&launch_repair_r<Rs>...};
};
template <int... Rs>
constexpr RepairLauncher RepairTable<Rs...>::table[sizeof...(Rs)];

template <int R>
cudaError_t launch_qsample_r(const QueryParams& p, uint32_t* hist_s, uint32_t j_target, cudaStream_t s) {
  auto kern = k_qsample<R>;
  const int64_t ns = ((p.d + 3) / 4 + kSampleQuads - 1) / kSampleQuads;
  launch(kern, persistent_grid(kern, ns, kBlock), kBlock, s, p, hist_s, j_target);
  return cudaGetLastError();
}

typedef cudaError_t (*SampleLauncher)(const QueryParams&, uint32_t*, uint32_t, cudaStream_t);

template <int... Rs>
struct SampleTable {
  static constexpr SampleLauncher table[sizeof...(Rs)] = {&launch_qsample_r<Rs>...};
};
template <int... Rs>
constexpr SampleLauncher SampleTable<Rs...>::table[sizeof...(Rs)];

// Rank, among the sampled keys, whose level-1 bin gives the prune key.  The sample holds n_s
// of the d coordinates; the number of them among the k - 1 keys above the k-th largest is
// at most hypergeometric with mean mu = k n_s / d.  Taking rank mu + 4 sqrt(mu) + 2 puts the
// sampled key below the k-th largest unless that count exceeds its mean by four standard
// deviations; for k below that rank it cannot exceed it at all.  0: no usable rank.
uint32_t sample_rank(int64_t d, int64_t k) {
  const int64_t ns = ((d + 3) / 4 + kSampleQuads - 1) / kSampleQuads;
  const int64_t last = (ns - 1) * kSampleQuads * 4;
  const int64_t n_s = 4 * (ns - 1) + (d - last < 4 ? d - last : 4);
  const double mu = (double)k * (double)n_s / (double)d;
  const double j = std::ceil(mu + 4.0 * std::sqrt(mu)) + 2.0;
  return j <= (double)n_s ? (uint32_t)j : 0u;
}

template <int R>
cudaError_t launch_gather_probe_r(const QueryParams& p, float* out, int64_t out_floats, cudaStream_t s) {
  auto kern = k_gather_probe<R>;
  const int grid = persistent_grid(k_query<R>, (p.d + 3) / 4, kBlock);  // the query's grid
  if (grid > out_floats) return cudaErrorInvalidValue;
  launch(kern, grid, kBlock, s, p, out);
  return cudaGetLastError();
}

typedef cudaError_t (*ProbeLauncher)(const QueryParams&, float*, int64_t, cudaStream_t);

template <int... Rs>
struct ProbeTable {
  static constexpr ProbeLauncher table[sizeof...(Rs)] = {&launch_gather_probe_r<Rs>...};
};
template <int... Rs>
constexpr ProbeLauncher ProbeTable<Rs...>::table[sizeof...(Rs)];

// Pruning applies on the fast path (c a power of two) with at least three rows, and from
// 2^22 coordinates up: below that the query takes a few tens of microseconds and the repair
// kernel's launch costs more than the skipped rows save (measured on the 2^20 workload).
constexpr int64_t kPruneMinDim = int64_t(1) << 22;
bool can_prune(int r, uint32_t c, int64_t d) { return is_pow2(c) && r >= 3 && r <= GS_MAX_ROWS && d >= kPruneMinDim; }

cudaError_t launch_query(const QueryParams& p, cudaStream_t s) {
  using T = QueryTable<1, 2, 3, 4, 5, 6, 7, 8, 9, 10, 11, 12, 13, 14, 15, 16>;
  if (is_pow2(p.c) && p.r >= 1 && p.r <= GS_MAX_ROWS) return T::table[p.r - 1](p, s);
  launch(k_query_generic, persistent_grid(k_query_generic, p.d, kBlock), kBlock, s, p);
  return cudaGetLastError();
}

QueryParams make_query_params(const float* merged, const HashCoeffs& h, int r, uint32_t c, int64_t d,
                              int64_t k, float* est, uint32_t* hist, SelectState* st) {
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
  qp.vec = (reinterpret_cast<uintptr_t>(est) & 15u) == 0 ? 1 : 0;
  qp.hist_on = 1;
  qp.prune = 0;
  qp.keys = nullptr;
  qp.theta = nullptr;
  qp.fill_seed = 0;
  qp.h = h;
  return qp;
}

// Layout of the caller's workspace for the candidate pipeline.
struct Workspace {
  float* est;         // d
  uint32_t* hist;     // 5 * kBins: levels 1-3, level 1 again for k_repair, the sample's level 1
  SelectState* st;
  uint2* cand;        // d (index, key) pairs: room for every coordinate
  uint32_t* gt_bm;    // nbw words
  uint32_t* eq_bm;    // nbw words
  uint32_t* blk;      // 4 * nblk
  int64_t nbw, nblk;
};

Workspace carve(void* base, int64_t d) {
  Workspace w;
  char* p = static_cast<char*>(base);
  w.nbw = (d + 31) / 32;
  w.nblk = (w.nbw + kBmWords - 1) / kBmWords;
  w.est = reinterpret_cast<float*>(p);
  p += align256((size_t)d * sizeof(float));
  w.hist = reinterpret_cast<uint32_t*>(p);
  p += align256(5 * kBins * sizeof(uint32_t));
  w.st = reinterpret_cast<SelectState*>(p);
  p += align256(sizeof(SelectState));
  w.cand = reinterpret_cast<uint2*>(p);
  p += align256((size_t)d * sizeof(uint2));
  w.gt_bm = reinterpret_cast<uint32_t*>(p);
  p += align256((size_t)w.nbw * sizeof(uint32_t));
  w.eq_bm = reinterpret_cast<uint32_t*>(p);
  p += align256((size_t)w.nbw * sizeof(uint32_t));
  w.blk = reinterpret_cast<uint32_t*>(p);
  return w;
}

}  // namespace

size_t query_topk_workspace_bytes(int64_t d, int64_t k) {
  (void)k;
  const int64_t nbw = (d + 31) / 32;
  const int64_t nblk = (nbw + kBmWords - 1) / kBmWords;
  return align256((size_t)d * sizeof(float)) + align256(5 * kBins * sizeof(uint32_t)) +
         align256(sizeof(SelectState)) + align256((size_t)d * sizeof(uint2)) +
         2 * align256((size_t)nbw * sizeof(uint32_t)) + align256((size_t)nblk * 4 * sizeof(uint32_t));
}

namespace {

// Records marks[i] on s when the caller passed marks and set that entry (while a plan is captured).
cudaError_t mark(const cudaEvent_t* marks, int i, cudaStream_t s) {
  return (marks && marks[i]) ? cudaEventRecordWithFlags(marks[i], s, cudaEventRecordExternal) : cudaSuccess;
}

// Histograms, state and both bitmaps back to zero.
cudaError_t clear_selection(const Workspace& w, cudaStream_t s) {
  cudaError_t err = cudaMemsetAsync(w.hist, 0, 5 * kBins * sizeof(uint32_t), s);
  if (err == cudaSuccess) err = cudaMemsetAsync(w.st, 0, sizeof(SelectState), s);
  // the two bitmaps are adjacent: clear both at once
  if (err == cudaSuccess)
    err = cudaMemsetAsync(w.gt_bm, 0, (size_t)(reinterpret_cast<char*>(w.blk) - reinterpret_cast<char*>(w.gt_bm)), s);
  return err;
}

// Levels 2 and 3 and the ordered output, after the level-1 histogram and pick of `src` keys.
cudaError_t select_from_keys(const Workspace& w, const float* src, int vec, uint32_t kmask, int64_t d, int64_t k,
                             int64_t* idx_out, cudaStream_t s) {
  launch(k_cand, persistent_grid(k_cand, (d + 3) / 4 / kU, kBlock), kBlock, s, src, d, vec, kmask, w.st,
                                                                                 w.hist + kBins, w.cand, w.gt_bm);
  const int small_grid = device_info().sms;
  launch(k_cand_hist3, small_grid, kBlock, s, w.cand, w.st, w.hist + 2 * kBins);
  launch(k_cand_mark, small_grid, kBlock, s, w.cand, w.st, w.gt_bm, w.eq_bm);
  uint32_t* blk_gt = w.blk;
  uint32_t* blk_eq = blk_gt + w.nblk;
  uint32_t* blk_base = blk_eq + w.nblk;
  uint32_t* blk_eqx = blk_base + w.nblk;
  const int nb = (int)w.nblk;
  launch(k_bm_count, nb, kBmThreads, s, w.gt_bm, w.eq_bm, w.nbw, blk_gt, blk_eq);
  launch(k_scan, 1, kScanThreads, s, blk_gt, blk_eq, w.nblk, w.st, blk_base, blk_eqx);
  launch(k_bm_write, nb, kBmThreads, s, w.gt_bm, w.eq_bm, w.nbw, w.st, blk_base, blk_eqx, idx_out, k);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_query_topk(const float* merged, const HashCoeffs& h, int r, uint32_t c,
                              int64_t d, int64_t k, int64_t* idx_out, float* est_out,
                              void* workspace, cudaStream_t s, const cudaEvent_t* marks) {
  Workspace w = carve(workspace, d);
  float* est = est_out ? est_out : w.est;
  cudaError_t err = clear_selection(w, s);
  if (err != cudaSuccess) return err;
  if ((err = mark(marks, 0, s)) != cudaSuccess) return err;

  QueryParams qp = make_query_params(merged, h, r, c, d, k, est, w.hist, w.st);
  // rows are pruned only while the estimate stays internal: a caller's est_out gets every value
  const uint32_t j_target = sample_rank(d, k);
  qp.prune = (!est_out && can_prune(r, c, d) && j_target > 0) ? 1 : 0;
  if (qp.prune) {
    using T = SampleTable<1, 2, 3, 4, 5, 6, 7, 8, 9, 10, 11, 12, 13, 14, 15, 16>;
    if ((err = T::table[r - 1](qp, w.hist + 4 * kBins, j_target, s)) != cudaSuccess) return err;
  }
  if (qp.prune && query_uses_bits(r, c)) {
    // the classes go in the candidate area, which the selection only uses after the query
    using T = BitsTable<1, 2, 3, 4, 5, 6, 7, 8, 9, 10, 11, 12, 13, 14, 15, 16>;
    if ((err = T::table[r - 1](qp, reinterpret_cast<uint32_t*>(w.cand), s)) != cudaSuccess) return err;
  } else if ((err = launch_query(qp, s)) != cudaSuccess) {
    return err;
  }
  if (qp.prune) {
    using T = RepairTable<1, 2, 3, 4, 5, 6, 7, 8, 9, 10, 11, 12, 13, 14, 15, 16>;
    if ((err = T::table[r - 1](qp, w.hist + 3 * kBins, s)) != cudaSuccess) return err;
  }
  if ((err = mark(marks, 1, s)) != cudaSuccess) return err;
  if ((err = select_from_keys(w, est, qp.vec, 0x7FFFFFFFu, d, k, idx_out, s)) != cudaSuccess) return err;
  return mark(marks, 2, s);
}

cudaError_t launch_query_ceiling_probe(const float* merged, const HashCoeffs& h, int r, uint32_t c, int64_t d,
                                       float* out, int64_t out_floats, cudaStream_t s) {
  if (!is_pow2(c) || r < 1 || r > GS_MAX_ROWS) return cudaErrorInvalidValue;
  const QueryParams qp = make_query_params(merged, h, r, c, d, 1, nullptr, nullptr, nullptr);
  using T = ProbeTable<1, 2, 3, 4, 5, 6, 7, 8, 9, 10, 11, 12, 13, 14, 15, 16>;
  return T::table[r - 1](qp, out, out_floats, s);
}

size_t heavymix_workspace_bytes(int64_t d, int64_t k) {
  return query_topk_workspace_bytes(d, k) + align256((size_t)d * sizeof(uint32_t)) + 256;
}

cudaError_t launch_query_heavymix(const float* merged, const HashCoeffs& h, int r, uint32_t c, int64_t d,
                                  int64_t k, uint64_t fill_seed, int64_t* idx_out, float* est_out, double* l2sq_out,
                                  void* workspace, cudaStream_t s, const cudaEvent_t* marks) {
  Workspace w = carve(workspace, d);
  char* extra = static_cast<char*>(workspace) + query_topk_workspace_bytes(d, k);
  uint32_t* keys = reinterpret_cast<uint32_t*>(extra);
  double* sumsq = reinterpret_cast<double*>(extra + align256((size_t)d * sizeof(uint32_t)));
  double* theta = sumsq + GS_MAX_ROWS;
  float* est = est_out ? est_out : w.est;
  cudaError_t err = clear_selection(w, s);
  if (err == cudaSuccess) err = cudaMemsetAsync(sumsq, 0, 256, s);
  if (err == cudaSuccess) err = mark(marks, 0, s);
  if (err != cudaSuccess) return err;

  // the threshold first (it reads only the table), so that the query can skip rows below it
  const int gx = (int)(((int64_t)c + kBlock - 1) / kBlock < 4 * device_info().sms ? ((int64_t)c + kBlock - 1) / kBlock
                                                                                  : 4 * device_info().sms);
  launch(k_row_sumsq, dim3(gx, r), kBlock, s, merged, c, sumsq);
  const int prune = (!est_out && can_prune(r, c, d)) ? 1 : 0;
  launch(k_heavy_theta, 1, 32, s, sumsq, r, k, theta, l2sq_out, w.st, prune);
  // the query stores each coordinate's composite key and picks on their level-1 histogram
  QueryParams qp = make_query_params(merged, h, r, c, d, k, est, w.hist, w.st);
  qp.prune = prune;
  qp.keys = keys;
  qp.theta = theta;
  qp.fill_seed = fill_seed;
  if ((err = launch_query(qp, s)) != cudaSuccess) return err;
  if ((err = mark(marks, 1, s)) != cudaSuccess) return err;
  if ((err = select_from_keys(w, reinterpret_cast<const float*>(keys), 1, 0xFFFFFFFFu, d, k, idx_out, s)) !=
      cudaSuccess)
    return err;
  return mark(marks, 2, s);
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

// Unique id of the context current on this thread (0 when none is current or the driver's
// entry points are unavailable).  A device reset or a rebuilt primary context gets a new id
// and a new load of this library's module, hence a new address of g_noalloc_scratch.  The
// two driver calls are reached through the runtime's entry-point query, so the library does
// not link the driver library itself.
unsigned long long current_context_id() {
  typedef CUresult (*GetCurrent)(CUcontext*);
  typedef CUresult (*GetId)(CUcontext, unsigned long long*);
  static GetCurrent get_current = nullptr;
  static GetId get_id = nullptr;
  static bool looked_up = false;
  if (!looked_up) {
    looked_up = true;
    void* f1 = nullptr;
    void* f2 = nullptr;
    cudaDriverEntryPointQueryResult q1, q2;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &f1, 12000, cudaEnableDefault, &q1) == cudaSuccess &&
        cudaGetDriverEntryPointByVersion("cuCtxGetId", &f2, 12000, cudaEnableDefault, &q2) == cudaSuccess &&
        q1 == cudaDriverEntryPointSuccess && q2 == cudaDriverEntryPointSuccess) {
      get_current = reinterpret_cast<GetCurrent>(f1);
      get_id = reinterpret_cast<GetId>(f2);
    }
    cudaGetLastError();
  }
  if (!get_current || !get_id) return 0;
  CUcontext ctx = nullptr;
  unsigned long long id = 0;
  if (get_current(&ctx) != CUDA_SUCCESS || !ctx || get_id(ctx, &id) != CUDA_SUCCESS) return 0;
  return id;
}

// Device address of g_noalloc_scratch on the current device.  It is looked up once per
// device and context (cudaGetSymbolAddress, a host-side query that allocates nothing) and
// cached under the context's id, so a reset device gets a fresh lookup.  Without a readable
// id the lookup runs on every call.
cudaError_t noalloc_scratch(void** out) {
  struct Entry {
    unsigned long long ctx;
    void* addr;
  };
  static std::mutex mu;
  static Entry cache[64] = {};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(mu);
  unsigned long long ctx = current_context_id();
  if (ctx != 0 && cache[dev].ctx == ctx && cache[dev].addr) {
    *out = cache[dev].addr;
    return cudaSuccess;
  }
  void* p = nullptr;
  e = cudaGetSymbolAddress(&p, g_noalloc_scratch);  // also makes the device's context current
  if (e != cudaSuccess) return e;
  if (ctx == 0) ctx = current_context_id();
  cache[dev].ctx = ctx;
  cache[dev].addr = ctx ? p : nullptr;
  *out = p;
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
  const int64_t nseg = (d + kSeg - 1) / kSeg;
  uint32_t* blk_gt = reinterpret_cast<uint32_t*>(p + kNoallocHistBytes + kNoallocStateBytes);
  uint32_t* blk_eq = blk_gt + nseg;
  uint32_t* blk_base = blk_eq + nseg;
  uint32_t* blk_eqx = blk_base + nseg;
  // the histograms and the state must start at zero; the segment counters are overwritten
  err = cudaMemsetAsync(hist, 0, kNoallocHistBytes, s);
  if (err == cudaSuccess) err = cudaMemsetAsync(st, 0, sizeof(SelectState), s);
  if (err != cudaSuccess) return err;

  const QueryParams qp = make_query_params(merged, h, r, c, d, k, est_out, hist, st);
  if ((err = launch_query(qp, s)) != cudaSuccess) return err;
  const int hgrid = persistent_grid(k_hist, (d + 3) / 4 / kU, kBlock);
  launch(k_hist, hgrid, kBlock, s, est_out, d, qp.vec, st, hist + kBins, kL2Shift, 11, 1);
  launch(k_hist, hgrid, kBlock, s, est_out, d, qp.vec, st, hist + 2 * kBins, 0, kL3Bits, 2);
  const int nb = (int)nseg;
  if (qp.vec) launch(k_count<true>, nb, kSegThreads, s, est_out, d, st, blk_gt, blk_eq);
  else launch(k_count<false>, nb, kSegThreads, s, est_out, d, st, blk_gt, blk_eq);
  launch(k_scan, 1, kScanThreads, s, blk_gt, blk_eq, nseg, st, blk_base, blk_eqx);
  if (qp.vec) launch(k_write<true>, nb, kSegThreads, s, est_out, d, st, blk_base, blk_eqx, idx_out, k);
  else launch(k_write<false>, nb, kSegThreads, s, est_out, d, st, blk_base, blk_eqx, idx_out, k);
  return cudaGetLastError();
}

}  // namespace gs
