// Internal declarations shared by the translation units of the gs-SGD compression library.
// Device-side Count Sketch hashing over the Mersenne prime 2^61 - 1, kernel parameter
// blocks and the host-side launcher entry points called by the C ABI in gs_api.cu.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "gs_sketch.h"

#include <utility>

namespace gs {

constexpr uint64_t kP61 = (1ull << 61) - 1;
constexpr int kMaxGroup = 16;       // widest worker group interleaved in one table
constexpr int kBlock = 256;         // threads per CTA for the streaming kernels

// Hash coefficients of every row: h_j uses (a[j], b[j]); s_j uses (a2[j], b2[j]).
struct HashCoeffs {
  uint64_t a[GS_MAX_ROWS], b[GS_MAX_ROWS], a2[GS_MAX_ROWS], b2[GS_MAX_ROWS];
};

// ---- Mersenne-prime arithmetic ----------------------------------------------------------
// x mod p is congruent to (x & p) + (x >> 61) because 2^61 = 1 (mod p).
__device__ __forceinline__ uint64_t fold61(uint64_t x) { return (x & kP61) + (x >> 61); }

// (a*i + b) mod p for a, b < p and i < 2^32.  a is split into 32-bit halves:
//   a*i = ahi*i*2^32 + alo*i,  and  ahi*i*2^32 = q*2^61 + rem*2^32 = q + rem*2^32 (mod p)
// with q = (ahi*i) >> 29 and rem = (ahi*i) mod 2^29.  Every partial sum stays below 2^63.
__device__ __forceinline__ uint64_t affine61(uint64_t a, uint64_t b, uint32_t i) {
  const uint64_t p0 = (uint64_t)(uint32_t)a * i;          // < 2^64
  const uint64_t p1 = (uint64_t)(uint32_t)(a >> 32) * i;  // < 2^61
  uint64_t s = (p1 >> 29) + ((p1 & ((1ull << 29) - 1)) << 32) + fold61(p0) + b;
  s = fold61(s);                                          // < p + 4
  return s >= kP61 ? s - kP61 : s;
}

// x + a mod p for x, a < p: the next coordinate's hash value in the incremental form
// (a*(i+1) + b) = (a*i + b) + a.
__device__ __forceinline__ uint64_t step61(uint64_t x, uint64_t a) {
  x += a;
  return x >= kP61 ? x - kP61 : x;
}

template <bool POW2>
__device__ __forceinline__ uint32_t bucket_of(uint64_t x, uint32_t c, uint32_t cmask) {
  if (POW2) return (uint32_t)x & cmask;
  return (uint32_t)(x % (uint64_t)c);
}

// Sign bit (bit 31 set for s = -1): s_j(i) = -1 when the second hash value is odd.
__device__ __forceinline__ uint32_t signbit_of(uint64_t y) { return ((uint32_t)y & 1u) << 31; }

__device__ __forceinline__ float apply_sign(float v, uint32_t sbit) {
  return __uint_as_float(__float_as_uint(v) ^ sbit);
}

// ---- fp32 reductions into L2-resident tables -------------------------------------------
__device__ __forceinline__ void red_add_f32(float* p, float v) {
  asm volatile("red.global.add.f32 [%0], %1;" ::"l"(p), "f"(v) : "memory");
}
__device__ __forceinline__ void red_add_v2(float* p, float v0, float v1) {
  asm volatile("red.global.add.v2.f32 [%0], {%1, %2};" ::"l"(p), "f"(v0), "f"(v1) : "memory");
}
__device__ __forceinline__ void red_add_v4(float* p, float v0, float v1, float v2, float v3) {
  asm volatile("red.global.add.v4.f32 [%0], {%1, %2, %3, %4};" ::"l"(p), "f"(v0), "f"(v1),
               "f"(v2), "f"(v3)
               : "memory");
}

// ---- L2 eviction priorities -------------------------------------------------------------
// Cache policies for the fused insert: its vector streams are read or written once
// (evict_first, not allocated in L1), while the sketch table receives every reduction and
// should stay in L2 (evict_last).  Measured on the BERT-large-sized table (64 MiB row slices
// next to 8 workers' streams): one group's five row passes 21.9 ms with these policies against
// 25.0 ms without; neutral at the other sizes.
__device__ __forceinline__ uint64_t policy_evict_first() {
  uint64_t pol;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
  return pol;
}
__device__ __forceinline__ uint64_t policy_evict_last() {
  uint64_t pol;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(pol));
  return pol;
}
__device__ __forceinline__ float4 ld_stream(const float* p, uint64_t pol) {
  float4 v;
  asm volatile("ld.global.L1::no_allocate.L2::cache_hint.v4.f32 {%0, %1, %2, %3}, [%4], %5;"
               : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
               : "l"(p), "l"(pol));
  return v;
}
__device__ __forceinline__ void st_stream(float* p, float4 v, uint64_t pol) {
  asm volatile("st.global.L1::no_allocate.L2::cache_hint.v4.f32 [%0], {%1, %2, %3, %4}, %5;" ::"l"(p), "f"(v.x),
               "f"(v.y), "f"(v.z), "f"(v.w), "l"(pol)
               : "memory");
}
__device__ __forceinline__ void red_add_v4_keep(float* p, float v0, float v1, float v2, float v3, uint64_t pol) {
  asm volatile("red.global.add.L2::cache_hint.v4.f32 [%0], {%1, %2, %3, %4}, %5;" ::"l"(p), "f"(v0), "f"(v1),
               "f"(v2), "f"(v3), "l"(pol)
               : "memory");
}

// ---- parameter blocks --------------------------------------------------------------------
struct InsertParams {
  float* u[kMaxGroup];
  float* e[kMaxGroup];
  const float* g[kMaxGroup];
  float* table;      // base of the group's interleaved table [r][c][W]
  int64_t d;
  int32_t nw;        // lanes of the group carrying a worker in this call
  int32_t lane;      // single-vector insert: the lane written
  int32_t r;
  int32_t j0, j1;    // rows inserted by this launch: [j0, j1)
  uint32_t c, cmask;
  float rho;
  int64_t winmask;   // request-ceiling probe only: vector offsets are taken modulo winmask + 1
  HashCoeffs h;
};

struct MergeParams {
  const float* tables;   // all groups, [group][r][c][W]
  float* merged;         // [r][c]
  int64_t cells;         // r*c
  int64_t group_stride;  // r*c*W floats
  int32_t P;
};

struct MergeListParams {
  const float* tables[GS_MAX_WORKERS];   // worker 0's table of each sketch, [r][c][lane_stride]
  int32_t lane_stride[GS_MAX_WORKERS];
  float* merged;                          // [r][c]
  int64_t cells;
  int32_t P;
};

struct GatherParams {
  float* u[GS_MAX_WORKERS];
  float* e[GS_MAX_WORKERS];
  const int64_t* idx;
  float* vals;
  float* w;          // weights to update with the gathered values (nullable)
  float lr;
  int64_t k, d;
  int32_t P;
};

// ---- launchers (return a cudaError_t from the launch) ------------------------------------
struct DeviceInfo {
  int sms;
};
DeviceInfo device_info();
// Resident CTAs per SM for `kernel` at `block` threads (cached per kernel address).
int blocks_per_sm(const void* kernel, int block);

cudaError_t launch_accumulate(float* u, float* e, const float* g, int64_t d, float rho,
                              cudaStream_t s);
// acc: accumulate (read g, u, e; write u, e) before inserting; otherwise insert e as it is.
cudaError_t launch_accumulate_insert(const InsertParams& p, int W, bool acc, bool vec, cudaStream_t s);
cudaError_t launch_insert_lane(const InsertParams& p, int W, cudaStream_t s);
// The fused insert's instruction stream with every vector access at offset i & p.winmask (the
// vectors are windows of winmask + 1 floats, 16-byte aligned): the same loads, stores and
// cell reductions, with the streams held in L2.  W in {4, 8, 16}, c a power of two.
cudaError_t launch_insert_ceiling_probe(const InsertParams& p, int W, bool acc, cudaStream_t s);
// Shared-memory-staged insert of the (already accumulated) vectors p.e[0..nw) into rows
// [j0, j1) of a W-wide group table; needs a tile of c * wt * 4 bytes (staged_tile_width).
constexpr size_t kStagedSmemBytes = size_t(200) << 10;
int staged_tile_width(uint32_t c, int W);   // workers per tile, 0 when no tile fits
cudaError_t launch_insert_staged(const InsertParams& p, int W, cudaStream_t s);
cudaError_t launch_hash_eval(const HashCoeffs& h, int r, uint32_t c, const int64_t* coords,
                             int64_t n, int32_t* bucket_out, int8_t* sign_out, cudaStream_t s);
cudaError_t launch_merge(const MergeParams& p, int W, cudaStream_t s);
cudaError_t launch_merge_list(const MergeListParams& p, cudaStream_t s);
cudaError_t launch_gather_and_zero(const GatherParams& p, cudaStream_t s);
cudaError_t launch_apply_update(float* w, int64_t d, const int64_t* idx, const float* vals, int64_t k, float lr,
                                cudaStream_t s);

size_t query_topk_workspace_bytes(int64_t d, int64_t k);

// momentum and error kept as sketches
cudaError_t launch_query_at(const float* T, const HashCoeffs& h, int r, uint32_t c, const int64_t* idx, int64_t k,
                            float* out, cudaStream_t s);
cudaError_t launch_add_sparse(float* T, const HashCoeffs& h, int r, uint32_t c, const int64_t* idx, const float* vals,
                              int64_t k, float scale, cudaStream_t s);
cudaError_t launch_take(const float* src, int64_t n, const int64_t* idx, int64_t k, float* out, cudaStream_t s);
// marks (nullable): three events recorded, when set, before the query, between the query
// (sample, median query, repair check) and the selection, and after the selection.
cudaError_t launch_query_topk(const float* merged, const HashCoeffs& h, int r, uint32_t c,
                              int64_t d, int64_t k, int64_t* idx_out, float* est_out,
                              void* workspace, cudaStream_t s, const cudaEvent_t* marks = nullptr);
// Request-ceiling probe of the median query: its loads (all r rows) without median, store or
// histogram; out receives one float per CTA (out_floats must cover the grid).  c a power of two.
cudaError_t launch_query_ceiling_probe(const float* merged, const HashCoeffs& h, int r, uint32_t c, int64_t d,
                                       float* out, int64_t out_floats, cudaStream_t s);
// HEAVYMIX selection (Alg. 2 as printed) from the merged table; l2sq_out (device double,
// nullable) receives the sketch's estimate of ||g||^2.
size_t heavymix_workspace_bytes(int64_t d, int64_t k);
cudaError_t launch_query_heavymix(const float* merged, const HashCoeffs& h, int r, uint32_t c, int64_t d,
                                  int64_t k, uint64_t fill_seed, int64_t* idx_out, float* est_out, double* l2sq_out,
                                  void* workspace, cudaStream_t s, const cudaEvent_t* marks = nullptr);

// Same pipeline with its scratch in a fixed device array (no allocation); est_out required,
// d <= GS_NOALLOC_MAX_DIM.  The first call on a device looks up the array's address.
cudaError_t launch_query_topk_noalloc(const float* merged, const HashCoeffs& h, int r, uint32_t c,
                                      int64_t d, int64_t k, int64_t* idx_out, float* est_out,
                                      cudaStream_t s);

inline bool is_pow2(uint32_t c) { return c && !(c & (c - 1)); }

// ---- launches -----------------------------------------------------------------------
// Every kernel of the library is launched with programmatic stream serialization (sm_90+):
// the next kernel in the stream may be scheduled before this one has finished, and it begins
// with grid_begin(), which waits until the grids it depends on have completed and their
// memory is visible (griddepcontrol.wait), then lets its own successor be scheduled
// (griddepcontrol.launch_dependents).  Launch latency and the ramp of the next grid overlap
// the tail of the previous one; no kernel touches memory before its wait.  A kernel launched
// after a memset, an event record or another library's kernel simply finds its wait satisfied.
__device__ __forceinline__ void grid_begin() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

template <typename... KArgs, typename... Args>
inline cudaError_t launch(void (*kernel)(KArgs...), dim3 grid, dim3 block, cudaStream_t s, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = 0;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

}  // namespace gs
