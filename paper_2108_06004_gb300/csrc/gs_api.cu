// C ABI of the gs-SGD compression library: argument validation, the sketch object, hash
// coefficient derivation, and composition of the kernels into the calls of gs_sketch.h.
#include <cstring>
#include <mutex>
#include <new>
#include <string>
#include <unordered_map>
#include <vector>

#include "gs_common.cuh"

struct gs_sketch {
  int32_t r, c, workers, W, groups;
  int32_t rows_per_pass;  // rows inserted per pass of the fused kernel (table slice <= L2 budget)
  uint64_t seed;
  gs::HashCoeffs h;
  float* tables;  // groups * r*c*W
  float* merged;  // r*c
  int device;
};

// Events recorded between the phases of a step while it is captured into a plan, where each
// becomes an event-record node of the graph: the insert phase, the query (sample, median
// query and repair check) and the selection that follows it.
enum PhaseMark { kInsertBegin, kInsertEnd, kQueryBegin, kQueryEnd, kSelectEnd, kMarks };

struct gs_plan {
  cudaGraph_t graph = nullptr;
  cudaGraphExec_t exec = nullptr;
  int32_t flags = 0;
  cudaGraphNode_t node[kMarks] = {};     // the event-record nodes of the marks in use
  std::vector<cudaEvent_t> ev[kMarks];   // their rings of events
  int64_t launches = 0;
  int device = 0;
};

namespace {

thread_local std::string g_err;

// Record the message of a failing call; a message that cannot be stored is dropped, so that
// the status still reaches the caller.
gs_status fail(gs_status st, const char* msg) noexcept {
  try {
    g_err = msg;
  } catch (...) {
    g_err.clear();
  }
  return st;
}

gs_status fail(gs_status st, const std::string& msg) noexcept { return fail(st, msg.c_str()); }

gs_status cuda_fail(cudaError_t e, const char* what) noexcept {
  try {
    g_err = std::string(what) + ": " + cudaGetErrorString(e);
  } catch (...) {
    g_err.clear();
  }
  return GS_ERR_CUDA;
}

gs_status ok() {
  return GS_OK;
}

// splitmix64 (Steele, Lea and Flood, OOPSLA 2014): advance the state by the golden-ratio
// increment and mix it with two xor-shift-multiply rounds.
uint64_t splitmix64_next(uint64_t& state) {
  state += 0x9E3779B97F4A7C15ull;
  uint64_t z = state;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

void derive_coefficients(int r, uint64_t seed, gs::HashCoeffs& h) {
  std::memset(&h, 0, sizeof(h));
  uint64_t state = seed;
  for (int j = 0; j < r; ++j) {
    h.a[j] = 1 + splitmix64_next(state) % (gs::kP61 - 1);
    h.b[j] = splitmix64_next(state) % gs::kP61;
    h.a2[j] = 1 + splitmix64_next(state) % (gs::kP61 - 1);
    h.b2[j] = splitmix64_next(state) % gs::kP61;
  }
}

// L2 budgets (GB300: 126 MB of L2 in two halves).  A group's table row must fit kRowBudget,
// else the group is narrowed; one insert pass updates at most kPassBudget of table, so that
// the slice stays resident in L2 while g, u and e stream past it.  Measured on the VGG-16 and
// BERT-large workloads: a 64 MB slice per pass is slower than a 32 MB one (L2 contention),
// and 96 MB thrashes; 8-wide groups with one 64 MB row per pass beat 4-wide groups.
constexpr size_t kRowBudget = size_t(64) << 20;
constexpr size_t kPassBudget = size_t(48) << 20;

// Widest group (up to 16, not wider than the worker count rounded up to a power of two) whose
// single table row fits the row budget.  16-wide groups are used only when the whole group
// table fits one pass: their 64-byte cells halve the reduction requests, but a 16-wide table
// that needs row passes re-reads e more often than two 8-wide groups do (measured slower).
int choose_group_width(int r, int c, int workers) {
  int W = 1;
  while (W < workers && W < gs::kMaxGroup) W *= 2;
  if (W == 16 && (size_t)r * (size_t)c * 16 * sizeof(float) > kPassBudget) W = 8;
  while (W > 1 && (size_t)c * (size_t)W * sizeof(float) > kRowBudget) W /= 2;
  return W;
}

int choose_rows_per_pass(int r, int c, int W) {
  const size_t row_bytes = (size_t)c * (size_t)W * sizeof(float);
  size_t n = kPassBudget / row_bytes;
  if (n < 1) n = 1;
  if (n > (size_t)r) n = (size_t)r;
  return (int)n;
}

// The row ranges of one group's insert passes, rows_per_pass rows each; the first pass also
// accumulates.
struct Pass {
  int j0, j1;
};

std::vector<Pass> insert_passes(const gs_sketch* sk) {
  std::vector<Pass> out;
  for (int j0 = 0; j0 < sk->r; j0 += sk->rows_per_pass)
    out.push_back({j0, (j0 + sk->rows_per_pass < sk->r) ? j0 + sk->rows_per_pass : sk->r});
  return out;
}

bool aligned(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) & (a - 1)) == 0; }

gs_status check_sketch(const gs_sketch* sk) {
  if (!sk) return fail(GS_ERR_INVALID_ARG, "sketch is NULL");
  int dev = -1;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
  if (dev != sk->device)
    return fail(GS_ERR_INVALID_ARG, "current device " + std::to_string(dev) +
                                        " differs from the sketch's device " + std::to_string(sk->device));
  return GS_OK;
}

gs_status check_d(int64_t d) {
  if (d < 1 || d > GS_MAX_DIM) return fail(GS_ERR_INVALID_ARG, "d must lie in [1, 2^31 - 1], got " + std::to_string(d));
  return GS_OK;
}

gs_status check_vec(const void* p, const char* name) {
  if (!p) return fail(GS_ERR_INVALID_ARG, std::string(name) + " is NULL");
  if (!aligned(p, 4)) return fail(GS_ERR_INVALID_ARG, std::string(name) + " is not 4-byte aligned");
  return GS_OK;
}

#define GS_TRY(expr)                  \
  do {                                \
    const gs_status st__ = (expr);    \
    if (st__ != GS_OK) return st__;   \
  } while (0)

#define GS_GUARD_BEGIN try {
#define GS_GUARD_END                                                  \
  }                                                                   \
  catch (const std::bad_alloc&) {                                     \
    return fail(GS_ERR_OOM, "host allocation failed");                \
  }                                                                   \
  catch (...) {                                                       \
    return fail(GS_ERR_INVALID_ARG, "unexpected host exception");     \
  }

cudaStream_t as_stream(gs_stream s) { return reinterpret_cast<cudaStream_t>(s); }

gs_status accumulate_insert_impl(gs_sketch* sk, int32_t first, int32_t n, float* const* m,
                                 float* const* e, const float* const* g, int64_t d, float rho,
                                 cudaStream_t s) {
  const int W = sk->W;
  const int end = first + n;
  for (int grp = first / W; grp * W < end; ++grp) {
    gs::InsertParams p;
    std::memset(&p, 0, sizeof(p));
    const int lo = grp * W;
    const int nw = (end - lo) < W ? (end - lo) : W;
    bool vec = true;
    for (int w = 0; w < nw; ++w) {
      const int a = lo + w - first;
      p.u[w] = m[a];
      p.e[w] = e[a];
      p.g[w] = g[a];
      vec = vec && aligned(m[a], 16) && aligned(e[a], 16) && aligned(g[a], 16);
    }
    p.table = sk->tables + (size_t)grp * sk->r * sk->c * W;
    p.d = d;
    p.nw = nw;
    p.r = sk->r;
    p.c = (uint32_t)sk->c;
    p.cmask = (uint32_t)sk->c - 1;
    p.rho = rho;
    p.h = sk->h;
    // first pass: accumulate and insert the first slice; later passes insert the remaining
    // slices from the updated error vectors
    bool first = true;
    for (const Pass& ps : insert_passes(sk)) {
      p.j0 = ps.j0;
      p.j1 = ps.j1;
      cudaError_t err = gs::launch_accumulate_insert(p, W, first, vec, s);
      if (err != cudaSuccess) return cuda_fail(err, "accumulate_insert launch");
      first = false;
    }
  }
  return GS_OK;
}

// Insert the vectors vec[p] (no accumulation) into the worker tables, all groups and passes.
gs_status insert_all_impl(gs_sketch* sk, const float* const* vec, int64_t d, cudaStream_t s) {
  const int W = sk->W;
  for (int grp = 0; grp * W < sk->workers; ++grp) {
    gs::InsertParams p;
    std::memset(&p, 0, sizeof(p));
    const int lo = grp * W;
    const int nw = (sk->workers - lo) < W ? (sk->workers - lo) : W;
    bool vec_ok = true;
    for (int w = 0; w < nw; ++w) {
      p.e[w] = const_cast<float*>(vec[lo + w]);
      vec_ok = vec_ok && aligned(vec[lo + w], 16);
    }
    p.table = sk->tables + (size_t)grp * sk->r * sk->c * W;
    p.d = d;
    p.nw = nw;
    p.r = sk->r;
    p.c = (uint32_t)sk->c;
    p.cmask = (uint32_t)sk->c - 1;
    p.h = sk->h;
    for (const Pass& ps : insert_passes(sk)) {
      p.j0 = ps.j0;
      p.j1 = ps.j1;
      cudaError_t err = gs::launch_accumulate_insert(p, W, false, vec_ok, s);
      if (err != cudaSuccess) return cuda_fail(err, "insert launch");
    }
  }
  return GS_OK;
}

bool same_family(const gs_sketch* a, const gs_sketch* b) {
  return a->r == b->r && a->c == b->c && a->seed == b->seed;
}

// Optional events recorded between the phases of a step (unset entries record nothing).  They
// are used only while a step is captured into a plan.
struct InsertMarks {
  cudaEvent_t ev[kMarks] = {};
};

cudaError_t mark(cudaEvent_t ev, cudaStream_t s) {
  return ev ? cudaEventRecordWithFlags(ev, s, cudaEventRecordExternal) : cudaSuccess;
}

// The selection of a step: the deterministic top-k (default), or HEAVYMIX (Alg. 2 as printed).
struct Selection {
  bool heavymix = false;
  uint64_t fill_seed = 0;
  double* l2sq_out = nullptr;
};

gs_status step_impl(gs_sketch* sk, float* const* m, float* const* e, const float* const* g,
                    int64_t d, float rho, int64_t k, int64_t* idx, float* vals, float* est,
                    void* ws, cudaStream_t s, float* weights = nullptr, float lr = 0.f,
                    InsertMarks marks = InsertMarks(), Selection sel = Selection()) {
  const size_t bytes = (size_t)sk->groups * sk->r * sk->c * sk->W * sizeof(float) +
                       (size_t)sk->r * sk->c * sizeof(float);
  cudaError_t err = cudaMemsetAsync(sk->tables, 0, bytes, s);
  if (err != cudaSuccess) return cuda_fail(err, "zero tables");
  if ((err = mark(marks.ev[kInsertBegin], s)) != cudaSuccess) return cuda_fail(err, "event record");
  GS_TRY(accumulate_insert_impl(sk, 0, sk->workers, m, e, g, d, rho, s));
  if ((err = mark(marks.ev[kInsertEnd], s)) != cudaSuccess) return cuda_fail(err, "event record");
  gs::MergeParams mp;
  mp.tables = sk->tables;
  mp.merged = sk->merged;
  mp.cells = (int64_t)sk->r * sk->c;
  mp.group_stride = (int64_t)sk->r * sk->c * sk->W;
  mp.P = sk->workers;
  if ((err = gs::launch_merge(mp, sk->W, s)) != cudaSuccess) return cuda_fail(err, "merge launch");
  if (sel.heavymix) {
    if ((err = gs::launch_query_heavymix(sk->merged, sk->h, sk->r, (uint32_t)sk->c, d, k, sel.fill_seed, idx, est,
                                         sel.l2sq_out, ws, s, &marks.ev[kQueryBegin])) != cudaSuccess)
      return cuda_fail(err, "HEAVYMIX query launch");
  } else if ((err = gs::launch_query_topk(sk->merged, sk->h, sk->r, (uint32_t)sk->c, d, k, idx, est, ws, s,
                                          &marks.ev[kQueryBegin])) != cudaSuccess) {
    return cuda_fail(err, "query/top-k launch");
  }
  gs::GatherParams gp;
  std::memset(&gp, 0, sizeof(gp));
  for (int p = 0; p < sk->workers; ++p) {
    gp.u[p] = m[p];
    gp.e[p] = e[p];
  }
  gp.idx = idx;
  gp.vals = vals;
  gp.w = weights;
  gp.lr = lr;
  gp.k = k;
  gp.d = d;
  gp.P = sk->workers;
  if ((err = gs::launch_gather_and_zero(gp, s)) != cudaSuccess) return cuda_fail(err, "gather launch");
  return GS_OK;
}

gs_status check_worker_arrays(int n, float* const* m, float* const* e, const float* const* g) {
  if (!m || !e) return fail(GS_ERR_INVALID_ARG, "pointer array is NULL");
  for (int w = 0; w < n; ++w) {
    GS_TRY(check_vec(m[w], "momentum[p]"));
    GS_TRY(check_vec(e[w], "error[p]"));
    if (g) GS_TRY(check_vec(g[w], "grad[p]"));
  }
  return GS_OK;
}

size_t step_ws_bytes(int64_t d, int64_t k) {
  return gs::query_topk_workspace_bytes(d, k) + (((size_t)k * 8 + 255) & ~size_t(255)) +
         (((size_t)k * 4 + 255) & ~size_t(255));
}

gs_status check_sketched_state(gs_sketch* workers, gs_sketch* momentum, gs_sketch* error, const float* const* grad,
                               int64_t d, int64_t k, int64_t* idx_out, float* vals_out, float* weights,
                               void* workspace, size_t workspace_bytes) {
  GS_TRY(check_sketch(workers));
  GS_TRY(check_sketch(momentum));
  GS_TRY(check_sketch(error));
  if (!same_family(workers, momentum) || !same_family(workers, error))
    return fail(GS_ERR_MISMATCH, "the three sketches must share r, c and seed");
  if (momentum == error || momentum == workers || error == workers)
    return fail(GS_ERR_INVALID_ARG, "workers, momentum and error must be three different sketches");
  GS_TRY(check_d(d));
  if (k < 1 || k > d) return fail(GS_ERR_INVALID_ARG, "k must lie in [1, d]");
  if (!grad) return fail(GS_ERR_INVALID_ARG, "grad array is NULL");
  for (int p = 0; p < workers->workers; ++p) GS_TRY(check_vec(grad[p], "grad[p]"));
  if (!idx_out || !aligned(idx_out, 8)) return fail(GS_ERR_INVALID_ARG, "idx_out is NULL or not 8-byte aligned");
  GS_TRY(check_vec(vals_out, "vals_out"));
  if (weights) GS_TRY(check_vec(weights, "weights"));
  if (!workspace || !aligned(workspace, 256)) return fail(GS_ERR_INVALID_ARG, "workspace is NULL or not 256-byte aligned");
  if (workspace_bytes < step_ws_bytes(d, k)) return fail(GS_ERR_INVALID_ARG, "workspace too small: use gs_step_workspace_size");
  return GS_OK;
}

// S = tree merge of S(g_p); U <- rho U + S, E <- E + U; top-k of the estimate from E; the
// extracted mass leaves E and U.  Arguments already checked.
gs_status sketched_state_impl(gs_sketch* workers, gs_sketch* momentum, gs_sketch* error, const float* const* grad,
                              int64_t d, float rho, int64_t k, int64_t* idx, float* vals, float* weights, float lr,
                              void* ws, cudaStream_t s, InsertMarks marks = InsertMarks()) {
  const int64_t cells = (int64_t)workers->r * workers->c;
  // S = tree merge of S(g_p)
  const size_t tbytes = ((size_t)workers->groups * workers->r * workers->c * workers->W + (size_t)cells) * sizeof(float);
  cudaError_t err = cudaMemsetAsync(workers->tables, 0, tbytes, s);
  if (err != cudaSuccess) return cuda_fail(err, "zero tables");
  if ((err = mark(marks.ev[kInsertBegin], s)) != cudaSuccess) return cuda_fail(err, "event record");
  GS_TRY(insert_all_impl(workers, grad, d, s));
  if ((err = mark(marks.ev[kInsertEnd], s)) != cudaSuccess) return cuda_fail(err, "event record");
  gs::MergeParams mp;
  mp.tables = workers->tables;
  mp.merged = workers->merged;
  mp.cells = cells;
  mp.group_stride = cells * workers->W;
  mp.P = workers->workers;
  if ((err = gs::launch_merge(mp, workers->W, s)) != cudaSuccess) return cuda_fail(err, "merge launch");
  // U <- rho U + S ; E <- E + U   (elementwise on the r*c cells)
  if ((err = gs::launch_accumulate(momentum->merged, error->merged, workers->merged, cells, rho, s)) != cudaSuccess)
    return cuda_fail(err, "sketch accumulate launch");
  // top-k of the estimate from E; delta = that estimate at the selected coordinates
  if ((err = gs::launch_query_topk(error->merged, error->h, error->r, (uint32_t)error->c, d, k, idx, nullptr,
                                   ws, s, &marks.ev[kQueryBegin])) != cudaSuccess)
    return cuda_fail(err, "query/top-k launch");
  const float* est = static_cast<const float*>(ws);  // the query keeps est at the ws start
  if ((err = gs::launch_take(est, d, idx, k, vals, s)) != cudaSuccess) return cuda_fail(err, "take launch");
  float* delta_u = reinterpret_cast<float*>(static_cast<char*>(ws) + gs::query_topk_workspace_bytes(d, k));
  if ((err = gs::launch_query_at(momentum->merged, momentum->h, momentum->r, (uint32_t)momentum->c, idx, k,
                                 delta_u, s)) != cudaSuccess)
    return cuda_fail(err, "query_at launch");
  // the extracted mass leaves both sketches
  if ((err = gs::launch_add_sparse(error->merged, error->h, error->r, (uint32_t)error->c, idx, vals, k, -1.f,
                                   s)) != cudaSuccess)
    return cuda_fail(err, "add_sparse launch");
  if ((err = gs::launch_add_sparse(momentum->merged, momentum->h, momentum->r, (uint32_t)momentum->c, idx, delta_u,
                                   k, -1.f, s)) != cudaSuccess)
    return cuda_fail(err, "add_sparse launch");
  if (weights && (err = gs::launch_apply_update(weights, d, idx, vals, k, lr, s)) != cudaSuccess)
    return cuda_fail(err, "update launch");
  return GS_OK;
}

gs_status check_step(gs_sketch* sk, float* const* momentum, float* const* error, const float* const* grad, int64_t d,
                     int64_t k, int64_t* idx_out, float* vals_out, float* est_out, void* workspace,
                     size_t workspace_bytes) {
  GS_TRY(check_sketch(sk));
  GS_TRY(check_d(d));
  if (k < 1 || k > d) return fail(GS_ERR_INVALID_ARG, "k must lie in [1, d]");
  if (!grad) return fail(GS_ERR_INVALID_ARG, "grad array is NULL");
  GS_TRY(check_worker_arrays(sk->workers, momentum, error, grad));
  if (!idx_out || !aligned(idx_out, 8)) return fail(GS_ERR_INVALID_ARG, "idx_out is NULL or not 8-byte aligned");
  GS_TRY(check_vec(vals_out, "vals_out"));
  if (est_out) GS_TRY(check_vec(est_out, "est_out"));
  if (!workspace || !aligned(workspace, 256)) return fail(GS_ERR_INVALID_ARG, "workspace is NULL or not 256-byte aligned");
  if (workspace_bytes < gs::query_topk_workspace_bytes(d, k)) return fail(GS_ERR_INVALID_ARG, "workspace too small");
  return GS_OK;
}

gs_status check_host_step(gs_sketch* sk, float* const* momentum, float* const* error, const float* const* grad_host,
                          float* const* grad_dev, int64_t d, int64_t k, int64_t* idx_host, float* vals_host,
                          void* workspace, size_t workspace_bytes) {
  GS_TRY(check_sketch(sk));
  GS_TRY(check_d(d));
  if (k < 1 || k > d) return fail(GS_ERR_INVALID_ARG, "k must lie in [1, d]");
  if (!grad_host || !grad_dev) return fail(GS_ERR_INVALID_ARG, "grad array is NULL");
  for (int p = 0; p < sk->workers; ++p)
    if (!grad_host[p]) return fail(GS_ERR_INVALID_ARG, "grad_host[p] is NULL");
  GS_TRY(check_worker_arrays(sk->workers, momentum, error, grad_dev));
  if (!idx_host || !vals_host) return fail(GS_ERR_INVALID_ARG, "host outputs are NULL");
  if (!workspace || !aligned(workspace, 256)) return fail(GS_ERR_INVALID_ARG, "workspace is NULL or not 256-byte aligned");
  if (workspace_bytes < step_ws_bytes(d, k)) return fail(GS_ERR_INVALID_ARG, "workspace too small: use gs_step_workspace_size");
  return GS_OK;
}

// Where the fused kernel reads each worker's host gradient: the gradient itself where the GPU
// can address it (pinned or registered host memory, device memory, or any host memory when
// the device has pageable-memory access), else nullptr: first copied into grad_dev[p].
void host_sources(const gs_sketch* sk, const float* const* grad_host, std::vector<const float*>& src) {
  int pageable = 0;
  cudaDeviceGetAttribute(&pageable, cudaDevAttrPageableMemoryAccess, sk->device);
  src.assign((size_t)sk->workers, nullptr);
  for (int p = 0; p < sk->workers; ++p) {
    cudaPointerAttributes attr;
    if (cudaPointerGetAttributes(&attr, grad_host[p]) != cudaSuccess) {
      cudaGetLastError();
      attr.type = cudaMemoryTypeUnregistered;
      attr.devicePointer = nullptr;
    }
    const float* direct = nullptr;
    if (attr.type == cudaMemoryTypeHost && attr.devicePointer) direct = static_cast<const float*>(attr.devicePointer);
    else if (attr.type == cudaMemoryTypeDevice || attr.type == cudaMemoryTypeManaged) direct = grad_host[p];
    else if (attr.type == cudaMemoryTypeUnregistered && pageable == 1) direct = grad_host[p];
    if (direct && aligned(direct, 4)) src[(size_t)p] = direct;
  }
}

// The host step on stream s: uploads where needed, the whole step, and the download of the
// k indices and values into the host outputs (not synchronised).
gs_status host_step_enqueue(gs_sketch* sk, float* const* momentum, float* const* error, const float* const* grad_host,
                            float* const* grad_dev, const std::vector<const float*>& src, int64_t d, float rho,
                            int64_t k, int64_t* idx_host, float* vals_host, void* workspace, cudaStream_t s,
                            InsertMarks marks = InsertMarks()) {
  const size_t qbytes = gs::query_topk_workspace_bytes(d, k);
  int64_t* idx_dev = reinterpret_cast<int64_t*>(static_cast<char*>(workspace) + qbytes);
  float* vals_dev = reinterpret_cast<float*>(reinterpret_cast<char*>(idx_dev) + (((size_t)k * 8 + 255) & ~size_t(255)));
  std::vector<const float*> gsrc(src);
  for (int p = 0; p < sk->workers; ++p) {
    if (gsrc[(size_t)p]) continue;
    cudaError_t e = cudaMemcpyAsync(grad_dev[p], grad_host[p], (size_t)d * sizeof(float), cudaMemcpyHostToDevice, s);
    if (e != cudaSuccess) return cuda_fail(e, "gradient upload");
    gsrc[(size_t)p] = grad_dev[p];
  }
  GS_TRY(step_impl(sk, momentum, error, gsrc.data(), d, rho, k, idx_dev, vals_dev, nullptr, workspace, s, nullptr, 0.f,
                   marks));
  cudaError_t e = cudaMemcpyAsync(idx_host, idx_dev, (size_t)k * sizeof(int64_t), cudaMemcpyDeviceToHost, s);
  if (e == cudaSuccess) e = cudaMemcpyAsync(vals_host, vals_dev, (size_t)k * sizeof(float), cudaMemcpyDeviceToHost, s);
  if (e != cudaSuccess) return cuda_fail(e, "result download");
  return GS_OK;
}

// A plan's events for the insert phase are a ring: launch n records into slot n mod kPlanRing.
constexpr int64_t kPlanRing = 1024;

void plan_free(gs_plan* p) {
  if (p->exec) cudaGraphExecDestroy(p->exec);
  if (p->graph) cudaGraphDestroy(p->graph);
  for (int m = 0; m < kMarks; ++m)
    for (cudaEvent_t ev : p->ev[m])
      if (ev) cudaEventDestroy(ev);
  delete p;
}

gs_status check_plan(const gs_plan* plan) {
  if (!plan) return fail(GS_ERR_INVALID_ARG, "plan is NULL");
  int dev = -1;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
  if (dev != plan->device) return fail(GS_ERR_INVALID_ARG, "current device differs from the plan's device");
  return GS_OK;
}

// The marks each plan flag records.
bool mark_in_use(int32_t flags, int m) {
  if (m == kInsertBegin || m == kInsertEnd) return (flags & GS_PLAN_TIME_INSERT) != 0;
  return (flags & GS_PLAN_TIME_QUERY) != 0;
}

// Capture body(stream, marks) on a private stream into a graph and instantiate it.  Every
// mark that the flags ask for becomes an event-record node whose event each launch re-points
// into the mark's ring.
template <class Body>
gs_status capture_plan(int device, int32_t flags, gs_plan** out, Body&& body) {
  if (!out) return fail(GS_ERR_INVALID_ARG, "plan_out is NULL");
  if (flags & ~int32_t(GS_PLAN_TIME_INSERT | GS_PLAN_TIME_QUERY)) return fail(GS_ERR_INVALID_ARG, "unknown plan flags");
  gs_plan* p = new gs_plan();
  p->device = device;
  p->flags = flags;
  cudaError_t e = cudaSuccess;
  InsertMarks marks;
  for (int m = 0; m < kMarks && e == cudaSuccess; ++m) {
    if (!mark_in_use(flags, m)) continue;
    p->ev[m].assign((size_t)kPlanRing, nullptr);
    for (size_t i = 0; i < (size_t)kPlanRing && e == cudaSuccess; ++i) e = cudaEventCreate(&p->ev[m][i]);
    marks.ev[m] = p->ev[m][0];
  }
  if (e != cudaSuccess) {
    plan_free(p);
    return cuda_fail(e, "cudaEventCreate");
  }
  cudaStream_t cs = nullptr;
  if ((e = cudaStreamCreateWithFlags(&cs, cudaStreamNonBlocking)) != cudaSuccess) {
    plan_free(p);
    return cuda_fail(e, "cudaStreamCreateWithFlags");
  }
  if ((e = cudaStreamBeginCapture(cs, cudaStreamCaptureModeThreadLocal)) != cudaSuccess) {
    cudaStreamDestroy(cs);
    plan_free(p);
    return cuda_fail(e, "cudaStreamBeginCapture");
  }
  const gs_status st = body(cs, marks);
  cudaGraph_t graph = nullptr;
  e = cudaStreamEndCapture(cs, &graph);
  p->graph = graph;
  if (st != GS_OK || e != cudaSuccess) {
    cudaStreamDestroy(cs);
    plan_free(p);
    return st != GS_OK ? st : cuda_fail(e, "stream capture");
  }
  if (flags) {
    size_t n = 0;
    e = cudaGraphGetNodes(graph, nullptr, &n);
    std::vector<cudaGraphNode_t> nodes(n);
    if (e == cudaSuccess && n) e = cudaGraphGetNodes(graph, nodes.data(), &n);
    for (size_t i = 0; i < n && e == cudaSuccess; ++i) {
      cudaGraphNodeType type;
      if ((e = cudaGraphNodeGetType(nodes[i], &type)) != cudaSuccess || type != cudaGraphNodeTypeEventRecord) continue;
      cudaEvent_t ev = nullptr;
      if ((e = cudaGraphEventRecordNodeGetEvent(nodes[i], &ev)) != cudaSuccess) break;
      for (int m = 0; m < kMarks; ++m)
        if (ev && ev == marks.ev[m]) p->node[m] = nodes[i];
    }
    for (int m = 0; m < kMarks && e == cudaSuccess; ++m) {
      if (mark_in_use(flags, m) && !p->node[m]) {
        cudaStreamDestroy(cs);
        plan_free(p);
        return fail(GS_ERR_CUDA, "stream capture: phase event nodes not found");
      }
    }
  }
  if (e == cudaSuccess) e = cudaGraphInstantiate(&p->exec, graph, 0);
  // upload now, so that the first launch does not pay for it
  if (e == cudaSuccess) e = cudaGraphUpload(p->exec, cs);
  if (e == cudaSuccess) e = cudaStreamSynchronize(cs);
  cudaStreamDestroy(cs);
  if (e != cudaSuccess) {
    plan_free(p);
    return cuda_fail(e, "graph instantiation");
  }
  *out = p;
  return GS_OK;
}

}  // namespace

namespace gs {

DeviceInfo device_info() {
  static std::mutex mu;
  static std::unordered_map<int, int> sms_of;
  int dev = 0;
  cudaGetDevice(&dev);
  std::lock_guard<std::mutex> lock(mu);
  auto it = sms_of.find(dev);
  if (it == sms_of.end()) {
    int sms = 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms < 1) sms = 1;
    it = sms_of.emplace(dev, sms).first;
  }
  return DeviceInfo{it->second};
}

int blocks_per_sm(const void* kernel, int block) {
  static std::mutex mu;
  static std::unordered_map<const void*, int> cache;
  std::lock_guard<std::mutex> lock(mu);
  auto it = cache.find(kernel);
  if (it != cache.end()) return it->second;
  int n = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, kernel, block, 0) != cudaSuccess || n < 1) {
    cudaGetLastError();
    n = 1;
  }
  cache.emplace(kernel, n);
  return n;
}

}  // namespace gs

extern "C" {

gs_status gs_sketch_create(int32_t r, int32_t c, uint64_t seed, int32_t workers, int32_t group_width,
                           gs_sketch** out) {
  GS_GUARD_BEGIN
  if (!out) return fail(GS_ERR_INVALID_ARG, "out is NULL");
  *out = nullptr;
  if (r < 1 || r > GS_MAX_ROWS) return fail(GS_ERR_INVALID_ARG, "r must lie in [1, 16]");
  if (c < 1 || c > GS_MAX_COLS) return fail(GS_ERR_INVALID_ARG, "c must lie in [1, 2^26]");
  if (workers < 1 || workers > GS_MAX_WORKERS) return fail(GS_ERR_INVALID_ARG, "workers must lie in [1, 64]");
  if (group_width != 0 && group_width != 1 && group_width != 2 && group_width != 4 && group_width != 8 &&
      group_width != 16)
    return fail(GS_ERR_INVALID_ARG, "group_width must be 0, 1, 2, 4, 8 or 16");
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
  const int W = group_width ? group_width : choose_group_width(r, c, workers);
  const int groups = (workers + W - 1) / W;
  const size_t table_floats = (size_t)groups * r * c * W;
  const size_t bytes = (table_floats + (size_t)r * c) * sizeof(float);
  float* mem = nullptr;
  e = cudaMalloc(&mem, bytes);
  if (e != cudaSuccess) {
    cudaGetLastError();
    return fail(e == cudaErrorMemoryAllocation ? GS_ERR_OOM : GS_ERR_CUDA,
                std::string("cudaMalloc of ") + std::to_string(bytes) + " bytes: " + cudaGetErrorString(e));
  }
  e = cudaMemset(mem, 0, bytes);
  if (e != cudaSuccess) {
    cudaFree(mem);
    return cuda_fail(e, "cudaMemset");
  }
  gs_sketch* sk = new gs_sketch;
  sk->r = r;
  sk->c = c;
  sk->workers = workers;
  sk->W = W;
  sk->groups = groups;
  sk->rows_per_pass = choose_rows_per_pass(r, c, W);
  sk->seed = seed;
  derive_coefficients(r, seed, sk->h);
  sk->tables = mem;
  sk->merged = mem + table_floats;
  sk->device = dev;
  *out = sk;
  return ok();
  GS_GUARD_END
}

gs_status gs_sketch_destroy(gs_sketch* sk) {
  GS_GUARD_BEGIN
  if (!sk) return GS_OK;
  int prev = -1;
  cudaGetDevice(&prev);
  if (prev != sk->device) cudaSetDevice(sk->device);
  cudaError_t e = cudaFree(sk->tables);
  if (prev >= 0 && prev != sk->device) cudaSetDevice(prev);
  delete sk;
  if (e != cudaSuccess) return cuda_fail(e, "cudaFree");
  return GS_OK;
  GS_GUARD_END
}

gs_status gs_sketch_info(const gs_sketch* sk, int32_t* r, int32_t* c, int32_t* workers, int32_t* group_width,
                         int32_t* rows_per_pass) {
  GS_GUARD_BEGIN
  if (!sk) return fail(GS_ERR_INVALID_ARG, "sketch is NULL");
  if (r) *r = sk->r;
  if (c) *c = sk->c;
  if (workers) *workers = sk->workers;
  if (group_width) *group_width = sk->W;
  if (rows_per_pass) *rows_per_pass = sk->rows_per_pass;
  return GS_OK;
  GS_GUARD_END
}

gs_status gs_sketch_coefficients(const gs_sketch* sk, uint64_t* out4r) {
  GS_GUARD_BEGIN
  if (!sk) return fail(GS_ERR_INVALID_ARG, "sketch is NULL");
  if (!out4r) return fail(GS_ERR_INVALID_ARG, "out4r is NULL");
  for (int j = 0; j < sk->r; ++j) {
    out4r[4 * j + 0] = sk->h.a[j];
    out4r[4 * j + 1] = sk->h.b[j];
    out4r[4 * j + 2] = sk->h.a2[j];
    out4r[4 * j + 3] = sk->h.b2[j];
  }
  return GS_OK;
  GS_GUARD_END
}

gs_status gs_sketch_zero(gs_sketch* sk, gs_stream stream) {
  GS_GUARD_BEGIN
  GS_TRY(check_sketch(sk));
  const size_t bytes = ((size_t)sk->groups * sk->r * sk->c * sk->W + (size_t)sk->r * sk->c) * sizeof(float);
  cudaError_t e = cudaMemsetAsync(sk->tables, 0, bytes, as_stream(stream));
  if (e != cudaSuccess) return cuda_fail(e, "cudaMemsetAsync");
  return GS_OK;
  GS_GUARD_END
}

gs_status gs_accumulate(float* momentum, float* error, const float* grad, int64_t d, float rho, gs_stream stream) {
  GS_GUARD_BEGIN
  GS_TRY(check_vec(momentum, "momentum"));
  GS_TRY(check_vec(error, "error"));
  GS_TRY(check_vec(grad, "grad"));
  GS_TRY(check_d(d));
  cudaError_t e = gs::launch_accumulate(momentum, error, grad, d, rho, as_stream(stream));
  if (e != cudaSuccess) return cuda_fail(e, "accumulate launch");
  return GS_OK;
  GS_GUARD_END
}

gs_status gs_sketch_insert(gs_sketch* sk, int32_t worker, const float* vec, int64_t d, gs_stream stream) {
  GS_GUARD_BEGIN
  GS_TRY(check_sketch(sk));
  GS_TRY(check_vec(vec, "vec"));
  GS_TRY(check_d(d));
  if (worker < 0 || worker >= sk->workers) return fail(GS_ERR_INVALID_ARG, "worker out of range");
  gs::InsertParams p;
  std::memset(&p, 0, sizeof(p));
  const int W = sk->W;
  p.e[0] = const_cast<float*>(vec);
  p.table = sk->tables + (size_t)(worker / W) * sk->r * sk->c * W;
  p.lane = worker % W;
  p.d = d;
  p.nw = 1;
  p.r = sk->r;
  p.j0 = 0;
  p.j1 = sk->r;
  p.c = (uint32_t)sk->c;
  p.cmask = (uint32_t)sk->c - 1;
  p.h = sk->h;
  cudaError_t e = gs::launch_insert_lane(p, W, as_stream(stream));
  if (e != cudaSuccess) return cuda_fail(e, "insert launch");
  return GS_OK;
  GS_GUARD_END
}

gs_status gs_accumulate_insert(gs_sketch* sk, int32_t first_worker, int32_t n_workers, float* const* momentum,
                               float* const* error, const float* const* grad, int64_t d, float rho,
                               gs_stream stream) {
  GS_GUARD_BEGIN
  GS_TRY(check_sketch(sk));
  GS_TRY(check_d(d));
  if (n_workers < 1 || first_worker < 0 || first_worker + n_workers > sk->workers)
    return fail(GS_ERR_INVALID_ARG, "worker range out of bounds");
  if (first_worker % sk->W != 0) return fail(GS_ERR_INVALID_ARG, "first_worker must be a multiple of the group width");
  const int end = first_worker + n_workers;
  if (end % sk->W != 0 && end != sk->workers)
    return fail(GS_ERR_INVALID_ARG, "the worker range must end on a group boundary or at the last worker");
  if (!grad) return fail(GS_ERR_INVALID_ARG, "grad array is NULL");
  GS_TRY(check_worker_arrays(n_workers, momentum, error, grad));
  return accumulate_insert_impl(sk, first_worker, n_workers, momentum, error, grad, d, rho, as_stream(stream));
  GS_GUARD_END
}

gs_status gs_accumulate_insert_staged(gs_sketch* sk, int32_t first_worker, int32_t n_workers, float* const* momentum,
                                      float* const* error, const float* const* grad, int64_t d, float rho,
                                      gs_stream stream) {
  GS_GUARD_BEGIN
  GS_TRY(check_sketch(sk));
  GS_TRY(check_d(d));
  if (n_workers < 1 || first_worker < 0 || first_worker + n_workers > sk->workers)
    return fail(GS_ERR_INVALID_ARG, "worker range out of bounds");
  if (first_worker % sk->W != 0) return fail(GS_ERR_INVALID_ARG, "first_worker must be a multiple of the group width");
  const int end = first_worker + n_workers;
  if (end % sk->W != 0 && end != sk->workers)
    return fail(GS_ERR_INVALID_ARG, "the worker range must end on a group boundary or at the last worker");
  if (!grad) return fail(GS_ERR_INVALID_ARG, "grad array is NULL");
  GS_TRY(check_worker_arrays(n_workers, momentum, error, grad));
  if (gs::staged_tile_width((uint32_t)sk->c, sk->W) == 0)
    return fail(GS_ERR_INVALID_ARG, "a table row of c = " + std::to_string(sk->c) +
                                        " cells does not fit a shared-memory tile (c * 4 bytes <= 200 KiB)");
  cudaStream_t s = as_stream(stream);
  for (int w = 0; w < n_workers; ++w) {
    cudaError_t e = gs::launch_accumulate(momentum[w], error[w], grad[w], d, rho, s);
    if (e != cudaSuccess) return cuda_fail(e, "accumulate launch");
  }
  const int W = sk->W;
  for (int grp = first_worker / W; grp * W < end; ++grp) {
    gs::InsertParams p;
    std::memset(&p, 0, sizeof(p));
    const int lo = grp * W;
    const int nw = (end - lo) < W ? (end - lo) : W;
    for (int w = 0; w < nw; ++w) p.e[w] = error[lo + w - first_worker];
    p.table = sk->tables + (size_t)grp * sk->r * sk->c * W;
    p.d = d;
    p.nw = nw;
    p.r = sk->r;
    p.c = (uint32_t)sk->c;
    p.cmask = (uint32_t)sk->c - 1;
    p.h = sk->h;
    p.j0 = 0;
    p.j1 = sk->r;
    cudaError_t e = gs::launch_insert_staged(p, W, s);
    if (e != cudaSuccess) return cuda_fail(e, "staged insert launch");
  }
  return GS_OK;
  GS_GUARD_END
}

gs_status gs_sketch_merge_tree(gs_sketch* sk, int32_t P, gs_stream stream) {
  GS_GUARD_BEGIN
  GS_TRY(check_sketch(sk));
  if (P < 1 || P > sk->workers) return fail(GS_ERR_INVALID_ARG, "P must lie in [1, workers]");
  gs::MergeParams mp;
  mp.tables = sk->tables;
  mp.merged = sk->merged;
  mp.cells = (int64_t)sk->r * sk->c;
  mp.group_stride = (int64_t)sk->r * sk->c * sk->W;
  mp.P = P;
  cudaError_t e = gs::launch_merge(mp, sk->W, as_stream(stream));
  if (e != cudaSuccess) return cuda_fail(e, "merge launch");
  return GS_OK;
  GS_GUARD_END
}

gs_status gs_sketch_merge_sketches(gs_sketch* const* sketches, int32_t P, gs_stream stream) {
  GS_GUARD_BEGIN
  if (!sketches) return fail(GS_ERR_INVALID_ARG, "sketches is NULL");
  if (P < 1 || P > GS_MAX_WORKERS) return fail(GS_ERR_INVALID_ARG, "P must lie in [1, 64]");
  for (int i = 0; i < P; ++i) {
    GS_TRY(check_sketch(sketches[i]));
    if (!same_family(sketches[0], sketches[i]))
      return fail(GS_ERR_MISMATCH, "sketch " + std::to_string(i) + " differs from sketch 0 in r, c or seed");
    for (int j = 0; j < i; ++j)
      if (sketches[j] == sketches[i]) return fail(GS_ERR_INVALID_ARG, "a sketch appears twice");
  }
  gs::MergeListParams mp;
  std::memset(&mp, 0, sizeof(mp));
  for (int i = 0; i < P; ++i) {
    mp.tables[i] = sketches[i]->tables;
    mp.lane_stride[i] = sketches[i]->W;
  }
  mp.merged = sketches[0]->merged;
  mp.cells = (int64_t)sketches[0]->r * sketches[0]->c;
  mp.P = P;
  cudaError_t e = gs::launch_merge_list(mp, as_stream(stream));
  if (e != cudaSuccess) return cuda_fail(e, "merge launch");
  return GS_OK;
  GS_GUARD_END
}

gs_status gs_query_topk_workspace_size(int64_t d, int64_t k, size_t* bytes) {
  GS_GUARD_BEGIN
  GS_TRY(check_d(d));
  if (k < 1 || k > d) return fail(GS_ERR_INVALID_ARG, "k must lie in [1, d]");
  if (!bytes) return fail(GS_ERR_INVALID_ARG, "bytes is NULL");
  *bytes = gs::query_topk_workspace_bytes(d, k);
  return GS_OK;
  GS_GUARD_END
}

gs_status gs_query_topk(const gs_sketch* sk, int64_t d, int64_t k, int64_t* idx_out, float* est_out,
                        void* workspace, size_t workspace_bytes, gs_stream stream) {
  GS_GUARD_BEGIN
  GS_TRY(check_sketch(sk));
  GS_TRY(check_d(d));
  if (k < 1 || k > d) return fail(GS_ERR_INVALID_ARG, "k must lie in [1, d]");
  if (!idx_out || !aligned(idx_out, 8)) return fail(GS_ERR_INVALID_ARG, "idx_out is NULL or not 8-byte aligned");
  if (est_out) GS_TRY(check_vec(est_out, "est_out"));
  if (!workspace || !aligned(workspace, 256)) return fail(GS_ERR_INVALID_ARG, "workspace is NULL or not 256-byte aligned");
  if (workspace_bytes < gs::query_topk_workspace_bytes(d, k))
    return fail(GS_ERR_INVALID_ARG, "workspace too small: need " + std::to_string(gs::query_topk_workspace_bytes(d, k)));
  cudaError_t e = gs::launch_query_topk(sk->merged, sk->h, sk->r, (uint32_t)sk->c, d, k, idx_out, est_out, workspace,
                                        as_stream(stream));
  if (e != cudaSuccess) return cuda_fail(e, "query/top-k launch");
  return GS_OK;
  GS_GUARD_END
}

gs_status gs_query_heavymix_workspace_size(int64_t d, int64_t k, size_t* bytes) {
  GS_GUARD_BEGIN
  GS_TRY(check_d(d));
  if (k < 1 || k > d) return fail(GS_ERR_INVALID_ARG, "k must lie in [1, d]");
  if (!bytes) return fail(GS_ERR_INVALID_ARG, "bytes is NULL");
  *bytes = gs::heavymix_workspace_bytes(d, k);
  return GS_OK;
  GS_GUARD_END
}

gs_status gs_query_heavymix(const gs_sketch* sk, int64_t d, int64_t k, uint64_t fill_seed, int64_t* idx_out,
                            float* est_out, double* l2sq_out, void* workspace, size_t workspace_bytes,
                            gs_stream stream) {
  GS_GUARD_BEGIN
  GS_TRY(check_sketch(sk));
  GS_TRY(check_d(d));
  if (k < 1 || k > d) return fail(GS_ERR_INVALID_ARG, "k must lie in [1, d]");
  if (!idx_out || !aligned(idx_out, 8)) return fail(GS_ERR_INVALID_ARG, "idx_out is NULL or not 8-byte aligned");
  if (est_out) GS_TRY(check_vec(est_out, "est_out"));
  if (l2sq_out && !aligned(l2sq_out, 8)) return fail(GS_ERR_INVALID_ARG, "l2sq_out is not 8-byte aligned");
  if (!workspace || !aligned(workspace, 256)) return fail(GS_ERR_INVALID_ARG, "workspace is NULL or not 256-byte aligned");
  if (workspace_bytes < gs::heavymix_workspace_bytes(d, k))
    return fail(GS_ERR_INVALID_ARG, "workspace too small: need " + std::to_string(gs::heavymix_workspace_bytes(d, k)));
  cudaError_t e = gs::launch_query_heavymix(sk->merged, sk->h, sk->r, (uint32_t)sk->c, d, k, fill_seed, idx_out,
                                            est_out, l2sq_out, workspace, as_stream(stream));
  if (e != cudaSuccess) return cuda_fail(e, "HEAVYMIX launch");
  return GS_OK;
  GS_GUARD_END
}

gs_status gs_query_topk_noalloc(const gs_sketch* sk, int64_t d, int64_t k, int64_t* idx_out, float* est_out,
                                gs_stream stream) {
  GS_GUARD_BEGIN
  GS_TRY(check_sketch(sk));
  GS_TRY(check_d(d));
  if (d > GS_NOALLOC_MAX_DIM)
    return fail(GS_ERR_INVALID_ARG, "d = " + std::to_string(d) + " exceeds GS_NOALLOC_MAX_DIM = " +
                                        std::to_string(GS_NOALLOC_MAX_DIM) +
                                        ", the size the fixed scratch serves; use gs_query_topk with a workspace");
  if (k < 1 || k > d) return fail(GS_ERR_INVALID_ARG, "k must lie in [1, d]");
  if (!idx_out || !aligned(idx_out, 8)) return fail(GS_ERR_INVALID_ARG, "idx_out is NULL or not 8-byte aligned");
  if (!est_out) return fail(GS_ERR_INVALID_ARG, "est_out is required by gs_query_topk_noalloc");
  GS_TRY(check_vec(est_out, "est_out"));
  cudaError_t e = gs::launch_query_topk_noalloc(sk->merged, sk->h, sk->r, (uint32_t)sk->c, d, k, idx_out, est_out,
                                                as_stream(stream));
  if (e != cudaSuccess) return cuda_fail(e, "query/top-k (no-allocation variant)");
  return GS_OK;
  GS_GUARD_END
}

gs_status gs_gather_and_zero(float* const* momentum, float* const* error, int32_t P, int64_t d, const int64_t* idx,
                             int64_t k, float* vals_out, gs_stream stream) {
  GS_GUARD_BEGIN
  if (P < 1 || P > GS_MAX_WORKERS) return fail(GS_ERR_INVALID_ARG, "P must lie in [1, 64]");
  GS_TRY(check_d(d));
  if (k < 1 || k > d) return fail(GS_ERR_INVALID_ARG, "k must lie in [1, d]");
  if (!idx || !aligned(idx, 8)) return fail(GS_ERR_INVALID_ARG, "idx is NULL or not 8-byte aligned");
  GS_TRY(check_vec(vals_out, "vals_out"));
  GS_TRY(check_worker_arrays(P, momentum, error, nullptr));
  gs::GatherParams gp;
  std::memset(&gp, 0, sizeof(gp));
  for (int p = 0; p < P; ++p) {
    gp.u[p] = momentum[p];
    gp.e[p] = error[p];
  }
  gp.idx = idx;
  gp.vals = vals_out;
  gp.w = nullptr;
  gp.lr = 0.f;
  gp.k = k;
  gp.d = d;
  gp.P = P;
  cudaError_t e = gs::launch_gather_and_zero(gp, as_stream(stream));
  if (e != cudaSuccess) return cuda_fail(e, "gather launch");
  return GS_OK;
  GS_GUARD_END
}

gs_status gs_gather_zero_update(float* const* momentum, float* const* error, int32_t P, int64_t d, const int64_t* idx,
                                int64_t k, float* vals_out, float* weights, float lr, gs_stream stream) {
  GS_GUARD_BEGIN
  if (P < 1 || P > GS_MAX_WORKERS) return fail(GS_ERR_INVALID_ARG, "P must lie in [1, 64]");
  GS_TRY(check_d(d));
  if (k < 1 || k > d) return fail(GS_ERR_INVALID_ARG, "k must lie in [1, d]");
  if (!idx || !aligned(idx, 8)) return fail(GS_ERR_INVALID_ARG, "idx is NULL or not 8-byte aligned");
  GS_TRY(check_vec(vals_out, "vals_out"));
  if (weights) GS_TRY(check_vec(weights, "weights"));
  GS_TRY(check_worker_arrays(P, momentum, error, nullptr));
  gs::GatherParams gp;
  std::memset(&gp, 0, sizeof(gp));
  for (int p = 0; p < P; ++p) {
    gp.u[p] = momentum[p];
    gp.e[p] = error[p];
  }
  gp.idx = idx;
  gp.vals = vals_out;
  gp.w = weights;
  gp.lr = lr;
  gp.k = k;
  gp.d = d;
  gp.P = P;
  cudaError_t e = gs::launch_gather_and_zero(gp, as_stream(stream));
  if (e != cudaSuccess) return cuda_fail(e, "gather launch");
  return GS_OK;
  GS_GUARD_END
}

gs_status gs_apply_update(float* weights, int64_t d, const int64_t* idx, const float* vals, int64_t k, float lr,
                          gs_stream stream) {
  GS_GUARD_BEGIN
  GS_TRY(check_vec(weights, "weights"));
  GS_TRY(check_d(d));
  if (k < 1 || k > d) return fail(GS_ERR_INVALID_ARG, "k must lie in [1, d]");
  if (!idx || !aligned(idx, 8)) return fail(GS_ERR_INVALID_ARG, "idx is NULL or not 8-byte aligned");
  GS_TRY(check_vec(vals, "vals"));
  cudaError_t e = gs::launch_apply_update(weights, d, idx, vals, k, lr, as_stream(stream));
  if (e != cudaSuccess) return cuda_fail(e, "update launch");
  return GS_OK;
  GS_GUARD_END
}

gs_status gs_step_workspace_size(int64_t d, int64_t k, size_t* bytes) {
  GS_GUARD_BEGIN
  GS_TRY(check_d(d));
  if (k < 1 || k > d) return fail(GS_ERR_INVALID_ARG, "k must lie in [1, d]");
  if (!bytes) return fail(GS_ERR_INVALID_ARG, "bytes is NULL");
  *bytes = step_ws_bytes(d, k);
  return GS_OK;
  GS_GUARD_END
}

gs_status gs_step(gs_sketch* sk, float* const* momentum, float* const* error, const float* const* grad, int64_t d,
                  float rho, int64_t k, int64_t* idx_out, float* vals_out, float* est_out, void* workspace,
                  size_t workspace_bytes, gs_stream stream) {
  GS_GUARD_BEGIN
  GS_TRY(check_step(sk, momentum, error, grad, d, k, idx_out, vals_out, est_out, workspace, workspace_bytes));
  return step_impl(sk, momentum, error, grad, d, rho, k, idx_out, vals_out, est_out, workspace, as_stream(stream));
  GS_GUARD_END
}

gs_status gs_train_step(gs_sketch* sk, float* weights, float lr, float* const* momentum, float* const* error,
                        const float* const* grad, int64_t d, float rho, int64_t k, int64_t* idx_out, float* vals_out,
                        float* est_out, void* workspace, size_t workspace_bytes, gs_stream stream) {
  GS_GUARD_BEGIN
  GS_TRY(check_vec(weights, "weights"));
  GS_TRY(check_step(sk, momentum, error, grad, d, k, idx_out, vals_out, est_out, workspace, workspace_bytes));
  return step_impl(sk, momentum, error, grad, d, rho, k, idx_out, vals_out, est_out, workspace, as_stream(stream),
                   weights, lr);
  GS_GUARD_END
}

gs_status gs_heavymix_step_workspace_size(int64_t d, int64_t k, size_t* bytes) {
  GS_GUARD_BEGIN
  GS_TRY(check_d(d));
  if (k < 1 || k > d) return fail(GS_ERR_INVALID_ARG, "k must lie in [1, d]");
  if (!bytes) return fail(GS_ERR_INVALID_ARG, "bytes is NULL");
  *bytes = gs::heavymix_workspace_bytes(d, k);
  return GS_OK;
  GS_GUARD_END
}

gs_status gs_heavymix_step(gs_sketch* sk, float* const* momentum, float* const* error, const float* const* grad,
                           int64_t d, float rho, int64_t k, uint64_t fill_seed, int64_t* idx_out, float* vals_out,
                           double* l2sq_out, void* workspace, size_t workspace_bytes, gs_stream stream) {
  GS_GUARD_BEGIN
  GS_TRY(check_step(sk, momentum, error, grad, d, k, idx_out, vals_out, nullptr, workspace, workspace_bytes));
  if (workspace_bytes < gs::heavymix_workspace_bytes(d, k))
    return fail(GS_ERR_INVALID_ARG, "workspace too small: use gs_heavymix_step_workspace_size");
  if (l2sq_out && !aligned(l2sq_out, 8)) return fail(GS_ERR_INVALID_ARG, "l2sq_out is not 8-byte aligned");
  Selection sel;
  sel.heavymix = true;
  sel.fill_seed = fill_seed;
  sel.l2sq_out = l2sq_out;
  return step_impl(sk, momentum, error, grad, d, rho, k, idx_out, vals_out, nullptr, workspace, as_stream(stream),
                   nullptr, 0.f, InsertMarks(), sel);
  GS_GUARD_END
}

gs_status gs_sketch_merged_table(const gs_sketch* sk, float** table_out) {
  GS_GUARD_BEGIN
  if (!sk) return fail(GS_ERR_INVALID_ARG, "sketch is NULL");
  if (!table_out) return fail(GS_ERR_INVALID_ARG, "table_out is NULL");
  *table_out = sk->merged;
  return GS_OK;
  GS_GUARD_END
}

gs_status gs_sketch_query_at(const gs_sketch* sk, const int64_t* idx, int64_t k, float* est_out, gs_stream stream) {
  GS_GUARD_BEGIN
  GS_TRY(check_sketch(sk));
  if (k < 1) return fail(GS_ERR_INVALID_ARG, "k must be positive");
  if (!idx || !aligned(idx, 8)) return fail(GS_ERR_INVALID_ARG, "idx is NULL or not 8-byte aligned");
  GS_TRY(check_vec(est_out, "est_out"));
  cudaError_t e = gs::launch_query_at(sk->merged, sk->h, sk->r, (uint32_t)sk->c, idx, k, est_out, as_stream(stream));
  if (e != cudaSuccess) return cuda_fail(e, "query_at launch");
  return GS_OK;
  GS_GUARD_END
}

gs_status gs_sketch_add_sparse(gs_sketch* sk, const int64_t* idx, const float* vals, int64_t k, float scale,
                               gs_stream stream) {
  GS_GUARD_BEGIN
  GS_TRY(check_sketch(sk));
  if (k < 1) return fail(GS_ERR_INVALID_ARG, "k must be positive");
  if (!idx || !aligned(idx, 8)) return fail(GS_ERR_INVALID_ARG, "idx is NULL or not 8-byte aligned");
  GS_TRY(check_vec(vals, "vals"));
  cudaError_t e = gs::launch_add_sparse(sk->merged, sk->h, sk->r, (uint32_t)sk->c, idx, vals, k, scale,
                                        as_stream(stream));
  if (e != cudaSuccess) return cuda_fail(e, "add_sparse launch");
  return GS_OK;
  GS_GUARD_END
}

gs_status gs_sketched_state_step(gs_sketch* workers, gs_sketch* momentum, gs_sketch* error, const float* const* grad,
                                 int64_t d, float rho, int64_t k, int64_t* idx_out, float* vals_out, float* weights,
                                 float lr, void* workspace, size_t workspace_bytes, gs_stream stream) {
  GS_GUARD_BEGIN
  GS_TRY(check_sketched_state(workers, momentum, error, grad, d, k, idx_out, vals_out, weights, workspace,
                              workspace_bytes));
  return sketched_state_impl(workers, momentum, error, grad, d, rho, k, idx_out, vals_out, weights, lr, workspace,
                             as_stream(stream));
  GS_GUARD_END
}

gs_status gs_step_host(gs_sketch* sk, float* const* momentum, float* const* error, const float* const* grad_host,
                       float* const* grad_dev, int64_t d, float rho, int64_t k, int64_t* idx_host, float* vals_host,
                       void* workspace, size_t workspace_bytes, gs_stream stream) {
  GS_GUARD_BEGIN
  GS_TRY(check_host_step(sk, momentum, error, grad_host, grad_dev, d, k, idx_host, vals_host, workspace,
                         workspace_bytes));
  std::vector<const float*> src;
  host_sources(sk, grad_host, src);
  cudaStream_t s = as_stream(stream);
  GS_TRY(host_step_enqueue(sk, momentum, error, grad_host, grad_dev, src, d, rho, k, idx_host, vals_host, workspace, s));
  cudaError_t e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return cuda_fail(e, "result download");
  return GS_OK;
  GS_GUARD_END
}

// ---- plans: one step captured into a CUDA graph -------------------------------------------

gs_status gs_step_plan_create(gs_sketch* sk, float* const* momentum, float* const* error, const float* const* grad,
                              int64_t d, float rho, int64_t k, int64_t* idx_out, float* vals_out, float* est_out,
                              float* weights, float lr, void* workspace, size_t workspace_bytes, int32_t flags,
                              gs_plan** plan_out) {
  GS_GUARD_BEGIN
  if (plan_out) *plan_out = nullptr;
  GS_TRY(check_step(sk, momentum, error, grad, d, k, idx_out, vals_out, est_out, workspace, workspace_bytes));
  if (weights) GS_TRY(check_vec(weights, "weights"));
  return capture_plan(sk->device, flags, plan_out, [&](cudaStream_t s, InsertMarks marks) {
    return step_impl(sk, momentum, error, grad, d, rho, k, idx_out, vals_out, est_out, workspace, s, weights, lr,
                     marks);
  });
  GS_GUARD_END
}

gs_status gs_heavymix_step_plan_create(gs_sketch* sk, float* const* momentum, float* const* error,
                                      const float* const* grad, int64_t d, float rho, int64_t k, uint64_t fill_seed,
                                      int64_t* idx_out, float* vals_out, double* l2sq_out, void* workspace,
                                      size_t workspace_bytes, int32_t flags, gs_plan** plan_out) {
  GS_GUARD_BEGIN
  if (plan_out) *plan_out = nullptr;
  GS_TRY(check_step(sk, momentum, error, grad, d, k, idx_out, vals_out, nullptr, workspace, workspace_bytes));
  if (workspace_bytes < gs::heavymix_workspace_bytes(d, k))
    return fail(GS_ERR_INVALID_ARG, "workspace too small: use gs_heavymix_step_workspace_size");
  if (l2sq_out && !aligned(l2sq_out, 8)) return fail(GS_ERR_INVALID_ARG, "l2sq_out is not 8-byte aligned");
  Selection sel;
  sel.heavymix = true;
  sel.fill_seed = fill_seed;
  sel.l2sq_out = l2sq_out;
  return capture_plan(sk->device, flags, plan_out, [&](cudaStream_t s, InsertMarks marks) {
    return step_impl(sk, momentum, error, grad, d, rho, k, idx_out, vals_out, nullptr, workspace, s, nullptr, 0.f,
                     marks, sel);
  });
  GS_GUARD_END
}

gs_status gs_step_host_plan_create(gs_sketch* sk, float* const* momentum, float* const* error,
                                   const float* const* grad_host, float* const* grad_dev, int64_t d, float rho,
                                   int64_t k, int64_t* idx_host, float* vals_host, void* workspace,
                                   size_t workspace_bytes, int32_t flags, gs_plan** plan_out) {
  GS_GUARD_BEGIN
  if (plan_out) *plan_out = nullptr;
  GS_TRY(check_host_step(sk, momentum, error, grad_host, grad_dev, d, k, idx_host, vals_host, workspace,
                         workspace_bytes));
  std::vector<const float*> src;
  host_sources(sk, grad_host, src);
  return capture_plan(sk->device, flags, plan_out, [&](cudaStream_t s, InsertMarks marks) {
    return host_step_enqueue(sk, momentum, error, grad_host, grad_dev, src, d, rho, k, idx_host, vals_host, workspace,
                             s, marks);
  });
  GS_GUARD_END
}

gs_status gs_sketched_state_plan_create(gs_sketch* workers, gs_sketch* momentum, gs_sketch* error,
                                        const float* const* grad, int64_t d, float rho, int64_t k, int64_t* idx_out,
                                        float* vals_out, float* weights, float lr, void* workspace,
                                        size_t workspace_bytes, int32_t flags, gs_plan** plan_out) {
  GS_GUARD_BEGIN
  if (plan_out) *plan_out = nullptr;
  GS_TRY(check_sketched_state(workers, momentum, error, grad, d, k, idx_out, vals_out, weights, workspace,
                              workspace_bytes));
  return capture_plan(workers->device, flags, plan_out, [&](cudaStream_t s, InsertMarks marks) {
    return sketched_state_impl(workers, momentum, error, grad, d, rho, k, idx_out, vals_out, weights, lr, workspace, s,
                               marks);
  });
  GS_GUARD_END
}

gs_status gs_plan_launch(gs_plan* plan, gs_stream stream) {
  GS_GUARD_BEGIN
  GS_TRY(check_plan(plan));
  cudaError_t e = cudaSuccess;
  const size_t slot = (size_t)(plan->launches % kPlanRing);
  for (int m = 0; m < kMarks && e == cudaSuccess; ++m)
    if (plan->node[m]) e = cudaGraphExecEventRecordNodeSetEvent(plan->exec, plan->node[m], plan->ev[m][slot]);
  if (e != cudaSuccess) return cuda_fail(e, "plan event update");
  e = cudaGraphLaunch(plan->exec, as_stream(stream));
  if (e != cudaSuccess) return cuda_fail(e, "cudaGraphLaunch");
  ++plan->launches;
  return GS_OK;
  GS_GUARD_END
}

}  // extern "C"

namespace {

// Elapsed ms between marks a and b over the last min(n, launches, ring) launches, oldest first.
gs_status plan_mark_times(gs_plan* plan, int a, int b, float* ms_out, int32_t n, int32_t* n_out) {
  int64_t m = n;
  if (m > plan->launches) m = plan->launches;
  if (m > kPlanRing) m = kPlanRing;
  *n_out = 0;
  if (m == 0) return GS_OK;
  cudaError_t e = cudaEventSynchronize(plan->ev[b][(size_t)((plan->launches - 1) % kPlanRing)]);
  for (int64_t t = 0; t < m && e == cudaSuccess; ++t) {
    const size_t slot = (size_t)((plan->launches - m + t) % kPlanRing);
    e = cudaEventElapsedTime(&ms_out[t], plan->ev[a][slot], plan->ev[b][slot]);
  }
  if (e != cudaSuccess) return cuda_fail(e, "plan event times");
  *n_out = (int32_t)m;
  return GS_OK;
}

}  // namespace

extern "C" {

gs_status gs_plan_insert_times(gs_plan* plan, float* ms_out, int32_t n, int32_t* n_out) {
  GS_GUARD_BEGIN
  GS_TRY(check_plan(plan));
  if (!(plan->flags & GS_PLAN_TIME_INSERT)) return fail(GS_ERR_INVALID_ARG, "the plan was created without GS_PLAN_TIME_INSERT");
  if (!ms_out || !n_out || n < 0) return fail(GS_ERR_INVALID_ARG, "ms_out or n_out is NULL, or n < 0");
  return plan_mark_times(plan, kInsertBegin, kInsertEnd, ms_out, n, n_out);
  GS_GUARD_END
}

gs_status gs_plan_query_times(gs_plan* plan, float* query_ms_out, float* select_ms_out, int32_t n, int32_t* n_out) {
  GS_GUARD_BEGIN
  GS_TRY(check_plan(plan));
  if (!(plan->flags & GS_PLAN_TIME_QUERY)) return fail(GS_ERR_INVALID_ARG, "the plan was created without GS_PLAN_TIME_QUERY");
  if (!query_ms_out || !select_ms_out || !n_out || n < 0)
    return fail(GS_ERR_INVALID_ARG, "an output pointer is NULL, or n < 0");
  int32_t n2 = 0;
  GS_TRY(plan_mark_times(plan, kQueryBegin, kQueryEnd, query_ms_out, n, n_out));
  GS_TRY(plan_mark_times(plan, kQueryEnd, kSelectEnd, select_ms_out, n, &n2));
  return GS_OK;
  GS_GUARD_END
}

gs_status gs_plan_destroy(gs_plan* plan) {
  GS_GUARD_BEGIN
  if (!plan) return GS_OK;
  cudaError_t e = cudaSuccess;
  if (plan->launches > 0) e = cudaDeviceSynchronize();
  plan_free(plan);
  if (e != cudaSuccess) return cuda_fail(e, "cudaDeviceSynchronize");
  return GS_OK;
  GS_GUARD_END
}

gs_status gs_insert_request_ceiling_window_size(const gs_sketch* sk, size_t* bytes) {
  GS_GUARD_BEGIN
  GS_TRY(check_sketch(sk));
  if (!bytes) return fail(GS_ERR_INVALID_ARG, "bytes is NULL");
  *bytes = (size_t)3 * sk->W * GS_CEILING_WINDOW_FLOATS * sizeof(float);
  return GS_OK;
  GS_GUARD_END
}

gs_status gs_insert_request_ceiling(gs_sketch* sk, int64_t d, void* window, size_t window_bytes, float* ms_out,
                                    gs_stream stream) {
  GS_GUARD_BEGIN
  GS_TRY(check_sketch(sk));
  GS_TRY(check_d(d));
  const size_t need = (size_t)3 * sk->W * GS_CEILING_WINDOW_FLOATS * sizeof(float);
  if (!window || !aligned(window, 256)) return fail(GS_ERR_INVALID_ARG, "window is NULL or not 256-byte aligned");
  if (window_bytes < need) return fail(GS_ERR_INVALID_ARG, "window too small: need " + std::to_string(need));
  if (!ms_out) return fail(GS_ERR_INVALID_ARG, "ms_out is NULL");
  if (sk->W < 4 || (sk->c & (sk->c - 1)) != 0)
    return fail(GS_ERR_INVALID_ARG, "the probe serves group widths 4, 8 and 16 with c a power of two");
  cudaStream_t s = as_stream(stream);
  cudaEvent_t ev[2] = {nullptr, nullptr};
  cudaError_t e = cudaEventCreate(&ev[0]);
  if (e == cudaSuccess) e = cudaEventCreate(&ev[1]);
  // zero windows keep every value finite; the requests do not depend on the values
  if (e == cudaSuccess) e = cudaMemsetAsync(window, 0, need, s);
  if (e == cudaSuccess) e = cudaEventRecord(ev[0], s);
  float* win = static_cast<float*>(window);
  const int W = sk->W;
  for (int grp = 0; e == cudaSuccess && grp * W < sk->workers; ++grp) {
    gs::InsertParams p;
    std::memset(&p, 0, sizeof(p));
    const int nw = (sk->workers - grp * W) < W ? (sk->workers - grp * W) : W;
    for (int w = 0; w < nw; ++w) {
      p.u[w] = win + (size_t)(3 * w + 0) * GS_CEILING_WINDOW_FLOATS;
      p.e[w] = win + (size_t)(3 * w + 1) * GS_CEILING_WINDOW_FLOATS;
      p.g[w] = win + (size_t)(3 * w + 2) * GS_CEILING_WINDOW_FLOATS;
    }
    p.table = sk->tables + (size_t)grp * sk->r * sk->c * W;
    p.d = d;
    p.nw = nw;
    p.r = sk->r;
    p.c = (uint32_t)sk->c;
    p.cmask = (uint32_t)sk->c - 1;
    p.rho = 0.9f;
    p.winmask = GS_CEILING_WINDOW_FLOATS - 1;
    p.h = sk->h;
    bool first = true;
    for (const Pass& ps : insert_passes(sk)) {
      if (e != cudaSuccess) break;
      p.j0 = ps.j0;
      p.j1 = ps.j1;
      e = gs::launch_insert_ceiling_probe(p, W, first, s);
      first = false;
    }
  }
  if (e == cudaSuccess) e = cudaEventRecord(ev[1], s);
  if (e == cudaSuccess) e = cudaEventSynchronize(ev[1]);
  if (e == cudaSuccess) e = cudaEventElapsedTime(ms_out, ev[0], ev[1]);
  for (cudaEvent_t x : ev)
    if (x) cudaEventDestroy(x);
  if (e != cudaSuccess) return cuda_fail(e, "insert request-ceiling probe");
  return GS_OK;
  GS_GUARD_END
}

gs_status gs_query_request_ceiling(const gs_sketch* sk, int64_t d, void* window, size_t window_bytes, float* ms_out,
                                   gs_stream stream) {
  GS_GUARD_BEGIN
  GS_TRY(check_sketch(sk));
  GS_TRY(check_d(d));
  if (!window || !aligned(window, 256)) return fail(GS_ERR_INVALID_ARG, "window is NULL or not 256-byte aligned");
  if (window_bytes < 65536) return fail(GS_ERR_INVALID_ARG, "window too small: need 65536 bytes");
  if (!ms_out) return fail(GS_ERR_INVALID_ARG, "ms_out is NULL");
  if ((sk->c & (sk->c - 1)) != 0) return fail(GS_ERR_INVALID_ARG, "the probe serves c a power of two");
  cudaStream_t s = as_stream(stream);
  cudaEvent_t ev[2] = {nullptr, nullptr};
  cudaError_t e = cudaEventCreate(&ev[0]);
  if (e == cudaSuccess) e = cudaEventCreate(&ev[1]);
  if (e == cudaSuccess) e = cudaEventRecord(ev[0], s);
  if (e == cudaSuccess)
    e = gs::launch_query_ceiling_probe(sk->merged, sk->h, sk->r, (uint32_t)sk->c, d, static_cast<float*>(window),
                                       (int64_t)(window_bytes / sizeof(float)), s);
  if (e == cudaSuccess) e = cudaEventRecord(ev[1], s);
  if (e == cudaSuccess) e = cudaEventSynchronize(ev[1]);
  if (e == cudaSuccess) e = cudaEventElapsedTime(ms_out, ev[0], ev[1]);
  for (cudaEvent_t x : ev)
    if (x) cudaEventDestroy(x);
  if (e != cudaSuccess) return cuda_fail(e, "query request-ceiling probe");
  return GS_OK;
  GS_GUARD_END
}

gs_status gs_hash_eval(const gs_sketch* sk, const int64_t* coords, int64_t n, int32_t* bucket_out, int8_t* sign_out,
                       gs_stream stream) {
  GS_GUARD_BEGIN
  GS_TRY(check_sketch(sk));
  if (n < 1) return fail(GS_ERR_INVALID_ARG, "n must be positive");
  if (!coords || !aligned(coords, 8)) return fail(GS_ERR_INVALID_ARG, "coords is NULL or not 8-byte aligned");
  if (!bucket_out || !aligned(bucket_out, 4) || !sign_out) return fail(GS_ERR_INVALID_ARG, "output is NULL or misaligned");
  cudaError_t e = gs::launch_hash_eval(sk->h, sk->r, (uint32_t)sk->c, coords, n, bucket_out, sign_out, as_stream(stream));
  if (e != cudaSuccess) return cuda_fail(e, "hash_eval launch");
  return GS_OK;
  GS_GUARD_END
}

gs_status gs_sketch_copy_to_host(const gs_sketch* sk, int32_t worker, float* host_out) {
  GS_GUARD_BEGIN
  GS_TRY(check_sketch(sk));
  if (!host_out) return fail(GS_ERR_INVALID_ARG, "host_out is NULL");
  if (worker < -1 || worker >= sk->workers) return fail(GS_ERR_INVALID_ARG, "worker out of range");
  cudaError_t e = cudaDeviceSynchronize();
  if (e != cudaSuccess) return cuda_fail(e, "cudaDeviceSynchronize");
  const size_t cells = (size_t)sk->r * sk->c;
  if (worker < 0) {
    e = cudaMemcpy(host_out, sk->merged, cells * sizeof(float), cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_fail(e, "cudaMemcpy");
    return GS_OK;
  }
  const int W = sk->W;
  std::vector<float> tmp(cells * W);
  e = cudaMemcpy(tmp.data(), sk->tables + (size_t)(worker / W) * cells * W, cells * W * sizeof(float),
                 cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(e, "cudaMemcpy");
  const int lane = worker % W;
  for (size_t q = 0; q < cells; ++q) host_out[q] = tmp[q * W + lane];
  return GS_OK;
  GS_GUARD_END
}

const char* gs_last_error(void) { return g_err.c_str(); }

}  // extern "C"
