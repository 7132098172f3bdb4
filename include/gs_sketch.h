/*
 * gs_sketch.h -- C ABI of the GB300 gs-SGD gradient-compression library.
 *
 * The library runs the per-step compression pipeline of global-sketching SGD
 * (Dai, Diao, Li, Xu, arXiv 2108.06004) for P data-parallel workers simulated on one
 * GPU:
 *
 *   accumulate    u_p <- rho*u_p + g_p,  e_p <- e_p + u_p       (momentum + error feedback)
 *   insert        T_p <- T_p + S(e_p), an r x c Count Sketch     (Alg. 1 step 5, Sec. III-A)
 *   merge         recursive-halving tree of the P sketches       (Alg. 1 steps 8-23)
 *   query + top-k est_i = median_j s_j(i) T[j][h_j(i)], top-k of |est|  (Alg. 2 steps 1-3)
 *   gather + zero v_t = sum_p e_p[I_t]; u_p[I_t] = e_p[I_t] = 0  (Alg. 2 step 4)
 *
 * Hash family (the paper names Count Sketch but prints no family): for row j,
 *   h_j(i) = ((a_j*i + b_j) mod (2^61 - 1)) mod c,
 *   s_j(i) = +1 if ((a'_j*i + b'_j) mod (2^61 - 1)) is even, else -1,
 * with (a_j, b_j, a'_j, b'_j) the next four outputs of splitmix64(seed) (Steele, Lea and
 * Flood, OOPSLA 2014) reduced as a = 1 + x mod (2^61 - 2), b = x mod (2^61 - 1).
 *
 * Conventions for every call
 *   - Vectors, index and value arrays and workspaces are CALLER-OWNED DEVICE pointers
 *     unless a parameter says "host".  The library owns only sketch tables.
 *   - Calls are asynchronous on `stream` (a cudaStream_t; NULL = the legacy default
 *     stream) except those documented as synchronous.  The current CUDA device must be
 *     the device the sketch was created on.
 *   - Arguments are validated on the host before any launch; a failed check returns
 *     GS_ERR_INVALID_ARG (or GS_ERR_MISMATCH) and launches nothing.  A CUDA error
 *     returns GS_ERR_CUDA.  gs_last_error() then gives a message (thread-local).
 *   - fp32 vectors must be 4-byte aligned; 16-byte alignment of every vector selects
 *     the vectorised path (results are identical either way).
 *   - Sizes: 1 <= r <= GS_MAX_ROWS, 1 <= c <= GS_MAX_COLS, 1 <= d <= GS_MAX_DIM,
 *     1 <= k <= d, 1 <= P <= GS_MAX_WORKERS.  Vector values must be finite.
 *   - No call waits on the device for a flag; nothing spins.  Kernels launch with
 *     programmatic stream serialization and wait in hardware for the grid before them.
 */
#ifndef GS_SKETCH_H
#define GS_SKETCH_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef int32_t gs_status;
#define GS_OK 0
#define GS_ERR_INVALID_ARG 1
#define GS_ERR_MISMATCH 2
#define GS_ERR_OOM 3
#define GS_ERR_CUDA 4
#define GS_ERR_TIMEOUT 5

#define GS_MAX_ROWS 16
#define GS_MAX_COLS (1 << 26)
#define GS_MAX_WORKERS 64
#define GS_MAX_DIM 2147483647LL /* d < 2^31 */

typedef struct gs_sketch gs_sketch; /* opaque */
typedef void* gs_stream;            /* a cudaStream_t */
typedef struct gs_plan gs_plan;     /* opaque: one step captured into a CUDA graph */

/* ---- sketch lifetime ------------------------------------------------------------- */

/* Create a set of `workers` Count Sketches of r rows x c columns sharing one hash family
 * drawn from `seed` (Sec. III-A: sketches combine by addition only when they share their
 * hash functions), plus the merged r x c table that gs_sketch_merge_tree writes.
 * All tables start at zero.  Worker tables are stored interleaved in groups of
 * `group_width` workers ([group][r][c][group_width] fp32) so that the group's values of a
 * cell are adjacent and are updated by 16-byte vector reductions (G = group_width/4 lanes
 * together write a whole cell in one instruction); group_width 0 lets the library choose
 * (up to 16, no wider than the worker count rounded up to a power of two; 16 only when the
 * whole group table fits 48 MiB of L2, and halved while one table row exceeds 64 MiB).  The
 * fused insert updates as many rows per pass as fit 48 MiB, and at least one.
 * On success *out owns device memory released by gs_sketch_destroy.
 * Errors: GS_ERR_INVALID_ARG (sizes, group_width not in {0,1,2,4,8,16}, out NULL),
 *         GS_ERR_OOM (allocation failed), GS_ERR_CUDA.  Synchronous. */
gs_status gs_sketch_create(int32_t r, int32_t c, uint64_t seed, int32_t workers,
                           int32_t group_width, gs_sketch** out);

/* Release a sketch and its device memory.  NULL is accepted.  Synchronous. */
gs_status gs_sketch_destroy(gs_sketch* sketch);

/* Shape query: any output pointer may be NULL.  rows_per_pass is the number of rows the
 * fused insert updates per pass over the vectors. */
gs_status gs_sketch_info(const gs_sketch* sketch, int32_t* r, int32_t* c, int32_t* workers,
                         int32_t* group_width, int32_t* rows_per_pass);

/* Host copy of the hash coefficients: out4r[4*j + {0,1,2,3}] = a_j, b_j, a'_j, b'_j
 * (host array of 4*r uint64).  Synchronous, no device work. */
gs_status gs_sketch_coefficients(const gs_sketch* sketch, uint64_t* out4r);

/* Zero every worker table and the merged table (start of a step). */
gs_status gs_sketch_zero(gs_sketch* sketch, gs_stream stream);

/* ---- step 1: accumulate ---------------------------------------------------------- */

/* u <- fl(fl(rho*u) + g); e <- fl(e + u) elementwise over d fp32 values, each operation
 * rounded to nearest in fp32 and never fused (momentum correction and error feedback,
 * Sec. II).  momentum and error are updated in place; grad is read only.  The three
 * arrays must not overlap. */
gs_status gs_accumulate(float* momentum, float* error, const float* grad, int64_t d,
                        float rho, gs_stream stream);

/* ---- step 2: sketch insert ------------------------------------------------------- */

/* T_worker[j][h_j(i)] += s_j(i) * vec[i] for all rows j and i < d (Alg. 1 step 5).
 * Cells are fp32 and updated with atomic additions, so their rounding order is not
 * fixed.  0 <= worker < workers. */
gs_status gs_sketch_insert(gs_sketch* sketch, int32_t worker, const float* vec, int64_t d,
                           gs_stream stream);

/* Fused steps 1+2 for workers first_worker .. first_worker+n_workers-1: for each such
 * worker p (array entry p - first_worker), gs_accumulate on (momentum, error, grad) and
 * then insert the updated error vector into T_p, in one pass over the vectors.  The
 * pointer arrays are HOST arrays of n_workers DEVICE pointers.  first_worker must be a
 * multiple of the group width, and the range must end on a group boundary or at the
 * last worker.  Per worker the result equals gs_accumulate followed by gs_sketch_insert
 * (up to the order of the fp32 atomic additions in the cells).  When the table is inserted
 * in several row passes, the first pass also accumulates and the later ones re-read the
 * updated error vectors. */
gs_status gs_accumulate_insert(gs_sketch* sketch, int32_t first_worker, int32_t n_workers,
                               float* const* momentum, float* const* error,
                               const float* const* grad, int64_t d, float rho,
                               gs_stream stream);

/* gs_accumulate_insert with the cell updates staged in shared memory: gs_accumulate for each
 * worker of the range, then one kernel per group in which every CTA holds one table row of up
 * to four of the group's workers in shared memory ([c][workers] fp32), adds a contiguous chunk
 * of the coordinates into it with shared-memory atomic additions, and flushes the tile into
 * the table with one vector reduction per touched bucket.  Same arguments, constraints and
 * result as gs_accumulate_insert (up to the order of the fp32 additions), but only for
 * sketches whose row of c cells fits a tile: c * 4 bytes <= 200 KiB (GS_ERR_INVALID_ARG
 * otherwise).  On GB300 it is slower than the direct reductions of gs_accumulate_insert at
 * every size where it applies; the library's steps use gs_accumulate_insert. */
gs_status gs_accumulate_insert_staged(gs_sketch* sketch, int32_t first_worker, int32_t n_workers,
                                      float* const* momentum, float* const* error,
                                      const float* const* grad, int64_t d, float rho,
                                      gs_stream stream);

/* ---- step 3: tree merge ---------------------------------------------------------- */

/* Merge the tables of workers 0..P-1 into the merged table by recursive halving
 * (Alg. 1 steps 8-23): in round l the workers whose rank is a multiple of 2^l take part
 * in rank order; each one at an even position adds the table of the next one to its own
 * ("sends = recvs + sends"); with an odd number of participants the largest rank sits the
 * round out (Sec. III-A).  ceil(log2 P) rounds; the fp32 additions follow exactly this
 * order for every cell.  Worker tables are left unchanged. */
gs_status gs_sketch_merge_tree(gs_sketch* sketch, int32_t P, gs_stream stream);

/* The same tree merge over P separately created sketches, for callers that keep one sketch per
 * worker (gs_sketch_create with workers = 1): the table of worker 0 of sketches[0..P-1], in that
 * rank order, is merged by the schedule of gs_sketch_merge_tree into the merged table of
 * sketches[0] (the table gs_query_topk reads).  sketches is a HOST array of P sketch pointers,
 * all on the current device.  GS_ERR_MISMATCH unless every sketch shares sketches[0]'s r, c and
 * seed; GS_ERR_INVALID_ARG for P outside [1, GS_MAX_WORKERS] or a sketch listed twice.  The
 * worker tables are left unchanged. */
gs_status gs_sketch_merge_sketches(gs_sketch* const* sketches, int32_t P, gs_stream stream);

/* ---- steps 4-5: median query and top-k ------------------------------------------- */

/* Device workspace bytes gs_query_topk needs for d coordinates and k selected. */
gs_status gs_query_topk_workspace_size(int64_t d, int64_t k, size_t* bytes);

/* From the merged table: est_i = median over rows j of s_j(i) * T[j][h_j(i)] (fp32; the
 * middle value for odd r, the mean of the two middle values for even r), then the k
 * coordinates of largest |est_i|, ties toward the smaller index, written to idx_out
 * (int64[k]) in ascending order (Alg. 2 steps 1-3).  est_out (fp32[d]) may be NULL.
 * workspace must hold gs_query_topk_workspace_size(d, k) bytes, 256-byte aligned (about
 * 12.3 bytes per coordinate: the estimate, room for a candidate list of (index, key) pairs,
 * and two d-bit bitmaps).
 * With est_out NULL, d >= 2^22, r >= 3 and c a power of two, the query may skip rows.  Rows
 * are read in order, and a coordinate stops once, with f = r/2 + 1, at least f of the cells
 * read are below a threshold t and at least f are above -t: then |est| < t whatever the
 * other rows hold, and it cannot be selected.  Its estimate is left in the workspace as the
 * marker -((32 g + n) * 2^-149): n the rows it examined (f <= n < r), g how many of those
 * cells were read from the table (where the classes of the first f rows' cells fit in shared
 * memory, f * c / 4 bytes <= 192 KiB, those cells are classified there and not read: g = n - f;
 * otherwise g = n).  The threshold is
 * taken by the same call before the main pass, from the full estimate of a fixed sample (the
 * first four coordinates of every 256): the level-1 bin edge below a rank of the sample chosen
 * so that the threshold lies under the k-th largest |est| except with negligible probability.
 * When it does not, the skipped estimates are recomputed.  idx_out is exactly the same as
 * without skipping; only the time differs.  The threshold lives in the workspace, so queries
 * on different streams with different workspaces are independent.
 * gs_step, gs_train_step, gs_step_host and gs_sketched_state_step query the same way. */
gs_status gs_query_topk(const gs_sketch* sketch, int64_t d, int64_t k, int64_t* idx_out,
                        float* est_out, void* workspace, size_t workspace_bytes,
                        gs_stream stream);

/* Device workspace bytes gs_query_heavymix needs. */
gs_status gs_query_heavymix_workspace_size(int64_t d, int64_t k, size_t* bytes);

/* HEAVYMIX selection from the merged table, as Alg. 2 prints it.  With est_i the median query
 * as in gs_query_topk and l2sq = the median over rows j of sum_b T[j][b]^2 (the sketch's
 * estimate of ||g||_2^2), H = {i : est_i^2 >= l2sq / k} and NH its complement (Alg. 2 step 2).
 * If |H| >= k the k coordinates of H with largest |est| are selected (ties to the smaller
 * index); otherwise all of H and l = k - |H| coordinates of NH drawn uniformly at random
 * (Alg. 2 step 3): those with the smallest xi_i = (i-th splitmix64 output of fill_seed) >> 33,
 * i counted from 0, ties to the smaller index.  idx_out (int64[k]) is ascending; est_out
 * (fp32[d]) and l2sq_out (one device double) may be NULL.  workspace must hold
 * gs_query_heavymix_workspace_size(d, k) bytes, 256-byte aligned.
 * With est_out NULL, d >= 2^22, r >= 3 and c a power of two, rows are skipped as in
 * gs_query_topk with t = sqrt(l2sq / k) (rounded down to a bin edge): a coordinate that stops
 * has est^2 below the threshold, so it can only enter through the fill, and its estimate is
 * left in the workspace as the marker -((32 n + n) * 2^-149), n the rows it read; idx_out is
 * the same as without skipping. */
gs_status gs_query_heavymix(const gs_sketch* sketch, int64_t d, int64_t k, uint64_t fill_seed,
                            int64_t* idx_out, float* est_out, double* l2sq_out, void* workspace,
                            size_t workspace_bytes, gs_stream stream);

/* Largest d that gs_query_topk_noalloc accepts. */
#define GS_NOALLOC_MAX_DIM (1LL << 30)

/* gs_query_topk for callers that cannot allocate device memory.  Some hosts hand a library
 * only the buffers it reads and writes: a framework whose memory pool already holds the
 * device memory (so a separate cudaMalloc would fail or escape its accounting), an
 * operator interface with no workspace argument, or a loop that must not pay for the
 * device-wide synchronisation that cudaMalloc and cudaFree can cause.  This variant
 * allocates nothing: its scratch (selection histograms, state and per-segment counters,
 * 1,073,408 bytes) is a fixed array in the library's device memory, which every GPU that
 * loads the library holds until the process exits.  The paper has no counterpart; this is
 * a service of the library, not a step of the method.
 * Same results as gs_query_topk, except that est_out is required (fp32[d], 4-byte aligned)
 * and d may not exceed GS_NOALLOC_MAX_DIM (larger d returns GS_ERR_INVALID_ARG and
 * launches nothing).  The first call on a device looks up the scratch array's device
 * address (a host-side query, no allocation); make that first call before any stream
 * capture.  Every call on a device shares the one array: each call clears the parts that
 * must start at zero, and calls whose work overlaps on the GPU (different streams, or
 * several threads) race on it, so order them on one stream. */
gs_status gs_query_topk_noalloc(const gs_sketch* sketch, int64_t d, int64_t k, int64_t* idx_out,
                                float* est_out, gs_stream stream);

/* ---- step 6: second round -------------------------------------------------------- */

/* vals_out[t] = sum over p = 0..P-1 (in that order, fp32) of error[p][idx[t]], then
 * momentum[p][idx[t]] = error[p][idx[t]] = 0 for every p (Alg. 2 step 4).  momentum and
 * error are HOST arrays of P DEVICE pointers.  idx holds k distinct indices in [0, d);
 * an index outside that range is skipped (no memory is touched) and its value is NaN. */
gs_status gs_gather_and_zero(float* const* momentum, float* const* error, int32_t P,
                             int64_t d, const int64_t* idx, int64_t k, float* vals_out,
                             gs_stream stream);

/* ---- step 7: weight update ------------------------------------------------------- */

/* w[idx[t]] <- fl(w[idx[t]] - fl(lr * vals[t])) for t < k: Alg. 1 step 26,
 * w_{t+1} = w_t - eta * G~_t, with G~_t the gathered values at the selected indices and zero
 * elsewhere (the values are sums over workers, so lr absorbs any averaging).  All workers hold
 * the same weights, so one vector is updated.  idx holds distinct indices; indices outside
 * [0, d) are skipped. */
gs_status gs_apply_update(float* weights, int64_t d, const int64_t* idx, const float* vals,
                          int64_t k, float lr, gs_stream stream);

/* gs_gather_and_zero and, when weights is not NULL, gs_apply_update with the gathered values,
 * in one kernel. */
gs_status gs_gather_zero_update(float* const* momentum, float* const* error, int32_t P,
                                int64_t d, const int64_t* idx, int64_t k, float* vals_out,
                                float* weights, float lr, gs_stream stream);

/* ---- whole step ------------------------------------------------------------------ */

/* Device workspace bytes gs_step needs (query workspace plus the step's own buffers). */
gs_status gs_step_workspace_size(int64_t d, int64_t k, size_t* bytes);

/* One full compression step for workers 0..P-1 (P = the sketch's worker count):
 * gs_sketch_zero, gs_accumulate_insert over all groups, gs_sketch_merge_tree(P),
 * gs_query_topk, gs_gather_and_zero -- all on `stream`, asynchronous.  All pointers are
 * device pointers (pointer arrays are host arrays of P device pointers); est_out may be
 * NULL. */
gs_status gs_step(gs_sketch* sketch, float* const* momentum, float* const* error,
                  const float* const* grad, int64_t d, float rho, int64_t k,
                  int64_t* idx_out, float* vals_out, float* est_out, void* workspace,
                  size_t workspace_bytes, gs_stream stream);

/* gs_step followed by the weight update of Alg. 1 step 26 (fused into the gather):
 * one training step of gs-SGD's compression and update for the simulated workers. */
gs_status gs_train_step(gs_sketch* sketch, float* weights, float lr, float* const* momentum,
                        float* const* error, const float* const* grad, int64_t d, float rho,
                        int64_t k, int64_t* idx_out, float* vals_out, float* est_out,
                        void* workspace, size_t workspace_bytes, gs_stream stream);

/* Device workspace bytes gs_heavymix_step needs. */
gs_status gs_heavymix_step_workspace_size(int64_t d, int64_t k, size_t* bytes);

/* gs_step with the HEAVYMIX selection of gs_query_heavymix (Alg. 2 steps 1-3 as printed, with
 * the fill drawn from fill_seed) in place of the deterministic top-k: gs_sketch_zero,
 * gs_accumulate_insert, gs_sketch_merge_tree, gs_query_heavymix (its estimate kept in the
 * workspace; l2sq_out, one device double, may be NULL), gs_gather_and_zero.  workspace:
 * gs_heavymix_step_workspace_size(d, k) bytes, 256-byte aligned. */
gs_status gs_heavymix_step(gs_sketch* sketch, float* const* momentum, float* const* error,
                           const float* const* grad, int64_t d, float rho, int64_t k,
                           uint64_t fill_seed, int64_t* idx_out, float* vals_out, double* l2sq_out,
                           void* workspace, size_t workspace_bytes, gs_stream stream);

/* ---- momentum and error kept as sketches ------------------------------------------ */
/* Sec. II notes that a linear sketch can carry momentum and error accumulation itself.  In
 * this variant the state is two r x c tables instead of 2P vectors of length d: the
 * merged tables of two sketches `momentum` (U) and `error` (E) created with the same r, c
 * and seed as the workers' sketch set (any worker count; only their merged tables are used,
 * and they start at zero). */

/* Device pointer of a sketch's merged table (fp32 [r][c], library-owned). */
gs_status gs_sketch_merged_table(const gs_sketch* sketch, float** table_out);

/* est_out[t] = median over rows j of s_j(idx[t]) * T[j][h_j(idx[t])] on the merged table,
 * for k coordinates (the query of Alg. 2 step 1 at given indices). */
gs_status gs_sketch_query_at(const gs_sketch* sketch, const int64_t* idx, int64_t k,
                             float* est_out, gs_stream stream);

/* merged[j][h_j(idx[t])] += scale * s_j(idx[t]) * vals[t] for every row and t < k: adds
 * scale * S(v) for the sparse vector v with vals at idx (fp32 atomic additions). */
gs_status gs_sketch_add_sparse(gs_sketch* sketch, const int64_t* idx, const float* vals,
                               int64_t k, float scale, gs_stream stream);

/* One step with sketched momentum and error:
 *   S = tree merge of S(grad[p]) over the workers' sketch set (steps 2-3 on raw gradients);
 *   U <- fl(fl(rho U) + S), E <- fl(E + U)           elementwise on the r*c cells;
 *   idx_out = the top-k of the estimate from E        (as gs_query_topk on E);
 *   vals_out = that estimate at idx_out                (delta; no per-coordinate exact
 *                                                      values exist in this variant);
 *   E <- E - S(delta), U <- U - S(delta_u), delta_u = the estimate from U at idx_out
 *                                                      (the extracted mass leaves both);
 *   weights (nullable) <- weights - lr * delta at idx_out.
 * workspace: gs_step_workspace_size(d, k) bytes.  GS_ERR_MISMATCH unless the three sketches
 * share r, c and seed. */
gs_status gs_sketched_state_step(gs_sketch* workers, gs_sketch* momentum, gs_sketch* error,
                                 const float* const* grad, int64_t d, float rho, int64_t k,
                                 int64_t* idx_out, float* vals_out, float* weights, float lr,
                                 void* workspace, size_t workspace_bytes, gs_stream stream);

/* gs_step with the gradients in HOST memory and the results returned to HOST memory, one
 * synchronous call per step.  Where the device can address grad_host[p] in place (memory
 * from cudaHostAlloc or cudaHostRegister, or any host memory on systems whose GPU has
 * pageable-memory access, such as Grace-based GB300 nodes), the fused accumulate+insert
 * kernel reads it directly over the CPU-GPU link and grad_dev[p] is left unused; otherwise
 * grad_host[p] is first copied into the device buffer grad_dev[p].  idx (int64[k]) and vals
 * (fp32[k]) are copied back to idx_host and vals_host, and `stream` is synchronized before
 * returning.  Momentum and error stay resident on the device.  workspace must hold
 * gs_step_workspace_size(d, k) bytes. */
gs_status gs_step_host(gs_sketch* sketch, float* const* momentum, float* const* error,
                       const float* const* grad_host, float* const* grad_dev, int64_t d,
                       float rho, int64_t k, int64_t* idx_host, float* vals_host,
                       void* workspace, size_t workspace_bytes, gs_stream stream);

/* ---- plans: a whole step captured once, launched many times ----------------------- */
/* A plan records one step's launch sequence (the same kernels, order and arguments as the
 * matching call above) into a CUDA graph, so that each later step is a single graph launch
 * instead of one launch per kernel and memset.  It has no counterpart in the paper: it only
 * removes host launch overhead and the gaps between dependent launches.
 *
 * A plan holds the POINTERS it was created with, not the data behind them: refill the
 * gradients in place between launches; momentum, error, sketch tables, workspace and outputs
 * are reused as in the direct calls.  All of them must stay allocated until
 * gs_plan_destroy.  The sketches must not be destroyed first.  A plan is not thread-safe.
 *
 * flags: 0, or any of GS_PLAN_TIME_INSERT, which brackets the insert phase (zeroed tables
 * excluded) with two event-record nodes, and GS_PLAN_TIME_QUERY, which records three: before
 * the median query (after its workspace is cleared), after it (its prune-key sample and repair
 * check included) and after the top-k selection.  Launch n records into slot n mod 1024 of a
 * ring of events per node; gs_plan_insert_times and gs_plan_query_times read them.
 *
 * Errors: the same argument checks as the direct call (GS_ERR_INVALID_ARG, GS_ERR_MISMATCH);
 * GS_ERR_CUDA if capture or instantiation fails (for example a host gradient that is neither
 * device-addressable nor pinned, whose upload cannot be captured).  Nothing is launched while
 * a plan is created. */
#define GS_PLAN_TIME_INSERT 1
#define GS_PLAN_TIME_QUERY 2

/* gs_step (weights == NULL) or gs_train_step (weights != NULL, with lr) as a plan. */
gs_status gs_step_plan_create(gs_sketch* sketch, float* const* momentum, float* const* error,
                              const float* const* grad, int64_t d, float rho, int64_t k,
                              int64_t* idx_out, float* vals_out, float* est_out, float* weights,
                              float lr, void* workspace, size_t workspace_bytes, int32_t flags,
                              gs_plan** plan_out);

/* gs_heavymix_step as a plan. */
gs_status gs_heavymix_step_plan_create(gs_sketch* sketch, float* const* momentum, float* const* error,
                                       const float* const* grad, int64_t d, float rho, int64_t k,
                                       uint64_t fill_seed, int64_t* idx_out, float* vals_out,
                                       double* l2sq_out, void* workspace, size_t workspace_bytes,
                                       int32_t flags, gs_plan** plan_out);

/* gs_step_host as a plan.  The uploads (where needed) and the download of idx and vals into
 * idx_host / vals_host are part of the graph; a launch does NOT synchronise: synchronise the
 * stream before reading the host outputs. */
gs_status gs_step_host_plan_create(gs_sketch* sketch, float* const* momentum, float* const* error,
                                   const float* const* grad_host, float* const* grad_dev,
                                   int64_t d, float rho, int64_t k, int64_t* idx_host,
                                   float* vals_host, void* workspace, size_t workspace_bytes,
                                   int32_t flags, gs_plan** plan_out);

/* gs_sketched_state_step as a plan. */
gs_status gs_sketched_state_plan_create(gs_sketch* workers, gs_sketch* momentum, gs_sketch* error,
                                        const float* const* grad, int64_t d, float rho, int64_t k,
                                        int64_t* idx_out, float* vals_out, float* weights, float lr,
                                        void* workspace, size_t workspace_bytes, int32_t flags,
                                        gs_plan** plan_out);

/* Enqueue one step on `stream` (asynchronous). */
gs_status gs_plan_launch(gs_plan* plan, gs_stream stream);

/* Insert-phase durations in ms of the last min(n, launches, 1024) launches, oldest first,
 * into ms_out (host); *n_out = how many.  Waits for the last launch to finish.
 * GS_ERR_INVALID_ARG if the plan was created without GS_PLAN_TIME_INSERT. */
gs_status gs_plan_insert_times(gs_plan* plan, float* ms_out, int32_t n, int32_t* n_out);

/* Median-query and selection durations in ms of the last min(n, launches, 1024) launches,
 * oldest first: query_ms_out[t] from before the query to after its repair check (steps 4),
 * select_ms_out[t] from there to after the top-k selection (steps 5), both HOST arrays of n
 * floats; *n_out = how many.  Waits for the last launch to finish.  GS_ERR_INVALID_ARG if the
 * plan was created without GS_PLAN_TIME_QUERY. */
gs_status gs_plan_query_times(gs_plan* plan, float* query_ms_out, float* select_ms_out, int32_t n,
                              int32_t* n_out);

/* Wait for the device to go idle if the plan was ever launched, then free it.  NULL is OK. */
gs_status gs_plan_destroy(gs_plan* plan);

/* ---- measurement aid --------------------------------------------------------------- */
/* The fused insert (gs_accumulate_insert over every group and row pass) is bound by the
 * requests its SMs send to L2: one cell reduction per (coordinate, row, group) and the
 * momentum and error stores, rather than by HBM bandwidth.  gs_insert_request_ceiling
 * measures the time of that request mix with HBM taken out: it runs the insert kernels of one
 * whole insert phase for d coordinates and all of the sketch's workers, with the same grids,
 * instructions, hash buckets and cell reductions, but with every vector access folded into an
 * L2-resident window (GS_CEILING_WINDOW_FLOATS floats per vector).  Not a step of the method
 * (the paper has no counterpart); it only gives the insert's roofline a measured second
 * bound.  window: a device buffer of gs_insert_request_ceiling_window_size bytes, 256-byte
 * aligned, overwritten.  The worker tables are left unspecified: zero them before the next
 * insert.  *ms_out (host) receives the elapsed time of the phase, measured with events on
 * `stream`; the call synchronizes with them.  GS_ERR_INVALID_ARG unless the group width is
 * 4, 8 or 16 and c is a power of two. */
#define GS_CEILING_WINDOW_FLOATS (1 << 17)

gs_status gs_insert_request_ceiling_window_size(const gs_sketch* sketch, size_t* bytes);

gs_status gs_insert_request_ceiling(gs_sketch* sketch, int64_t d, void* window, size_t window_bytes,
                                    float* ms_out, gs_stream stream);

/* The median query is bound by its r scattered 4-byte reads per coordinate from the merged
 * table (each one a separate sector request from L1 to L2), not by HBM.  This probe runs the
 * query kernel's loads alone for d coordinates (all r rows, the same grid and hash buckets,
 * no median, no estimate store, no histogram), so that d*r requests over *ms_out (host) is a
 * measured ceiling of that request stream.  window: at least 65536 bytes of device memory,
 * 256-byte aligned, overwritten (one float per CTA).  The call synchronizes with its events.
 * Not a step of the method.  GS_ERR_INVALID_ARG unless c is a power of two. */
gs_status gs_query_request_ceiling(const gs_sketch* sketch, int64_t d, void* window, size_t window_bytes,
                                   float* ms_out, gs_stream stream);

/* ---- inspection hooks ------------------------------------------------------------ */

/* Buckets and signs of n coordinates for every row: bucket_out[j*n + t] = h_j(coords[t]),
 * sign_out[j*n + t] = s_j(coords[t]) (int32 / int8 device arrays of r*n).  Coordinates
 * must lie in [0, 2^31); others give bucket -1 and sign 0. */
gs_status gs_hash_eval(const gs_sketch* sketch, const int64_t* coords, int64_t n,
                       int32_t* bucket_out, int8_t* sign_out, gs_stream stream);

/* Copy one table to HOST memory host_out (fp32 [r][c]): worker >= 0 gives that worker's
 * table, worker == -1 the merged table.  Synchronous (waits for all prior device work). */
gs_status gs_sketch_copy_to_host(const gs_sketch* sketch, int32_t worker, float* host_out);

/* Message for the last non-OK status returned on this thread ("" if none). */
const char* gs_last_error(void);

#ifdef __cplusplus
}
#endif

#endif /* GS_SKETCH_H */
