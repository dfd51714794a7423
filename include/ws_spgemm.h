/*
 * ws_spgemm.h -- C ABI of the GB300 (sm_103a) sparse x sparse -> sparse
 * matrix multiply, C = A * B, with A, B and C in CSR.
 *
 * The operation is the sparse product whose parallel form is Gustavson's
 * algorithm (Sec. 5.1, Fig. "SpGEMM implemented in WingSpan"): every output
 * row C[i,:] = sum over stored A[i,k] of A[i,k] * B[k,:] is owned by exactly
 * one worker, which accumulates it in a private workspace and then writes its
 * own, disjoint segment of C (the shard level of Sec. 4, used for SpGEMM in
 * Sec. 5.1).  The output must satisfy the compressed-format invariants the
 * paper singles out (Sec. 1 and Sec. 3.1: monotone prefix-sum position
 * arrays over contiguous buffers).  The calls follow the tensor lifecycle of
 * Sec. 4 (declare -> update -> freeze): a symbolic pass sizes C and fills its
 * row pointer, the caller allocates C's index and value arrays, and a numeric
 * pass fills them.
 *
 * CSR layout used by every call (0-based):
 *   rowptr  int64_t[nrows + 1], rowptr[0] = 0, non-decreasing, rowptr[nrows] = nnz
 *   colidx  int32_t[nnz], strictly increasing within each row, in [0, ncols)
 *   vals    float[nnz] or double[nnz] (ws_dtype_t)
 * All array pointers are DEVICE pointers on the current CUDA device and are
 * borrowed: the library never frees them, and the caller keeps them alive
 * until the last call that uses the handle has completed on its stream.
 *
 * Result semantics:
 *   - structure: C holds (i, j) iff some stored A[i,k] meets a stored B[k,j]
 *     (structural product; an entry whose sum is exactly zero is kept, stored
 *     zeros in A or B count as entries);
 *   - column indices of every row of C are strictly increasing;
 *   - values are accumulated in the value type of A and B; the order of the
 *     additions is unspecified (results agree with an ordered sequential sum
 *     up to rounding).
 *
 * Errors: every call returns a ws_status_t; no call throws or aborts.
 * Argument, shape and dtype errors are detected on the host before any work
 * is queued.  Failures detected by a kernel are recorded in a status word
 * that the library reads at its next synchronisation point (the end of
 * ws_spgemm_symbolic, or ws_spgemm_wait).  Kernels never trap and every
 * device loop is bounded.  ws_last_error() gives a one-line description of
 * the most recent failure on the calling thread.
 *
 * Threading: handles are not thread-safe.  One output handle serves one
 * product at a time; use separate output handles for products that run
 * concurrently.
 */
#ifndef WS_SPGEMM_H
#define WS_SPGEMM_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Same type as cudaStream_t; NULL is the legacy default stream. */
typedef struct CUstream_st* ws_stream_t;

typedef struct ws_csr_s* ws_csr_t;

typedef enum {
  WS_F32 = 1, /* float  */
  WS_F64 = 2  /* double */
} ws_dtype_t;

typedef enum {
  WS_OK = 0,
  WS_ERR_INVALID_ARG = 1, /* NULL handle/pointer, negative size, bad enum        */
  WS_ERR_INVALID_CSR = 2, /* validation found broken CSR invariants              */
  WS_ERR_SHAPE = 3,       /* operand or output shapes do not fit the operation    */
  WS_ERR_DTYPE = 4,       /* A, B and C do not share one value type              */
  WS_ERR_OVERFLOW = 5,    /* a size exceeds what the index types can hold         */
  WS_ERR_ALLOC = 6,       /* device or pinned-host allocation failed             */
  WS_ERR_CUDA = 7,        /* a CUDA runtime call failed                          */
  WS_ERR_DEVICE = 8,      /* a kernel gave up (bounded loop ran out) -- internal  */
  WS_ERR_STATE = 9        /* calls out of order (numeric before symbolic, ...)   */
} ws_status_t;

/*
 * ws_csr_create -- wraps borrowed device CSR arrays in a handle.
 *   out      receives the handle (set to NULL on failure)
 *   nrows, ncols  matrix shape, 0 <= nrows, 0 <= ncols <= INT32_MAX
 *   nnz      number of stored entries (ignored for an output handle, pass 0)
 *   rowptr   int64[nrows + 1] device array (required, also for C: the
 *            symbolic pass writes C's row pointer into it)
 *   colidx   int32[nnz] device array; may be NULL when nnz == 0 or for an
 *            output handle before ws_spgemm_numeric
 *   vals     value array of type dtype; same NULL rule as colidx
 *   dtype    WS_F32 or WS_F64
 *   validate non-zero: check the CSR invariants listed above on the device
 *            (O(nrows + nnz) work, synchronises `stream`); a violation gives
 *            WS_ERR_INVALID_CSR and no handle.  Pass 0 for an output handle.
 *   stream   stream for the validation kernel
 * The handle owns only library scratch (released by ws_csr_destroy).
 * Passage: the compressed-format invariants of Sec. 1 ("Complex Data
 * Structure Invariants": CSR is prefix sums over contiguous buffers) and
 * Sec. 3.1 (position arrays are cumulative sums that must stay monotonically
 * non-decreasing); validation checks exactly those plus sorted, in-range
 * column indices.
 */
ws_status_t ws_csr_create(ws_csr_t* out, int64_t nrows, int64_t ncols, int64_t nnz, int64_t* rowptr,
                          int32_t* colidx, void* vals, ws_dtype_t dtype, int validate,
                          ws_stream_t stream);

/*
 * ws_spgemm_symbolic -- structure pass of C = A * B.
 * Computes, for every row i, the number of distinct columns of
 * sum_k A[i,k] B[k,:], writes C.rowptr (exclusive prefix sum, C.rowptr[0] = 0)
 * into the rowptr array given to C's handle, and returns nnz(C) in *nnz_out
 * (host pointer).  C must be an output handle of shape A.nrows x B.ncols and
 * the same dtype.  Work is queued on `stream`; the call returns after the
 * stream has reached the end of the pass (it synchronises `stream`), because
 * the caller needs nnz(C) to allocate C's arrays.  The row plan (row classes,
 * per-row workspaces) is kept in C's handle for ws_spgemm_numeric.
 * Device scratch is allocated stream-ordered on `stream` and cached in C's
 * handle across calls.  The first call on a device sets the release
 * threshold of that device's default stream-ordered memory pool to its
 * maximum, so memory freed by destroyed handles stays in the pool for the
 * next ones (it is returned to the system when the process exits).
 * Passage: Sec. 5.1 (Gustavson's SpGEMM, parallel over output fibers: the
 * count of row i is the number of distinct fibers that row's worker will
 * write under the shard level) and the `declare` step of the lifecycle in
 * Sec. 4 ("Building on Finch": the output is initialised and sized before it
 * is updated).
 */
ws_status_t ws_spgemm_symbolic(ws_csr_t A, ws_csr_t B, ws_csr_t C, int64_t* nnz_out, ws_stream_t stream);

/*
 * ws_spgemm_numeric -- value pass of C = A * B.
 *   c_colidx  device int32[nnz(C)] written with C's column indices
 *   c_vals    device value array [nnz(C)] of C's dtype
 * Requires a completed ws_spgemm_symbolic for the same A, B and C (and A, B
 * unchanged since).  Asynchronous: work is queued on `stream` and the call
 * returns without waiting; device-side failures are reported by
 * ws_spgemm_wait.  The two arrays are recorded in C's handle.
 * Passage: Sec. 5.1 (Gustavson's loop: w[j] += A[i,k] * B[k,j] in a per-row
 * workspace, then row i of C is written from w in sorted column order) and
 * the `update` -> `freeze` steps of Sec. 4 (the pass updates C's disjoint row
 * segments and leaves C in read mode).
 */
ws_status_t ws_spgemm_numeric(ws_csr_t A, ws_csr_t B, ws_csr_t C, int32_t* c_colidx, void* c_vals,
                              ws_stream_t stream);

/*
 * ws_spgemm_outer_symbolic / ws_spgemm_outer_numeric -- C = A * B as the
 * outer-product SpGEMM (Sec. 5.1, Fig. "SpGEMM implemented in WingSpan",
 * outer product, with the merge level and its coalesce step of Sec. 4): the
 * k range is split into `parts` contiguous blocks K_p; block p contributes the
 * partial product A[:, K_p] * B[K_p, :] (a worker's own copy of C) and the
 * copies are coalesced by pairwise sparse additions.  C's structure equals
 * the row-wise product's (a sum of exactly 0.0 is kept); values agree up to
 * summation order (sums per block, then block sums).
 *   parts  >= 1 (clamped to the number of columns of A; 1 is the row-wise
 *          product itself), else WS_ERR_INVALID_ARG
 * Same two-pass contract as ws_spgemm_symbolic / ws_spgemm_numeric: the
 * symbolic call writes C.rowptr, returns nnz(C) and synchronises `stream`;
 * it computes every block's partial product and every merge except the value
 * pass of the last one, in library-owned scratch allocated stream-ordered on
 * `stream` (B's row blocks are views of B, A's column blocks share one buffer
 * of nnz(A) entries).  The numeric call (asynchronous) writes C's column
 * indices and values and releases that scratch stream-ordered.  A and B must
 * stay unchanged in between.  Errors as for the row-wise calls; a device-side
 * failure in any step gives WS_ERR_DEVICE.
 */
ws_status_t ws_spgemm_outer_symbolic(ws_csr_t A, ws_csr_t B, ws_csr_t C, int parts, int64_t* nnz_out,
                                     ws_stream_t stream);
ws_status_t ws_spgemm_outer_numeric(ws_csr_t A, ws_csr_t B, ws_csr_t C, int32_t* c_colidx, void* c_vals,
                                    ws_stream_t stream);

/* Elementwise operations (Sec. 5.2, "Sparse Linear Algebra": C = A op B). */
typedef enum {
  WS_EWISE_ADD = 1, /* SpAdd: C = A + B on the union of the two patterns            */
  WS_EWISE_MUL = 2  /* Hadamard product: C = A .* B on the intersection of the two */
} ws_ewise_op_t;

/*
 * ws_ewise_symbolic -- structure pass of the elementwise operation C = A op B
 * (Sec. 5.2, "Sparse Linear Algebra", where SpAdd and the Hadamard product
 * use the sharded sparse list: distinct rows of C go to distinct workers).
 *   op   WS_EWISE_ADD: C holds (i, j) iff A or B stores (i, j), with
 *        C[i,j] = A[i,j] + B[i,j] (a missing entry contributes nothing; a sum
 *        of exactly 0.0 is kept);
 *        WS_EWISE_MUL: C holds (i, j) iff both store (i, j), with
 *        C[i,j] = A[i,j] * B[i,j].
 * A and B have the same shape and dtype; C is an output handle of that shape
 * and dtype.  Writes C.rowptr into the rowptr array of C's handle and returns
 * nnz(C) in *nnz_out (host pointer).  Work is queued on `stream` and the call
 * synchronises it (the caller needs nnz(C) to allocate C).  The chunk plan
 * (rows cut into pieces of their merged column lists) is kept in C's handle
 * for ws_ewise_numeric; device scratch is allocated stream-ordered on
 * `stream` and cached in the handle.  Errors: WS_ERR_SHAPE, WS_ERR_DTYPE,
 * WS_ERR_INVALID_ARG (NULL pointer, unknown op), WS_ERR_DEVICE (a kernel found
 * inconsistent input, e.g. unsorted columns).
 */
ws_status_t ws_ewise_symbolic(ws_csr_t A, ws_csr_t B, ws_csr_t C, int op, int64_t* nnz_out, ws_stream_t stream);

/*
 * ws_ewise_numeric -- value pass of C = A op B.
 *   c_colidx  device int32[nnz(C)] written with C's column indices
 *   c_vals    device value array [nnz(C)] of C's dtype
 * Requires a completed ws_ewise_symbolic for the same A, B and C (A and B
 * unchanged since).  Asynchronous on `stream`; device-side failures are
 * reported by ws_spgemm_wait.  Values are computed in the value type: one
 * rounding per entry.
 */
ws_status_t ws_ewise_numeric(ws_csr_t A, ws_csr_t B, ws_csr_t C, int32_t* c_colidx, void* c_vals,
                             ws_stream_t stream);

/*
 * ws_spmspv -- sparse matrix - sparse vector product y = A x (Sec. 5.2,
 * "Sparse Linear Algebra": SpMSpV, where x's stored entries select columns of
 * A and the columns are accumulated into a sparse byte-map over y that a
 * merge level protects).
 *   At      handle of A^T in CSR, i.e. A by columns: At is n x m for an m x n
 *           A, and row j of At lists the rows i of A's entries in column j
 *           (ascending) with their values
 *   nnz_x   stored entries of x, 0 <= nnz_x <= n
 *   x_idx   device int32[nnz_x], strictly increasing, in [0, n)
 *   x_vals  device values [nnz_x] of At's dtype
 *   y_idx   device int32[m] (capacity m): receives y's indices, increasing
 *   y_vals  device values [m] of At's dtype: receives y's values
 *   nnz_y   host pointer: receives the number of stored entries of y
 * y holds i iff some stored A[i,j] has j stored in x (structural: a sum of
 * exactly 0.0 is kept), y[i] = sum of A[i,j] x[j] accumulated in the value
 * type in unspecified order.  Work is queued on `stream` and the call
 * synchronises it (to return nnz_y).  Device scratch (an accumulator and a
 * byte-map of length m, offsets per x entry) is allocated stream-ordered and
 * cached in At's handle.  Errors: WS_ERR_INVALID_ARG (NULL pointers, nnz_x out
 * of range), WS_ERR_DEVICE (an index of x or of At out of range: those entries
 * are skipped and flagged).
 */
ws_status_t ws_spmspv(ws_csr_t At, int64_t nnz_x, const int32_t* x_idx, const void* x_vals, int32_t* y_idx,
                      void* y_vals, int64_t* nnz_y, ws_stream_t stream);

/*
 * ws_csr_submatrix_symbolic / ws_csr_submatrix_numeric -- S = A[r0:r1, c0:c1]
 * as a CSR matrix of shape (r1 - r0) x (c1 - c0) with columns shifted by -c0.
 * This is the layout step of the outer-product SpGEMM (Sec. 5.1, Fig.
 * "SpGEMM implemented in WingSpan": the k loop split over workers, worker p
 * multiplying the column block A[:, K_p] by the row block B[K_p, :] into its
 * own copy of C before a merge level coalesces the copies).
 *   0 <= r0 <= r1 <= A.nrows, 0 <= c0 <= c1 <= A.ncols (else WS_ERR_INVALID_ARG)
 *   S   output handle of shape (r1 - r0) x (c1 - c0) and A's dtype
 * The symbolic call writes S.rowptr and returns nnz(S) (it synchronises
 * `stream`); the numeric call (asynchronous) fills the caller's s_colidx
 * (int32[nnz(S)]) and s_vals from the same A, unchanged in between.
 */
ws_status_t ws_csr_submatrix_symbolic(ws_csr_t A, int64_t r0, int64_t r1, int64_t c0, int64_t c1, ws_csr_t S,
                                      int64_t* nnz_out, ws_stream_t stream);
ws_status_t ws_csr_submatrix_numeric(ws_csr_t A, ws_csr_t S, int32_t* s_colidx, void* s_vals, ws_stream_t stream);

/*
 * ws_spgemm_wait -- synchronises `stream` and returns the device status
 * recorded by the last symbolic/numeric pass of C (WS_OK if none failed);
 * serves the elementwise passes too.
 */
ws_status_t ws_spgemm_wait(ws_csr_t C, ws_stream_t stream);

/*
 * ws_csr_destroy -- releases the handle and the scratch it owns (never the
 * borrowed arrays).  NULL-safe.  Synchronises the device if the handle owns
 * scratch, so pending work that uses it completes first; device scratch goes
 * back to the stream-ordered pool and the pinned host summary to a
 * process-wide free list.
 * Passage: the end of the lifecycle of Sec. 4 ("Building on Finch"): once C is
 * frozen, the workspaces the passes declared are no longer needed.  The
 * paper has no explicit release call; this one frees the library's share.
 */
ws_status_t ws_csr_destroy(ws_csr_t handle);

/* Short static description of a status code. */
const char* ws_status_string(ws_status_t status);

/* One-line description of the most recent failure on the calling thread ("" if none). */
const char* ws_last_error(void);

/*
 * ws_csr_nnz -- number of entries of a handle (for C: nnz(C) after symbolic,
 * -1 before).  Returns WS_ERR_INVALID_ARG for a NULL handle or pointer.
 */
ws_status_t ws_csr_nnz(ws_csr_t handle, int64_t* nnz_out);

/*
 * ws_spgemm_plan_info -- counts from the last symbolic pass of C, for
 * diagnostics and tests: info[0] empty rows, info[1] single-entry (direct
 * copy) rows, info[2] hash rows, info[3] hash rows re-routed to the sorting
 * path, info[4] dense-window rows, info[5] dense-window slices,
 * info[6] total products (sum over rows of the product count),
 * info[7] number of kernel launches queued by the last symbolic pass,
 * info[8] number queued by the last numeric pass, info[9] bitmap rows,
 * info[10] heavy rows on the dense column-slice path, info[11] heavy rows
 * on the wide-bitmap path.
 * `n` is the length of `info` (at most 12 values are written).
 */
ws_status_t ws_spgemm_plan_info(ws_csr_t C, int64_t* info, int n);

/*
 * ws_set_tuning -- test/diagnostic knob, process-wide.
 *   key 1: largest product count of a row that uses the shared-memory hash
 *          path (default 4096; smaller values send more rows to the
 *          dense-window path, 0 sends every multi-entry row there)
 *   key 2: longest run of occupied slots a row's hash table may hold
 *          (default 64; a row with a longer run, or whose probes wrap
 *          around the table, uses the sorting path; smaller values send
 *          more rows there)
 *   key 3: dense-window slice width in columns (default 8192 for double,
 *          16384 for float; must be a multiple of 1024, 0 = default)
 *   key 4: widest column range of a row that uses the bitmap path
 *          (default and maximum 65536; 0 disables the bitmap path)
 *   key 5: most stored A entries of a row that uses the one-warp register
 *          bitmap path (default and maximum 16; 0 disables that path)
 *   key 6: most stored A entries of a heavy row that uses the dense
 *          column-slice path (default and maximum 8192; 0 disables it)
 *   key 7: widest column range of a heavy row that uses the wide-bitmap path
 *          (default and maximum 1048576; 0 disables it)
 *   key 8: elementwise operations, lanes per row chunk: -1 (default:
 *          automatic, 2 for rows averaging under 64 merged entries, 64
 *          otherwise), 1 (one thread merges a chunk entry by entry from
 *          global memory), 2 (the same from shared-memory copies of the
 *          input runs of a warp's 32 chunks, chunks of at most 16 merged
 *          entries), 4, 8, 16 or 32 (a lane group merges windows of that
 *          many entries), 0 (lane group sized from the mean row length), 64
 *          (a warp per 64-entry chunk ranks every entry by binary search)
 *   key 9: elementwise operations with one lane per chunk: merged entries
 *          per chunk (default 64, range [2, 1048576]; with key 8 = 2 at
 *          most 16 are used)
 * Returns WS_ERR_INVALID_ARG for an unknown key or out-of-range value.
 */
ws_status_t ws_set_tuning(int key, int64_t value);

/*
 * ws_rowptr_scan_static -- builds a CSR row pointer from per-row counts
 * without allocating any memory.  (The paper has no counterpart: this is a
 * service for callers of this library that cannot allocate device memory at
 * this point, for example code inside a framework that owns all device
 * memory and forbids outside allocations, or a latency-critical loop where
 * cudaMalloc/cudaFree would block on the whole device.)
 *   rowptr  device int64[nrows + 1]; on entry rowptr[i + 1] holds the entry
 *           count of row i (rowptr[0] is ignored); on exit rowptr[0] = 0 and
 *           rowptr[i + 1] = rowptr[i] + count_i, so rowptr[nrows] = nnz.
 *   nrows   0 <= nrows <= 16,777,216 (the fixed scratch holds one partial
 *           sum per 4096 rows); larger values return WS_ERR_OVERFLOW.
 *   stream  the work is queued on it; the call does not wait.
 * Scratch lives in a fixed array compiled into the library (about 33 KB),
 * which every GPU that loads the library keeps until the process exits.  The
 * call itself calls no cudaMalloc, cudaFree or other allocating routine.
 * The first call on a device looks up that array's device address and
 * keeps it for the life of the process; make that first call before any
 * stream capture, and do not call this function again on a device after
 * cudaDeviceReset (or anything else that destroys the device's primary
 * context), because the kept address then names freed memory.  All calls
 * share the array:
 * calls that may run at the same time on the GPU (on unordered streams) race
 * and give wrong results.  Returns WS_ERR_INVALID_ARG for a NULL rowptr or a
 * negative nrows, WS_ERR_CUDA if a CUDA call fails.
 */
ws_status_t ws_rowptr_scan_static(int64_t* rowptr, int64_t nrows, ws_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* WS_SPGEMM_H */
