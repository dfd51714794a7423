// Internal declarations shared by the CUDA translation units of the SpGEMM library.
//
// Row classes.  The symbolic pass sorts every output row i of C = A*B into one
// class by its product count ub_i = sum over stored A[i,k] of |B[k,:]| (the
// work of the row, which is data dependent and unknown before the pass --
// the load-balance problem of Sec. 1):
//   empty         ub_i = 0                       -> no output
//   direct        exactly one stored A[i,k]      -> C[i,:] = A[i,k] * B[k,:]
//   bitmap bin b  column range of the row at most 32 << log_words(b) columns and
//                 min(ub_i, range) <= cap(b)     -> bitmap + rank workspace
//   hash bin b    ub_i <= 32 << b (b = 0..7)     -> shared-memory hash workspace of
//                                                  64 << b slots, sort-free ranking
//   sort          a hash row whose table showed a long run of occupied slots
//                 (or wrapped) -> shared-memory hash + bitonic sort
//   dense window  ub_i above the hash limit      -> column slices of the row, each a
//                                                  dense bitmap + value workspace
// Each class is a different realisation of the per-row workspace w of
// Gustavson's algorithm (Sec. 5.1); every row is written by exactly one
// thread team (or, for dense-window rows, each column slice by one team),
// so C's segments are disjoint (the shard pattern, Sec. 4).
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

namespace wsk {

constexpr int kNumHashBins = 8;
constexpr int kMinHashLog = 6;  // bin b uses a table of 1 << (kMinHashLog + b) slots
constexpr int kMaxHashProducts = 32 << (kNumHashBins - 1);  // 4096

// Bitmap bins: bitmap of 1 << log_words 32-bit words (the row's column range
// is at most 32 << log_words columns) and a staging array of cap entries.
struct BitmapBin {
  int log_words;
  int cap;
};
constexpr int kNumBitmapBins = 5;
constexpr BitmapBin kBitmapBins[kNumBitmapBins] = {{6, 256}, {9, 512}, {11, 512}, {11, 1024}, {11, 8192}};
constexpr int kMaxBitmapSpan = 32 << 11;  // 65,536 columns
__host__ __device__ constexpr int bitmap_log_words(int b) {
  return b == 0 ? kBitmapBins[0].log_words : b == 1 ? kBitmapBins[1].log_words : b == 2 ? kBitmapBins[2].log_words
       : b == 3 ? kBitmapBins[3].log_words : kBitmapBins[4].log_words;
}
__host__ __device__ constexpr int bitmap_cap(int b) {
  return b == 0 ? kBitmapBins[0].cap : b == 1 ? kBitmapBins[1].cap : b == 2 ? kBitmapBins[2].cap
       : b == 3 ? kBitmapBins[3].cap : kBitmapBins[4].cap;
}

// Register bitmap bins: rows with at most kBmrMaxA stored A entries whose B
// rows fit one lane group; bitmap of 1 << bmr_log_words(b) words (column
// ranges of at most 4096, 16,384 and 65,536 columns).
constexpr int kNumBmrBins = 3;
constexpr int kBmrPlannedBin = kNumBmrBins;  // launch_bmr: numeric pass of the rows ranked by the planning pass
constexpr int kBmrMaxA = 16;
constexpr int kBmrCap = 512;  // >= kBmrMaxA * 32 products
constexpr int kBmrSlots = 512;  // rank slots per register bitmap row (one per possible product)
__host__ __device__ constexpr int bmr_log_words(int b) { return b == 0 ? 7 : b == 1 ? 9 : 11; }
// Smallest register bitmap bin whose bitmap covers `span` columns (span <= kMaxBitmapSpan).
__host__ __device__ constexpr int bmr_bin_for_span(long long span) {
  return span <= (32ll << bmr_log_words(0)) ? 0 : span <= (32ll << bmr_log_words(1)) ? 1 : 2;
}

// Row class codes stored per row (uint8).
constexpr uint8_t kClsEmpty = 0;
constexpr uint8_t kClsDirect = 1;
constexpr uint8_t kClsBmr0 = 2;                            // .. + kNumBmrBins - 1
constexpr uint8_t kClsBitmap0 = kClsBmr0 + kNumBmrBins;    // .. + kNumBitmapBins - 1
constexpr uint8_t kClsHash0 = kClsBitmap0 + kNumBitmapBins;  // .. + kNumHashBins - 1
constexpr uint8_t kClsDense = kClsHash0 + kNumHashBins;
constexpr uint8_t kClsSort = kClsDense + 1;
constexpr uint8_t kClsBmrWide = kClsSort + 1;  // register bitmap rows counted by the planning pass
constexpr uint8_t kClsRcd = kClsBmrWide + 1;    // heavy rows, dense column-slice workspace, CTA per row
constexpr uint8_t kClsWb = kClsRcd + 1;         // heavy rows, wide bitmap workspace, CTA per row

// Heavy-row limits.
constexpr int kRcdMaxA = 8192;            // stored A entries a dense row may have (cursor slots)
constexpr int kRcdDefaultMaxA = 8192;     // default limit used by the classification
constexpr int kRcdWidthBytes = 65536;     // dense value window per slice
// Dense-window slices of a dense heavy row (its span is at most kMaxBitmapSpan columns).
template <typename T>
constexpr int rcd_slices() {
  return (kMaxBitmapSpan + kRcdWidthBytes / static_cast<int>(sizeof(T)) - 1) / (kRcdWidthBytes / static_cast<int>(sizeof(T)));
}
constexpr int kWbMaxSpan = 1 << 20;       // widest column range of a wide-bitmap row

// Segments of the row permutation: direct rows, register bitmap bins, bitmap
// bins, hash bins, dense-window rows.
constexpr int kSegDirect = 0;
constexpr int kSegBmr0 = 1;
constexpr int kSegBitmap0 = kSegBmr0 + kNumBmrBins;
constexpr int kSegHash0 = kSegBitmap0 + kNumBitmapBins;
constexpr int kSegDense = kSegHash0 + kNumHashBins;
constexpr int kSegBmrWide = kSegDense + 1;
constexpr int kSegRcd = kSegBmrWide + 1;
constexpr int kSegWb = kSegRcd + 1;
constexpr int kNumSegs = kSegWb + 1;

// Device error flags (OR-ed into DevSummary::status).
enum DevError : int {
  kErrProbe = 1,       // a hash insert ran through a whole table (cannot happen at load <= 1/2)
  kErrRank = 2,        // a run of occupied slots longer than the ranking limit in the numeric pass
  kErrCount = 4,       // the numeric pass found a different entry count than the symbolic pass
  kErrInvalidCsr = 8,  // validation found broken CSR invariants
  kErrSortCap = 16,    // a sort-path row exceeded its workspace
};

// Counters shared between the kernels of one product and read back by the host.
struct DevSummary {
  long long nnz;       // nnz(C), written by the scan
  long long products;  // sum of ub_i
  long long dense_slices;
  long long slice_cursor;
  long long rcd_mega_entries;  // stored A entries of the dense heavy rows split into (row, slice) items
  int status;
  int n_sort;
  int n_long;   // rows analysed by a CTA each (queued from the back of the long-row list)
  int n_mid;    // rows analysed by a warp each (queued from the front)
  int n_empty;
  int bad_row;
  int n_pending;  // rows the planning pass left to the analysis kernel
  int seg_count[kNumSegs];
  int seg_cursor[kNumSegs];
};

// Read-only view of an input CSR matrix.
template <typename T>
struct CsrView {
  const int64_t* rowptr;
  const int32_t* colidx;
  const T* vals;
};

// Everything the row kernels need about one product.
template <typename T>
struct RowPlan {
  CsrView<T> A;
  CsrView<T> B;
  int64_t* c_rowptr;   // C.rowptr; symbolic writes counts to [i + 1] then scans in place
  int32_t* c_colidx;   // numeric only
  T* c_vals;           // numeric only
  int32_t* perm;       // rows grouped by segment
  uint8_t* cls;        // row class per row
  int32_t* lo;         // smallest column any product of the row can hit
  int32_t* hi;         // largest such column
  int32_t* sort_list;  // rows rerouted to the sorting path
  const int32_t* slice_row;    // dense-window slices: row, slice index, first slice of the row
  const int32_t* slice_idx;
  const int32_t* slice_first;
  int32_t* slice_cnt;          // entries per dense-window slice
  uint16_t* ranks;             // register bitmap rows: output position of every product, kBmrSlots per row
  int32_t* rcd_scnt;           // dense heavy rows: entries per dense-window slice, rcd_slices<T>() per row
  int32_t* rcd_mega;           // dense heavy rows with more than 256 stored A entries (segment positions)
  int32_t* rcd_nmega;          // their number
  int32_t* rcd_ctr;            // two work counters of the numeric kernel (zeroed before it)
  int64_t* rcd_moff;           // per mega row: first of its entries in the slice-start table
  int32_t* rcd_mna;            // per mega row: its stored A entries when the table was sized
  int32_t* rcd_bnd;            // slice-start table of the mega rows' B rows (numeric only)
  DevSummary* sum;
  int64_t seg_begin;   // first position in perm of the segment a kernel processes
  int64_t seg_len;     // rows in that segment
  int log2_group;      // lanes per stored A entry when walking B rows (1 << log2_group)
  int run_limit;       // longest occupied run a hash row may hold (longer: sorting path)
  int dense_width;     // dense-window slice width in columns
};

// Elementwise operations C = A op B on CSR matrices of one shape.
constexpr int kEwiseAdd = 1;  // SpAdd: pattern union, values added
constexpr int kEwiseMul = 2;  // Hadamard product: pattern intersection, values multiplied
constexpr int kEwiseRankGroup = 64;  // EwisePlan::group of the warp-per-chunk ranking kernels
constexpr int kEwiseTileGroup = 2;   // EwisePlan::group of the warp-staged tile kernels (a lane per chunk)
constexpr int kEwiseTileDiag = 16;   // their largest chunk (merged positions)
constexpr int kEwiseRankChunk = 64;  // their merged positions per chunk

template <typename T>
struct EwisePlan {
  CsrView<T> A;
  CsrView<T> B;
  int64_t m;
  int64_t* c_rowptr;
  int32_t* c_colidx;     // numeric only
  T* c_vals;             // numeric only
  int64_t* chunk_begin;  // [m + 1]: first chunk of each row (chunks per row, then scanned in place)
  int32_t* chunk_row;    // [nc_max]: row of each chunk
  int64_t* chunk_off;    // [nc_max + 1]: C offset of each chunk (counts, then scanned in place)
  int64_t* chunk_split;  // [nc_max + 1]: 2 * (A entries before the chunk) + (1 if an equal pair straddles its start);
                         // warp-staged tiles: the chunk's first position in A's arrays ([nc]: the end of A)
  int64_t* chunk_bpos;   // [nc_max + 1]: warp-staged tiles: the chunk's first position in B's arrays
  int64_t nc_max;        // bound on the number of chunks: m + (nnz(A) + nnz(B)) / diag + 1
  int64_t* partials;     // scan scratch for max(m, nc_max) entries
  DevSummary* sum;
  int64_t diag;          // merged positions per chunk
  int group;             // lanes per chunk (1: one thread merges entry by entry; kEwiseTileGroup: the same
                         // from shared-memory copies of a warp's 32 chunks; 4, 8, 16, 32: windows;
                         // kEwiseRankGroup: a warp per chunk ranks every entry by binary search)
  int op;                // kEwiseAdd or kEwiseMul
};
template <typename T>
void launch_ewise_symbolic(const EwisePlan<T>& p, int num_sms, cudaStream_t s, int* launches);
template <typename T>
void launch_ewise_numeric(const EwisePlan<T>& p, int num_sms, cudaStream_t s, int* launches);

// Sparse matrix - sparse vector product y = A x, A given by columns (At = A^T in CSR).
template <typename T>
struct SpmspvPlan {
  CsrView<T> At;         // n x m: row j holds column j of A
  int64_t n;             // columns of A (rows of At)
  int64_t m;             // rows of A = length of y
  int64_t nnz_a;
  int64_t nx;            // stored entries of x
  const int32_t* x_idx;  // strictly increasing in [0, n)
  const T* x_vals;
  int64_t* off;          // [nx + 1]: products per x entry, then scanned in place
  int64_t* first;        // [nx]: first entry of each x entry's column in At
  T* acc;                // [m]: dense accumulator (zeroed by the host)
  uint8_t* mark;         // [tiles * 4096]: 1 at the positions of y hit (zeroed by the host)
  int64_t* cnt;          // [tiles + 1]: set bits per compaction tile, then scanned in place
  int64_t* partials;     // scan scratch for max(nx, tiles) entries
  DevSummary* sum;
  int32_t* y_idx;        // [cap]
  T* y_vals;             // [cap]
  int64_t cap;           // capacity of y (m)
};
int64_t spmspv_tiles(int64_t m);
template <typename T>
void launch_spmspv(const SpmspvPlan<T>& p, int num_sms, cudaStream_t s, int* launches);

// Submatrix S = A[r0:r1, c0:c1]: per-row counts into s_rowptr[1..rows], then the copy.
void launch_submatrix_count(const int64_t* rowptr, const int32_t* colidx, int64_t r0, int64_t rows, int64_t c0,
                            int64_t c1, int64_t* s_rowptr, int num_sms, cudaStream_t s, int* launches);
template <typename T>
void launch_submatrix_copy(const int64_t* rowptr, const int32_t* colidx, const T* vals, int64_t r0, int64_t rows,
                           int64_t c0, const int64_t* s_rowptr, int32_t* s_colidx, T* s_vals, DevSummary* sum,
                           int num_sms, cudaStream_t s, int* launches);

// Host-side launchers (one translation unit each).
struct AnalyzeParams {
  int64_t m;
  int64_t hash_max;    // largest ub that uses a hash bin
  int64_t bitmap_span; // largest column range that uses a bitmap bin (0: none)
  int group;           // lanes per stored A entry in the register bitmap kernels
  int bmr_max_a;       // most stored A entries of a register bitmap row (0: none)
  int rcd_max_a;       // most stored A entries of a dense heavy row (0: no dense heavy rows)
  int64_t wb_span;     // widest column range of a wide-bitmap heavy row (0: none)
  int dense_width;
  int long_threshold;
};
// rows == nullptr: every row of A; otherwise the first sum->n_pending entries of rows.
template <typename T>
void launch_analyze(const RowPlan<T>& p, const AnalyzeParams& ap, int32_t* long_rows, const int32_t* rows,
                    int num_sms, cudaStream_t s, int* launches);
template <typename T>
void launch_bmr_plan(const RowPlan<T>& p, const AnalyzeParams& ap, int64_t ncols, int32_t* pending, int num_sms,
                     cudaStream_t s, int* launches);
template <typename T>
void launch_scatter(const RowPlan<T>& p, int64_t m, const int64_t* seg_offset, int num_sms, cudaStream_t s,
                    int* launches);
template <typename T>
void launch_dense_slices(const RowPlan<T>& p, int32_t* slice_row, int32_t* slice_idx, int32_t* slice_first,
                         int num_sms, cudaStream_t s, int* launches);
template <typename T>
void launch_hash(const RowPlan<T>& p, int bin, bool numeric, int num_sms, cudaStream_t s, int* launches);
template <typename T>
void launch_bmr(const RowPlan<T>& p, int bin, bool numeric, int num_sms, cudaStream_t s, int* launches);
template <typename T>
void launch_bitmap(const RowPlan<T>& p, int bin, bool numeric, int num_sms, cudaStream_t s, int* launches);
template <typename T>
void launch_rcd(const RowPlan<T>& p, bool numeric, int num_sms, cudaStream_t s, int* launches);
template <typename T>
void launch_rcd_bounds(const RowPlan<T>& p, int num_sms, cudaStream_t s, int* launches);
template <typename T>
void launch_wb(const RowPlan<T>& p, bool numeric, int num_sms, cudaStream_t s, int* launches);
template <typename T>
void launch_dense(const RowPlan<T>& p, int64_t nslices, bool numeric, int num_sms, cudaStream_t s,
                  int* launches);
template <typename T>
void launch_direct(const RowPlan<T>& p, int num_sms, cudaStream_t s, int* launches);
template <typename T>
void launch_sort(const RowPlan<T>& p, int64_t nrows, int num_sms, cudaStream_t s, int* launches);

// skip != nullptr: the scan does nothing when *skip != 0 (read on the device).
void launch_scan(int64_t* rowptr, int64_t m, int64_t* partials, DevSummary* sum, cudaStream_t s, int* launches,
                 const int* skip = nullptr);
int64_t scan_partials_needed(int64_t m);

void launch_validate(const int64_t* rowptr, const int32_t* colidx, int64_t nrows, int64_t ncols, int64_t nnz,
                     DevSummary* sum, int num_sms, cudaStream_t s);

// Dynamic shared memory needed by the dense-window kernel and the sort kernel.
size_t dense_smem_bytes(int width, size_t value_bytes, bool numeric);
size_t sort_smem_bytes(size_t value_bytes);
constexpr int kSortTableLog = 13;  // sort path: 8192-slot table, up to 4096 entries

// Exclusive prefix sum over the threads of a CTA of blockDim.x threads
// (a multiple of 32, at most 1024).  `scratch` holds 32 values; returns this
// thread's exclusive prefix and stores the CTA total in *total.  Every thread
// of the CTA must call it.
template <typename V>
__device__ __forceinline__ V block_exclusive_scan(V x, V* scratch, V* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
  V incl = x;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const V y = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += y;
  }
  if (lane == 31) scratch[warp] = incl;
  __syncthreads();
  if (warp == 0) {
    V w = lane < nwarps ? scratch[lane] : V(0);
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const V y = __shfl_up_sync(0xffffffffu, w, o);
      if (lane >= o) w += y;
    }
    if (lane < nwarps) scratch[lane] = w;  // inclusive scan of warp totals
  }
  __syncthreads();
  const V warp_prefix = warp > 0 ? scratch[warp - 1] : V(0);
  *total = scratch[nwarps - 1];
  __syncthreads();
  return warp_prefix + incl - x;
}

}  // namespace wsk
