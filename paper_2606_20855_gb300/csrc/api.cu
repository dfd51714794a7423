// C ABI of the SpGEMM library (declared in include/ws_spgemm.h).
//
// Symbolic pass (ws_spgemm_symbolic), all on the caller's stream:
//   1. analyze   per-row product count, column range, class       (2 launches)
//   -- read the class counts back (one small copy + stream sync)
//   2. scatter   group rows by class                                (1 launch)
//   3. dense     expand dense-window rows into column slices, count (2 launches)
//   4. hash      count distinct columns per hash bin                (1 launch per non-empty bin)
//   5. scan      counts -> C.rowptr                                 (3 launches)
//   -- read nnz(C) and the status word back (one small copy + stream sync)
// Numeric pass (ws_spgemm_numeric): one launch per non-empty class, no sync.
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <new>
#include <string>
#include <vector>

#include "ws_internal.cuh"
#include "ws_spgemm.h"

using namespace wsk;

namespace {

thread_local std::string g_last_error;

// Process-wide tuning (ws_set_tuning).
int64_t g_hash_max = kMaxHashProducts;
int64_t g_bitmap_span = kMaxBitmapSpan;
int g_bmr_max_a = kBmrMaxA;
int g_rcd_max_a = kRcdDefaultMaxA;
int64_t g_wb_span = kWbMaxSpan;
int g_run_limit = 64;
int g_dense_width = 0;  // 0 = default per value type
int g_ewise_lanes = -1;  // elementwise: lanes per chunk (0 = lane groups from the mean row length, -1 = automatic)
int64_t g_ewise_diag = 64;  // elementwise, one thread per chunk: merged positions per chunk
constexpr int kLongRowThreshold = 16;  // rows with more stored entries are analysed by a warp or a CTA

ws_status_t fail(ws_status_t st, const char* fmt, ...) __attribute__((format(printf, 2, 3)));
ws_status_t fail(ws_status_t st, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  g_last_error = buf;
  return st;
}

ws_status_t cuda_fail(cudaError_t e, const char* what) {
  return fail(WS_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

#define WS_CUDA(call, what)                     \
  do {                                          \
    cudaError_t e_ = (call);                    \
    if (e_ != cudaSuccess) return cuda_fail(e_, what); \
  } while (0)

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// Grow-only stream-ordered device buffer.
struct DevBuf {
  void* ptr = nullptr;
  size_t bytes = 0;
  ws_status_t reserve(size_t need, cudaStream_t s) {
    if (need <= bytes) return WS_OK;
    if (ptr) {
      cudaError_t e = cudaFreeAsync(ptr, s);
      ptr = nullptr;
      bytes = 0;
      if (e != cudaSuccess) return cuda_fail(e, "cudaFreeAsync");
    }
    size_t want = need + need / 8;
    cudaError_t e = cudaMallocAsync(&ptr, want, s);
    if (e != cudaSuccess) {
      ptr = nullptr;
      return fail(WS_ERR_ALLOC, "cudaMallocAsync(%zu bytes): %s", want, cudaGetErrorString(e));
    }
    bytes = want;
    return WS_OK;
  }
  // Returns the memory to the stream-ordered pool (callers synchronise the
  // device first, so no queued work still uses it).
  void release() {
    if (ptr) cudaFreeAsync(ptr, nullptr);
    ptr = nullptr;
    bytes = 0;
  }
};

// Pinned host copies of the summary block, recycled across handles: a
// cudaMallocHost / cudaFreeHost pair per handle costs more than a small
// product.  Blocks are allocated 64 at a time and kept until the process
// exits.
std::mutex g_host_sum_mutex;
std::vector<DevSummary*> g_host_sum_free;

DevSummary* acquire_host_sum() {
  std::lock_guard<std::mutex> lock(g_host_sum_mutex);
  if (g_host_sum_free.empty()) {
    constexpr int kBlocks = 64;
    const size_t each = (sizeof(DevSummary) + 255) / 256 * 256;
    char* base = nullptr;
    if (cudaMallocHost(reinterpret_cast<void**>(&base), each * kBlocks) != cudaSuccess) return nullptr;
    for (int i = kBlocks - 1; i >= 0; --i) g_host_sum_free.push_back(reinterpret_cast<DevSummary*>(base + i * each));
  }
  DevSummary* h = g_host_sum_free.back();
  g_host_sum_free.pop_back();
  return h;
}

void release_host_sum(DevSummary* h) {
  if (!h) return;
  std::lock_guard<std::mutex> lock(g_host_sum_mutex);
  g_host_sum_free.push_back(h);
}

// Once per device: let the default stream-ordered pool keep freed memory
// (its default releases it to the system at every synchronisation, so the
// next handle's scratch would be allocated from scratch again).  This is a
// setting of this process's pool, not of the GPU.
void keep_pool_memory(int dev) {
  static std::mutex m;
  static bool done[64] = {};
  std::lock_guard<std::mutex> lock(m);
  if (dev < 0 || dev >= 64 || done[dev]) return;
  cudaMemPool_t pool;
  if (cudaDeviceGetDefaultMemPool(&pool, dev) == cudaSuccess) {
    uint64_t keep = UINT64_MAX;
    cudaMemPoolSetAttribute(pool, cudaMemPoolAttrReleaseThreshold, &keep);
  }
  done[dev] = true;
}

enum PlanKind { kPlanNone = 0, kPlanSpgemm = 1, kPlanEwise = 2, kPlanSub = 3 };

struct Plan {
  DevBuf rows;    // per-row arrays + summary + scan partials
  DevBuf slices;  // dense-window slice arrays
  DevBuf ranks;   // register bitmap rows: kBmrSlots uint16 ranks per row of A
  DevBuf ew;      // elementwise operations: summary, chunk arrays, scan partials
  DevBuf sv;      // sparse matrix - sparse vector product (in A^T's handle): accumulator, byte-map, offsets
  DevBuf rcd;     // dense heavy rows: per-slice counts, mega-row list, work counters
  DevBuf rcdb;    // dense heavy rows: slice starts of the mega rows' B rows
  int kind = kPlanNone;  // which symbolic pass filled this plan
  // elementwise plan (kPlanEwise)
  int ew_op = 0, ew_group = 32;
  int64_t ew_diag = 0, ew_nc_max = 0;
  int64_t* ew_chunk_begin = nullptr;
  int32_t* ew_chunk_row = nullptr;
  int64_t* ew_chunk_off = nullptr;
  int64_t* ew_chunk_split = nullptr;
  int64_t* ew_chunk_bpos = nullptr;
  int64_t* ew_partials = nullptr;
  int32_t* rcd_scnt = nullptr;
  int32_t* rcd_mega = nullptr;
  int32_t* rcd_nmega = nullptr;
  int32_t* rcd_ctr = nullptr;
  int64_t* rcd_moff = nullptr;
  int32_t* rcd_mna = nullptr;
  long long rcd_mega_entries = 0;
  // submatrix plan (kPlanSub): the block the symbolic pass counted
  int64_t sub_r0 = 0, sub_r1 = 0, sub_c0 = 0, sub_c1 = 0;
  DevSummary* host_sum = nullptr;  // pinned
  // carved pointers
  DevSummary* dsum = nullptr;
  int32_t* perm = nullptr;
  uint8_t* cls = nullptr;
  int32_t* lo = nullptr;
  int32_t* hi = nullptr;
  int32_t* long_rows = nullptr;
  int32_t* sort_list = nullptr;
  int32_t* pending = nullptr;
  int64_t* partials = nullptr;
  int32_t* slice_row = nullptr;
  int32_t* slice_idx = nullptr;
  int32_t* slice_first = nullptr;
  int32_t* slice_cnt = nullptr;
  // results of the last symbolic pass
  bool ready = false;
  const void* A = nullptr;
  const void* B = nullptr;
  int64_t a_nnz = -1, b_nnz = -1;
  int64_t seg_count[kNumSegs] = {};
  int64_t seg_offset[kNumSegs + 1] = {};
  int64_t n_sort = 0, n_empty = 0, dense_slices = 0, products = 0;
  int log2_group = 5;
  bool all_planned = false;  // the planning pass took every row: its segment is rows 0..m-1 in order
  int dense_width = 0;
  int run_limit = 64;
  int sym_launches = 0, num_launches = 0;
  struct OuterState* outer = nullptr;  // outer-product SpGEMM between its two passes
};

}  // namespace

struct ws_csr_s {
  int64_t nrows = 0, ncols = 0, nnz = 0;
  int64_t* rowptr = nullptr;
  int32_t* colidx = nullptr;
  void* vals = nullptr;
  ws_dtype_t dtype = WS_F64;
  int device = 0;
  Plan* plan = nullptr;
};

namespace {

int num_sms_of(int device) {
  static int cached_dev = -1, cached = 0;
  if (cached_dev != device) {
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, device) != cudaSuccess || n <= 0) n = 1;
    cached = n;
    cached_dev = device;
  }
  return cached;
}

int log2_group_for(const ws_csr_s* B) {
  const double avg = B->nrows > 0 ? static_cast<double>(B->nnz) / static_cast<double>(B->nrows) : 0.0;
  if (avg <= 4.0) return 2;
  if (avg <= 8.0) return 3;
  if (avg <= 16.0) return 4;
  return 5;
}

ws_status_t read_summary(Plan* pl, cudaStream_t s) {
  WS_CUDA(cudaMemcpyAsync(pl->host_sum, pl->dsum, sizeof(DevSummary), cudaMemcpyDeviceToHost, s),
          "cudaMemcpyAsync(summary)");
  WS_CUDA(cudaStreamSynchronize(s), "cudaStreamSynchronize");
  return WS_OK;
}

ws_status_t device_status(const DevSummary& hs) {
  if (hs.status == 0) return WS_OK;
  return fail(WS_ERR_DEVICE, "device status 0x%x (probe=%d rank=%d count=%d sortcap=%d)", hs.status,
              !!(hs.status & kErrProbe), !!(hs.status & kErrRank), !!(hs.status & kErrCount),
              !!(hs.status & kErrSortCap));
}

template <typename T>
RowPlan<T> make_rowplan(const ws_csr_s* A, const ws_csr_s* B, ws_csr_s* C, Plan* pl) {
  RowPlan<T> p{};
  p.A = {A->rowptr, A->colidx, static_cast<const T*>(A->vals)};
  p.B = {B->rowptr, B->colidx, static_cast<const T*>(B->vals)};
  p.c_rowptr = C->rowptr;
  p.c_colidx = C->colidx;
  p.c_vals = static_cast<T*>(C->vals);
  p.perm = pl->perm;
  p.cls = pl->cls;
  p.lo = pl->lo;
  p.hi = pl->hi;
  p.sort_list = pl->sort_list;
  p.slice_row = pl->slice_row;
  p.slice_idx = pl->slice_idx;
  p.slice_first = pl->slice_first;
  p.slice_cnt = pl->slice_cnt;
  p.ranks = static_cast<uint16_t*>(pl->ranks.ptr);
  p.sum = pl->dsum;
  p.log2_group = pl->log2_group;
  p.run_limit = pl->run_limit;
  p.dense_width = pl->dense_width;
  return p;
}

ws_status_t carve_rows(Plan* pl, int64_t m, cudaStream_t s) {
  const int64_t nb = scan_partials_needed(m);
  size_t off = 0;
  const size_t o_sum = off; off = align_up(off + sizeof(DevSummary), 256);
  const size_t o_perm = off; off = align_up(off + 4 * static_cast<size_t>(m), 256);
  const size_t o_lo = off; off = align_up(off + 4 * static_cast<size_t>(m), 256);
  const size_t o_hi = off; off = align_up(off + 4 * static_cast<size_t>(m), 256);
  const size_t o_long = off; off = align_up(off + 4 * static_cast<size_t>(m), 256);
  const size_t o_sort = off; off = align_up(off + 4 * static_cast<size_t>(m), 256);
  const size_t o_pend = off; off = align_up(off + 4 * static_cast<size_t>(m), 256);
  const size_t o_part = off; off = align_up(off + 8 * static_cast<size_t>(nb + 1), 256);
  const size_t o_cls = off; off = align_up(off + static_cast<size_t>(m), 256);
  ws_status_t st = pl->rows.reserve(off, s);
  if (st != WS_OK) return st;
  char* b = static_cast<char*>(pl->rows.ptr);
  pl->dsum = reinterpret_cast<DevSummary*>(b + o_sum);
  pl->perm = reinterpret_cast<int32_t*>(b + o_perm);
  pl->lo = reinterpret_cast<int32_t*>(b + o_lo);
  pl->hi = reinterpret_cast<int32_t*>(b + o_hi);
  pl->long_rows = reinterpret_cast<int32_t*>(b + o_long);
  pl->sort_list = reinterpret_cast<int32_t*>(b + o_sort);
  pl->pending = reinterpret_cast<int32_t*>(b + o_pend);
  pl->partials = reinterpret_cast<int64_t*>(b + o_part);
  pl->cls = reinterpret_cast<uint8_t*>(b + o_cls);
  return WS_OK;
}

ws_status_t carve_slices(Plan* pl, int64_t nslices, cudaStream_t s) {
  const size_t n = static_cast<size_t>(nslices > 0 ? nslices : 1);
  const size_t each = align_up(4 * n, 256);
  ws_status_t st = pl->slices.reserve(4 * each, s);
  if (st != WS_OK) return st;
  char* b = static_cast<char*>(pl->slices.ptr);
  pl->slice_row = reinterpret_cast<int32_t*>(b);
  pl->slice_idx = reinterpret_cast<int32_t*>(b + each);
  pl->slice_first = reinterpret_cast<int32_t*>(b + 2 * each);
  pl->slice_cnt = reinterpret_cast<int32_t*>(b + 3 * each);
  return WS_OK;
}

// Second half of the symbolic pass when some rows were not ranked by the
// planning pass: group the rows by segment, run the per-bin symbolic kernels,
// scan the counts into C's row pointer and read the summary back.
template <typename T>
ws_status_t symbolic_bins(const ws_csr_s* A, const ws_csr_s* B, ws_csr_s* C, Plan* pl, RowPlan<T> p, int64_t off,
                          int sms, cudaStream_t s) {
  const int64_t m = A->nrows;
  ws_status_t st = WS_OK;
  if (off > 0) {
    launch_scatter<T>(p, m, pl->seg_offset, sms, s, &pl->sym_launches);
  }
  int64_t bmr_rows = 0;
  for (int b = 0; b < kNumBmrBins; ++b) bmr_rows += pl->seg_count[kSegBmr0 + b];
  if (bmr_rows > 0) {
    st = pl->ranks.reserve(static_cast<size_t>(m) * kBmrSlots * sizeof(uint16_t), s);
    if (st != WS_OK) return st;
    p.ranks = static_cast<uint16_t*>(pl->ranks.ptr);
  }
  if (pl->seg_count[kSegDense] > 0) {
    st = carve_slices(pl, pl->dense_slices, s);
    if (st != WS_OK) return st;
    p = make_rowplan<T>(A, B, C, pl);
    p.seg_begin = pl->seg_offset[kSegDense];
    p.seg_len = pl->seg_count[kSegDense];
    launch_dense_slices<T>(p, pl->slice_row, pl->slice_idx, pl->slice_first, sms, s, &pl->sym_launches);
    launch_dense<T>(p, pl->dense_slices, false, sms, s, &pl->sym_launches);
  }
  if (pl->seg_count[kSegRcd] > 0) {
    const int64_t nr = pl->seg_count[kSegRcd];
    const size_t o_scnt = 0;
    const size_t o_mega = align_up(o_scnt + 4 * static_cast<size_t>(nr) * rcd_slices<T>(), 256);
    const size_t o_moff = align_up(o_mega + 4 * static_cast<size_t>(nr), 256);
    const size_t o_mna = align_up(o_moff + 8 * static_cast<size_t>(nr), 256);
    const size_t o_cnt = align_up(o_mna + 4 * static_cast<size_t>(nr), 256);
    st = pl->rcd.reserve(o_cnt + 256, s);
    if (st != WS_OK) return st;
    char* b = static_cast<char*>(pl->rcd.ptr);
    pl->rcd_scnt = reinterpret_cast<int32_t*>(b + o_scnt);
    pl->rcd_mega = reinterpret_cast<int32_t*>(b + o_mega);
    pl->rcd_moff = reinterpret_cast<int64_t*>(b + o_moff);
    pl->rcd_mna = reinterpret_cast<int32_t*>(b + o_mna);
    pl->rcd_nmega = reinterpret_cast<int32_t*>(b + o_cnt);
    pl->rcd_ctr = pl->rcd_nmega + 1;
    WS_CUDA(cudaMemsetAsync(pl->rcd_nmega, 0, sizeof(int32_t), s), "cudaMemsetAsync(rcd counters)");
    p.rcd_scnt = pl->rcd_scnt;
    p.rcd_mega = pl->rcd_mega;
    p.rcd_moff = pl->rcd_moff;
    p.rcd_mna = pl->rcd_mna;
    p.rcd_nmega = pl->rcd_nmega;
    p.rcd_ctr = pl->rcd_ctr;
    p.seg_begin = pl->seg_offset[kSegRcd];
    p.seg_len = nr;
    launch_rcd<T>(p, false, sms, s, &pl->sym_launches);
  }
  if (pl->seg_count[kSegWb] > 0) {
    p.seg_begin = pl->seg_offset[kSegWb];
    p.seg_len = pl->seg_count[kSegWb];
    launch_wb<T>(p, false, sms, s, &pl->sym_launches);
  }
  for (int b = 0; b < kNumBmrBins; ++b) {
    const int g = kSegBmr0 + b;
    if (pl->seg_count[g] == 0) continue;
    p.seg_begin = pl->seg_offset[g];
    p.seg_len = pl->seg_count[g];
    launch_bmr<T>(p, b, false, sms, s, &pl->sym_launches);
  }
  for (int b = 0; b < kNumBitmapBins; ++b) {
    const int g = kSegBitmap0 + b;
    if (pl->seg_count[g] == 0) continue;
    p.seg_begin = pl->seg_offset[g];
    p.seg_len = pl->seg_count[g];
    launch_bitmap<T>(p, b, false, sms, s, &pl->sym_launches);
  }
  for (int b = 0; b < kNumHashBins; ++b) {
    const int g = kSegHash0 + b;
    if (pl->seg_count[g] == 0) continue;
    p.seg_begin = pl->seg_offset[g];
    p.seg_len = pl->seg_count[g];
    launch_hash<T>(p, b, false, sms, s, &pl->sym_launches);
  }
  launch_scan(C->rowptr, m, pl->partials, pl->dsum, s, &pl->sym_launches);
  WS_CUDA(cudaGetLastError(), "symbolic launches");
  st = read_summary(pl, s);
  if (st != WS_OK) return st;
  return WS_OK;
}

template <typename T>
ws_status_t symbolic_impl(const ws_csr_s* A, const ws_csr_s* B, ws_csr_s* C, Plan* pl, cudaStream_t s,
                          int64_t* nnz_out) {
  const int64_t m = A->nrows;
  const int dev = C->device;
  const int sms = num_sms_of(dev);
  pl->ready = false;
  pl->kind = kPlanSpgemm;
  pl->sym_launches = 0;
  pl->num_launches = 0;
  pl->log2_group = log2_group_for(B);
  pl->run_limit = g_run_limit;
  pl->dense_width = g_dense_width > 0 ? g_dense_width : (sizeof(T) == 8 ? 8192 : 16384);

  ws_status_t st = carve_rows(pl, m, s);
  if (st != WS_OK) return st;
  WS_CUDA(cudaMemsetAsync(pl->dsum, 0, sizeof(DevSummary), s), "cudaMemsetAsync(summary)");
  WS_CUDA(cudaMemsetAsync(C->rowptr, 0, sizeof(int64_t), s), "cudaMemsetAsync(rowptr[0])");

  RowPlan<T> p = make_rowplan<T>(A, B, C, pl);
  if (m > 0) {
    AnalyzeParams ap{m,           g_hash_max, g_bitmap_span,   1 << pl->log2_group, g_bmr_max_a,
                     g_rcd_max_a, g_wb_span,  pl->dense_width, kLongRowThreshold};
    // When every row of C fits the widest register bitmap (B has at most
    // 65,536 columns), the planning pass counts the eligible rows in its first
    // read of A and only the remaining rows go through the analysis kernel.
    const bool plan_pass = g_bmr_max_a > 0 && B->ncols > 0 && B->ncols <= kMaxBitmapSpan && g_bitmap_span >= B->ncols;
    if (plan_pass) {
      st = pl->ranks.reserve(static_cast<size_t>(m) * kBmrSlots * sizeof(uint16_t), s);
      if (st != WS_OK) return st;
      p.ranks = static_cast<uint16_t*>(pl->ranks.ptr);
      launch_bmr_plan<T>(p, ap, B->ncols, pl->pending, sms, s, &pl->sym_launches);
      launch_analyze<T>(p, ap, pl->long_rows, pl->pending, sms, s, &pl->sym_launches);
      // If the planning pass took every row, all counts are in place now: a
      // scan queued here (a no-op otherwise) saves the second read-back.
      launch_scan(C->rowptr, m, pl->partials, pl->dsum, s, &pl->sym_launches, &pl->dsum->n_pending);
    } else {
      launch_analyze<T>(p, ap, pl->long_rows, nullptr, sms, s, &pl->sym_launches);
    }
    WS_CUDA(cudaGetLastError(), "analyze launch");
  }
  st = read_summary(pl, s);
  if (st != WS_OK) return st;
  const DevSummary& hs = *pl->host_sum;
  int64_t off = 0;
  for (int g = 0; g < kNumSegs; ++g) {
    pl->seg_count[g] = hs.seg_count[g];
    pl->seg_offset[g] = off;
    off += hs.seg_count[g];
  }
  pl->seg_offset[kNumSegs] = off;
  pl->n_empty = hs.n_empty;
  pl->products = hs.products;
  pl->dense_slices = hs.dense_slices;
  if (pl->dense_slices > INT32_MAX) return fail(WS_ERR_OVERFLOW, "too many dense-window slices (%lld)", (long long)pl->dense_slices);
  pl->all_planned = m > 0 && hs.n_pending == 0 && pl->seg_count[kSegBmrWide] == m;
  if (!pl->all_planned) {
    st = symbolic_bins<T>(A, B, C, pl, p, off, sms, s);
    if (st != WS_OK) return st;
  }
  st = device_status(*pl->host_sum);
  if (st != WS_OK) return st;
  pl->n_sort = pl->host_sum->n_sort;
  pl->rcd_mega_entries = pl->all_planned ? 0 : pl->host_sum->rcd_mega_entries;
  C->nnz = m > 0 ? pl->host_sum->nnz : 0;
  pl->A = A;
  pl->B = B;
  pl->a_nnz = A->nnz;
  pl->b_nnz = B->nnz;
  pl->ready = true;
  *nnz_out = C->nnz;
  return WS_OK;
}

template <typename T>
ws_status_t numeric_impl(const ws_csr_s* A, const ws_csr_s* B, ws_csr_s* C, Plan* pl, cudaStream_t s) {
  const int sms = num_sms_of(C->device);
  pl->num_launches = 0;
  RowPlan<T> p = make_rowplan<T>(A, B, C, pl);
  if (pl->seg_count[kSegDirect] > 0) {
    p.seg_begin = pl->seg_offset[kSegDirect];
    p.seg_len = pl->seg_count[kSegDirect];
    launch_direct<T>(p, sms, s, &pl->num_launches);
  }
  if (pl->seg_count[kSegBmrWide] > 0) {
    p.seg_begin = pl->seg_offset[kSegBmrWide];
    p.seg_len = pl->seg_count[kSegBmrWide];
    if (pl->all_planned) p.perm = nullptr;  // rows in order, no permutation was built
    launch_bmr<T>(p, kBmrPlannedBin, true, sms, s, &pl->num_launches);
    p.perm = pl->perm;
  }
  if (pl->seg_count[kSegRcd] > 0) {
    WS_CUDA(cudaMemsetAsync(pl->rcd_ctr, 0, 2 * sizeof(int32_t), s), "cudaMemsetAsync(rcd work counters)");
    p.rcd_scnt = pl->rcd_scnt;
    p.rcd_mega = pl->rcd_mega;
    p.rcd_moff = pl->rcd_moff;
    p.rcd_mna = pl->rcd_mna;
    p.rcd_nmega = pl->rcd_nmega;
    p.rcd_ctr = pl->rcd_ctr;
    p.seg_begin = pl->seg_offset[kSegRcd];
    p.seg_len = pl->seg_count[kSegRcd];
    if (pl->rcd_mega_entries > 0) {  // slice starts of the mega rows' B rows, found once per entry
      const size_t need = static_cast<size_t>(pl->rcd_mega_entries) * (rcd_slices<T>() - 1) * sizeof(int32_t);
      ws_status_t st = pl->rcdb.reserve(need > 0 ? need : 4, s);
      if (st != WS_OK) return st;
      p.rcd_bnd = static_cast<int32_t*>(pl->rcdb.ptr);
      launch_rcd_bounds<T>(p, sms, s, &pl->num_launches);
    }
    launch_rcd<T>(p, true, sms, s, &pl->num_launches);
  }
  if (pl->seg_count[kSegWb] > 0) {
    p.seg_begin = pl->seg_offset[kSegWb];
    p.seg_len = pl->seg_count[kSegWb];
    launch_wb<T>(p, true, sms, s, &pl->num_launches);
  }
  for (int b = 0; b < kNumBmrBins; ++b) {
    const int g = kSegBmr0 + b;
    if (pl->seg_count[g] == 0) continue;
    p.seg_begin = pl->seg_offset[g];
    p.seg_len = pl->seg_count[g];
    launch_bmr<T>(p, b, true, sms, s, &pl->num_launches);
  }
  for (int b = 0; b < kNumBitmapBins; ++b) {
    const int g = kSegBitmap0 + b;
    if (pl->seg_count[g] == 0) continue;
    p.seg_begin = pl->seg_offset[g];
    p.seg_len = pl->seg_count[g];
    launch_bitmap<T>(p, b, true, sms, s, &pl->num_launches);
  }
  for (int b = 0; b < kNumHashBins; ++b) {
    const int g = kSegHash0 + b;
    if (pl->seg_count[g] == 0) continue;
    p.seg_begin = pl->seg_offset[g];
    p.seg_len = pl->seg_count[g];
    launch_hash<T>(p, b, true, sms, s, &pl->num_launches);
  }
  if (pl->n_sort > 0) launch_sort<T>(p, pl->n_sort, sms, s, &pl->num_launches);
  if (pl->seg_count[kSegDense] > 0) {
    p.seg_begin = pl->seg_offset[kSegDense];
    p.seg_len = pl->seg_count[kSegDense];
    launch_dense<T>(p, pl->dense_slices, true, sms, s, &pl->num_launches);
  }
  WS_CUDA(cudaGetLastError(), "numeric launches");
  return WS_OK;
}

// ----------------------------------------------------- elementwise operations

// Lanes per chunk from the mean merged row length (entries of A and B per row).
int ewise_group_for(int64_t m, int64_t merged) {
  const double avg = m > 0 ? static_cast<double>(merged) / static_cast<double>(m) : 0.0;
  if (avg <= 8.0) return 4;
  if (avg <= 16.0) return 8;
  if (avg <= 32.0) return 16;
  return 32;
}

ws_status_t carve_ewise(Plan* pl, int64_t m, int64_t nc_max, cudaStream_t s) {
  const int64_t nb = scan_partials_needed(m > nc_max ? m : nc_max);
  size_t off = 0;
  const size_t o_sum = off; off = align_up(off + sizeof(DevSummary), 256);
  const size_t o_begin = off; off = align_up(off + 8 * static_cast<size_t>(m + 1), 256);
  const size_t o_row = off; off = align_up(off + 4 * static_cast<size_t>(nc_max), 256);
  const size_t o_off = off; off = align_up(off + 8 * static_cast<size_t>(nc_max + 1), 256);
  const size_t o_split = off; off = align_up(off + 8 * static_cast<size_t>(nc_max + 1), 256);
  const size_t o_bpos = off; off = align_up(off + 8 * static_cast<size_t>(nc_max + 1), 256);
  const size_t o_part = off; off = align_up(off + 8 * static_cast<size_t>(nb + 1), 256);
  ws_status_t st = pl->ew.reserve(off, s);
  if (st != WS_OK) return st;
  char* b = static_cast<char*>(pl->ew.ptr);
  pl->dsum = reinterpret_cast<DevSummary*>(b + o_sum);
  pl->ew_chunk_begin = reinterpret_cast<int64_t*>(b + o_begin);
  pl->ew_chunk_row = reinterpret_cast<int32_t*>(b + o_row);
  pl->ew_chunk_off = reinterpret_cast<int64_t*>(b + o_off);
  pl->ew_chunk_split = reinterpret_cast<int64_t*>(b + o_split);
  pl->ew_chunk_bpos = reinterpret_cast<int64_t*>(b + o_bpos);
  pl->ew_partials = reinterpret_cast<int64_t*>(b + o_part);
  return WS_OK;
}

template <typename T>
EwisePlan<T> make_ewise(const ws_csr_s* A, const ws_csr_s* B, ws_csr_s* C, const Plan* pl) {
  EwisePlan<T> p{};
  p.A = {A->rowptr, A->colidx, static_cast<const T*>(A->vals)};
  p.B = {B->rowptr, B->colidx, static_cast<const T*>(B->vals)};
  p.m = A->nrows;
  p.c_rowptr = C->rowptr;
  p.c_colidx = C->colidx;
  p.c_vals = static_cast<T*>(C->vals);
  p.chunk_begin = pl->ew_chunk_begin;
  p.chunk_row = pl->ew_chunk_row;
  p.chunk_off = pl->ew_chunk_off;
  p.chunk_split = pl->ew_chunk_split;
  p.chunk_bpos = pl->ew_chunk_bpos;
  p.nc_max = pl->ew_nc_max;
  p.partials = pl->ew_partials;
  p.sum = pl->dsum;
  p.diag = pl->ew_diag;
  p.group = pl->ew_group;
  p.op = pl->ew_op;
  return p;
}

template <typename T>
ws_status_t ewise_symbolic_impl(const ws_csr_s* A, const ws_csr_s* B, ws_csr_s* C, Plan* pl, int op,
                                cudaStream_t s, int64_t* nnz_out) {
  const int64_t m = A->nrows;
  pl->ready = false;
  pl->kind = kPlanEwise;
  pl->sym_launches = 0;
  pl->num_launches = 0;
  pl->ew_op = op;
  const int64_t merged = A->nnz + B->nnz;
  // automatic: a lane per chunk of a warp-staged tile for short rows
  // (power-law graphs), a warp per 64-position chunk once rows average a
  // whole chunk
  const bool long_rows = m > 0 && merged >= static_cast<int64_t>(kEwiseRankChunk) * m;
  pl->ew_group = g_ewise_lanes > 0 ? g_ewise_lanes
               : g_ewise_lanes == 0 ? ewise_group_for(m, merged) : (long_rows ? kEwiseRankGroup : kEwiseTileGroup);
  pl->ew_diag = pl->ew_group == 1 ? g_ewise_diag
              : pl->ew_group == kEwiseTileGroup ? (g_ewise_diag < kEwiseTileDiag ? g_ewise_diag : kEwiseTileDiag)
              : pl->ew_group == kEwiseRankGroup ? kEwiseRankChunk : 16 * static_cast<int64_t>(pl->ew_group);
  pl->ew_nc_max = m + merged / pl->ew_diag + 1;  // row i has at most 1 + len_i / diag chunks
  ws_status_t st = carve_ewise(pl, m, pl->ew_nc_max, s);
  if (st != WS_OK) return st;
  WS_CUDA(cudaMemsetAsync(pl->dsum, 0, sizeof(DevSummary), s), "cudaMemsetAsync(summary)");
  WS_CUDA(cudaMemsetAsync(C->rowptr, 0, sizeof(int64_t), s), "cudaMemsetAsync(rowptr[0])");
  WS_CUDA(cudaMemsetAsync(pl->ew_chunk_begin, 0, sizeof(int64_t), s), "cudaMemsetAsync(chunk_begin[0])");
  WS_CUDA(cudaMemsetAsync(pl->ew_chunk_off, 0, sizeof(int64_t), s), "cudaMemsetAsync(chunk_off[0])");
  if (m > 0) {
    launch_ewise_symbolic<T>(make_ewise<T>(A, B, C, pl), num_sms_of(C->device), s, &pl->sym_launches);
    WS_CUDA(cudaGetLastError(), "elementwise symbolic launches");
  }
  st = read_summary(pl, s);
  if (st != WS_OK) return st;
  st = device_status(*pl->host_sum);
  if (st != WS_OK) return st;
  C->nnz = m > 0 ? pl->host_sum->nnz : 0;
  pl->products = merged;
  pl->A = A;
  pl->B = B;
  pl->a_nnz = A->nnz;
  pl->b_nnz = B->nnz;
  pl->ready = true;
  *nnz_out = C->nnz;
  return WS_OK;
}

// ------------------------------------------ sparse matrix - sparse vector

// Creates a handle's plan and its pinned summary if missing.
ws_status_t ensure_plan(ws_csr_s* h) {
  if (!h->plan) {
    h->plan = new (std::nothrow) Plan;
    if (!h->plan) return fail(WS_ERR_ALLOC, "host allocation failed");
  }
  if (!h->plan->host_sum) {
    keep_pool_memory(h->device);
    h->plan->host_sum = acquire_host_sum();
    if (!h->plan->host_sum) return fail(WS_ERR_ALLOC, "cudaMallocHost failed");
  }
  return WS_OK;
}

template <typename T>
ws_status_t spmspv_impl(ws_csr_s* At, int64_t nx, const int32_t* x_idx, const void* x_vals, int32_t* y_idx,
                        void* y_vals, int64_t* nnz_y, cudaStream_t s) {
  Plan* pl = At->plan;
  const int64_t m = At->ncols, n = At->nrows;
  const int64_t tiles = spmspv_tiles(m);
  const int64_t mark_bytes = tiles * 4096;  // the byte-map, padded to whole compaction tiles
  const int64_t nb = scan_partials_needed(nx > tiles ? nx : tiles);
  size_t off = 0;
  const size_t o_sum = off; off = align_up(off + sizeof(DevSummary), 256);
  const size_t o_acc = off; off = align_up(off + sizeof(T) * static_cast<size_t>(m), 256);
  const size_t o_mark = off; off = align_up(off + static_cast<size_t>(mark_bytes), 256);
  const size_t o_off = off; off = align_up(off + 8 * static_cast<size_t>(nx + 1), 256);
  const size_t o_first = off; off = align_up(off + 8 * static_cast<size_t>(nx), 256);
  const size_t o_cnt = off; off = align_up(off + 8 * static_cast<size_t>(tiles + 1), 256);
  const size_t o_part = off; off = align_up(off + 8 * static_cast<size_t>(nb + 1), 256);
  ws_status_t st = pl->sv.reserve(off, s);
  if (st != WS_OK) return st;
  char* b = static_cast<char*>(pl->sv.ptr);
  SpmspvPlan<T> p{};
  p.At = {At->rowptr, At->colidx, static_cast<const T*>(At->vals)};
  p.n = n;
  p.m = m;
  p.nnz_a = At->nnz;
  p.nx = nx;
  p.x_idx = x_idx;
  p.x_vals = static_cast<const T*>(x_vals);
  p.sum = reinterpret_cast<DevSummary*>(b + o_sum);
  p.acc = reinterpret_cast<T*>(b + o_acc);
  p.mark = reinterpret_cast<uint8_t*>(b + o_mark);
  p.off = reinterpret_cast<int64_t*>(b + o_off);
  p.first = reinterpret_cast<int64_t*>(b + o_first);
  p.cnt = reinterpret_cast<int64_t*>(b + o_cnt);
  p.partials = reinterpret_cast<int64_t*>(b + o_part);
  p.y_idx = y_idx;
  p.y_vals = static_cast<T*>(y_vals);
  p.cap = m;
  pl->dsum = p.sum;
  pl->sym_launches = 0;
  pl->num_launches = 0;
  // zero the summary, the accumulator and the byte-map (contiguous), and the scan heads
  WS_CUDA(cudaMemsetAsync(b, 0, o_off, s), "cudaMemsetAsync(spmspv scratch)");
  WS_CUDA(cudaMemsetAsync(p.off, 0, sizeof(int64_t), s), "cudaMemsetAsync(off[0])");
  WS_CUDA(cudaMemsetAsync(p.cnt, 0, sizeof(int64_t), s), "cudaMemsetAsync(cnt[0])");
  if (m > 0) {
    launch_spmspv<T>(p, num_sms_of(At->device), s, &pl->num_launches);
    WS_CUDA(cudaGetLastError(), "spmspv launches");
  }
  st = read_summary(pl, s);
  if (st != WS_OK) return st;
  st = device_status(*pl->host_sum);
  if (st != WS_OK) return st;
  *nnz_y = m > 0 ? pl->host_sum->nnz : 0;
  return WS_OK;
}

// Shared checks of the operand and output handles; creates C's plan.
ws_status_t prepare_output(const ws_csr_s* A, const ws_csr_s* B, ws_csr_s* C) {
  if (C == A || C == B) return fail(WS_ERR_INVALID_ARG, "C must be a separate output handle");
  if (A->dtype != B->dtype || C->dtype != A->dtype) return fail(WS_ERR_DTYPE, "A, B and C dtypes differ");
  if (!C->plan) {
    C->plan = new (std::nothrow) Plan;
    if (!C->plan) return fail(WS_ERR_ALLOC, "host allocation failed");
  }
  Plan* pl = C->plan;
  if (!pl->host_sum) {
    keep_pool_memory(C->device);
    pl->host_sum = acquire_host_sum();
    if (!pl->host_sum) return fail(WS_ERR_ALLOC, "cudaMallocHost failed");
  }
  return WS_OK;
}

ws_status_t check_handle(const ws_csr_s* h, const char* name) {
  if (!h) return fail(WS_ERR_INVALID_ARG, "%s is NULL", name);
  return WS_OK;
}

// ------------------------------------------------------ outer-product SpGEMM
//
// C = A*B with the k loop split over P workers (Sec. 5.1, Fig. "SpGEMM
// implemented in WingSpan", outer product): worker p multiplies the column
// block A[:, K_p] by the row block B[K_p, :] into its own copy of C, and a
// merge level coalesces the copies (Sec. 4, coalesce).  On one GPU every
// block's product already fills the device, so the blocks run one after
// another on the caller's stream:
//   - B[K_p, :] is a view of B's rows (no copy);
//   - A[:, K_p] is extracted (count, scan, copy) into one library buffer of
//     nnz(A) entries that every block reuses, so its size needs no read-back;
//   - the partial product is the row-wise product of the two blocks;
//   - the partial products are merged pairwise by sparse additions (a sum of
//     exactly 0.0 is kept, so C's structure equals the row-wise product's).
// The symbolic call runs everything but the value pass of the last merge,
// whose structure pass writes C.rowptr; the numeric call runs that value pass.

// A CSR matrix whose arrays the library owns (stream-ordered allocations).
struct Owned {
  ws_csr_s h;
  void* rp_mem = nullptr;  // row pointer
  void* cv_mem = nullptr;  // column indices and values
};

struct OuterState {
  int parts = 1;
  const ws_csr_s* A = nullptr;
  const ws_csr_s* B = nullptr;
  int64_t a_nnz = 0, b_nnz = 0;
  Owned* x = nullptr;  // operands of the last merge (parts >= 2)
  Owned* y = nullptr;
};

// Frees a plan's scratch stream-ordered on s (no device synchronisation).
void release_plan_async(Plan* pl, cudaStream_t s);

void release_owned(Owned* o, cudaStream_t s) {
  if (!o) return;
  release_plan_async(o->h.plan, s);
  o->h.plan = nullptr;
  if (o->rp_mem) cudaFreeAsync(o->rp_mem, s);
  if (o->cv_mem) cudaFreeAsync(o->cv_mem, s);
  delete o;
}

void release_outer(Plan* pl, cudaStream_t s) {
  if (!pl || !pl->outer) return;
  release_owned(pl->outer->x, s);
  release_owned(pl->outer->y, s);
  delete pl->outer;
  pl->outer = nullptr;
}

void release_plan_async(Plan* pl, cudaStream_t s) {
  if (!pl) return;
  release_outer(pl, s);
  DevBuf* bufs[] = {&pl->rows, &pl->slices, &pl->ranks, &pl->ew, &pl->sv, &pl->rcd, &pl->rcdb};
  for (DevBuf* b : bufs) {
    if (b->ptr) cudaFreeAsync(b->ptr, s);
    b->ptr = nullptr;
    b->bytes = 0;
  }
  release_host_sum(pl->host_sum);
  delete pl;
}

// An owned m x n matrix with its row pointer allocated; entries come later.
ws_status_t new_owned(int64_t m, int64_t n, ws_dtype_t dt, int dev, cudaStream_t s, Owned** out) {
  *out = nullptr;
  Owned* o = new (std::nothrow) Owned;
  if (!o) return fail(WS_ERR_ALLOC, "host allocation failed");
  o->h.nrows = m;
  o->h.ncols = n;
  o->h.nnz = 0;
  o->h.dtype = dt;
  o->h.device = dev;
  const cudaError_t e = cudaMallocAsync(&o->rp_mem, 8 * static_cast<size_t>(m + 1), s);
  if (e != cudaSuccess) {
    delete o;
    return fail(WS_ERR_ALLOC, "cudaMallocAsync(row pointer): %s", cudaGetErrorString(e));
  }
  o->h.rowptr = static_cast<int64_t*>(o->rp_mem);
  ws_status_t st = ensure_plan(&o->h);
  if (st != WS_OK) {
    release_owned(o, s);
    return st;
  }
  *out = o;
  return WS_OK;
}

// Room for cap entries (column indices and values) of an owned matrix.
ws_status_t owned_entries(Owned* o, int64_t cap, cudaStream_t s) {
  const size_t vs = o->h.dtype == WS_F64 ? 8 : 4;
  const size_t o_val = align_up(4 * static_cast<size_t>(cap > 0 ? cap : 1), 256);
  const cudaError_t e = cudaMallocAsync(&o->cv_mem, o_val + vs * static_cast<size_t>(cap > 0 ? cap : 1), s);
  if (e != cudaSuccess) return fail(WS_ERR_ALLOC, "cudaMallocAsync(%lld entries): %s", (long long)cap, cudaGetErrorString(e));
  o->h.colidx = static_cast<int32_t*>(o->cv_mem);
  o->h.vals = static_cast<char*>(o->cv_mem) + o_val;
  return WS_OK;
}

// Device status word of a plan whose queued work has completed.
ws_status_t plan_status(const Plan* pl) {
  int st = 0;
  WS_CUDA(cudaMemcpy(&st, &pl->dsum->status, sizeof(int), cudaMemcpyDeviceToHost), "cudaMemcpy(status)");
  if (st != 0) return fail(WS_ERR_DEVICE, "device status 0x%x in an outer-product step", st);
  return WS_OK;
}

template <typename T>
ws_status_t outer_symbolic_impl(const ws_csr_s* A, const ws_csr_s* B, ws_csr_s* C, int parts, cudaStream_t s,
                                int64_t* nnz_out) {
  Plan* pl = C->plan;
  release_outer(pl, s);
  const int64_t m = A->nrows, K = A->ncols, n = B->ncols;
  const int P = static_cast<int>(parts < 1 ? 1 : (parts > K ? (K > 0 ? K : 1) : parts));
  OuterState* os = new (std::nothrow) OuterState;
  if (!os) return fail(WS_ERR_ALLOC, "host allocation failed");
  os->parts = P;
  os->A = A;
  os->B = B;
  os->a_nnz = A->nnz;
  os->b_nnz = B->nnz;
  if (P == 1) {  // one block: the row-wise product itself
    ws_status_t st = symbolic_impl<T>(A, B, C, pl, s, nnz_out);
    if (st != WS_OK) {
      delete os;
      return st;
    }
    pl->outer = os;
    return WS_OK;
  }
  const int sms = num_sms_of(C->device);
  int launches = 0;
  std::vector<Owned*> partial;
  Owned* ab = nullptr;  // the current column block of A
  void* ex_mem = nullptr;  // the extraction's summary and scan partials
  ws_status_t st = WS_OK;
  auto cleanup = [&]() {
    for (Owned* o : partial) release_owned(o, s);
    release_owned(ab, s);
    if (ex_mem) cudaFreeAsync(ex_mem, s);
    delete os;
  };
  const size_t o_part = align_up(sizeof(DevSummary), 256);
  cudaError_t e = cudaMallocAsync(&ex_mem, o_part + 8 * static_cast<size_t>(scan_partials_needed(m) + 1), s);
  if (e != cudaSuccess) {
    ex_mem = nullptr;
    cleanup();
    return fail(WS_ERR_ALLOC, "cudaMallocAsync(extraction scratch): %s", cudaGetErrorString(e));
  }
  DevSummary* ex_sum = static_cast<DevSummary*>(ex_mem);
  int64_t* ex_part = reinterpret_cast<int64_t*>(static_cast<char*>(ex_mem) + o_part);
  if (cudaMemsetAsync(ex_sum, 0, sizeof(DevSummary), s) != cudaSuccess ||
      (st = new_owned(m, 1, A->dtype, C->device, s, &ab)) != WS_OK || (st = owned_entries(ab, A->nnz, s)) != WS_OK) {
    cleanup();
    return st != WS_OK ? st : fail(WS_ERR_CUDA, "cudaMemsetAsync(extraction summary)");
  }
  ab->h.nnz = A->nnz;  // capacity: the block's own count stays on the device
  for (int p = 0; p < P && st == WS_OK; ++p) {
    const int64_t k0 = K * p / P, k1 = K * (p + 1) / P;
    // A[:, k0:k1], columns shifted by -k0
    ab->h.ncols = k1 - k0;
    if (cudaMemsetAsync(ab->h.rowptr, 0, sizeof(int64_t), s) != cudaSuccess) {
      st = fail(WS_ERR_CUDA, "cudaMemsetAsync(block row pointer)");
      break;
    }
    if (m > 0) {
      launch_submatrix_count(A->rowptr, A->colidx, 0, m, k0, k1, ab->h.rowptr, sms, s, &launches);
      launch_scan(ab->h.rowptr, m, ex_part, ex_sum, s, &launches);
      launch_submatrix_copy<T>(A->rowptr, A->colidx, static_cast<const T*>(A->vals), 0, m, k0, ab->h.rowptr,
                               ab->h.colidx, static_cast<T*>(ab->h.vals), ex_sum, sms, s, &launches);
    }
    // B[k0:k1, :]: a view of B's rows (positions stay absolute in B's arrays)
    ws_csr_s bp = *B;
    bp.plan = nullptr;
    bp.nrows = k1 - k0;
    bp.rowptr = B->rowptr + k0;
    bp.nnz = K > 0 ? B->nnz * (k1 - k0) / K : 0;  // estimate: only the lane-group choice reads it
    // the worker's partial product
    Owned* cp = nullptr;
    if ((st = new_owned(m, n, A->dtype, C->device, s, &cp)) != WS_OK) break;
    partial.push_back(cp);
    int64_t nnz_p = 0;
    if ((st = symbolic_impl<T>(&ab->h, &bp, &cp->h, cp->h.plan, s, &nnz_p)) != WS_OK) break;
    cp->h.nnz = nnz_p;
    if ((st = owned_entries(cp, nnz_p, s)) != WS_OK) break;
    if ((st = numeric_impl<T>(&ab->h, &bp, &cp->h, cp->h.plan, s)) != WS_OK) break;
    launches += cp->h.plan->sym_launches + cp->h.plan->num_launches;
  }
  if (st == WS_OK) {  // every extraction has completed (each block's structure pass synchronised)
    int ex_status = 0;
    if (cudaMemcpy(&ex_status, &ex_sum->status, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess)
      st = fail(WS_ERR_CUDA, "cudaMemcpy(extraction status)");
    else if (ex_status != 0)
      st = fail(WS_ERR_DEVICE, "device status 0x%x in a column-block extraction", ex_status);
  }
  release_owned(ab, s);
  ab = nullptr;
  // merge levels: pairwise sparse additions until two copies are left
  while (st == WS_OK && partial.size() > 2) {
    std::vector<Owned*> next;
    size_t i = 0;
    for (; i + 1 < partial.size() && st == WS_OK; i += 2) {
      Owned* x = partial[i];
      Owned* y = partial[i + 1];
      Owned* z = nullptr;
      if ((st = new_owned(m, n, A->dtype, C->device, s, &z)) != WS_OK) break;
      next.push_back(z);
      int64_t nz = 0;
      if ((st = ewise_symbolic_impl<T>(&x->h, &y->h, &z->h, z->h.plan, kEwiseAdd, s, &nz)) != WS_OK) break;
      if ((st = plan_status(x->h.plan)) != WS_OK || (st = plan_status(y->h.plan)) != WS_OK) break;
      z->h.nnz = nz;
      if ((st = owned_entries(z, nz, s)) != WS_OK) break;
      if (nz > 0) launch_ewise_numeric<T>(make_ewise<T>(&x->h, &y->h, &z->h, z->h.plan), sms, s, &launches);
      launches += z->h.plan->sym_launches;
      release_owned(x, s);  // stream-ordered: the value pass above still reads them
      release_owned(y, s);
      partial[i] = partial[i + 1] = nullptr;
    }
    for (; i < partial.size(); ++i) {
      if (partial[i]) next.push_back(partial[i]);
      partial[i] = nullptr;
    }
    for (Owned* o : partial) release_owned(o, s);
    partial.swap(next);
  }
  if (st == WS_OK) {  // the last merge's structure pass writes C.rowptr
    st = ewise_symbolic_impl<T>(&partial[0]->h, &partial[1]->h, C, pl, kEwiseAdd, s, nnz_out);
    if (st == WS_OK && (st = plan_status(partial[0]->h.plan)) == WS_OK) st = plan_status(partial[1]->h.plan);
  }
  cudaFreeAsync(ex_mem, s);
  ex_mem = nullptr;
  if (st != WS_OK) {
    cleanup();
    return st;
  }
  os->x = partial[0];
  os->y = partial[1];
  partial.clear();
  pl->outer = os;
  pl->sym_launches += launches;
  return WS_OK;
}

template <typename T>
ws_status_t outer_numeric_impl(ws_csr_s* C, cudaStream_t s) {
  Plan* pl = C->plan;
  OuterState* os = pl->outer;
  if (os->parts == 1) return numeric_impl<T>(os->A, os->B, C, pl, s);
  pl->num_launches = 0;
  if (C->nnz > 0)
    launch_ewise_numeric<T>(make_ewise<T>(&os->x->h, &os->y->h, C, pl), num_sms_of(C->device), s, &pl->num_launches);
  WS_CUDA(cudaGetLastError(), "outer-product merge launch");
  release_outer(pl, s);  // stream-ordered: the copies stay valid for the pass just queued
  return WS_OK;
}

}  // namespace

extern "C" {

ws_status_t ws_csr_create(ws_csr_t* out, int64_t nrows, int64_t ncols, int64_t nnz, int64_t* rowptr,
                          int32_t* colidx, void* vals, ws_dtype_t dtype, int validate, ws_stream_t stream) {
  g_last_error.clear();
  if (!out) return fail(WS_ERR_INVALID_ARG, "out is NULL");
  *out = nullptr;
  if (nrows < 0 || ncols < 0 || nnz < 0) return fail(WS_ERR_INVALID_ARG, "negative size");
  if (nrows > INT32_MAX - 1 || ncols > INT32_MAX)
    return fail(WS_ERR_OVERFLOW, "nrows/ncols exceed the int32 index range");
  if (dtype != WS_F32 && dtype != WS_F64) return fail(WS_ERR_INVALID_ARG, "unknown dtype %d", (int)dtype);
  if (!rowptr) return fail(WS_ERR_INVALID_ARG, "rowptr is NULL");
  if (nnz > 0 && (!colidx || !vals)) return fail(WS_ERR_INVALID_ARG, "colidx/vals NULL with nnz > 0");
  int dev = 0;
  WS_CUDA(cudaGetDevice(&dev), "cudaGetDevice");
  if (validate) {
    DevSummary* d = nullptr;
    DevSummary h{};
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    WS_CUDA(cudaMallocAsync(reinterpret_cast<void**>(&d), sizeof(DevSummary), s), "cudaMallocAsync(validate)");
    h.bad_row = INT32_MAX;
    cudaError_t e = cudaMemcpyAsync(d, &h, sizeof(h), cudaMemcpyHostToDevice, s);
    if (e == cudaSuccess && nrows > 0) {
      launch_validate(rowptr, colidx, nrows, ncols, nnz, d, num_sms_of(dev), s);
      e = cudaGetLastError();
    }
    if (e == cudaSuccess) e = cudaMemcpyAsync(&h, d, sizeof(h), cudaMemcpyDeviceToHost, s);
    cudaFreeAsync(d, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return cuda_fail(e, "validation");
    if (nrows == 0) {
      int64_t r0 = -1;
      WS_CUDA(cudaMemcpy(&r0, rowptr, sizeof(r0), cudaMemcpyDeviceToHost), "cudaMemcpy(rowptr[0])");
      if (r0 != 0 || nnz != 0) return fail(WS_ERR_INVALID_CSR, "empty matrix needs rowptr[0] = 0 and nnz = 0");
    }
    if (h.status & kErrInvalidCsr)
      return fail(WS_ERR_INVALID_CSR, "CSR invariants violated (first bad row %d)", h.bad_row);
  }
  ws_csr_s* hnd = new (std::nothrow) ws_csr_s;
  if (!hnd) return fail(WS_ERR_ALLOC, "host allocation failed");
  hnd->nrows = nrows;
  hnd->ncols = ncols;
  hnd->nnz = nnz;
  hnd->rowptr = rowptr;
  hnd->colidx = colidx;
  hnd->vals = vals;
  hnd->dtype = dtype;
  hnd->device = dev;
  *out = hnd;
  return WS_OK;
}

ws_status_t ws_spgemm_symbolic(ws_csr_t A, ws_csr_t B, ws_csr_t C, int64_t* nnz_out, ws_stream_t stream) {
  g_last_error.clear();
  ws_status_t st;
  if ((st = check_handle(A, "A")) != WS_OK || (st = check_handle(B, "B")) != WS_OK ||
      (st = check_handle(C, "C")) != WS_OK)
    return st;
  if (!nnz_out) return fail(WS_ERR_INVALID_ARG, "nnz_out is NULL");
  if (C == A || C == B) return fail(WS_ERR_INVALID_ARG, "C must be a separate output handle");
  if (A->ncols != B->nrows)
    return fail(WS_ERR_SHAPE, "A is %lldx%lld but B is %lldx%lld", (long long)A->nrows, (long long)A->ncols,
                (long long)B->nrows, (long long)B->ncols);
  if (C->nrows != A->nrows || C->ncols != B->ncols)
    return fail(WS_ERR_SHAPE, "C is %lldx%lld, expected %lldx%lld", (long long)C->nrows, (long long)C->ncols,
                (long long)A->nrows, (long long)B->ncols);
  if (A->dtype != B->dtype || C->dtype != A->dtype) return fail(WS_ERR_DTYPE, "A, B and C dtypes differ");
  if (A->nnz > 0 && B->nrows == 0) return fail(WS_ERR_INVALID_CSR, "A has entries but B has no rows");
  if ((st = prepare_output(A, B, C)) != WS_OK) return st;
  Plan* pl = C->plan;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  release_outer(pl, s);
  C->nnz = -1;
  if (A->dtype == WS_F64) return symbolic_impl<double>(A, B, C, pl, s, nnz_out);
  return symbolic_impl<float>(A, B, C, pl, s, nnz_out);
}

ws_status_t ws_spgemm_numeric(ws_csr_t A, ws_csr_t B, ws_csr_t C, int32_t* c_colidx, void* c_vals,
                              ws_stream_t stream) {
  g_last_error.clear();
  ws_status_t st;
  if ((st = check_handle(A, "A")) != WS_OK || (st = check_handle(B, "B")) != WS_OK ||
      (st = check_handle(C, "C")) != WS_OK)
    return st;
  Plan* pl = C->plan;
  if (!pl || !pl->ready || pl->kind != kPlanSpgemm)
    return fail(WS_ERR_STATE, "numeric called before a successful SpGEMM symbolic pass");
  if (pl->A != A || pl->B != B || pl->a_nnz != A->nnz || pl->b_nnz != B->nnz)
    return fail(WS_ERR_STATE, "numeric called with other operands than the symbolic pass");
  if (C->nnz > 0 && (!c_colidx || !c_vals)) return fail(WS_ERR_INVALID_ARG, "c_colidx/c_vals NULL with nnz(C) > 0");
  C->colidx = c_colidx;
  C->vals = c_vals;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (A->dtype == WS_F64) return numeric_impl<double>(A, B, C, pl, s);
  return numeric_impl<float>(A, B, C, pl, s);
}

ws_status_t ws_spgemm_outer_symbolic(ws_csr_t A, ws_csr_t B, ws_csr_t C, int parts, int64_t* nnz_out,
                                     ws_stream_t stream) {
  g_last_error.clear();
  ws_status_t st;
  if ((st = check_handle(A, "A")) != WS_OK || (st = check_handle(B, "B")) != WS_OK ||
      (st = check_handle(C, "C")) != WS_OK)
    return st;
  if (!nnz_out) return fail(WS_ERR_INVALID_ARG, "nnz_out is NULL");
  if (parts < 1) return fail(WS_ERR_INVALID_ARG, "parts must be at least 1, got %d", parts);
  if (C == A || C == B) return fail(WS_ERR_INVALID_ARG, "C must be a separate output handle");
  if (A->ncols != B->nrows)
    return fail(WS_ERR_SHAPE, "A is %lldx%lld but B is %lldx%lld", (long long)A->nrows, (long long)A->ncols,
                (long long)B->nrows, (long long)B->ncols);
  if (C->nrows != A->nrows || C->ncols != B->ncols)
    return fail(WS_ERR_SHAPE, "C is %lldx%lld, expected %lldx%lld", (long long)C->nrows, (long long)C->ncols,
                (long long)A->nrows, (long long)B->ncols);
  if (A->dtype != B->dtype || C->dtype != A->dtype) return fail(WS_ERR_DTYPE, "A, B and C dtypes differ");
  if (A->nnz > 0 && B->nrows == 0) return fail(WS_ERR_INVALID_CSR, "A has entries but B has no rows");
  if ((st = prepare_output(A, B, C)) != WS_OK) return st;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  C->nnz = -1;
  if (A->dtype == WS_F64) return outer_symbolic_impl<double>(A, B, C, parts, s, nnz_out);
  return outer_symbolic_impl<float>(A, B, C, parts, s, nnz_out);
}

ws_status_t ws_spgemm_outer_numeric(ws_csr_t A, ws_csr_t B, ws_csr_t C, int32_t* c_colidx, void* c_vals,
                                    ws_stream_t stream) {
  g_last_error.clear();
  ws_status_t st;
  if ((st = check_handle(A, "A")) != WS_OK || (st = check_handle(B, "B")) != WS_OK ||
      (st = check_handle(C, "C")) != WS_OK)
    return st;
  Plan* pl = C->plan;
  if (!pl || !pl->ready || !pl->outer)
    return fail(WS_ERR_STATE, "numeric called before a successful outer-product symbolic pass");
  const OuterState* os = pl->outer;
  if (os->A != A || os->B != B || os->a_nnz != A->nnz || os->b_nnz != B->nnz)
    return fail(WS_ERR_STATE, "numeric called with other operands than the symbolic pass");
  if (C->nnz > 0 && (!c_colidx || !c_vals)) return fail(WS_ERR_INVALID_ARG, "c_colidx/c_vals NULL with nnz(C) > 0");
  C->colidx = c_colidx;
  C->vals = c_vals;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (A->dtype == WS_F64) return outer_numeric_impl<double>(C, s);
  return outer_numeric_impl<float>(C, s);
}

ws_status_t ws_ewise_symbolic(ws_csr_t A, ws_csr_t B, ws_csr_t C, int op, int64_t* nnz_out, ws_stream_t stream) {
  g_last_error.clear();
  ws_status_t st;
  if ((st = check_handle(A, "A")) != WS_OK || (st = check_handle(B, "B")) != WS_OK ||
      (st = check_handle(C, "C")) != WS_OK)
    return st;
  if (!nnz_out) return fail(WS_ERR_INVALID_ARG, "nnz_out is NULL");
  if (op != WS_EWISE_ADD && op != WS_EWISE_MUL) return fail(WS_ERR_INVALID_ARG, "unknown elementwise op %d", op);
  if (A->nrows != B->nrows || A->ncols != B->ncols)
    return fail(WS_ERR_SHAPE, "A is %lldx%lld but B is %lldx%lld", (long long)A->nrows, (long long)A->ncols,
                (long long)B->nrows, (long long)B->ncols);
  if (C->nrows != A->nrows || C->ncols != A->ncols)
    return fail(WS_ERR_SHAPE, "C is %lldx%lld, expected %lldx%lld", (long long)C->nrows, (long long)C->ncols,
                (long long)A->nrows, (long long)A->ncols);
  if ((st = prepare_output(A, B, C)) != WS_OK) return st;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  release_outer(C->plan, s);
  C->nnz = -1;
  const int kop = op == WS_EWISE_ADD ? kEwiseAdd : kEwiseMul;
  if (A->dtype == WS_F64) return ewise_symbolic_impl<double>(A, B, C, C->plan, kop, s, nnz_out);
  return ewise_symbolic_impl<float>(A, B, C, C->plan, kop, s, nnz_out);
}

ws_status_t ws_ewise_numeric(ws_csr_t A, ws_csr_t B, ws_csr_t C, int32_t* c_colidx, void* c_vals,
                             ws_stream_t stream) {
  g_last_error.clear();
  ws_status_t st;
  if ((st = check_handle(A, "A")) != WS_OK || (st = check_handle(B, "B")) != WS_OK ||
      (st = check_handle(C, "C")) != WS_OK)
    return st;
  Plan* pl = C->plan;
  if (!pl || !pl->ready || pl->kind != kPlanEwise)
    return fail(WS_ERR_STATE, "numeric called before a successful elementwise symbolic pass");
  if (pl->A != A || pl->B != B || pl->a_nnz != A->nnz || pl->b_nnz != B->nnz)
    return fail(WS_ERR_STATE, "numeric called with other operands than the symbolic pass");
  if (C->nnz > 0 && (!c_colidx || !c_vals)) return fail(WS_ERR_INVALID_ARG, "c_colidx/c_vals NULL with nnz(C) > 0");
  C->colidx = c_colidx;
  C->vals = c_vals;
  pl->num_launches = 0;
  if (C->nnz == 0) return WS_OK;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const int sms = num_sms_of(C->device);
  if (A->dtype == WS_F64) {
    launch_ewise_numeric<double>(make_ewise<double>(A, B, C, pl), sms, s, &pl->num_launches);
  } else {
    launch_ewise_numeric<float>(make_ewise<float>(A, B, C, pl), sms, s, &pl->num_launches);
  }
  WS_CUDA(cudaGetLastError(), "elementwise numeric launch");
  return WS_OK;
}

ws_status_t ws_spmspv(ws_csr_t At, int64_t nnz_x, const int32_t* x_idx, const void* x_vals, int32_t* y_idx,
                      void* y_vals, int64_t* nnz_y, ws_stream_t stream) {
  g_last_error.clear();
  ws_status_t st;
  if ((st = check_handle(At, "At")) != WS_OK) return st;
  if (!nnz_y) return fail(WS_ERR_INVALID_ARG, "nnz_y is NULL");
  if (nnz_x < 0 || nnz_x > At->nrows) return fail(WS_ERR_INVALID_ARG, "nnz_x must be in [0, %lld]", (long long)At->nrows);
  if (nnz_x > 0 && (!x_idx || !x_vals)) return fail(WS_ERR_INVALID_ARG, "x_idx/x_vals NULL with nnz_x > 0");
  if (At->ncols > 0 && (!y_idx || !y_vals)) return fail(WS_ERR_INVALID_ARG, "y_idx/y_vals NULL");
  if ((st = ensure_plan(At)) != WS_OK) return st;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (At->dtype == WS_F64) return spmspv_impl<double>(At, nnz_x, x_idx, x_vals, y_idx, y_vals, nnz_y, s);
  return spmspv_impl<float>(At, nnz_x, x_idx, x_vals, y_idx, y_vals, nnz_y, s);
}

ws_status_t ws_csr_submatrix_symbolic(ws_csr_t A, int64_t r0, int64_t r1, int64_t c0, int64_t c1, ws_csr_t S,
                                      int64_t* nnz_out, ws_stream_t stream) {
  g_last_error.clear();
  ws_status_t st;
  if ((st = check_handle(A, "A")) != WS_OK || (st = check_handle(S, "S")) != WS_OK) return st;
  if (!nnz_out) return fail(WS_ERR_INVALID_ARG, "nnz_out is NULL");
  if (S == A) return fail(WS_ERR_INVALID_ARG, "S must be a separate output handle");
  if (r0 < 0 || r0 > r1 || r1 > A->nrows || c0 < 0 || c0 > c1 || c1 > A->ncols)
    return fail(WS_ERR_INVALID_ARG, "block [%lld:%lld, %lld:%lld] outside the %lldx%lld matrix", (long long)r0,
                (long long)r1, (long long)c0, (long long)c1, (long long)A->nrows, (long long)A->ncols);
  if (S->nrows != r1 - r0 || S->ncols != c1 - c0)
    return fail(WS_ERR_SHAPE, "S is %lldx%lld, expected %lldx%lld", (long long)S->nrows, (long long)S->ncols,
                (long long)(r1 - r0), (long long)(c1 - c0));
  if (S->dtype != A->dtype) return fail(WS_ERR_DTYPE, "A and S dtypes differ");
  if ((st = ensure_plan(S)) != WS_OK) return st;
  Plan* pl = S->plan;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const int64_t rows = r1 - r0;
  const int64_t nb = scan_partials_needed(rows);
  const size_t o_part = align_up(sizeof(DevSummary), 256);
  if ((st = pl->ew.reserve(o_part + 8 * static_cast<size_t>(nb + 1), s)) != WS_OK) return st;
  char* b = static_cast<char*>(pl->ew.ptr);
  pl->dsum = reinterpret_cast<DevSummary*>(b);
  int64_t* partials = reinterpret_cast<int64_t*>(b + o_part);
  pl->ready = false;
  pl->kind = kPlanSub;
  pl->sym_launches = 0;
  pl->num_launches = 0;
  S->nnz = -1;
  WS_CUDA(cudaMemsetAsync(pl->dsum, 0, sizeof(DevSummary), s), "cudaMemsetAsync(summary)");
  WS_CUDA(cudaMemsetAsync(S->rowptr, 0, sizeof(int64_t), s), "cudaMemsetAsync(rowptr[0])");
  if (rows > 0) {
    const int sms = num_sms_of(S->device);
    launch_submatrix_count(A->rowptr, A->colidx, r0, rows, c0, c1, S->rowptr, sms, s, &pl->sym_launches);
    launch_scan(S->rowptr, rows, partials, pl->dsum, s, &pl->sym_launches);
    WS_CUDA(cudaGetLastError(), "submatrix symbolic launches");
  }
  st = read_summary(pl, s);
  if (st != WS_OK) return st;
  S->nnz = rows > 0 ? pl->host_sum->nnz : 0;
  pl->A = A;
  pl->B = nullptr;
  pl->a_nnz = A->nnz;
  pl->sub_r0 = r0;
  pl->sub_r1 = r1;
  pl->sub_c0 = c0;
  pl->sub_c1 = c1;
  pl->ready = true;
  *nnz_out = S->nnz;
  return WS_OK;
}

ws_status_t ws_csr_submatrix_numeric(ws_csr_t A, ws_csr_t S, int32_t* s_colidx, void* s_vals, ws_stream_t stream) {
  g_last_error.clear();
  ws_status_t st;
  if ((st = check_handle(A, "A")) != WS_OK || (st = check_handle(S, "S")) != WS_OK) return st;
  Plan* pl = S->plan;
  if (!pl || !pl->ready || pl->kind != kPlanSub)
    return fail(WS_ERR_STATE, "numeric called before a successful submatrix symbolic pass");
  if (pl->A != A || pl->a_nnz != A->nnz)
    return fail(WS_ERR_STATE, "numeric called with another matrix than the symbolic pass");
  if (S->nnz > 0 && (!s_colidx || !s_vals)) return fail(WS_ERR_INVALID_ARG, "s_colidx/s_vals NULL with nnz(S) > 0");
  S->colidx = s_colidx;
  S->vals = s_vals;
  pl->num_launches = 0;
  if (S->nnz == 0) return WS_OK;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const int sms = num_sms_of(S->device);
  const int64_t rows = pl->sub_r1 - pl->sub_r0;
  if (A->dtype == WS_F64) {
    launch_submatrix_copy<double>(A->rowptr, A->colidx, static_cast<const double*>(A->vals), pl->sub_r0, rows,
                                  pl->sub_c0, S->rowptr, s_colidx, static_cast<double*>(s_vals), pl->dsum, sms, s,
                                  &pl->num_launches);
  } else {
    launch_submatrix_copy<float>(A->rowptr, A->colidx, static_cast<const float*>(A->vals), pl->sub_r0, rows,
                                 pl->sub_c0, S->rowptr, s_colidx, static_cast<float*>(s_vals), pl->dsum, sms, s,
                                 &pl->num_launches);
  }
  WS_CUDA(cudaGetLastError(), "submatrix numeric launch");
  return WS_OK;
}

ws_status_t ws_spgemm_wait(ws_csr_t C, ws_stream_t stream) {
  g_last_error.clear();
  if (!C) return fail(WS_ERR_INVALID_ARG, "C is NULL");
  Plan* pl = C->plan;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (!pl || !pl->host_sum || !pl->dsum) {
    WS_CUDA(cudaStreamSynchronize(s), "cudaStreamSynchronize");
    return WS_OK;
  }
  ws_status_t st = read_summary(pl, s);
  if (st != WS_OK) return st;
  return device_status(*pl->host_sum);
}

ws_status_t ws_csr_destroy(ws_csr_t h) {
  if (!h) return WS_OK;
  if (h->plan) {
    if (h->plan->rows.ptr || h->plan->slices.ptr || h->plan->ranks.ptr || h->plan->ew.ptr || h->plan->sv.ptr ||
        h->plan->rcd.ptr || h->plan->rcdb.ptr || h->plan->outer)
      cudaDeviceSynchronize();
    release_outer(h->plan, nullptr);
    h->plan->rows.release();
    h->plan->slices.release();
    h->plan->ranks.release();
    h->plan->ew.release();
    h->plan->sv.release();
    h->plan->rcd.release();
    h->plan->rcdb.release();
    release_host_sum(h->plan->host_sum);
    delete h->plan;
  }
  delete h;
  return WS_OK;
}

const char* ws_status_string(ws_status_t st) {
  switch (st) {
    case WS_OK: return "ok";
    case WS_ERR_INVALID_ARG: return "invalid argument";
    case WS_ERR_INVALID_CSR: return "invalid CSR matrix";
    case WS_ERR_SHAPE: return "shape mismatch";
    case WS_ERR_DTYPE: return "dtype mismatch";
    case WS_ERR_OVERFLOW: return "size overflow";
    case WS_ERR_ALLOC: return "allocation failed";
    case WS_ERR_CUDA: return "CUDA error";
    case WS_ERR_DEVICE: return "device-side failure";
    case WS_ERR_STATE: return "calls out of order";
  }
  return "unknown status";
}

const char* ws_last_error(void) { return g_last_error.c_str(); }

ws_status_t ws_csr_nnz(ws_csr_t h, int64_t* nnz_out) {
  if (!h || !nnz_out) return fail(WS_ERR_INVALID_ARG, "NULL argument");
  *nnz_out = h->nnz;
  return WS_OK;
}

ws_status_t ws_spgemm_plan_info(ws_csr_t C, int64_t* info, int n) {
  if (!C || !info || n < 0) return fail(WS_ERR_INVALID_ARG, "NULL argument");
  const Plan* pl = C->plan;
  int64_t v[12] = {0, 0, 0, 0, 0, 0, 0, 0, 0, 0, 0, 0};
  if (pl) {
    int64_t hash_rows = 0, bitmap_rows = 0;
    for (int b = 0; b < kNumHashBins; ++b) hash_rows += pl->seg_count[kSegHash0 + b];
    for (int b = 0; b < kNumBitmapBins; ++b) bitmap_rows += pl->seg_count[kSegBitmap0 + b];
    for (int b = 0; b < kNumBmrBins; ++b) bitmap_rows += pl->seg_count[kSegBmr0 + b];
    bitmap_rows += pl->seg_count[kSegBmrWide];
    v[0] = pl->n_empty;
    v[1] = pl->seg_count[kSegDirect];
    v[2] = hash_rows;
    v[3] = pl->n_sort;
    v[4] = pl->seg_count[kSegDense];
    v[5] = pl->dense_slices;
    v[6] = pl->products;
    v[7] = pl->sym_launches;
    v[8] = pl->num_launches;
    v[9] = bitmap_rows;
    v[10] = pl->seg_count[kSegRcd];
    v[11] = pl->seg_count[kSegWb];
  }
  for (int i = 0; i < n && i < 12; ++i) info[i] = v[i];
  return WS_OK;
}

ws_status_t ws_set_tuning(int key, int64_t value) {
  switch (key) {
    case 1:
      if (value < 0 || value > kMaxHashProducts) return fail(WS_ERR_INVALID_ARG, "hash limit out of range");
      g_hash_max = value;
      return WS_OK;
    case 2:
      if (value < 1 || value > 4096) return fail(WS_ERR_INVALID_ARG, "run limit out of range");
      g_run_limit = static_cast<int>(value);
      return WS_OK;
    case 3:
      if (value != 0 && (value < 1024 || value > 16384 || value % 1024 != 0))
        return fail(WS_ERR_INVALID_ARG, "dense width must be 0 or a multiple of 1024 in [1024, 16384]");
      g_dense_width = static_cast<int>(value);
      return WS_OK;
    case 4:
      if (value < 0 || value > kMaxBitmapSpan) return fail(WS_ERR_INVALID_ARG, "bitmap span out of range");
      g_bitmap_span = value;
      return WS_OK;
    case 5:
      if (value < 0 || value > kBmrMaxA) return fail(WS_ERR_INVALID_ARG, "register-row entry limit out of range");
      g_bmr_max_a = static_cast<int>(value);
      return WS_OK;
    case 6:
      if (value < 0 || value > kRcdMaxA) return fail(WS_ERR_INVALID_ARG, "dense-row entry limit out of range");
      g_rcd_max_a = static_cast<int>(value);
      return WS_OK;
    case 7:
      if (value < 0 || value > kWbMaxSpan) return fail(WS_ERR_INVALID_ARG, "wide-bitmap span out of range");
      g_wb_span = value;
      return WS_OK;
    case 8:
      if (value != -1 && value != 0 && value != 1 && value != kEwiseTileGroup && value != 4 && value != 8 &&
          value != 16 && value != 32 && value != kEwiseRankGroup)
        return fail(WS_ERR_INVALID_ARG, "elementwise lanes per chunk must be -1, 0, 1, 2, 4, 8, 16, 32 or 64");
      g_ewise_lanes = static_cast<int>(value);
      return WS_OK;
    case 9:
      if (value < 2 || value > (int64_t{1} << 20)) return fail(WS_ERR_INVALID_ARG, "elementwise chunk length out of range");
      g_ewise_diag = value;
      return WS_OK;
  }
  return fail(WS_ERR_INVALID_ARG, "unknown tuning key %d", key);
}

}  // extern "C"
