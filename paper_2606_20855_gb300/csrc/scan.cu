// Device-wide prefix sum that turns per-row entry counts into C's row
// pointer (the monotone position array of the compressed format, Sec. 1 and
// Sec. 3.1): on entry rowptr[i + 1] holds nnz(C[i,:]) and rowptr[0] = 0; on
// exit rowptr[i + 1] = sum_{r <= i} nnz(C[r,:]).
//
// Reduce-then-scan in three launches (tile sums, scan of the tile sums in one
// CTA, scan of each tile plus its offset); arrays of at most 16,384 entries
// are scanned by one CTA in one launch.  No CTA waits on another, so the
// scan cannot stall however the CTAs are scheduled.  With a `skip` flag the
// three kernels do nothing when *skip != 0 (a scan queued before the host
// knows whether every count is in place).
#include "ws_internal.cuh"

namespace wsk {

namespace {

constexpr int kScanThreads = 256;
constexpr int kScanItems = 16;
constexpr int kTile = kScanThreads * kScanItems;

__global__ void __launch_bounds__(kScanThreads) scan_reduce_kernel(const int64_t* x, int64_t n, int64_t* partial,
                                                                    const int* skip) {
  if (skip && *skip) return;
  __shared__ long long scratch[32];
  const int64_t tile0 = static_cast<int64_t>(blockIdx.x) * kTile;
  long long s = 0;
  for (int j = 0; j < kScanItems; ++j) {
    const int64_t i = tile0 + static_cast<int64_t>(j) * kScanThreads + threadIdx.x;
    if (i < n) s += x[i];
  }
  long long total;
  block_exclusive_scan(s, scratch, &total);
  if (threadIdx.x == 0) partial[blockIdx.x] = total;
}

// Exclusive scan of the tile sums, in place, by one CTA of 1024 threads.
__global__ void __launch_bounds__(1024) scan_partials_kernel(int64_t* partial, int64_t nb, const int* skip) {
  if (skip && *skip) return;
  __shared__ long long scratch[32];
  long long carry = 0;
  for (int64_t b0 = 0; b0 < nb; b0 += blockDim.x) {
    const int64_t b = b0 + threadIdx.x;
    const long long v = b < nb ? partial[b] : 0;
    long long total;
    const long long ex = block_exclusive_scan(v, scratch, &total);
    if (b < nb) partial[b] = carry + ex;
    carry += total;
  }
}

__global__ void __launch_bounds__(kScanThreads) scan_apply_kernel(int64_t* x, int64_t n, const int64_t* partial,
                                                                   DevSummary* sum, const int* skip) {
  if (skip && *skip) return;
  __shared__ long long scratch[32];
  const int64_t tile0 = static_cast<int64_t>(blockIdx.x) * kTile;
  // Each thread owns kScanItems consecutive elements.
  const int64_t my0 = tile0 + static_cast<int64_t>(threadIdx.x) * kScanItems;
  long long v[kScanItems];
  long long s = 0;
#pragma unroll
  for (int j = 0; j < kScanItems; ++j) {
    v[j] = (my0 + j < n) ? x[my0 + j] : 0;
    s += v[j];
  }
  long long total;
  long long run = block_exclusive_scan(s, scratch, &total) + partial[blockIdx.x];
#pragma unroll
  for (int j = 0; j < kScanItems; ++j) {
    run += v[j];
    if (my0 + j < n) x[my0 + j] = run;
    if (my0 + j == n - 1) sum->nnz = run;
  }
}

// Short arrays (n <= kSmallScan): one CTA of 1024 threads scans the whole
// array (the loop carries a running total, but one round covers kSmallScan).
constexpr int kSmallThreads = 1024;
constexpr int64_t kSmallScan = static_cast<int64_t>(kSmallThreads) * kScanItems;  // one round

__global__ void __launch_bounds__(kSmallThreads) scan_small_kernel(int64_t* x, int64_t n, DevSummary* sum,
                                                                   const int* skip) {
  if (skip && *skip) return;
  __shared__ long long scratch[32];
  long long carry = 0;
  for (int64_t r0 = 0; r0 < n; r0 += static_cast<int64_t>(kSmallThreads) * kScanItems) {
    const int64_t my0 = r0 + static_cast<int64_t>(threadIdx.x) * kScanItems;
    long long v[kScanItems];
    long long s = 0;
#pragma unroll
    for (int j = 0; j < kScanItems; ++j) {
      v[j] = (my0 + j < n) ? x[my0 + j] : 0;
      s += v[j];
    }
    long long total;
    long long run = block_exclusive_scan(s, scratch, &total) + carry;
#pragma unroll
    for (int j = 0; j < kScanItems; ++j) {
      run += v[j];
      if (my0 + j < n) x[my0 + j] = run;
      if (my0 + j == n - 1) sum->nnz = run;
    }
    carry += total;
  }
}

}  // namespace

int64_t scan_partials_needed(int64_t m) { return (m + kTile - 1) / kTile; }

void launch_scan(int64_t* rowptr, int64_t m, int64_t* partials, DevSummary* sum, cudaStream_t s, int* launches,
                 const int* skip) {
  if (m <= 0) return;
  if (m <= kSmallScan) {  // one launch instead of three
    scan_small_kernel<<<1, kSmallThreads, 0, s>>>(rowptr + 1, m, sum, skip);
    *launches += 1;
    return;
  }
  const int64_t nb = scan_partials_needed(m);
  scan_reduce_kernel<<<static_cast<int>(nb), kScanThreads, 0, s>>>(rowptr + 1, m, partials, skip);
  scan_partials_kernel<<<1, 1024, 0, s>>>(partials, nb, skip);
  scan_apply_kernel<<<static_cast<int>(nb), kScanThreads, 0, s>>>(rowptr + 1, m, partials, sum, skip);
  *launches += 3;
}

}  // namespace wsk
