// Submatrix extraction S = A[r0:r1, c0:c1] (CSR in, CSR out, columns shifted
// by -c0).  It is the layout step of the outer-product SpGEMM (Sec. 5.1, Fig.
// "SpGEMM implemented in WingSpan", outer product: the k loop is split over
// workers, worker p multiplies the column block A[:, K_p] by the row block
// B[K_p, :] into its own copy of C, and a merge level coalesces the copies).
//
// Count: one thread per output row finds, by binary search in the sorted row
// of A, the first column >= c0 and the first >= c1; their distance is the
// row's entry count (then scanned into S.rowptr).  Copy: a group of 32 lanes
// per row copies that contiguous range with coalesced loads and stores.
#include "ws_internal.cuh"

namespace wsk {

namespace {

constexpr int kSubThreads = 256;

// First position in cols[0..n) with cols[pos] >= c (n if none).
__device__ __forceinline__ int64_t lower_bound_col(const int32_t* cols, int64_t n, int64_t c) {
  int64_t lo = 0, hi = n;
  while (lo < hi) {  // O(log n) probes
    const int64_t mid = (lo + hi) >> 1;
    if (cols[mid] < c) {
      lo = mid + 1;
    } else {
      hi = mid;
    }
  }
  return lo;
}

__global__ void __launch_bounds__(kSubThreads) sub_count_kernel(const int64_t* rowptr, const int32_t* colidx,
                                                                int64_t r0, int64_t rows, int64_t c0, int64_t c1,
                                                                int64_t* s_rowptr) {
  for (int64_t r = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; r < rows;
       r += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t a0 = rowptr[r0 + r], n = rowptr[r0 + r + 1] - a0;
    const int32_t* cols = colidx + a0;
    s_rowptr[r + 1] = lower_bound_col(cols, n, c1) - lower_bound_col(cols, n, c0);
  }
}

template <typename T>
__global__ void __launch_bounds__(kSubThreads) sub_copy_kernel(const int64_t* rowptr, const int32_t* colidx,
                                                               const T* vals, int64_t r0, int64_t rows, int64_t c0,
                                                               const int64_t* s_rowptr, int32_t* s_colidx, T* s_vals,
                                                               DevSummary* sum) {
  const int lane = threadIdx.x & 31;
  const int64_t warp = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int64_t warps = (static_cast<int64_t>(gridDim.x) * blockDim.x) >> 5;
  for (int64_t r = warp; r < rows; r += warps) {
    const int64_t a0 = rowptr[r0 + r], n = rowptr[r0 + r + 1] - a0;
    // the row's first column >= c0, found by the warp: a 32-way search
    int64_t lo = 0, hi = n;  // answer in [lo, hi]
    for (int level = 0; level < 16 && lo < hi; ++level) {
      const int64_t step = (hi - lo + 31) / 32;
      const int64_t pos = lo + static_cast<int64_t>(lane) * step;
      const unsigned below = __ballot_sync(0xffffffffu, pos < hi && colidx[a0 + pos] < c0);
      const int cnt = __popc(below);  // probes below c0 form a prefix of the lanes
      lo = lo + (cnt > 0 ? static_cast<int64_t>(cnt - 1) * step + 1 : 0);
      const int64_t nhi = lo + step - 1;
      hi = hi < nhi ? hi : nhi;
    }
    const int64_t o0 = s_rowptr[r], len = s_rowptr[r + 1] - o0;
    if (lo + len > n) {  // inconsistent with the count pass (input changed in between)
      if (lane == 0) atomicOr(&sum->status, kErrCount);
      continue;
    }
    for (int64_t e = lane; e < len; e += 32) {
      s_colidx[o0 + e] = static_cast<int32_t>(colidx[a0 + lo + e] - c0);
      s_vals[o0 + e] = vals[a0 + lo + e];
    }
  }
}

int grid_for(int64_t work, int per_block, int num_sms, int per_sm) {
  const int64_t want = (work + per_block - 1) / per_block;
  const int64_t cap = static_cast<int64_t>(num_sms) * per_sm;
  return static_cast<int>(want < 1 ? 1 : (want > cap ? cap : want));
}

}  // namespace

void launch_submatrix_count(const int64_t* rowptr, const int32_t* colidx, int64_t r0, int64_t rows, int64_t c0,
                            int64_t c1, int64_t* s_rowptr, int num_sms, cudaStream_t s, int* launches) {
  sub_count_kernel<<<grid_for(rows, kSubThreads, num_sms, 8), kSubThreads, 0, s>>>(rowptr, colidx, r0, rows, c0, c1,
                                                                                   s_rowptr);
  *launches += 1;
}

template <typename T>
void launch_submatrix_copy(const int64_t* rowptr, const int32_t* colidx, const T* vals, int64_t r0, int64_t rows,
                           int64_t c0, const int64_t* s_rowptr, int32_t* s_colidx, T* s_vals, DevSummary* sum,
                           int num_sms, cudaStream_t s, int* launches) {
  sub_copy_kernel<T><<<grid_for(rows * 32, kSubThreads, num_sms, 8), kSubThreads, 0, s>>>(
      rowptr, colidx, vals, r0, rows, c0, s_rowptr, s_colidx, s_vals, sum);
  *launches += 1;
}

template void launch_submatrix_copy<float>(const int64_t*, const int32_t*, const float*, int64_t, int64_t, int64_t,
                                           const int64_t*, int32_t*, float*, DevSummary*, int, cudaStream_t, int*);
template void launch_submatrix_copy<double>(const int64_t*, const int32_t*, const double*, int64_t, int64_t, int64_t,
                                            const int64_t*, int32_t*, double*, DevSummary*, int, cudaStream_t, int*);

}  // namespace wsk
