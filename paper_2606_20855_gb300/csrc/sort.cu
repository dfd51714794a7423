// Sorting path for hash rows whose monotone-hash table could not be ranked
// without a sort (a wrap-around or a long run of occupied slots, which skewed
// column distributions produce).  One CTA per row:
//   1. accumulate into a shared-memory hash table (multiplicative hash,
//      linear probing) -- the workspace w of Gustavson's algorithm (Sec. 5.1);
//   2. compact the occupied slots into a list;
//   3. bitonic-sort the list by column and write the row.
// These rows have at most kMaxHashProducts products, so the table (8192
// slots) is at most half full and the list holds at most 4096 entries.
#include <climits>

#include "ws_internal.cuh"

namespace wsk {

namespace {

constexpr int kSortThreads = 256;
constexpr int kTable = 1 << kSortTableLog;
constexpr int kList = kTable / 2;
constexpr int kEmptyKey = -1;

template <typename T>
__global__ void __launch_bounds__(kSortThreads) sort_rows_kernel(const RowPlan<T> p, int64_t nrows) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  int* keys = reinterpret_cast<int*>(smem_raw);
  T* vals = reinterpret_cast<T*>(keys + kTable);
  int* lkeys = reinterpret_cast<int*>(vals + kTable);
  T* lvals = reinterpret_cast<T*>(lkeys + kList);
  __shared__ int s_n;
  __shared__ int s_err;

  for (int64_t r = blockIdx.x; r < nrows; r += gridDim.x) {
    const int32_t row = p.sort_list[r];
    const int64_t base = p.c_rowptr[row];
    const int64_t cnt = p.c_rowptr[row + 1] - base;
    for (int s = threadIdx.x; s < kTable; s += kSortThreads) {
      keys[s] = kEmptyKey;
      vals[s] = T(0);
    }
    if (threadIdx.x == 0) {
      s_n = 0;
      s_err = 0;
    }
    __syncthreads();

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t pa_end = p.A.rowptr[row + 1];
    for (int64_t pa = p.A.rowptr[row] + warp; pa < pa_end; pa += kSortThreads / 32) {
      const int k = p.A.colidx[pa];
      const T av = p.A.vals[pa];
      const int64_t qe = p.B.rowptr[k + 1];
      for (int64_t q = p.B.rowptr[k] + lane; q < qe; q += 32) {
        const int c = p.B.colidx[q];
        const T v = av * p.B.vals[q];
        uint32_t h = (static_cast<uint32_t>(c) * 0x9E3779B1u) >> (32 - kSortTableLog);
        volatile int* vk = keys;
        bool done = false;
        for (int n = 0; n < kTable && !done; ++n) {
          int cur = vk[h];
          if (cur == kEmptyKey) cur = atomicCAS(&keys[h], kEmptyKey, c);
          if (cur == kEmptyKey || cur == c) {
            atomicAdd(&vals[h], v);
            done = true;
          } else {
            h = (h + 1) & (kTable - 1);
          }
        }
        if (!done) s_err = 1;
      }
    }
    __syncthreads();

    // Compact.
    for (int s = threadIdx.x; s < kTable; s += kSortThreads) {
      const int key = keys[s];
      if (key != kEmptyKey) {
        const int idx = atomicAdd(&s_n, 1);
        if (idx < kList) {
          lkeys[idx] = key;
          lvals[idx] = vals[s];
        }
      }
    }
    __syncthreads();
    const int n = s_n;
    if (n != cnt || n > kList || s_err) {
      if (threadIdx.x == 0) atomicOr(&p.sum->status, n > kList ? kErrSortCap : (s_err ? kErrProbe : kErrCount));
      __syncthreads();
      continue;
    }
    int np2 = 1;
    while (np2 < n) np2 <<= 1;
    for (int s = n + threadIdx.x; s < np2; s += kSortThreads) lkeys[s] = INT_MAX;
    __syncthreads();

    // Bitonic sort of lkeys[0, np2) ascending, values follow their keys.
    for (int k = 2; k <= np2; k <<= 1) {
      for (int j = k >> 1; j > 0; j >>= 1) {
        for (int i = threadIdx.x; i < np2; i += kSortThreads) {
          const int ixj = i ^ j;
          if (ixj > i) {
            const int a = lkeys[i], b = lkeys[ixj];
            const bool up = (i & k) == 0;
            if ((a > b) == up) {
              lkeys[i] = b;
              lkeys[ixj] = a;
              const T t = lvals[i];
              lvals[i] = lvals[ixj];
              lvals[ixj] = t;
            }
          }
        }
        __syncthreads();
      }
    }
    for (int s = threadIdx.x; s < n; s += kSortThreads) {
      p.c_colidx[base + s] = lkeys[s];
      p.c_vals[base + s] = lvals[s];
    }
    __syncthreads();
  }
}

}  // namespace

size_t sort_smem_bytes(size_t value_bytes) {
  return static_cast<size_t>(kTable) * (sizeof(int) + value_bytes) + static_cast<size_t>(kList) * (sizeof(int) + value_bytes);
}

template <typename T>
void launch_sort(const RowPlan<T>& p, int64_t nrows, int num_sms, cudaStream_t s, int* launches) {
  const size_t smem = sort_smem_bytes(sizeof(T));
  static bool configured = false;
  if (!configured) {
    cudaFuncSetAttribute(sort_rows_kernel<T>, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
    configured = true;
  }
  int64_t grid = nrows;
  if (grid > num_sms) grid = num_sms;
  if (grid < 1) grid = 1;
  sort_rows_kernel<T><<<static_cast<int>(grid), kSortThreads, smem, s>>>(p, nrows);
  *launches += 1;
}

template void launch_sort<float>(const RowPlan<float>&, int64_t, int, cudaStream_t, int*);
template void launch_sort<double>(const RowPlan<double>&, int64_t, int, cudaStream_t, int*);

}  // namespace wsk
