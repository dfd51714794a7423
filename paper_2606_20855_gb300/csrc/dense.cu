// Dense-window rows: rows with more products than the hash bins take.
//
// The row's column range [lo, hi] is cut into slices of `dense_width`
// columns; one CTA owns one slice at a time.  Its workspace is a dense
// bitmap of touched columns plus a dense value array over the slice -- the
// sparse byte-map workspace of Gustavson's SpGEMM (Sec. 5.1), with one bit
// per column in place of one byte.  Because every stored B row is sorted, a
// binary search finds the part of B[k,:] inside the slice.  Scanning the
// bitmap in column order yields the slice's entries already sorted, so no
// sort is needed.  Distinct slices of a row write disjoint, consecutive parts
// of the row's output segment (each slice is a shard of the row, Sec. 4);
// the symbolic pass stores every slice's entry count, and the numeric pass
// starts a slice's output after the counts of the row's earlier slices.
#include "ws_internal.cuh"

namespace wsk {

namespace {

constexpr int kDenseThreads = 256;

__host__ __device__ __forceinline__ size_t bitmap_bytes(int width) {
  return ((static_cast<size_t>(width) / 32) * sizeof(uint32_t) + 15) & ~static_cast<size_t>(15);
}

template <typename T, bool NUMERIC>
__global__ void __launch_bounds__(kDenseThreads) dense_rows_kernel(const RowPlan<T> p, int64_t nslices) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  __shared__ long long s_scan[32];
  __shared__ long long s_red[32];
  const int width = p.dense_width;
  const int nwords = width >> 5;
  uint32_t* bits = reinterpret_cast<uint32_t*>(smem_raw);
  T* vals = reinterpret_cast<T*>(smem_raw + bitmap_bytes(width));

  for (int w = threadIdx.x; w < nwords; w += kDenseThreads) bits[w] = 0u;
  if constexpr (NUMERIC) {
    for (int c = threadIdx.x; c < width; c += kDenseThreads) vals[c] = T(0);
  }
  __syncthreads();

  const int lg = p.log2_group;
  const int gsize = 1 << lg;
  const int grp = threadIdx.x >> lg;
  const int gl = threadIdx.x & (gsize - 1);
  const int ngrp = kDenseThreads >> lg;

  for (int64_t item = blockIdx.x; item < nslices; item += gridDim.x) {
    const int32_t row = p.slice_row[item];
    const int32_t sidx = p.slice_idx[item];
    const int32_t first = p.slice_first[item];
    const long long c0 = static_cast<long long>(p.lo[row]) + static_cast<long long>(sidx) * width;
    const long long c1 = min(c0 + width, static_cast<long long>(p.hi[row]) + 1);

    // Accumulate the products whose column falls in [c0, c1).
    const int64_t pa_end = p.A.rowptr[row + 1];
    for (int64_t pa = p.A.rowptr[row] + grp; pa < pa_end; pa += ngrp) {
      const int k = p.A.colidx[pa];
      T av = T(0);
      if constexpr (NUMERIC) av = p.A.vals[pa];
      int64_t lo = p.B.rowptr[k], hi = p.B.rowptr[k + 1];
      const int64_t qe = hi;
      while (lo < hi) {  // first position with column >= c0
        const int64_t mid = (lo + hi) >> 1;
        if (p.B.colidx[mid] < c0) lo = mid + 1;
        else hi = mid;
      }
      for (int64_t q = lo + gl; q < qe; q += gsize) {
        const int c = p.B.colidx[q];
        if (c >= c1) break;
        const int off = static_cast<int>(c - c0);
        atomicOr(&bits[off >> 5], 1u << (off & 31));
        if constexpr (NUMERIC) atomicAdd(&vals[off], av * p.B.vals[q]);
      }
    }
    __syncthreads();

    if constexpr (!NUMERIC) {
      long long cnt = 0;
      for (int w = threadIdx.x; w < nwords; w += kDenseThreads) {
        cnt += __popc(bits[w]);
        bits[w] = 0u;
      }
      long long total;
      block_exclusive_scan(cnt, s_scan, &total);
      if (threadIdx.x == 0) {
        p.slice_cnt[item] = static_cast<int32_t>(total);
        if (total) atomicAdd(reinterpret_cast<unsigned long long*>(&p.c_rowptr[row + 1]),
                             static_cast<unsigned long long>(total));
      }
    } else {
      // Start of this slice inside the row's output segment.
      long long before = 0;
      for (int s = threadIdx.x; s < sidx; s += kDenseThreads) before += p.slice_cnt[first + s];
      long long tot_before;
      block_exclusive_scan(before, s_red, &tot_before);
      const int64_t row_base = p.c_rowptr[row];
      const int64_t row_end = p.c_rowptr[row + 1];
      const int64_t base = row_base + tot_before;
      const long long expect = p.slice_cnt[item];
      long long emitted_total = 0;
      bool bad = false;
      for (int wb = 0; wb < nwords; wb += kDenseThreads) {
        const int w = wb + threadIdx.x;
        uint32_t word = w < nwords ? bits[w] : 0u;
        long long round_total;
        const long long excl = block_exclusive_scan(static_cast<long long>(__popc(word)), s_scan, &round_total);
        int64_t pos = base + emitted_total + excl;
        while (word) {
          const int b = __ffs(word) - 1;
          word &= word - 1;
          const int off = (w << 5) + b;
          if (pos < row_end && emitted_total + round_total <= expect) {
            p.c_colidx[pos] = static_cast<int32_t>(c0 + off);
            p.c_vals[pos] = vals[off];
          } else {
            bad = true;
          }
          vals[off] = T(0);
          ++pos;
        }
        if (w < nwords) bits[w] = 0u;
        emitted_total += round_total;
      }
      if (emitted_total != expect) bad = true;
      if (bad) atomicOr(&p.sum->status, kErrCount);
    }
    __syncthreads();
  }
}

}  // namespace

size_t dense_smem_bytes(int width, size_t value_bytes, bool numeric) {
  return bitmap_bytes(width) + (numeric ? static_cast<size_t>(width) * value_bytes : 0);
}

template <typename T>
void launch_dense(const RowPlan<T>& p, int64_t nslices, bool numeric, int num_sms, cudaStream_t s,
                  int* launches) {
  const size_t smem = dense_smem_bytes(p.dense_width, sizeof(T), numeric);
  auto kern = numeric ? dense_rows_kernel<T, true> : dense_rows_kernel<T, false>;
  cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  int per_sm = 0;
  cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kDenseThreads, smem);
  if (per_sm < 1) per_sm = 1;
  int64_t grid = nslices;
  const int64_t cap = static_cast<int64_t>(num_sms) * per_sm;
  if (grid > cap) grid = cap;
  if (grid < 1) grid = 1;
  kern<<<static_cast<int>(grid), kDenseThreads, smem, s>>>(p, nslices);
  *launches += 1;
}

template void launch_dense<float>(const RowPlan<float>&, int64_t, bool, int, cudaStream_t, int*);
template void launch_dense<double>(const RowPlan<double>&, int64_t, bool, int, cudaStream_t, int*);

}  // namespace wsk
