// Row analysis and binning (first step of the symbolic pass), plus CSR validation.
//
// For every row i of C = A*B:
//   nnzA_i = A.rowptr[i+1] - A.rowptr[i]
//   ub_i   = sum over stored A[i,k] of (B.rowptr[k+1] - B.rowptr[k])   (products of the row)
//   lo_i   = min over those k of the first column of B[k,:]
//   hi_i   = max over those k of the last column of B[k,:]
// (B's rows are sorted, so every product of the row lands in [lo_i, hi_i].)
// The row's class follows from (nnzA_i, ub_i); the counts per class go to
// DevSummary so the host can size the per-class launches.  The work per row
// is not known before this pass (Sec. 1, irregular compute balance); the
// binning replaces the static/dynamic loop schedules of Sec. 4 with a
// partition of rows by their work.
#include <climits>

#include "ws_internal.cuh"

namespace wsk {

namespace {

__device__ __forceinline__ int ceil_log2_ll(long long x) {  // x >= 1
  return x <= 1 ? 0 : 64 - __clzll(x - 1);
}

// Class of a row from its stored-entry count, product count and column range.
// Bitmap bins take rows whose range fits a bitmap that is not much larger
// than the row's products (at most 8 words per product plus 64).
// Rows with at most bmr_max_a entries whose B rows fit one lane group take the
// register bitmap bins; other narrow rows with at most 1024 entries the
// bitmap bins.  Heavy rows (more entries than those) go to the dense rows
// (narrow range, few stored A entries: long B rows), the 8192-entry bitmap
// bin, the hash bins, the wide bitmap (range up to 2^20) and finally the
// column-sliced dense window.
__device__ __forceinline__ uint8_t classify(long long nnza, long long ub, int lo, int hi, int maxlen,
                                            const AnalyzeParams& ap) {
  if (ub == 0) return kClsEmpty;
  if (nnza == 1) return kClsDirect;
  const long long span = static_cast<long long>(hi) - lo + 1;
  const long long est = ub < span ? ub : span;  // entries of the row are at most this
  const bool bitmap_ok = span <= ap.bitmap_span && ((span + 31) >> 5) <= 8 * ub + 64;
  if (bitmap_ok) {
    if (nnza <= ap.bmr_max_a && maxlen <= ap.group) {
#pragma unroll
      for (int b = 0; b < kNumBmrBins; ++b) {
        if (span <= (32ll << bmr_log_words(b))) return static_cast<uint8_t>(kClsBmr0 + b);
      }
    }
#pragma unroll
    for (int b = 0; b < kNumBitmapBins - 1; ++b) {
      if (span <= (32ll << bitmap_log_words(b)) && est <= bitmap_cap(b)) return static_cast<uint8_t>(kClsBitmap0 + b);
    }
  }
  const bool heavy = ub > 4096 || (bitmap_ok && est > bitmap_cap(kNumBitmapBins - 2));
  if (heavy && span <= kMaxBitmapSpan && nnza <= ap.rcd_max_a) return kClsRcd;
  if (bitmap_ok && span <= (32ll << bitmap_log_words(kNumBitmapBins - 1)) && est <= bitmap_cap(kNumBitmapBins - 1))
    return static_cast<uint8_t>(kClsBitmap0 + kNumBitmapBins - 1);
  if (ub <= ap.hash_max) {
    int b = ceil_log2_ll(ub) - (kMinHashLog - 1);
    b = b < 0 ? 0 : b;
    return static_cast<uint8_t>(kClsHash0 + b);
  }
  if (span <= ap.wb_span) return kClsWb;
  return kClsDense;
}

__device__ __forceinline__ int segment_of(uint8_t cls) {
  if (cls == kClsDirect) return kSegDirect;
  if (cls == kClsDense) return kSegDense;
  if (cls == kClsBmrWide) return kSegBmrWide;
  if (cls == kClsRcd) return kSegRcd;
  if (cls == kClsWb) return kSegWb;
  if (cls < kClsBitmap0) return kSegBmr0 + (cls - kClsBmr0);      // register bitmap bins
  if (cls < kClsHash0) return kSegBitmap0 + (cls - kClsBitmap0);  // bitmap bins
  return kSegHash0 + (cls - kClsHash0);                            // hash bins
}

// Stores the class and column range of row i (and its count if it is known
// already) and returns the class.
template <typename T>
__device__ __forceinline__ uint8_t store_row(const RowPlan<T>& p, const AnalyzeParams& ap, int64_t i, long long nnza,
                                             long long ub, int lo, int hi, int maxlen, long long* s_slices) {
  const uint8_t c = classify(nnza, ub, lo, hi, maxlen, ap);
  p.cls[i] = c;
  // Direct rows know their count already; the others start at 0 and are
  // filled by the hash / dense-window symbolic kernels.
  p.c_rowptr[i + 1] = (c == kClsDirect) ? ub : 0;
  if (c != kClsEmpty) {
    p.lo[i] = lo;
    p.hi[i] = hi;
    if (c == kClsDense) {
      const long long span = static_cast<long long>(hi) - lo + 1;
      atomicAdd(reinterpret_cast<unsigned long long*>(s_slices),
                static_cast<unsigned long long>((span + ap.dense_width - 1) / ap.dense_width));
    }
  }
  return c;
}

// store_row for one row analysed by a single thread, with its counts added
// to the CTA's counters.
template <typename T>
__device__ __forceinline__ void record_row(const RowPlan<T>& p, const AnalyzeParams& ap, int64_t i, long long nnza,
                                           long long ub, int lo, int hi, int maxlen, int* s_seg, long long* s_prod,
                                           long long* s_slices, int* s_empty) {
  const uint8_t c = store_row(p, ap, i, nnza, ub, lo, hi, maxlen, s_slices);
  if (c == kClsEmpty) {
    atomicAdd(s_empty, 1);
  } else {
    atomicAdd(&s_seg[segment_of(c)], 1);
  }
  atomicAdd(reinterpret_cast<unsigned long long*>(s_prod), static_cast<unsigned long long>(ub));
}

template <typename T>
__device__ __forceinline__ void flush_counts(const RowPlan<T>& p, int* s_seg, long long* s_prod,
                                             long long* s_slices, int* s_empty) {
  if (threadIdx.x < kNumSegs && s_seg[threadIdx.x]) atomicAdd(&p.sum->seg_count[threadIdx.x], s_seg[threadIdx.x]);
  if (threadIdx.x == 0) {
    if (*s_prod) atomicAdd(reinterpret_cast<unsigned long long*>(&p.sum->products),
                           static_cast<unsigned long long>(*s_prod));
    if (*s_slices) atomicAdd(reinterpret_cast<unsigned long long*>(&p.sum->dense_slices),
                             static_cast<unsigned long long>(*s_slices));
    if (*s_empty) atomicAdd(&p.sum->n_empty, *s_empty);
  }
}

// Longest row a warp analyses; longer rows take a whole CTA.
constexpr int64_t kMidRowMax = 2048;

// One thread per row for rows with at most long_threshold stored entries;
// longer rows are queued in long_rows for analyze_long_kernel: rows up to
// kMidRowMax entries from the front (a warp per row), the others from the back
// (a CTA per row).
template <typename T>
__global__ void __launch_bounds__(256) analyze_kernel(const RowPlan<T> p, const AnalyzeParams ap,
                                                      int32_t* long_rows, const int32_t* rows) {
  __shared__ int s_seg[kNumSegs];
  __shared__ long long s_prod, s_slices;
  __shared__ int s_empty;
  if (threadIdx.x < kNumSegs) s_seg[threadIdx.x] = 0;
  if (threadIdx.x == 0) {
    s_prod = 0;
    s_slices = 0;
    s_empty = 0;
  }
  __syncthreads();
  const int64_t nrows = rows ? static_cast<int64_t>(*reinterpret_cast<volatile int*>(&p.sum->n_pending)) : ap.m;
  // Whole warps walk the rows (lane l takes row t0 + l), so that the counts
  // per class can be added once per warp and class: every row adding to the
  // same few CTA counters serialised on the shared-memory atomics.
  const int lane = threadIdx.x & 31;
  unsigned long long prod = 0;
  for (int64_t t0 = static_cast<int64_t>(blockIdx.x) * blockDim.x + (threadIdx.x & ~31); t0 < nrows;
       t0 += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t t = t0 + lane;
    int seg = -2;  // no row, or a long row (queued)
    if (t < nrows) {
      const int64_t i = rows ? rows[t] : t;
      const int64_t s = p.A.rowptr[i], e = p.A.rowptr[i + 1];
      if (e - s > ap.long_threshold) {
        if (e - s <= kMidRowMax) {
          long_rows[atomicAdd(&p.sum->n_mid, 1)] = static_cast<int32_t>(i);
        } else {
          long_rows[ap.m - 1 - atomicAdd(&p.sum->n_long, 1)] = static_cast<int32_t>(i);
        }
      } else {
        long long ub = 0;
        int lo = INT_MAX, hi = -1, maxlen = 0;
#pragma unroll 4
        for (int64_t q = s; q < e; ++q) {
          const int k = p.A.colidx[q];
          const int64_t bs = p.B.rowptr[k], be = p.B.rowptr[k + 1];
          if (be > bs) {
            ub += be - bs;
            maxlen = max(maxlen, static_cast<int>(min(be - bs, static_cast<int64_t>(INT_MAX))));
            lo = min(lo, p.B.colidx[bs]);
            hi = max(hi, p.B.colidx[be - 1]);
          }
        }
        const uint8_t c = store_row(p, ap, i, e - s, ub, lo, hi, maxlen, &s_slices);
        seg = c == kClsEmpty ? -1 : segment_of(c);
        prod += static_cast<unsigned long long>(ub);
      }
    }
    const unsigned peers = __match_any_sync(0xffffffffu, seg);
    if (seg >= -1 && lane == __ffs(peers) - 1) {
      if (seg < 0) {
        atomicAdd(&s_empty, __popc(peers));
      } else {
        atomicAdd(&s_seg[seg], __popc(peers));
      }
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) prod += __shfl_xor_sync(0xffffffffu, prod, o);
  if (lane == 0 && prod) atomicAdd(reinterpret_cast<unsigned long long*>(&s_prod), prod);
  __syncthreads();
  flush_counts(p, s_seg, &s_prod, &s_slices, &s_empty);
}

// Rows queued by analyze_kernel.  First one CTA per long row (a power-law
// row can hold tens of thousands of entries, and its three dependent loads
// per entry are a latency chain), then one warp per row of long_threshold + 1
// .. kMidRowMax entries (the lanes stride over the entries, eight in flight
// each, and warp reductions give the product count and the column range).
// For a long row:
// threads stride over the row's stored entries, eight in flight each, and
// the CTA reduces the product count and column range.
template <typename T>
__global__ void __launch_bounds__(256) analyze_long_kernel(const RowPlan<T> p, const AnalyzeParams ap,
                                                           const int32_t* long_rows) {
  __shared__ int s_seg[kNumSegs];
  __shared__ long long s_prod, s_slices;
  __shared__ int s_empty;
  __shared__ long long s_ub[8];
  __shared__ int s_lo[8], s_hi[8];
  if (threadIdx.x < kNumSegs) s_seg[threadIdx.x] = 0;
  if (threadIdx.x == 0) {
    s_prod = 0;
    s_slices = 0;
    s_empty = 0;
  }
  __syncthreads();
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int nlong = *reinterpret_cast<volatile int*>(&p.sum->n_long);
  for (int64_t w = blockIdx.x; w < nlong; w += gridDim.x) {
    const int64_t i = long_rows[ap.m - 1 - w];  // long rows fill the list from the back
    const int64_t s = p.A.rowptr[i], e = p.A.rowptr[i + 1];
    long long ub = 0;
    int lo = INT_MAX, hi = -1;
#pragma unroll 8
    for (int64_t q = s + threadIdx.x; q < e; q += blockDim.x) {
      const int k = p.A.colidx[q];
      const int64_t bs = p.B.rowptr[k], be = p.B.rowptr[k + 1];
      if (be > bs) {
        ub += be - bs;
        lo = min(lo, p.B.colidx[bs]);
        hi = max(hi, p.B.colidx[be - 1]);
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      ub += __shfl_xor_sync(0xffffffffu, ub, o);
      lo = min(lo, __shfl_xor_sync(0xffffffffu, lo, o));
      hi = max(hi, __shfl_xor_sync(0xffffffffu, hi, o));
    }
    if (lane == 0) {
      s_ub[warp] = ub;
      s_lo[warp] = lo;
      s_hi[warp] = hi;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      for (int w2 = 1; w2 < static_cast<int>(blockDim.x >> 5); ++w2) {
        ub += s_ub[w2];
        lo = min(lo, s_lo[w2]);
        hi = max(hi, s_hi[w2]);
      }
      record_row(p, ap, i, e - s, ub, lo, hi, INT_MAX, s_seg, &s_prod, &s_slices, &s_empty);
    }
    __syncthreads();  // s_ub/s_lo/s_hi are reused by the next row
  }
  const int nmid = *reinterpret_cast<volatile int*>(&p.sum->n_mid);
  const int64_t gw = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int64_t nw = (static_cast<int64_t>(gridDim.x) * blockDim.x) >> 5;
  for (int64_t w = gw; w < nmid; w += nw) {
    const int64_t i = long_rows[w];
    const int64_t s = p.A.rowptr[i], e = p.A.rowptr[i + 1];
    long long ub = 0;
    int lo = INT_MAX, hi = -1;
#pragma unroll 8
    for (int64_t q = s + lane; q < e; q += 32) {
      const int k = p.A.colidx[q];
      const int64_t bs = p.B.rowptr[k], be = p.B.rowptr[k + 1];
      if (be > bs) {
        ub += be - bs;
        lo = min(lo, p.B.colidx[bs]);
        hi = max(hi, p.B.colidx[be - 1]);
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      ub += __shfl_xor_sync(0xffffffffu, ub, o);
      lo = min(lo, __shfl_xor_sync(0xffffffffu, lo, o));
      hi = max(hi, __shfl_xor_sync(0xffffffffu, hi, o));
    }
    if (lane == 0) record_row(p, ap, i, e - s, ub, lo, hi, INT_MAX, s_seg, &s_prod, &s_slices, &s_empty);
  }
  __syncthreads();
  flush_counts(p, s_seg, &s_prod, &s_slices, &s_empty);
}

struct SegOffsets {
  long long off[kNumSegs];
};

// Groups non-empty rows by segment: perm[seg_offset[s] .. + seg_count[s]).
// Rows of one block keep their relative order inside each segment.
template <typename T>
__global__ void __launch_bounds__(256) scatter_kernel(const RowPlan<T> p, int64_t m, const SegOffsets so) {
  __shared__ int s_cnt[kNumSegs];
  __shared__ int s_base[kNumSegs];
  for (int64_t tile = static_cast<int64_t>(blockIdx.x) * blockDim.x; tile < m;
       tile += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    if (threadIdx.x < kNumSegs) s_cnt[threadIdx.x] = 0;
    __syncthreads();
    const int64_t i = tile + threadIdx.x;
    int seg = -1, rank = 0;
    if (i < m) {
      const uint8_t c = p.cls[i];
      if (c != kClsEmpty) {
        seg = segment_of(c);
        rank = atomicAdd(&s_cnt[seg], 1);
      }
    }
    __syncthreads();
    if (threadIdx.x < kNumSegs && s_cnt[threadIdx.x])
      s_base[threadIdx.x] = atomicAdd(&p.sum->seg_cursor[threadIdx.x], s_cnt[threadIdx.x]);
    __syncthreads();
    if (seg >= 0) p.perm[so.off[seg] + s_base[seg] + rank] = static_cast<int32_t>(i);
    __syncthreads();
  }
}

// Expands every dense-window row into its column slices.
template <typename T>
__global__ void __launch_bounds__(256) dense_slices_kernel(const RowPlan<T> p, int32_t* slice_row,
                                                           int32_t* slice_idx, int32_t* slice_first) {
  for (int64_t r = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; r < p.seg_len;
       r += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int32_t row = p.perm[p.seg_begin + r];
    const long long span = static_cast<long long>(p.hi[row]) - p.lo[row] + 1;
    const long long ns = (span + p.dense_width - 1) / p.dense_width;
    const long long first =
        static_cast<long long>(atomicAdd(reinterpret_cast<unsigned long long*>(&p.sum->slice_cursor),
                                         static_cast<unsigned long long>(ns)));
    for (long long s = 0; s < ns; ++s) {
      slice_row[first + s] = row;
      slice_idx[first + s] = static_cast<int32_t>(s);
      slice_first[first + s] = static_cast<int32_t>(first);
    }
  }
}

// Checks the CSR invariants of one matrix; records the smallest offending row.
__global__ void __launch_bounds__(256) validate_kernel(const int64_t* rowptr, const int32_t* colidx, int64_t nrows,
                                                       int64_t ncols, int64_t nnz, DevSummary* sum) {
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < nrows;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t s = rowptr[i], e = rowptr[i + 1];
    bool bad = s < 0 || e < s || e > nnz || (i == 0 && s != 0) || (i == nrows - 1 && e != nnz);
    if (!bad) {
      int prev = -1;
      for (int64_t q = s; q < e; ++q) {
        const int c = colidx[q];
        if (c <= prev || c >= ncols) {
          bad = true;
          break;
        }
        prev = c;
      }
    }
    if (bad) {
      atomicOr(&sum->status, kErrInvalidCsr);
      atomicMin(&sum->bad_row, static_cast<int>(i < INT_MAX ? i : INT_MAX));
    }
  }
}

int grid_for(int64_t work, int per_block, int num_sms, int blocks_per_sm) {
  int64_t g = (work + per_block - 1) / per_block;
  const int64_t cap = static_cast<int64_t>(num_sms) * blocks_per_sm;
  if (g > cap) g = cap;
  if (g < 1) g = 1;
  return static_cast<int>(g);
}

}  // namespace

template <typename T>
void launch_analyze(const RowPlan<T>& p, const AnalyzeParams& ap, int32_t* long_rows, const int32_t* rows,
                    int num_sms, cudaStream_t s, int* launches) {
  analyze_kernel<T><<<grid_for(ap.m, 256, num_sms, 8), 256, 0, s>>>(p, ap, long_rows, rows);
  analyze_long_kernel<T><<<num_sms * 8, 256, 0, s>>>(p, ap, long_rows);
  *launches += 2;
}

template <typename T>
void launch_scatter(const RowPlan<T>& p, int64_t m, const int64_t* seg_offset, int num_sms, cudaStream_t s,
                    int* launches) {
  SegOffsets so;
  for (int i = 0; i < kNumSegs; ++i) so.off[i] = seg_offset[i];
  scatter_kernel<T><<<grid_for(m, 256, num_sms, 8), 256, 0, s>>>(p, m, so);
  *launches += 1;
}

template <typename T>
void launch_dense_slices(const RowPlan<T>& p, int32_t* slice_row, int32_t* slice_idx, int32_t* slice_first,
                         int num_sms, cudaStream_t s, int* launches) {
  dense_slices_kernel<T><<<grid_for(p.seg_len, 256, num_sms, 4), 256, 0, s>>>(p, slice_row, slice_idx,
                                                                              slice_first);
  *launches += 1;
}

void launch_validate(const int64_t* rowptr, const int32_t* colidx, int64_t nrows, int64_t ncols, int64_t nnz,
                     DevSummary* sum, int num_sms, cudaStream_t s) {
  validate_kernel<<<grid_for(nrows, 256, num_sms, 8), 256, 0, s>>>(rowptr, colidx, nrows, ncols, nnz, sum);
}

#define WS_INST(T)                                                                                          \
  template void launch_analyze<T>(const RowPlan<T>&, const AnalyzeParams&, int32_t*, const int32_t*, int,      \
                                  cudaStream_t, int*);                                                       \
  template void launch_scatter<T>(const RowPlan<T>&, int64_t, const int64_t*, int, cudaStream_t, int*);      \
  template void launch_dense_slices<T>(const RowPlan<T>&, int32_t*, int32_t*, int32_t*, int, cudaStream_t, int*);
WS_INST(float)
WS_INST(double)
#undef WS_INST

}  // namespace wsk
