// Elementwise operations on CSR matrices of one shape (Sec. 5.2, "Sparse
// Linear Algebra": C = A op B with op in {+, elementwise product}):
//   SpAdd     C = A + B   pattern union, a sum of exactly 0.0 is kept;
//   Hadamard  C = A .* B  pattern intersection.
// Row i of C depends only on rows i of A and B, so distinct output positions
// go to distinct workers -- the sharded sparse list of Sec. 5.2 -- and no
// worker ever waits on another.
//
// Work units.  Row i is seen as the merge of its two sorted column lists
// (length na_i + nb_i) and cut into chunks of `diag` merged positions
// (merge-path diagonals; at least one chunk per row, so an empty row has one
// empty chunk).  A chunk boundary is placed by a binary search on the two
// lists, with the entry of A ahead of an equal entry of B and an equal pair
// never cut apart, so every chunk is the merge of a contiguous part of each
// list and no position of C is produced by two chunks.  Chunks balance long
// rows (power-law graphs) across the GPU.
//
// Merging a chunk.  A group of G lanes loads G entries of each list (a
// window), finds for every entry the number of entries of the other window
// below it (a binary search through shuffles) and whether it has an equal
// partner, and emits every entry not above the smaller of the two window
// maxima (entries above it may interleave with entries not yet loaded).  An
// output's position is the count of outputs before it: for the A entry of lane
// l, l plus the B-only entries below it; for a B-only entry, the A entries
// below it plus the B-only entries of lower lanes.  Each window step consumes
// at least one full window unless a list is exhausted.
//
// Symbolic pass: chunks per row -> scan -> chunk -> row map -> count per
// chunk -> scan (chunk output offsets, nnz(C)) -> C.rowptr[i] = offset of the
// first chunk of row i.  Numeric pass: every chunk merges again and writes its
// entries from its offset.
#include <climits>

#include "ws_internal.cuh"

namespace wsk {

namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr int kEwThreads = 256;

// Largest i such that the first d merged positions hold a[0..i) and
// b[0..d-i), with a[x] ahead of an equal b[y]; an equal pair straddling the
// cut moves to the left part (j + 1).  O(log na) probes.
__device__ __forceinline__ void merge_split(const int32_t* a, int64_t na, const int32_t* b, int64_t nb, int64_t d,
                                            int64_t* i_out, int64_t* j_out) {
  int64_t lo = d - nb > 0 ? d - nb : 0;
  int64_t hi = d < na ? d : na;
  while (lo < hi) {
    const int64_t mid = (lo + hi + 1) >> 1;
    if (d - mid >= nb || a[mid - 1] <= b[d - mid]) {
      lo = mid;
    } else {
      hi = mid - 1;
    }
  }
  int64_t j = d - lo;
  if (lo > 0 && j < nb && a[lo - 1] == b[j]) ++j;
  *i_out = lo;
  *j_out = j;
}

template <int G>
__device__ __forceinline__ unsigned group_bits(unsigned ballot, int g) {
  if constexpr (G == 32) {
    return ballot;
  } else {
    return (ballot >> (g * G)) & ((1u << G) - 1u);
  }
}

__device__ __forceinline__ unsigned below_mask(int k) { return k >= 32 ? kFull : (1u << k) - 1u; }

// Merges a[0..na) with b[0..nb) in windows of G entries; returns the number of
// outputs.  FILL: writes output q to (out_c[q], out_v[q]) for q < cap.
template <typename T, int G, int OP, bool FILL>
__device__ int64_t merge_chunk(const int32_t* a, const T* va, int64_t na, const int32_t* b, const T* vb, int64_t nb,
                               int g, int gl, unsigned gmask, int32_t* out_c, T* out_v, int64_t cap, bool* bad) {
  int64_t pa = 0, pb = 0, out = 0;
  const int64_t rounds = (na + G - 1) / G + (nb + G - 1) / G + 1;  // every window step consumes >= 1 entry
  for (int64_t r = 0; r < rounds && (pa < na || pb < nb); ++r) {
    const int64_t ia = pa + gl, ib = pb + gl;
    const int ca = ia < na ? a[ia] : INT_MAX;  // INT_MAX: past the end (no column reaches it)
    const int cb = ib < nb ? b[ib] : INT_MAX;
    T xa = T(0), xb = T(0);
    if constexpr (FILL) {
      xa = ia < na ? va[ia] : T(0);
      xb = ib < nb ? vb[ib] : T(0);
    }
    const int limit = min(__shfl_sync(gmask, ca, G - 1, G), __shfl_sync(gmask, cb, G - 1, G));
    // la = #{b window < ca}, lb = #{a window < cb}
    int la = 0, lb = 0;
#pragma unroll
    for (int s = G / 2; s > 0; s >>= 1) {
      if (__shfl_sync(gmask, cb, la + s - 1, G) < ca) la += s;
      if (__shfl_sync(gmask, ca, lb + s - 1, G) < cb) lb += s;
    }
    if (__shfl_sync(gmask, cb, la, G) < ca) ++la;
    if (__shfl_sync(gmask, ca, lb, G) < cb) ++lb;
    // every lane of the group takes part in each shuffle, so both run before the tests
    const int cb_at = __shfl_sync(gmask, cb, la & (G - 1), G);
    const int ca_at = __shfl_sync(gmask, ca, lb & (G - 1), G);
    const bool a_eq = la < G && cb_at == ca && ca != INT_MAX;
    const bool b_eq = lb < G && ca_at == cb && cb != INT_MAX;
    T xb_at = T(0);
    if constexpr (FILL) xb_at = __shfl_sync(gmask, xb, la & (G - 1), G);
    const bool a_take = ca != INT_MAX && ca <= limit;
    const bool b_take = cb != INT_MAX && cb <= limit;
    const unsigned ma = group_bits<G>(__ballot_sync(gmask, a_take), g);
    const unsigned mb = group_bits<G>(__ballot_sync(gmask, b_take), g);
    const unsigned below = below_mask(gl);
    if constexpr (OP == kEwiseAdd) {
      const unsigned mbu = group_bits<G>(__ballot_sync(gmask, b_take && !b_eq), g);  // B-only entries
      if constexpr (FILL) {
        if (a_take) {
          const int64_t q = out + gl + __popc(mbu & below_mask(la));
          if (q < cap) {
            out_c[q] = ca;
            out_v[q] = a_eq ? xa + xb_at : xa;
          } else {
            *bad = true;
          }
        }
        if (b_take && !b_eq) {
          const int64_t q = out + lb + __popc(mbu & below);
          if (q < cap) {
            out_c[q] = cb;
            out_v[q] = xb;
          } else {
            *bad = true;
          }
        }
      }
      out += __popc(ma) + __popc(mbu);
    } else {
      const unsigned md = group_bits<G>(__ballot_sync(gmask, a_take && a_eq), g);
      if constexpr (FILL) {
        if (a_take && a_eq) {
          const int64_t q = out + __popc(md & below);
          if (q < cap) {
            out_c[q] = ca;
            out_v[q] = xa * xb_at;
          } else {
            *bad = true;
          }
        }
      }
      out += __popc(md);
    }
    pa += __popc(ma);
    pb += __popc(mb);
  }
  if (pa < na || pb < nb) *bad = true;  // only for unsorted input: the step bound ran out
  return out;
}

__global__ void __launch_bounds__(kEwThreads) ew_chunks_per_row_kernel(int64_t m, const int64_t* arp,
                                                                       const int64_t* brp, int64_t diag,
                                                                       int64_t* chunk_begin) {
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < m;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t len = (arp[i + 1] - arp[i]) + (brp[i + 1] - brp[i]);
    chunk_begin[i + 1] = len > diag ? (len + diag - 1) / diag : 1;
  }
}

__global__ void __launch_bounds__(kEwThreads) ew_chunk_rows_kernel(int64_t m, const int64_t* chunk_begin,
                                                                   int64_t nc_max, int32_t* chunk_row) {
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < m;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t c1 = chunk_begin[i + 1] < nc_max ? chunk_begin[i + 1] : nc_max;
    for (int64_t c = chunk_begin[i]; c < c1; ++c) chunk_row[c] = static_cast<int32_t>(i);
  }
}

// One group of G lanes per chunk.  Counting: chunk_off[c + 1] = outputs of
// chunk c (0 for c beyond the last chunk).  FILL: writes chunk c's outputs
// from C offset chunk_off[c].
template <typename T, int G, int OP, bool FILL>
__global__ void __launch_bounds__(kEwThreads) ew_merge_kernel(const EwisePlan<T> p) {
  constexpr int kGroups = 32 / G;
  const int lane = threadIdx.x & 31;
  const int g = lane / G, gl = lane % G;
  const unsigned gmask = G == 32 ? kFull : (((1u << G) - 1u) << (g * G));
  const int64_t warp = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int64_t warps = (static_cast<int64_t>(gridDim.x) * blockDim.x) >> 5;
  const int64_t nc = p.chunk_begin[p.m];  // chunks in use (<= nc_max)
  bool bad = false;
  for (int64_t c = warp * kGroups + g; c < p.nc_max; c += warps * kGroups) {
    if (c >= nc) {
      if (!FILL && gl == 0) p.chunk_off[c + 1] = 0;
      continue;
    }
    const int32_t row = p.chunk_row[c];
    const int64_t k = c - p.chunk_begin[row];
    const int64_t a0 = p.A.rowptr[row], na = p.A.rowptr[row + 1] - a0;
    const int64_t b0 = p.B.rowptr[row], nb = p.B.rowptr[row + 1] - b0;
    const int32_t* a = p.A.colidx + a0;
    const int32_t* b = p.B.colidx + b0;
    const int64_t d0 = k * p.diag;
    const int64_t d1 = d0 + p.diag < na + nb ? d0 + p.diag : na + nb;
    int64_t i0 = 0, j0 = 0, i1 = na, j1 = nb;
    if (d0 > 0) merge_split(a, na, b, nb, d0, &i0, &j0);
    if (d1 < na + nb) merge_split(a, na, b, nb, d1, &i1, &j1);
    if constexpr (FILL) {
      const int64_t o0 = p.chunk_off[c];
      const int64_t cap = p.chunk_off[c + 1] - o0;
      const int64_t n = merge_chunk<T, G, OP, true>(a + i0, p.A.vals + a0 + i0, i1 - i0, b + j0, p.B.vals + b0 + j0,
                                                    j1 - j0, g, gl, gmask, p.c_colidx + o0, p.c_vals + o0, cap, &bad);
      if (n != cap) bad = true;
    } else {
      const int64_t n = merge_chunk<T, G, OP, false>(a + i0, nullptr, i1 - i0, b + j0, nullptr, j1 - j0, g, gl,
                                                     gmask, nullptr, nullptr, 0, &bad);
      if (gl == 0) p.chunk_off[c + 1] = n;
    }
  }
  if (bad) atomicOr(&p.sum->status, kErrCount);
}

// C.rowptr[i] = output offset of the first chunk of row i (i = 0..m; the
// first chunk past row m - 1 is the end).
__global__ void __launch_bounds__(kEwThreads) ew_rowptr_kernel(int64_t m, const int64_t* chunk_begin,
                                                               const int64_t* chunk_off, int64_t* c_rowptr) {
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i <= m;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x)
    c_rowptr[i] = chunk_off[chunk_begin[i]];
}

int grid_for(int64_t work, int per_block, int num_sms, int per_sm) {
  const int64_t want = (work + per_block - 1) / per_block;
  const int64_t cap = static_cast<int64_t>(num_sms) * per_sm;
  return static_cast<int>(want < 1 ? 1 : (want > cap ? cap : want));
}

template <typename T, int G, int OP, bool FILL>
void launch_merge(const EwisePlan<T>& p, int num_sms, cudaStream_t s) {
  const int grid = grid_for(p.nc_max, kEwThreads / 32 * (32 / G), num_sms, 8);
  ew_merge_kernel<T, G, OP, FILL><<<grid, kEwThreads, 0, s>>>(p);
}

template <typename T, int OP, bool FILL>
void launch_merge_g(const EwisePlan<T>& p, int num_sms, cudaStream_t s) {
  switch (p.group) {
    case 4: launch_merge<T, 4, OP, FILL>(p, num_sms, s); break;
    case 8: launch_merge<T, 8, OP, FILL>(p, num_sms, s); break;
    case 16: launch_merge<T, 16, OP, FILL>(p, num_sms, s); break;
    default: launch_merge<T, 32, OP, FILL>(p, num_sms, s); break;
  }
}

}  // namespace

template <typename T>
void launch_ewise_symbolic(const EwisePlan<T>& p, int num_sms, cudaStream_t s, int* launches) {
  ew_chunks_per_row_kernel<<<grid_for(p.m, kEwThreads, num_sms, 8), kEwThreads, 0, s>>>(p.m, p.A.rowptr, p.B.rowptr,
                                                                                        p.diag, p.chunk_begin);
  launch_scan(p.chunk_begin, p.m, p.partials, p.sum, s, launches);
  ew_chunk_rows_kernel<<<grid_for(p.m, kEwThreads, num_sms, 8), kEwThreads, 0, s>>>(p.m, p.chunk_begin, p.nc_max,
                                                                                    p.chunk_row);
  if (p.op == kEwiseAdd) {
    launch_merge_g<T, kEwiseAdd, false>(p, num_sms, s);
  } else {
    launch_merge_g<T, kEwiseMul, false>(p, num_sms, s);
  }
  launch_scan(p.chunk_off, p.nc_max, p.partials, p.sum, s, launches);
  ew_rowptr_kernel<<<grid_for(p.m + 1, kEwThreads, num_sms, 8), kEwThreads, 0, s>>>(p.m, p.chunk_begin, p.chunk_off,
                                                                                    p.c_rowptr);
  *launches += 4;
}

template <typename T>
void launch_ewise_numeric(const EwisePlan<T>& p, int num_sms, cudaStream_t s, int* launches) {
  if (p.op == kEwiseAdd) {
    launch_merge_g<T, kEwiseAdd, true>(p, num_sms, s);
  } else {
    launch_merge_g<T, kEwiseMul, true>(p, num_sms, s);
  }
  *launches += 1;
}

template void launch_ewise_symbolic<float>(const EwisePlan<float>&, int, cudaStream_t, int*);
template void launch_ewise_symbolic<double>(const EwisePlan<double>&, int, cudaStream_t, int*);
template void launch_ewise_numeric<float>(const EwisePlan<float>&, int, cudaStream_t, int*);
template void launch_ewise_numeric<double>(const EwisePlan<double>&, int, cudaStream_t, int*);

}  // namespace wsk
