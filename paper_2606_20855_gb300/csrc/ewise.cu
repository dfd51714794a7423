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
// (merge-path diagonals; an empty row has none).  A chunk boundary is placed
// by a binary search on the two lists, with the entry of A ahead of an equal
// entry of B and an equal pair
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
// chunk (the chunk's split, found by the binary search, is kept) -> scan
// (chunk output offsets, nnz(C)) -> C.rowptr[i] = offset of the first chunk
// of row i (of the next chunk for an empty row).  Numeric pass: every chunk
// reads its split and the next chunk's, merges again and writes its entries
// from its offset.  The default for short rows merges one chunk per lane
// from shared-memory copies of a warp's 32 chunks (ew_tile_kernel); its
// count keeps each chunk's absolute start in A and B instead of the split.
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
    // Counting needs only the equal pairs (found from the A side); writing a
    // union also needs the place of every B entry among the A entries.
    constexpr bool kBSide = FILL && OP == kEwiseAdd;
    int la = 0, lb = 0;
#pragma unroll
    for (int s = G / 2; s > 0; s >>= 1) {
      if (__shfl_sync(gmask, cb, la + s - 1, G) < ca) la += s;
      if constexpr (kBSide) {
        if (__shfl_sync(gmask, ca, lb + s - 1, G) < cb) lb += s;
      }
    }
    if (__shfl_sync(gmask, cb, la, G) < ca) ++la;
    // every lane of the group takes part in each shuffle, so they run before the tests
    const int cb_at = __shfl_sync(gmask, cb, la & (G - 1), G);
    const bool a_eq = la < G && cb_at == ca && ca != INT_MAX;
    bool b_eq = false;
    if constexpr (kBSide) {
      if (__shfl_sync(gmask, ca, lb, G) < cb) ++lb;
      const int ca_at = __shfl_sync(gmask, ca, lb & (G - 1), G);
      b_eq = lb < G && ca_at == cb && cb != INT_MAX;
    }
    T xb_at = T(0);
    if constexpr (FILL) xb_at = __shfl_sync(gmask, xb, la & (G - 1), G);
    const bool a_take = ca != INT_MAX && ca <= limit;
    const bool b_take = cb != INT_MAX && cb <= limit;
    const unsigned ma = group_bits<G>(__ballot_sync(gmask, a_take), g);
    const unsigned mb = group_bits<G>(__ballot_sync(gmask, b_take), g);
    const unsigned below = below_mask(gl);
    if constexpr (OP == kEwiseAdd && !FILL) {
      // union size: every A and B entry taken, less one per equal pair
      out += __popc(ma) + __popc(mb) - __popc(group_bits<G>(__ballot_sync(gmask, a_take && a_eq), g));
    } else if constexpr (OP == kEwiseAdd) {
      const unsigned mbu = group_bits<G>(__ballot_sync(gmask, b_take && !b_eq), g);  // B-only entries
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

// Output writer of one thread: entries go out four at a time as 16-byte
// stores once the position is a multiple of four (vec), singly before that
// and for the last partial group.  Positions past `cap` are dropped and
// flagged.
template <typename T>
struct SeqWriter {
  int32_t* c;
  T* v;
  int64_t cap, n = 0, head = 0;
  bool vec;
  int bc0 = 0, bc1 = 0, bc2 = 0, bc3 = 0;
  T bv0 = T(0), bv1 = T(0), bv2 = T(0), bv3 = T(0);

  __device__ SeqWriter(int32_t* c_, T* v_, int64_t cap_, int64_t abs0, bool vec_) : c(c_), v(v_), cap(cap_), vec(vec_) {
    head = vec ? ((4 - (abs0 & 3)) & 3) : cap;  // entries before the first 16-byte boundary
  }
  __device__ void put(int col, T val, bool* bad) {
    if (n >= cap) {
      *bad = true;
      return;
    }
    if (n < head) {
      c[n] = col;
      v[n] = val;
    } else {
      const int slot = static_cast<int>((n - head) & 3);
      bc0 = slot == 0 ? col : bc0;
      bc1 = slot == 1 ? col : bc1;
      bc2 = slot == 2 ? col : bc2;
      bc3 = slot == 3 ? col : bc3;
      bv0 = slot == 0 ? val : bv0;
      bv1 = slot == 1 ? val : bv1;
      bv2 = slot == 2 ? val : bv2;
      bv3 = slot == 3 ? val : bv3;
      if (slot == 3) {
        const int64_t q = n - 3;
        *reinterpret_cast<int4*>(c + q) = make_int4(bc0, bc1, bc2, bc3);
        if constexpr (sizeof(T) == 4) {
          *reinterpret_cast<float4*>(v + q) = make_float4(bv0, bv1, bv2, bv3);
        } else {
          reinterpret_cast<double2*>(v + q)[0] = make_double2(bv0, bv1);
          reinterpret_cast<double2*>(v + q)[1] = make_double2(bv2, bv3);
        }
      }
    }
    ++n;
  }
  __device__ void flush() {
    if (n <= head) return;
    const int rest = static_cast<int>((n - head) & 3);
    const int64_t q = n - rest;
    if (rest > 0) { c[q] = bc0; v[q] = bv0; }
    if (rest > 1) { c[q + 1] = bc1; v[q + 1] = bv1; }
    if (rest > 2) { c[q + 2] = bc2; v[q + 2] = bv2; }
  }
};

// One thread merges a[0..na) with b[0..nb) entry by entry (the two lists sit
// in a few cache lines each, so the loads after the first hit L1); returns
// the number of outputs.  FILL: writes them through `w`.
template <typename T, int OP, bool FILL>
__device__ int64_t merge_seq(const int32_t* a, const T* va, int64_t na, const int32_t* b, const T* vb, int64_t nb,
                             SeqWriter<T>* w, bool* bad) {
  int64_t i = 0, j = 0, out = 0;
  int ca = na > 0 ? a[0] : INT_MAX;
  int cb = nb > 0 ? b[0] : INT_MAX;
  for (int64_t step = 0; step < na + nb && (i < na || j < nb); ++step) {
    const bool take_a = ca <= cb, take_b = cb <= ca;
    if constexpr (OP == kEwiseAdd) {
      if constexpr (FILL) w->put(take_a ? ca : cb, take_a && take_b ? va[i] + vb[j] : (take_a ? va[i] : vb[j]), bad);
      ++out;
    } else if (take_a && take_b) {
      if constexpr (FILL) w->put(ca, va[i] * vb[j], bad);
      ++out;
    }
    if (take_a) {
      ++i;
      ca = i < na ? a[i] : INT_MAX;
    }
    if (take_b) {
      ++j;
      cb = j < nb ? b[j] : INT_MAX;
    }
  }
  if (i < na || j < nb) *bad = true;  // only for unsorted input: the step bound ran out
  if constexpr (FILL) w->flush();
  return out;
}

// SpAdd fill of one chunk: every merge step emits one entry of the union,
// so after a scalar head up to the first 16-byte boundary of C the steps go
// four at a time into registers with fixed slots and leave as one 16-byte
// store of columns and one (fp32) or two (fp64) of values; the tail is
// scalar again.  `cap` is the chunk's entry count from the symbolic pass.
template <typename T>
__device__ int64_t merge_add_fill(const int32_t* a, const T* va, int64_t na, const int32_t* b, const T* vb,
                                  int64_t nb, int32_t* c, T* v, int64_t cap, int64_t abs0, bool vec, bool* bad) {
  int64_t i = 0, j = 0, n = 0;
  int ca = na > 0 ? a[0] : INT_MAX;
  int cb = nb > 0 ? b[0] : INT_MAX;
  // One merge step: the smaller head (both when equal, values added).
  auto step = [&](int* col, T* val) {
    const bool take_a = ca <= cb, take_b = cb <= ca;
    *col = take_a ? ca : cb;
    const T x = take_a ? va[i] : T(0);
    const T y = take_b ? vb[j] : T(0);
    *val = take_a ? (take_b ? x + y : x) : y;
    if (take_a) {
      ++i;
      ca = i < na ? a[i] : INT_MAX;
    }
    if (take_b) {
      ++j;
      cb = j < nb ? b[j] : INT_MAX;
    }
  };
  auto more = [&]() { return i < na || j < nb; };
  if (vec) {
    for (int h = 0; h < 3 && more() && n < cap && ((abs0 + n) & 3); ++h, ++n) step(c + n, v + n);
    for (int64_t g = 0; g < (na + nb) / 4 + 1 && n + 4 <= cap; ++g, n += 4) {
      int c0, c1, c2, c3;
      T v0, v1, v2, v3;
      // n + 4 <= cap: four more entries exist unless the lists changed since the count
      if (!more()) break;
      step(&c0, &v0);
      if (!more()) { *bad = true; break; }
      step(&c1, &v1);
      if (!more()) { *bad = true; break; }
      step(&c2, &v2);
      if (!more()) { *bad = true; break; }
      step(&c3, &v3);
      *reinterpret_cast<int4*>(c + n) = make_int4(c0, c1, c2, c3);
      if constexpr (sizeof(T) == 4) {
        *reinterpret_cast<float4*>(v + n) = make_float4(v0, v1, v2, v3);
      } else {
        reinterpret_cast<double2*>(v + n)[0] = make_double2(v0, v1);
        reinterpret_cast<double2*>(v + n)[1] = make_double2(v2, v3);
      }
    }
  }
  for (int64_t guard = 0; guard <= na + nb && more(); ++guard, ++n) {
    int col;
    T val;
    step(&col, &val);
    if (n < cap) {
      c[n] = col;
      v[n] = val;
    } else {
      *bad = true;
    }
  }
  return n;
}

// The chunk's ranges a[i0..i1) and b[j0..j1) (merged positions d0..d1 of
// the row).  The symbolic pass finds the split at d0 by binary search and
// keeps it in chunk_split as 2 * i0 + (j0 - (d0 - i0)) (an equal pair
// straddling the cut puts j0 one past d0 - i0); the numeric pass reads its
// own and the next chunk's split from there, clamped to the lists (if the
// input changed in between, the ranges stay inside them and the count check
// reports it).
template <bool FILL, typename T>
__device__ __forceinline__ void chunk_bounds(const EwisePlan<T>& p, int64_t c, const int32_t* a, int64_t na,
                                             const int32_t* b, int64_t nb, int64_t d0, int64_t d1, int64_t* i0,
                                             int64_t* j0, int64_t* i1, int64_t* j1, bool writer) {
  auto decode = [&](int64_t d, int64_t code, int64_t* i, int64_t* j) {
    const int64_t lo = d - nb > 0 ? d - nb : 0, hi = d < na ? d : na;
    const int64_t x = code >> 1;
    *i = x < lo ? lo : (x > hi ? hi : x);
    const int64_t y = d - *i + (code & 1);
    *j = y > nb ? nb : y;
  };
  if constexpr (!FILL) {
    if (d0 > 0) merge_split(a, na, b, nb, d0, i0, j0);
    if (d1 < na + nb) merge_split(a, na, b, nb, d1, i1, j1);
    if (writer) p.chunk_split[c] = 2 * *i0 + (*j0 - (d0 - *i0));
  } else {
    decode(d0, p.chunk_split[c], i0, j0);
    if (d1 < na + nb) decode(d1, p.chunk_split[c + 1], i1, j1);  // the next chunk belongs to this row
  }
}

// One thread per chunk, same contract as ew_merge_kernel.
template <typename T, int OP, bool FILL>
__global__ void __launch_bounds__(kEwThreads, FILL ? 4 : 6) ew_merge_seq_kernel(const EwisePlan<T> p) {
  const int64_t nc = p.chunk_begin[p.m];
  bool bad = false;
  // 16-byte stores need 16-byte aligned C arrays (any allocation is)
  const bool vec = ((reinterpret_cast<uintptr_t>(p.c_colidx) | reinterpret_cast<uintptr_t>(p.c_vals)) & 15u) == 0;
  for (int64_t c = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; c < p.nc_max;
       c += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    if (c >= nc) {
      if (!FILL) p.chunk_off[c + 1] = 0;
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
    chunk_bounds<FILL>(p, c, a, na, b, nb, d0, d1, &i0, &j0, &i1, &j1, threadIdx.x % p.group == 0);
    if constexpr (FILL) {
      const int64_t o0 = p.chunk_off[c];
      const int64_t cap = p.chunk_off[c + 1] - o0;
      int64_t n;
      if constexpr (OP == kEwiseAdd) {
        n = merge_add_fill<T>(a + i0, p.A.vals + a0 + i0, i1 - i0, b + j0, p.B.vals + b0 + j0, j1 - j0,
                              p.c_colidx + o0, p.c_vals + o0, cap, o0, vec, &bad);
      } else {
        SeqWriter<T> w(p.c_colidx + o0, p.c_vals + o0, cap, o0, vec);
        n = merge_seq<T, OP, true>(a + i0, p.A.vals + a0 + i0, i1 - i0, b + j0, p.B.vals + b0 + j0, j1 - j0, &w,
                                   &bad);
      }
      if (n != cap) bad = true;
    } else {
      p.chunk_off[c + 1] = merge_seq<T, OP, false>(a + i0, nullptr, i1 - i0, b + j0, nullptr, j1 - j0, nullptr, &bad);
    }
  }
  if (bad) atomicOr(&p.sum->status, kErrCount);
}

// Warp-staged tiles: a warp takes 32 consecutive chunks, one per lane.  The
// chunks' parts of A and of B are contiguous runs of A's and B's arrays
// (consecutive chunks of a row continue each other; the rows between two
// chunks are empty), so the warp first copies the two runs into shared
// memory with coalesced loads; every lane then merges its chunk from there,
// with no dependent global loads in the merge loop.  A lane whose bounds
// fall outside the staged runs (only if the inputs changed since the
// symbolic pass) merges from global memory; the count check then reports it.
constexpr int kTileWarps = 4;
constexpr int kTileCap = 32 * kEwiseTileDiag;  // staged entries per list and warp

// Values are staged for the union's fill only: an intersection reads the
// values of its (few) equal pairs from global memory.
template <int OP, bool FILL>
constexpr bool tile_stages_values() { return FILL && OP == kEwiseAdd; }
template <typename T, int OP, bool FILL>
constexpr size_t tile_warp_bytes() {
  return 2 * static_cast<size_t>(kTileCap) * (sizeof(int32_t) + (tile_stages_values<OP, FILL>() ? sizeof(T) : 0));
}

template <typename T, int OP, bool FILL>
__global__ void __launch_bounds__(32 * kTileWarps) ew_tile_kernel(const EwisePlan<T> p) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  constexpr bool kVals = tile_stages_values<OP, FILL>();
  // per warp: A values, B values (when staged), then A columns, B columns
  unsigned char* ws = smem_raw + static_cast<size_t>(warp) * tile_warp_bytes<T, OP, FILL>();
  T* sva = reinterpret_cast<T*>(ws);
  T* svb = sva + (kVals ? kTileCap : 0);
  int32_t* sca = reinterpret_cast<int32_t*>(svb + (kVals ? kTileCap : 0));
  int32_t* scb = sca + kTileCap;
  const int64_t nc = p.chunk_begin[p.m];
  bool bad = false;
  const bool vec = ((reinterpret_cast<uintptr_t>(p.c_colidx) | reinterpret_cast<uintptr_t>(p.c_vals)) & 15u) == 0;
  const int64_t ntiles = (p.nc_max + 31) / 32;
  for (int64_t tile = static_cast<int64_t>(blockIdx.x) * kTileWarps + warp; tile < ntiles;
       tile += static_cast<int64_t>(gridDim.x) * kTileWarps) {
    const int64_t c = tile * 32 + lane;
    if (!FILL && c >= nc && c < p.nc_max) p.chunk_off[c + 1] = 0;
    if (!FILL && c == nc) {  // end positions, read as the bounds after the last chunk
      p.chunk_split[nc] = p.A.rowptr[p.m];
      p.chunk_bpos[nc] = p.B.rowptr[p.m];
    }
    const bool valid = c < nc;
    const unsigned vmask = __ballot_sync(kFull, valid);
    if (vmask == 0u) continue;  // past the last chunk (the counts above are zeroed all the same)
    // The chunk's parts of A and B as absolute positions [ga0, ga1), [gb0, gb1).
    int64_t ga0 = 0, ga1 = 0, gb0 = 0, gb1 = 0;
    if (valid) {
      if constexpr (FILL) {
        // kept by the symbolic pass; chunk c + 1 (or the end) bounds chunk c
        ga0 = p.chunk_split[c];
        gb0 = p.chunk_bpos[c];
        ga1 = p.chunk_split[c + 1];
        gb1 = p.chunk_bpos[c + 1];
        // A changed input could leave the bounds out of order or outside the
        // lists: clamp them (the count check then reports the difference).
        const int64_t a_end = p.A.rowptr[p.m], b_end = p.B.rowptr[p.m];
        ga0 = ga0 < 0 ? 0 : (ga0 > a_end ? a_end : ga0);
        ga1 = ga1 < ga0 ? ga0 : (ga1 > a_end ? a_end : ga1);
        gb0 = gb0 < 0 ? 0 : (gb0 > b_end ? b_end : gb0);
        gb1 = gb1 < gb0 ? gb0 : (gb1 > b_end ? b_end : gb1);
      } else {
        const int32_t row = p.chunk_row[c];
        const int64_t k = c - p.chunk_begin[row];
        const int64_t a0 = p.A.rowptr[row], na = p.A.rowptr[row + 1] - a0;
        const int64_t b0 = p.B.rowptr[row], nb = p.B.rowptr[row + 1] - b0;
        const int64_t d0 = k * p.diag;
        const int64_t d1 = d0 + p.diag < na + nb ? d0 + p.diag : na + nb;
        int64_t i0 = 0, j0 = 0, i1 = na, j1 = nb;
        chunk_bounds<false>(p, c, p.A.colidx + a0, na, p.B.colidx + b0, nb, d0, d1, &i0, &j0, &i1, &j1, false);
        ga0 = a0 + i0;
        ga1 = a0 + i1;
        gb0 = b0 + j0;
        gb1 = b0 + j1;
        p.chunk_split[c] = ga0;
        p.chunk_bpos[c] = gb0;
      }
    }
    // The tile's runs: from the first lane's start to the last valid lane's end.
    const int last = 31 - __clz(vmask);
    const int64_t alo = __shfl_sync(kFull, ga0, 0), ahi = __shfl_sync(kFull, ga1, last);
    const int64_t blo = __shfl_sync(kFull, gb0, 0), bhi = __shfl_sync(kFull, gb1, last);
    const bool staged = ahi - alo <= kTileCap && bhi - blo <= kTileCap && ahi >= alo && bhi >= blo;
    if (staged) {
      const int n_a = static_cast<int>(ahi - alo), n_b = static_cast<int>(bhi - blo);
      for (int t = lane; t < n_a; t += 32) {
        sca[t] = p.A.colidx[alo + t];
        if constexpr (kVals) sva[t] = p.A.vals[alo + t];
      }
      for (int t = lane; t < n_b; t += 32) {
        scb[t] = p.B.colidx[blo + t];
        if constexpr (kVals) svb[t] = p.B.vals[blo + t];
      }
    }
    __syncwarp();
    if (valid) {
      const bool mine = staged && ga0 >= alo && ga1 <= ahi && gb0 >= blo && gb1 <= bhi;
      const int64_t na = ga1 - ga0, nb = gb1 - gb0;
      // The same merge for staged lists and (after a changed input) for the
      // global arrays; separate calls keep the staged one on shared-memory loads.
      auto merge = [&](const int32_t* a, const T* va, const int32_t* b, const T* vb) {
        if constexpr (FILL) {
          const int64_t o0 = p.chunk_off[c];
          const int64_t cap = p.chunk_off[c + 1] - o0;
          int64_t n;
          if constexpr (OP == kEwiseAdd) {
            n = merge_add_fill<T>(a, va, na, b, vb, nb, p.c_colidx + o0, p.c_vals + o0, cap, o0, vec, &bad);
          } else {
            SeqWriter<T> w(p.c_colidx + o0, p.c_vals + o0, cap, o0, vec);
            n = merge_seq<T, OP, true>(a, va, na, b, vb, nb, &w, &bad);
          }
          if (n != cap) bad = true;
        } else {
          p.chunk_off[c + 1] = merge_seq<T, OP, false>(a, nullptr, na, b, nullptr, nb, nullptr, &bad);
        }
      };
      if (mine) {
        merge(sca + (ga0 - alo), kVals ? sva + (ga0 - alo) : p.A.vals + ga0, scb + (gb0 - blo),
              kVals ? svb + (gb0 - blo) : p.B.vals + gb0);
      } else {
        merge(p.A.colidx + ga0, p.A.vals + ga0, p.B.colidx + gb0, p.B.vals + gb0);
      }
    }
    __syncwarp();  // the next tile rewrites the staging
  }
  if (bad) atomicOr(&p.sum->status, kErrCount);
}

__global__ void __launch_bounds__(kEwThreads) ew_chunks_per_row_kernel(int64_t m, const int64_t* arp,
                                                                       const int64_t* brp, int64_t diag,
                                                                       int64_t* chunk_begin) {
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < m;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t len = (arp[i + 1] - arp[i]) + (brp[i + 1] - brp[i]);
    chunk_begin[i + 1] = (len + diag - 1) / diag;  // an empty row has no chunk
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
__global__ void __launch_bounds__(kEwThreads, FILL ? 4 : 6) ew_merge_kernel(const EwisePlan<T> p) {
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
    chunk_bounds<FILL>(p, c, a, na, b, nb, d0, d1, &i0, &j0, &i1, &j1, threadIdx.x % p.group == 0);
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

// A warp per chunk, chunks taken 32 at a time (kEwiseRankChunk merged
// positions each).  Lane l first fetches the bounds of chunk t0 + l (row, the split of
// each list, C offset), so the dependent loads of 32 chunks overlap; then the
// warp takes the chunks in turn.  A chunk's parts of the two lists are staged
// in shared memory with coalesced loads (the next chunk's are loaded while the
// current one is merged), and every entry finds its place by a binary search
// in the other part: for A entry x, lb = #B entries below it and whether B
// holds its column; for B entry y, the same against A.  Ballots over the
// "has an equal partner" flags give the pairs below each entry, so
//   SpAdd:    rank(A x) = x + lb - pairs below x          (value a + b at a pair)
//             rank(B y) = y + lb - pairs below y, B entries with a partner skipped
//   Hadamard: rank(A x) = pairs below x, A entries without a partner skipped
// and the count is na + nb - pairs (SpAdd) or pairs (Hadamard).  The outputs
// of a chunk are one contiguous run of C written in order.
constexpr int kRankSlots = 96;  // staged entries per list (a chunk part holds at most kEwiseRankChunk + 1)
static_assert(kEwiseRankChunk + 1 <= kRankSlots, "a chunk's part of a list fits the staging");
constexpr int kRankWarps = kEwThreads / 32;

// First position in s[0..n) holding a value >= x (n if none).
__device__ __forceinline__ int lower_bound_smem(const int* s, int n, int x) {
  int lo = 0, hi = n;
#pragma unroll 1
  while (lo < hi) {
    const int mid = (lo + hi) >> 1;
    if (s[mid] < x) {
      lo = mid + 1;
    } else {
      hi = mid;
    }
  }
  return lo;
}

template <typename T, int OP, bool FILL>
__global__ void __launch_bounds__(kEwThreads) ew_rank_kernel(const EwisePlan<T> p) {
  __shared__ int s_ac[kRankWarps][kRankSlots], s_bc[kRankWarps][kRankSlots];
  __shared__ T s_av[kRankWarps][FILL ? kRankSlots : 1], s_bv[kRankWarps][FILL ? kRankSlots : 1];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  int* ac = s_ac[w];
  int* bc = s_bc[w];
  T* av = s_av[w];
  T* bv = s_bv[w];
  const int64_t nc = p.chunk_begin[p.m];
  const int64_t gwarp = static_cast<int64_t>(blockIdx.x) * kRankWarps + w;
  const int64_t nwarps = static_cast<int64_t>(gridDim.x) * kRankWarps;
  bool bad = false;
  for (int64_t t0 = gwarp * 32; t0 < p.nc_max; t0 += nwarps * 32) {
    // bounds of chunk t0 + lane
    const int64_t c = t0 + lane;
    int64_t ga = 0, gb = 0, o0 = 0, cap = 0;
    int na = 0, nb = 0;
    const bool valid = c < nc;
    if (!FILL && c >= nc && c < p.nc_max) p.chunk_off[c + 1] = 0;
    if (valid) {
      const int32_t row = p.chunk_row[c];
      const int64_t k = c - p.chunk_begin[row];
      const int64_t a0 = p.A.rowptr[row], ra = p.A.rowptr[row + 1] - a0;
      const int64_t b0 = p.B.rowptr[row], rb = p.B.rowptr[row + 1] - b0;
      const int32_t* a = p.A.colidx + a0;
      const int32_t* b = p.B.colidx + b0;
      const int64_t d0 = k * p.diag;
      const int64_t d1 = d0 + p.diag < ra + rb ? d0 + p.diag : ra + rb;
      int64_t i0 = 0, j0 = 0, i1 = ra, j1 = rb;
      if constexpr (!FILL) {
        if (d0 > 0) merge_split(a, ra, b, rb, d0, &i0, &j0);
        if (d1 < ra + rb) merge_split(a, ra, b, rb, d1, &i1, &j1);
        p.chunk_split[c] = 2 * i0 + (j0 - (d0 - i0));
      } else {
        auto decode = [&](int64_t d, int64_t code, int64_t* i, int64_t* j) {
          const int64_t lo = d - rb > 0 ? d - rb : 0, hi = d < ra ? d : ra;
          const int64_t x = code >> 1;
          *i = x < lo ? lo : (x > hi ? hi : x);
          const int64_t y = d - *i + (code & 1);
          *j = y > rb ? rb : y;
        };
        decode(d0, p.chunk_split[c], &i0, &j0);
        if (d1 < ra + rb) decode(d1, p.chunk_split[c + 1], &i1, &j1);
        o0 = p.chunk_off[c];
        cap = p.chunk_off[c + 1] - o0;
      }
      ga = a0 + i0;
      gb = b0 + j0;
      const int64_t la = i1 - i0 > 0 ? i1 - i0 : 0, lb = j1 - j0 > 0 ? j1 - j0 : 0;
      if (la > kRankSlots || lb > kRankSlots) bad = true;  // cannot happen for kEwiseRankChunk-position chunks
      na = static_cast<int>(la < kRankSlots ? la : kRankSlots);
      nb = static_cast<int>(lb < kRankSlots ? lb : kRankSlots);
    }
    const unsigned vmask = __ballot_sync(kFull, valid);
    const int nq = 32 - __clz(vmask);  // chunks of this tile in use (a prefix of the lanes)
    // entries of chunk q held in registers: lane l takes positions l, l + 32, l + 64
    int pac[3], pbc[3];
    T pav[3], pbv[3];
    auto fetch = [&](int q) {
      const int64_t cga = __shfl_sync(kFull, ga, q), cgb = __shfl_sync(kFull, gb, q);
      const int cna = __shfl_sync(kFull, na, q), cnb = __shfl_sync(kFull, nb, q);
#pragma unroll
      for (int r = 0; r < 3; ++r) {
        const int e = lane + 32 * r;
        pac[r] = e < cna ? p.A.colidx[cga + e] : 0;
        pbc[r] = e < cnb ? p.B.colidx[cgb + e] : 0;
        if constexpr (FILL) {
          pav[r] = e < cna ? p.A.vals[cga + e] : T(0);
          pbv[r] = e < cnb ? p.B.vals[cgb + e] : T(0);
        }
      }
    };
    if (nq > 0) fetch(0);
    for (int q = 0; q < nq; ++q) {
      const int cna = __shfl_sync(kFull, na, q), cnb = __shfl_sync(kFull, nb, q);
      const int64_t co0 = __shfl_sync(kFull, o0, q), ccap = __shfl_sync(kFull, cap, q);
#pragma unroll
      for (int r = 0; r < 3; ++r) {
        ac[lane + 32 * r] = pac[r];
        bc[lane + 32 * r] = pbc[r];
        if constexpr (FILL) {
          av[lane + 32 * r] = pav[r];
          bv[lane + 32 * r] = pbv[r];
        }
      }
      __syncwarp();
      if (q + 1 < nq) fetch(q + 1);  // in flight while this chunk is ranked
      // A side: position in B and equal partner
      int lbA[3];
      unsigned eqA[3];
#pragma unroll
      for (int r = 0; r < 3; ++r) {
        const int x = lane + 32 * r;
        lbA[r] = 0;
        bool eq = false;
        if (x < cna) {
          const int col = ac[x];
          lbA[r] = lower_bound_smem(bc, cnb, col);
          eq = lbA[r] < cnb && bc[lbA[r]] == col;
        }
        eqA[r] = __ballot_sync(kFull, eq);
      }
      const int pairs = __popc(eqA[0]) + __popc(eqA[1]) + __popc(eqA[2]);
      const int count = OP == kEwiseAdd ? cna + cnb - pairs : pairs;
      if constexpr (!FILL) {
        if (lane == q) p.chunk_off[c + 1] = count;
      } else {
        if (count != ccap) bad = true;
        const unsigned below = (1u << lane) - 1u;
#pragma unroll
        for (int r = 0; r < 3; ++r) {
          const int x = lane + 32 * r;
          if (x >= cna) continue;
          int pb = __popc(eqA[r] & below);  // pairs below x
          for (int r2 = 0; r2 < r; ++r2) pb += __popc(eqA[r2]);
          const bool eq = (eqA[r] >> lane) & 1u;
          if (OP == kEwiseAdd) {
            const int64_t rank = x + lbA[r] - pb;
            if (rank < ccap) {
              p.c_colidx[co0 + rank] = ac[x];
              p.c_vals[co0 + rank] = eq ? av[x] + bv[lbA[r]] : av[x];
            }
          } else if (eq) {
            if (pb < ccap) {
              p.c_colidx[co0 + pb] = ac[x];
              p.c_vals[co0 + pb] = av[x] * bv[lbA[r]];
            }
          }
        }
        if constexpr (OP == kEwiseAdd) {
          // B side: entries without a partner, placed among A
          int lbB[3];
          unsigned eqB[3];
#pragma unroll
          for (int r = 0; r < 3; ++r) {
            const int y = lane + 32 * r;
            lbB[r] = 0;
            bool eq = false;
            if (y < cnb) {
              const int col = bc[y];
              lbB[r] = lower_bound_smem(ac, cna, col);
              eq = lbB[r] < cna && ac[lbB[r]] == col;
            }
            eqB[r] = __ballot_sync(kFull, eq);
          }
#pragma unroll
          for (int r = 0; r < 3; ++r) {
            const int y = lane + 32 * r;
            if (y >= cnb || ((eqB[r] >> lane) & 1u)) continue;
            int pb = __popc(eqB[r] & below);
            for (int r2 = 0; r2 < r; ++r2) pb += __popc(eqB[r2]);
            const int64_t rank = y + lbB[r] - pb;
            if (rank < ccap) {
              p.c_colidx[co0 + rank] = bc[y];
              p.c_vals[co0 + rank] = bv[y];
            }
          }
        }
      }
      __syncwarp();  // the staged parts are overwritten by the next chunk
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
  if (p.group == kEwiseRankGroup) {
    ew_rank_kernel<T, OP, FILL><<<grid_for((p.nc_max + 31) / 32, kRankWarps, num_sms, 8), kEwThreads, 0, s>>>(p);
    return;
  }
  if (p.group == 1) {
    ew_merge_seq_kernel<T, OP, FILL><<<grid_for(p.nc_max, kEwThreads, num_sms, 8), kEwThreads, 0, s>>>(p);
    return;
  }
  if (p.group == kEwiseTileGroup) {
    constexpr size_t smem = kTileWarps * tile_warp_bytes<T, OP, FILL>();
    static bool configured = false;
    if (!configured) {
      cudaFuncSetAttribute(ew_tile_kernel<T, OP, FILL>, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
      configured = true;
    }
    int per_sm = 0;
    cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, ew_tile_kernel<T, OP, FILL>, 32 * kTileWarps, smem);
    const int grid = grid_for((p.nc_max + 31) / 32, kTileWarps, num_sms, per_sm > 0 ? per_sm : 1);
    ew_tile_kernel<T, OP, FILL><<<grid, 32 * kTileWarps, smem, s>>>(p);
    return;
  }
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
