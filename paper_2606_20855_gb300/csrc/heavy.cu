// Heavy rows: rows with too many products for the one-warp workspaces.  One
// CTA owns one row, or one (row, column slice) item of a row with many
// stored entries (the shard pattern of Sec. 4), so every output segment is
// written by one CTA and no CTA waits on another.
//
// Dense rows (kClsRcd): the row's column range is at most 65,536 columns and
// it has at most kRcdMaxA stored A entries (typically hub rows: few stored A
// entries whose B rows are long).  This is the dense workspace of Gustavson's
// algorithm (Sec. 5.1) -- a value per column plus a flag per column, the
// sparse byte-map workspace -- over column slices:
//   symbolic: every product stores 1 into the flag byte of its column (plain
//             byte stores, no atomics: the store is idempotent); nnz of the
//             row is the number of set flags.
//   numeric:  for each slice of `width` columns, groups of lanes walk the B
//             rows of the stored A entries from their cursors (where the
//             previous slice stopped) and add a * b into the dense value
//             window with shared-memory atomics (the atomic level of Sec. 4).
//             The flags of the slice are then scanned in column order, so the
//             slice's entries are written sorted.  A row whose output fits
//             one or two windows indexes the window by output rank instead
//             (a bitmap of its columns and word ranks; rcd_compact_row) and
//             needs no slices.
//
// Wide rows (kClsWb): column range up to 2^20 columns.  A bitmap over the
// whole range (one bit per column) is the workspace:
//   symbolic: atomicOr every product column, count the bits that were 0.
//   numeric:  set the bits, rank the bitmap in 128-bit chunks, write C's
//             column indices in order straight from the bitmap, zero C's
//             values, and let every product add its value at the rank of its
//             column in C (global atomic add; the row's segment is private).
#include <climits>

#include "ws_internal.cuh"

namespace wsk {

namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr int kRcdThreads = 512;
constexpr int kRcdNumThreads = 512;
constexpr int kWbThreads = 1024;  // one CTA per SM (its 128 KB bitmap), so 32 warps hide the gathers
constexpr int kWbBatch = 4;  // stored A entries a lane group has in flight in the wide-bitmap kernel

// ---------------------------------------------------------------- dense rows

constexpr int kRcdCacheA = 1024;  // stored A entries of a row kept in shared memory (and of a batch)
// Rows with more stored A entries are split into (row, slice) items (256 was
// faster than 64 or 1024 on the R-MAT inputs; splitting every row was 1.8x slower).
constexpr int kRcdMegaA = 256;
static_assert(kRcdMegaA <= kRcdCacheA, "rows done whole keep all entries in shared memory");

// Counts the non-zero bytes of 16 bytes.
__device__ __forceinline__ int nonzero_bytes(const uint4 v) {
  return __popc(__vcmpne4(v.x, 0u) & 0x01010101u) + __popc(__vcmpne4(v.y, 0u) & 0x01010101u) +
         __popc(__vcmpne4(v.z, 0u) & 0x01010101u) + __popc(__vcmpne4(v.w, 0u) & 0x01010101u);
}

template <typename T>
__global__ void __launch_bounds__(kRcdThreads, 3) rcd_symbolic_kernel(const RowPlan<T> p) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  uint8_t* flags = smem_raw;  // kMaxBitmapSpan bytes
  uint4* flags4 = reinterpret_cast<uint4*>(smem_raw);
  __shared__ long long s_scan[32];
  constexpr int kS = rcd_slices<T>();
  __shared__ int s_slice[kS];  // entries per dense-window slice of the row
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  constexpr int kWarps = kRcdThreads / 32;
  for (int i = threadIdx.x; i < kMaxBitmapSpan / 16; i += kRcdThreads) flags4[i] = make_uint4(0u, 0u, 0u, 0u);
  if (threadIdx.x < kS) s_slice[threadIdx.x] = 0;
  __syncthreads();
  for (int64_t r = blockIdx.x; r < p.seg_len; r += gridDim.x) {
    const int32_t row = p.perm[p.seg_begin + r];
    const int lo = p.lo[row];
    const int span = p.hi[row] - lo + 1;
    const int64_t ra = p.A.rowptr[row], re = p.A.rowptr[row + 1];
    // A warp takes four stored A entries per round, one per group of 8
    // lanes: a B row of at most 32 entries is flagged by its group in one
    // round of loads (four per lane), longer ones by the whole warp after.
    for (int64_t pa0 = ra + static_cast<int64_t>(warp) * 4; pa0 < re; pa0 += kWarps * 4) {
      const int64_t pa = pa0 + (lane >> 3);
      int64_t qb = 0, qe = 0;
      if (pa < re) {
        const int k = p.A.colidx[pa];
        qb = p.B.rowptr[k];
        qe = p.B.rowptr[k + 1];
      }
      const bool lng = qe - qb > 32;
      const unsigned longs = __ballot_sync(kFull, lng && (lane & 7) == 0);
      if (!lng) {
        int c[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int64_t t = qb + (lane & 7) + 8 * u;
          c[u] = t < qe ? p.B.colidx[t] : -1;
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          if (c[u] >= 0) flags[c[u] - lo] = 1;
        }
      }
      for (unsigned m = longs; m; m &= m - 1u) {
        const int src = __ffs(m) - 1;
        const int64_t be = __shfl_sync(kFull, qe, src);
        int64_t q = __shfl_sync(kFull, qb, src) + lane;
        for (; q + 96 < be; q += 128) {  // four loads in flight per lane
          const int c0 = p.B.colidx[q], c1 = p.B.colidx[q + 32], c2 = p.B.colidx[q + 64], c3 = p.B.colidx[q + 96];
          flags[c0 - lo] = 1;
          flags[c1 - lo] = 1;
          flags[c2 - lo] = 1;
          flags[c3 - lo] = 1;
        }
        for (; q < be; q += 32) flags[p.B.colidx[q] - lo] = 1;
      }
    }
    __syncthreads();
    long long cnt = 0;
    const int n16 = (span + 15) >> 4;
    constexpr int kChunksPerSlice = kRcdWidthBytes / static_cast<int>(sizeof(T)) / 16;
    static_assert(kChunksPerSlice % 32 == 0, "a warp's 32 chunks lie in one slice");
    // Lane l of warp w reads chunk i0 + l; the warp's chunks share one slice,
    // so their counts are summed in the warp and added with one atomic.
    for (int i0 = threadIdx.x & ~31; i0 < n16; i0 += kRcdThreads) {
      const int i = i0 + (threadIdx.x & 31);
      const int n = i < n16 ? nonzero_bytes(flags4[i]) : 0;
      cnt += n;
      const int wsum = __reduce_add_sync(kFull, n);
      if ((threadIdx.x & 31) == 0 && wsum) atomicAdd(&s_slice[i0 / kChunksPerSlice], wsum);
      if (i < n16) flags4[i] = make_uint4(0u, 0u, 0u, 0u);
    }
    long long total;
    block_exclusive_scan(cnt, s_scan, &total);
    if (threadIdx.x == 0) {
      p.c_rowptr[row + 1] = total;
      if (re - ra > kRcdMegaA) {
        const int idx = atomicAdd(p.rcd_nmega, 1);
        p.rcd_mega[idx] = static_cast<int32_t>(r);
        p.rcd_mna[idx] = static_cast<int32_t>(re - ra);
        p.rcd_moff[idx] = static_cast<int64_t>(
            atomicAdd(reinterpret_cast<unsigned long long*>(&p.sum->rcd_mega_entries), static_cast<unsigned long long>(re - ra)));
      }
    }
    if (threadIdx.x < kS) {
      p.rcd_scnt[r * kS + threadIdx.x] = s_slice[threadIdx.x];
      s_slice[threadIdx.x] = 0;
    }
    __syncthreads();
  }
}

// Slice starts of the mega rows' B rows, found once per stored A entry
// instead of once per (row, slice) item.  Blocks (b, y) take mega rows b,
// b + gridDim.x, ...; thread t of block (b, y) the row's entries
// y * blockDim.x + t, stepping by gridDim.y * blockDim.x (the gridDim.y blocks
// of a row share its entries, so one long row is no tail): for
// every slice start lo + s * width (s = 1 .. ns - 1) the first position of the
// sorted B row at or past it, the ns - 1 binary searches run in lockstep so
// their loads are in flight together.  Row idx's table holds (kS - 1) arrays
// of its na entries, slice by slice, from rcd_moff[idx] * (kS - 1).
template <typename T>
__global__ void __launch_bounds__(kRcdNumThreads) rcd_bounds_kernel(const RowPlan<T> p, int width) {
  constexpr int kS = rcd_slices<T>();
  const int n_mega = *p.rcd_nmega;
  for (int idx = blockIdx.x; idx < n_mega; idx += gridDim.x) {
    const int32_t row = p.perm[p.seg_begin + p.rcd_mega[idx]];
    const long long lo = p.lo[row], hi = p.hi[row];
    const int ns = static_cast<int>((hi - lo + width) / width);
    const int64_t ra = p.A.rowptr[row];
    const int na = p.rcd_mna[idx];
    if (p.A.rowptr[row + 1] - ra != na) continue;  // the input changed: the numeric item reports it
    int32_t* tab = p.rcd_bnd + p.rcd_moff[idx] * (kS - 1);
    for (int j = blockIdx.y * blockDim.x + threadIdx.x; j < na; j += gridDim.y * blockDim.x) {
      const int k = p.A.colidx[ra + j];
      const int64_t b0 = p.B.rowptr[k];
      const int len = static_cast<int>(p.B.rowptr[k + 1] - b0);
      const int32_t* cols = p.B.colidx + b0;
      int slo[kS], shi[kS];
#pragma unroll
      for (int q = 1; q < kS; ++q) {
        slo[q] = 0;
        shi[q] = q < ns ? len : 0;
      }
      for (int round = 0; round < 64; ++round) {  // each search halves its interval: <= 32 rounds
        int v[kS];
        bool open = false;
#pragma unroll
        for (int q = 1; q < kS; ++q) {
          v[q] = 0;
          if (slo[q] < shi[q]) {
            open = true;
            v[q] = cols[(slo[q] + shi[q]) >> 1];
          }
        }
        if (!open) break;
#pragma unroll
        for (int q = 1; q < kS; ++q) {
          if (slo[q] < shi[q]) {
            const int mid = (slo[q] + shi[q]) >> 1;
            if (v[q] < lo + static_cast<long long>(q) * width) {
              slo[q] = mid + 1;
            } else {
              shi[q] = mid;
            }
          }
        }
      }
#pragma unroll
      for (int q = 1; q < kS; ++q) {
        if (q < ns) tab[static_cast<int64_t>(q - 1) * na + j] = slo[q];
      }
    }
  }
}

// Numeric pass of the dense heavy rows.  Two kinds of work, taken from two
// counters so CTAs balance themselves:
//   1. mega rows (more than kRcdMegaA stored A entries, typically the hub
//      rows of a power-law matrix): every (row, slice) pair is a separate
//      item, so one row's slices run on several CTAs at once.  An item reads
//      the part of each entry's B row inside its slice from the table of
//      slice starts (rcd_bounds_kernel), walks the long parts with a warp
//      each and the short ones with a group of lanes each, and emits the
//      slice from the offset the symbolic pass's per-slice counts give.
//   2. the other rows, one CTA per row.  A row whose output fits one or two
//      value windows takes the compact window (rcd_compact_row: no column
//      slices); the others go slice by slice, each entry's B-row position,
//      end and A value staying in shared memory for the whole row and every
//      slice continuing where the last one stopped.
constexpr int kRcdShort = 32;  // parts of B rows walked by one group of kShortLanes lanes
constexpr int kShortLanes = 8;  // lanes walking one short part, four entries each
static_assert(kShortLanes * 4 >= kRcdShort, "a short part takes one round of loads");

// Emits one slice of the dense window in column order: thread t owns the
// contiguous 16-byte flag chunks [t * cpt, (t + 1) * cpt); it counts their set
// flags, the CTA scans the counts, and every thread writes its entries in
// order from `pos0` and clears its chunks and values.  Returns the count.
template <typename T>
__device__ long long rcd_emit(const RowPlan<T>& p, T* dense, uint8_t* flags, int w, long long c0, int64_t pos0,
                              int64_t cend, long long* s_scan, bool* bad) {
  const int nq = (w + 15) >> 4;
  const int cpt = (nq + kRcdNumThreads - 1) / kRcdNumThreads;
  const int q0 = threadIdx.x * cpt;
  const int q1 = min(q0 + cpt, nq);
  uint4* f4 = reinterpret_cast<uint4*>(flags);
  long long mine = 0;
  for (int q = q0; q < q1; ++q) mine += nonzero_bytes(f4[q]);
  long long total;
  const long long before = block_exclusive_scan(mine, s_scan, &total);
  int64_t pos = pos0 + before;
  for (int q = q0; q < q1; ++q) {
    const uint4 v = f4[q];
    const uint32_t words[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int h = 0; h < 4; ++h) {
      // bytes of this word that are set, lowest column first
      for (uint32_t m = __vcmpne4(words[h], 0u) & 0x01010101u; m; m &= m - 1u) {
        const int i = (q << 4) + (h << 2) + ((__ffs(m) - 1) >> 3);
        if (pos < cend) {
          p.c_colidx[pos] = static_cast<int32_t>(c0 + i);
          p.c_vals[pos] = dense[i];
        } else {
          *bad = true;
        }
        dense[i] = T(0);
        ++pos;
      }
    }
    f4[q] = make_uint4(0u, 0u, 0u, 0u);
  }
  return total;
}

// Adds a * B[., c] for the B entries [b, b + n) (all inside [c0, c1)) into the
// window, a warp at a time, four loads in flight per lane.
template <typename T>
__device__ __forceinline__ void rcd_warp_add(const RowPlan<T>& p, T* dense, uint8_t* flags, long long b, long long n,
                                             T av, long long c0, int lane) {
  for (long long t0 = 0; t0 < n; t0 += 128) {
    int cc[4];
    T bv[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const long long t = t0 + u * 32 + lane;
      cc[u] = t < n ? p.B.colidx[b + t] : -1;
      bv[u] = t < n ? p.B.vals[b + t] : T(0);
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      if (cc[u] >= 0) {
        const int off = static_cast<int>(cc[u] - c0);
        atomicAdd(dense + off, av * bv[u]);
        flags[off] = 1;
      }
    }
  }
}

// Compact window for a dense heavy row whose output fits a few value windows
// (nnz(row) <= kCompactPasses * width): the window is indexed by output
// position instead of column, so the row needs no column slices; a row with
// more entries than one window takes one pass of step 4-5 per window of
// positions.  The flag bytes serve as a bitmap over the row's range
// (8 * width bits >= 65,536 columns).
//   1. warp 0 lists the stored A entries and cuts their whole B rows into
//      pieces of kRcdPiece entries (scan of the piece counts into e_pp);
//   2. the warps share the pieces and set the bit of every product column;
//   3. each thread ranks four consecutive bitmap words (one barrier for
//      the CTA scan) and keeps the rank of every word (uint16);
//   4. the warps take the pieces again and add a * b at the rank of each
//      column (shared-memory atomics); the product that set a column's bit
//      in step 2 (its flag is kept per piece and lane) writes the column
//      index of C there (rows with too many pieces for the flags write the
//      column indices from the bitmap in step 3 instead);
//   5. the window is copied to C's values with coalesced stores and cleared;
//      after the last pass every thread clears its bitmap words.
// All threads of the CTA call it; the caller's barrier follows.  Returns
// false, having written only the entry cache, when the extra walks of a
// multi-pass row would cost more than column slices.
constexpr int kRcdPiece = 256;  // B entries of one warp-sized piece
constexpr int kCompactPre = 6400;  // byte offset of the word ranks in the entry cache
constexpr int kCompactFresh = kCompactPre + kMaxBitmapSpan / 32 * 2;  // byte offset of the fresh flags
constexpr int kCompactPasses = 2;  // value windows a compact row may take
constexpr long long kCompactExtraProducts = 65536;  // products re-walked by the extra passes, at most

template <typename T>
__device__ bool rcd_compact_row(const RowPlan<T>& p, T* dense, uint8_t* flags, unsigned char* cache, int width,
                                int64_t ra, int na, long long lo, long long hi, int64_t cbase, int64_t cend,
                                long long* s_cnt, int* s_work, bool* bad) {
  constexpr int kWarps = kRcdNumThreads / 32;
  constexpr int kPerLane = kRcdMegaA / 32;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  long long* e_b0 = reinterpret_cast<long long*>(cache);              // kRcdMegaA B row starts
  T* e_av = reinterpret_cast<T*>(cache + kRcdMegaA * 8);              // kRcdMegaA A values
  int* e_pp = reinterpret_cast<int*>(cache + kRcdMegaA * 16);         // first piece of every entry
  int* e_len = e_pp + kRcdMegaA + 1;                                  // B row lengths
  uint16_t* pre = reinterpret_cast<uint16_t*>(cache + kCompactPre);  // rank of every bitmap word
  // Per piece and lane, which of the lane's products set its column's bit
  // first (one byte: bit u for the product at u * 32 + lane of the piece).
  // That product writes the column index of C in step 4; a row with more
  // pieces than the array holds writes them from the bitmap in step 3.
  uint8_t* fresh = cache + kCompactFresh;
  const int cache_bytes = kRcdCacheA * static_cast<int>(2 * sizeof(long long) + sizeof(T) + sizeof(int));
  uint32_t* bm = reinterpret_cast<uint32_t*>(flags);
  const int nnz = static_cast<int>(cend - cbase);
  // 1. entries and pieces
  if (warp == 0) {
    int np[kPerLane];
    int run = 0;
#pragma unroll
    for (int u = 0; u < kPerLane; ++u) {
      const int j = lane * kPerLane + u;
      np[u] = 0;
      if (j < na) {
        const int k = p.A.colidx[ra + j];
        const long long b0 = p.B.rowptr[k];
        const int len = static_cast<int>(p.B.rowptr[k + 1] - b0);
        e_b0[j] = b0;
        e_av[j] = p.A.vals[ra + j];
        e_len[j] = len;
        np[u] = (len + kRcdPiece - 1) / kRcdPiece;
      }
      run += np[u];
    }
    int incl = run;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(kFull, incl, o);
      if (lane >= o) incl += y;
    }
    int at = incl - run;
#pragma unroll
    for (int u = 0; u < kPerLane; ++u) {
      const int j = lane * kPerLane + u;
      if (j < na) e_pp[j] = at;
      at += np[u];
    }
    if (lane == 31) s_work[0] = incl;
    long long prod = 0;  // the row's products
#pragma unroll
    for (int u = 0; u < kPerLane; ++u) {
      const int j = lane * kPerLane + u;
      if (j < na) prod += e_len[j];
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) prod += __shfl_xor_sync(kFull, prod, o);
    if (lane == 0) s_work[1] = static_cast<int>(min(prod, static_cast<long long>(INT_MAX)));
  }
  __syncthreads();
  const int npieces = s_work[0];
  const bool by_fresh = static_cast<long long>(npieces) * 32 <= cache_bytes - kCompactFresh;
  // Every window pass after the first walks all products again; past the
  // budget the column-sliced path (one walk) is cheaper.
  const int passes = (nnz + width - 1) / width;
  if (static_cast<long long>(passes - 1) * s_work[1] > kCompactExtraProducts) return false;
  // 2. bitmap of the product columns
  for (int pc = warp; pc < npieces; pc += kWarps) {
    int jl = 0, jh = na - 1;  // the entry of the piece: last one whose first piece is <= pc
    while (jl < jh) {         // O(log na) probes of shared memory
      const int mid = (jl + jh + 1) >> 1;
      if (e_pp[mid] <= pc) {
        jl = mid;
      } else {
        jh = mid - 1;
      }
    }
    const int t0 = (pc - e_pp[jl]) * kRcdPiece + lane;
    const int e = min((pc - e_pp[jl] + 1) * kRcdPiece, e_len[jl]);
    const long long b = e_b0[jl];
    int cc[kRcdPiece / 32];
#pragma unroll
    for (int u = 0; u < kRcdPiece / 32; ++u) cc[u] = t0 + u * 32 < e ? p.B.colidx[b + t0 + u * 32] : -1;
    uint32_t first = 0;
#pragma unroll
    for (int u = 0; u < kRcdPiece / 32; ++u) {
      const long long off = cc[u] - lo;
      if (cc[u] >= 0) {
        if (off >= 0 && off <= hi - lo) {
          const uint32_t bit = 1u << (off & 31);
          if ((atomicOr(bm + (off >> 5), bit) & bit) == 0u) first |= 1u << u;
        } else {
          *bad = true;
        }
      }
    }
    if (by_fresh) fresh[pc * 32 + lane] = static_cast<uint8_t>(first);
  }
  __syncthreads();
  // 3. word ranks and C's column indices; thread t owns the bitmap words
  // [4 t, 4 t + 4) (the range has at most 4 * kRcdNumThreads words; words
  // past it are zero)
  const int w0 = threadIdx.x * 4;
  const uint4 v4 = *reinterpret_cast<const uint4*>(bm + w0);
  const uint32_t wv[4] = {v4.x, v4.y, v4.z, v4.w};
  const int mine = __popc(wv[0]) + __popc(wv[1]) + __popc(wv[2]) + __popc(wv[3]);
  int incl = mine;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(kFull, incl, o);
    if (lane >= o) incl += y;
  }
  if (lane == 31) s_cnt[warp] = incl;
  __syncthreads();
  int run = incl - mine, total = 0;
#pragma unroll
  for (int v = 0; v < kWarps; ++v) {
    const int n = static_cast<int>(s_cnt[v]);
    run += v < warp ? n : 0;
    total += n;
  }
  if (total != nnz) *bad = true;
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    pre[w0 + q] = static_cast<uint16_t>(run);
    run += __popc(wv[q]);
  }
  __syncthreads();
  // Rows with too many pieces for the fresh flags: column indices in order,
  // thread t writing those of the words t, t + 512, t + 1024, t + 1536
  // (strided, so a dense stretch of columns is shared out).
#pragma unroll
  for (int q = 0; q < 4 && !by_fresh; ++q) {
    const int w = q * kRcdNumThreads + threadIdx.x;
    const long long col0 = lo + (static_cast<long long>(w) << 5) - 1;
    int at = pre[w];
    for (uint32_t m = bm[w]; m; m &= m - 1u) {
      if (at < nnz) p.c_colidx[cbase + at] = static_cast<int32_t>(col0 + __ffs(m));
      ++at;
    }
  }
  // 4. values at the ranks of their columns, one window of ranks per pass
  for (int q0 = 0; q0 < nnz; q0 += width) {
    for (int pc = warp; pc < npieces; pc += kWarps) {
      int jl = 0, jh = na - 1;
      while (jl < jh) {  // O(log na) probes of shared memory
        const int mid = (jl + jh + 1) >> 1;
        if (e_pp[mid] <= pc) {
          jl = mid;
        } else {
          jh = mid - 1;
        }
      }
      const int t0 = (pc - e_pp[jl]) * kRcdPiece + lane;
      const int e = min((pc - e_pp[jl] + 1) * kRcdPiece, e_len[jl]);
      const long long b = e_b0[jl];
      const T av = e_av[jl];
      int cc[kRcdPiece / 32];
      T bv[kRcdPiece / 32];
#pragma unroll
      for (int u = 0; u < kRcdPiece / 32; ++u) {
        const int t = t0 + u * 32;
        cc[u] = t < e ? p.B.colidx[b + t] : -1;
        bv[u] = t < e ? p.B.vals[b + t] : T(0);
      }
      const uint32_t first = by_fresh ? fresh[pc * 32 + lane] : 0u;
#pragma unroll
      for (int u = 0; u < kRcdPiece / 32; ++u) {
        const long long off = cc[u] - lo;
        if (cc[u] >= 0 && off >= 0 && off <= hi - lo) {
          const int w = static_cast<int>(off >> 5);
          const int rank = pre[w] + __popc(bm[w] & ((1u << (off & 31)) - 1u)) - q0;
          if (rank >= 0 && rank < width) {
            atomicAdd(dense + rank, av * bv[u]);
            if ((first >> u) & 1u) p.c_colidx[cbase + q0 + rank] = cc[u];
          }
        }
      }
    }
    __syncthreads();
    // 5. copy the window out and clear it
    const int n = min(width, nnz - q0);
    for (int i = threadIdx.x; i < n; i += kRcdNumThreads) {
      p.c_vals[cbase + q0 + i] = dense[i];
      dense[i] = T(0);
    }
    __syncthreads();
  }
  *reinterpret_cast<uint4*>(bm + w0) = make_uint4(0u, 0u, 0u, 0u);
  return true;
}

template <typename T>
__global__ void __launch_bounds__(kRcdNumThreads, 2) rcd_numeric_kernel(const RowPlan<T> p, int width) {
  constexpr int kS = rcd_slices<T>();
  static_assert(kRcdCacheA * (2 * sizeof(long long) + sizeof(T) + sizeof(int)) <= kRcdMaxA * sizeof(int),
                "the entry cache fits the space after the window");
  static_assert(kRcdMegaA * 16 + (2 * kRcdMegaA + 1) * static_cast<int>(sizeof(int)) <= kCompactPre &&
                    kCompactPre + kMaxBitmapSpan / 32 * sizeof(uint16_t) <=
                        kRcdCacheA * (2 * sizeof(long long) + sizeof(T) + sizeof(int)),
                "the compact-window layout fits the entry cache");
  static_assert(kMaxBitmapSpan <= 65536, "a row has at most 65,536 entries, so word ranks fit uint16");
  static_assert(kRcdWidthBytes / static_cast<int>(sizeof(T)) * 8 >= kMaxBitmapSpan &&
                    kMaxBitmapSpan / 32 == 4 * kRcdNumThreads,
                "the flag bytes hold a bitmap of the range; four bitmap words per thread");
  extern __shared__ __align__(16) unsigned char smem_raw[];
  T* dense = reinterpret_cast<T*>(smem_raw);                           // width values
  uint8_t* flags = smem_raw + static_cast<size_t>(width) * sizeof(T);  // width bytes
  long long* c_pos = reinterpret_cast<long long*>(flags + width);      // per entry: position in B,
  long long* c_end = c_pos + kRcdCacheA;                               //   end of the B row (or of the part),
  T* c_av = reinterpret_cast<T*>(c_end + kRcdCacheA);                  //   the A value,
  int* c_long = reinterpret_cast<int*>(c_av + kRcdCacheA);             //   and the list of long parts
  __shared__ long long s_scan[32];
  __shared__ int s_item, s_next, s_next2, s_nlong, s_work[2];
  __shared__ long long s_out0;
  const int lane = threadIdx.x & 31;
  for (int i = threadIdx.x; i < width; i += kRcdNumThreads) {
    dense[i] = T(0);
    flags[i] = 0;
  }
  bool bad = false;
  const int n_mega = *p.rcd_nmega;

  // 1. (mega row, slice) items
  for (int guard = 0; guard <= n_mega * kS; ++guard) {
    __syncthreads();  // the previous item is done with the shared state
    if (threadIdx.x == 0) {
      s_item = atomicAdd(p.rcd_ctr, 1);
      s_nlong = 0;
    }
    __syncthreads();
    const int item = s_item;
    if (item >= n_mega * kS) break;
    const int r = p.rcd_mega[item / kS], sl = item % kS;
    const int32_t row = p.perm[p.seg_begin + r];
    const long long lo = p.lo[row], hi = p.hi[row];
    const long long c0 = lo + static_cast<long long>(sl) * width;
    if (c0 > hi) continue;
    const long long c1 = min(c0 + width, hi + 1);
    if (threadIdx.x == 0) {
      long long o = p.c_rowptr[row];
      for (int t = 0; t < sl; ++t) o += p.rcd_scnt[static_cast<int64_t>(r) * kS + t];
      s_out0 = o;
    }
    const int64_t ra = p.A.rowptr[row];
    const int na = static_cast<int>(p.A.rowptr[row + 1] - ra);
    const int ns = static_cast<int>((hi - lo + width) / width);
    const int32_t* tab = p.rcd_bnd + p.rcd_moff[item / kS] * (kS - 1);
    if (na != p.rcd_mna[item / kS]) {  // the input changed since the symbolic pass
      bad = true;
      continue;
    }
    for (int e0 = 0; e0 < na; e0 += kRcdCacheA) {
      const int nb = min(kRcdCacheA, na - e0);
      // the part of each entry's B row inside the slice, from the table of
      // slice starts (rcd_bounds_kernel)
      for (int j = threadIdx.x; j < nb; j += kRcdNumThreads) {
        const int e = e0 + j;
        const int k = p.A.colidx[ra + e];
        const long long b0 = p.B.rowptr[k], len = p.B.rowptr[k + 1] - b0;
        const long long st = sl == 0 ? 0 : tab[static_cast<int64_t>(sl - 1) * na + e];
        const long long en = sl + 1 < ns ? tab[static_cast<int64_t>(sl) * na + e] : len;
        c_pos[j] = b0 + st;
        c_end[j] = b0 + en;
        c_av[j] = p.A.vals[ra + e];
        if (en - st > kRcdShort) c_long[atomicAdd(&s_nlong, 1)] = j;
      }
      if (threadIdx.x == 0) {
        s_next = 0;
        s_next2 = 0;
      }
      __syncthreads();
      const int nl = s_nlong;
      for (int g2 = 0; g2 <= nl; ++g2) {  // long parts: a warp each
        int t = 0;
        if (lane == 0) t = atomicAdd(&s_next, 1);
        t = __shfl_sync(kFull, t, 0);
        if (t >= nl) break;
        const int j = c_long[t];
        rcd_warp_add(p, dense, flags, c_pos[j], c_end[j] - c_pos[j], c_av[j], c0, lane);
      }
      // short parts: a group of kShortLanes lanes each, every lane loading up
      // to four of the part's entries at once (one round of loads per part)
      constexpr int kGroupsPerWarp = 32 / kShortLanes;
      for (int g2 = 0; g2 <= nb / kGroupsPerWarp + 1; ++g2) {
        int base = 0;
        if (lane == 0) base = atomicAdd(&s_next2, kGroupsPerWarp);
        base = __shfl_sync(kFull, base, 0);
        if (base >= nb) break;
        const int j = base + lane / kShortLanes;
        if (j < nb && c_end[j] - c_pos[j] <= kRcdShort) {
          const T av = c_av[j];
          const long long t0 = c_pos[j] + lane % kShortLanes, e = c_end[j];
          int cc[4];
          T bv[4];
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const long long t = t0 + u * kShortLanes;
            cc[u] = t < e ? p.B.colidx[t] : -1;
            bv[u] = t < e ? p.B.vals[t] : T(0);
          }
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            if (cc[u] >= 0) {
              const int off = static_cast<int>(cc[u] - c0);
              atomicAdd(dense + off, av * bv[u]);
              flags[off] = 1;
            }
          }
        }
      }
      __syncthreads();
      if (threadIdx.x == 0) s_nlong = 0;
      __syncthreads();
    }
    const int64_t want = p.rcd_scnt[static_cast<int64_t>(r) * kS + sl];
    const long long got = rcd_emit(p, dense, flags, static_cast<int>(c1 - c0), c0, s_out0, s_out0 + want, s_scan, &bad);
    if (threadIdx.x == 0 && got != want) bad = true;
  }

  // 2. the other rows, one CTA each
  for (int guard = 0; guard <= p.seg_len; ++guard) {
    __syncthreads();
    if (threadIdx.x == 0) {
      s_item = atomicAdd(p.rcd_ctr + 1, 1);
      s_nlong = 0;
      s_next = 0;
      s_next2 = 0;
    }
    __syncthreads();
    const int r = s_item;
    if (r >= p.seg_len) break;
    const int32_t row = p.perm[p.seg_begin + r];
    const int64_t ra = p.A.rowptr[row];
    const int na = static_cast<int>(p.A.rowptr[row + 1] - ra);
    if (na > kRcdMegaA) continue;  // a mega row: done in part 1
    const long long lo = p.lo[row], hi = p.hi[row];
    const int64_t cbase = p.c_rowptr[row];
    const int64_t cend = p.c_rowptr[row + 1];
    if (cend - cbase <= static_cast<int64_t>(kCompactPasses) * width &&
        rcd_compact_row(p, dense, flags, reinterpret_cast<unsigned char*>(c_pos), width, ra, na, lo, hi, cbase, cend,
                        s_scan, s_work, &bad))
      continue;  // done without column slices
    for (int j = threadIdx.x; j < na; j += kRcdNumThreads) {
      const int k = p.A.colidx[ra + j];
      c_pos[j] = p.B.rowptr[k];
      c_end[j] = p.B.rowptr[k + 1];
      c_av[j] = p.A.vals[ra + j];
    }
    __syncthreads();
    int64_t emitted = 0;
    for (long long c0 = lo; c0 <= hi; c0 += width) {
      const long long c1 = min(c0 + width, hi + 1);
      // Warps take stored A entries one at a time from a shared counter and
      // walk each B row from where the last slice stopped, four loads in
      // flight per lane; the columns of one B row are distinct, entries of
      // different warps meet in shared-memory atomics.
      for (int g2 = 0; g2 <= na; ++g2) {
        int j = 0;
        if (lane == 0) j = atomicAdd(&s_next, 1);
        j = __shfl_sync(kFull, j, 0);
        if (j >= na) break;
        const long long pos = c_pos[j], end = c_end[j];
        const T av = c_av[j];
        long long stop = end;
        for (long long t0 = pos; t0 < end; t0 += 128) {
          int cc[4];
          T bv[4];
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const long long t = t0 + u * 32 + lane;
            cc[u] = t < end ? p.B.colidx[t] : INT_MAX;
            bv[u] = t < end ? p.B.vals[t] : T(0);
          }
          bool past = false;
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const long long t = t0 + u * 32 + lane;
            if (cc[u] < c1) {
              const int off = static_cast<int>(cc[u] - c0);
              atomicAdd(dense + off, av * bv[u]);
              flags[off] = 1;
            } else if (t < end) {
              stop = min(stop, t);
              past = true;
            }
          }
          if (__any_sync(kFull, past)) break;  // the rest of this B row lies past the slice
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) stop = min(stop, __shfl_xor_sync(kFull, stop, o));
        if (lane == 0) c_pos[j] = stop;
      }
      __syncthreads();
      emitted += rcd_emit(p, dense, flags, static_cast<int>(c1 - c0), c0, cbase + emitted, cend, s_scan, &bad);
      if (threadIdx.x == 0) s_next = 0;  // every warp has left this slice's entry loop
      __syncthreads();
    }
    if (threadIdx.x == 0 && emitted != cend - cbase) bad = true;
  }
  if (bad) atomicOr(&p.sum->status, kErrCount);
}

// ----------------------------------------------------------------- wide rows

template <typename T, bool NUMERIC>
__global__ void __launch_bounds__(kWbThreads, 1) wb_kernel(const RowPlan<T> p) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  uint32_t* bm = reinterpret_cast<uint32_t*>(smem_raw);          // kWbMaxSpan / 32 words
  uint4* bm4 = reinterpret_cast<uint4*>(smem_raw);
  uint32_t* pre = bm + kWbMaxSpan / 32;                           // one prefix per 128-bit chunk
  __shared__ long long s_scan[32];
  const int lg = p.log2_group;
  const int gsize = 1 << lg;
  const int grp = threadIdx.x >> lg;
  const int gl = threadIdx.x & (gsize - 1);
  const int ngrp = kWbThreads >> lg;
  for (int i = threadIdx.x; i < kWbMaxSpan / 128; i += kWbThreads) bm4[i] = make_uint4(0u, 0u, 0u, 0u);
  __syncthreads();
  for (int64_t r = blockIdx.x; r < p.seg_len; r += gridDim.x) {
    const int32_t row = p.perm[p.seg_begin + r];
    const int lo = p.lo[row];
    const int span = p.hi[row] - lo + 1;
    const int nchunks = (span + 127) >> 7;
    const int64_t ra = p.A.rowptr[row], re = p.A.rowptr[row + 1];
    int64_t cbase = 0, cend = 0;
    if constexpr (NUMERIC) {
      cbase = p.c_rowptr[row];
      cend = p.c_rowptr[row + 1];
      for (int64_t i = cbase + threadIdx.x; i < cend; i += kWbThreads) p.c_vals[i] = T(0);
    }
    // Set the bit of every product column.  A group takes kWbBatch stored A
    // entries per round, so their row-pointer and column loads are in flight
    // together (a hub row has tens of thousands of entries).
    long long fresh = 0;
    for (int64_t pa0 = ra + grp; pa0 < re; pa0 += static_cast<int64_t>(kWbBatch) * ngrp) {
      int64_t qb[kWbBatch], qe[kWbBatch];
#pragma unroll
      for (int u = 0; u < kWbBatch; ++u) {
        const int64_t pa = pa0 + static_cast<int64_t>(u) * ngrp;
        qb[u] = 0;
        qe[u] = 0;
        if (pa < re) {
          const int k = p.A.colidx[pa];
          qb[u] = p.B.rowptr[k];
          qe[u] = p.B.rowptr[k + 1];
        }
      }
#pragma unroll
      for (int u = 0; u < kWbBatch; ++u) {
        for (int64_t q = qb[u] + gl; q < qe[u]; q += gsize) {
          const uint32_t off = static_cast<uint32_t>(p.B.colidx[q] - lo);
          const uint32_t bit = 1u << (off & 31u);
          if constexpr (NUMERIC) {
            atomicOr(bm + (off >> 5), bit);
          } else {
            fresh += (atomicOr(bm + (off >> 5), bit) & bit) == 0u;
          }
        }
      }
    }
    __syncthreads();
    if constexpr (!NUMERIC) {
      long long total;
      block_exclusive_scan(fresh, s_scan, &total);
      if (threadIdx.x == 0) p.c_rowptr[row + 1] = total;
      for (int i = threadIdx.x; i < nchunks; i += kWbThreads) bm4[i] = make_uint4(0u, 0u, 0u, 0u);
      __syncthreads();
    } else {
      // Rank the chunks: thread t owns a run of consecutive chunks.
      const int per = (nchunks + kWbThreads - 1) / kWbThreads;
      const int my0 = threadIdx.x * per;
      const int my1 = min(my0 + per, nchunks);
      long long mine = 0;
      for (int i = my0; i < my1; ++i) {
        const uint4 v = bm4[i];
        mine += __popc(v.x) + __popc(v.y) + __popc(v.z) + __popc(v.w);
      }
      long long total;
      long long run = block_exclusive_scan(mine, s_scan, &total);
      bool bad = total != cend - cbase;
      // Write the column indices in order and keep each chunk's prefix.
      for (int i = my0; i < my1; ++i) {
        pre[i] = static_cast<uint32_t>(run);
        const uint4 v = bm4[i];
        const uint32_t wv[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          uint32_t x = wv[q];
          while (x) {
            const int b = __ffs(x) - 1;
            x &= x - 1u;
            const int64_t pos = cbase + run;
            if (pos < cend) p.c_colidx[pos] = lo + (i << 7) + (q << 5) + b;
            ++run;
          }
        }
      }
      __syncthreads();  // prefixes and the zeroed values are visible to the CTA
      for (int64_t pa0 = ra + grp; pa0 < re; pa0 += static_cast<int64_t>(kWbBatch) * ngrp) {
        int64_t qb[kWbBatch], qe[kWbBatch];
        T avs[kWbBatch];
#pragma unroll
        for (int u = 0; u < kWbBatch; ++u) {
          const int64_t pa = pa0 + static_cast<int64_t>(u) * ngrp;
          qb[u] = 0;
          qe[u] = 0;
          avs[u] = T(0);
          if (pa < re) {
            const int k = p.A.colidx[pa];
            avs[u] = p.A.vals[pa];
            qb[u] = p.B.rowptr[k];
            qe[u] = p.B.rowptr[k + 1];
          }
        }
#pragma unroll
        for (int u = 0; u < kWbBatch; ++u) {
        const T av = avs[u];
        for (int64_t q = qb[u] + gl; q < qe[u]; q += gsize) {
          const uint32_t off = static_cast<uint32_t>(p.B.colidx[q] - lo);
          const uint32_t i = off >> 7;
          const uint4 v = bm4[i];
          const uint32_t wq = (off >> 5) & 3u;
          const uint32_t wd = wq == 0 ? v.x : wq == 1 ? v.y : wq == 2 ? v.z : v.w;
          const int64_t pos = cbase + pre[i] + (wq > 0 ? __popc(v.x) : 0) + (wq > 1 ? __popc(v.y) : 0) +
                              (wq > 2 ? __popc(v.z) : 0) + __popc(wd & ((1u << (off & 31u)) - 1u));
          if (pos < cend) {
            atomicAdd(p.c_vals + pos, av * p.B.vals[q]);
          } else {
            bad = true;
          }
        }
        }
      }
      if (bad) atomicOr(&p.sum->status, kErrCount);
      __syncthreads();
      for (int i = threadIdx.x; i < nchunks; i += kWbThreads) bm4[i] = make_uint4(0u, 0u, 0u, 0u);
      __syncthreads();
    }
  }
}

template <typename K>
int occupancy(K kern, int threads, size_t smem) {
  cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  int n = 0;
  cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, kern, threads, smem);
  return n > 0 ? n : 1;
}

int grid_of(int64_t rows, int num_sms, int per_sm) {
  int64_t g = rows;
  const int64_t cap = static_cast<int64_t>(num_sms) * per_sm;
  if (g > cap) g = cap;
  if (g < 1) g = 1;
  return static_cast<int>(g);
}

}  // namespace

size_t rcd_numeric_smem(int width, size_t value_bytes) {
  return static_cast<size_t>(width) * (value_bytes + 1) +
         static_cast<size_t>(kRcdCacheA) * (2 * sizeof(long long) + value_bytes + sizeof(int));
}

template <typename T>
void launch_rcd(const RowPlan<T>& p, bool numeric, int num_sms, cudaStream_t s, int* launches) {
  if (!numeric) {
    const size_t smem = kMaxBitmapSpan;
    static int per_sm = 0;
    if (per_sm == 0) per_sm = occupancy(rcd_symbolic_kernel<T>, kRcdThreads, smem);
    rcd_symbolic_kernel<T><<<grid_of(p.seg_len, num_sms, per_sm), kRcdThreads, smem, s>>>(p);
  } else {
    const int width = kRcdWidthBytes / static_cast<int>(sizeof(T));
    const size_t smem = rcd_numeric_smem(width, sizeof(T));
    static int per_sm = 0;
    if (per_sm == 0) per_sm = occupancy(rcd_numeric_kernel<T>, kRcdNumThreads, smem);
    rcd_numeric_kernel<T><<<grid_of(p.seg_len, num_sms, per_sm), kRcdNumThreads, smem, s>>>(p, width);
  }
  *launches += 1;
}

template <typename T>
void launch_rcd_bounds(const RowPlan<T>& p, int num_sms, cudaStream_t s, int* launches) {
  const int width = kRcdWidthBytes / static_cast<int>(sizeof(T));
  constexpr int kBlocksPerRow = 8;
  const dim3 grid(grid_of(p.seg_len, num_sms, 1), kBlocksPerRow);
  rcd_bounds_kernel<T><<<grid, kRcdNumThreads, 0, s>>>(p, width);
  *launches += 1;
}

template <typename T>
void launch_wb(const RowPlan<T>& p, bool numeric, int num_sms, cudaStream_t s, int* launches) {
  const size_t smem = kWbMaxSpan / 8 + (kWbMaxSpan / 128) * 4;
  auto kern = numeric ? wb_kernel<T, true> : wb_kernel<T, false>;
  static int per_sm[2] = {0, 0};
  if (per_sm[numeric] == 0) per_sm[numeric] = occupancy(kern, kWbThreads, smem);
  kern<<<grid_of(p.seg_len, num_sms, per_sm[numeric]), kWbThreads, smem, s>>>(p);
  *launches += 1;
}

template void launch_rcd<float>(const RowPlan<float>&, bool, int, cudaStream_t, int*);
template void launch_rcd<double>(const RowPlan<double>&, bool, int, cudaStream_t, int*);
template void launch_rcd_bounds<float>(const RowPlan<float>&, int, cudaStream_t, int*);
template void launch_rcd_bounds<double>(const RowPlan<double>&, int, cudaStream_t, int*);
template void launch_wb<float>(const RowPlan<float>&, bool, int, cudaStream_t, int*);
template void launch_wb<double>(const RowPlan<double>&, bool, int, cudaStream_t, int*);

}  // namespace wsk
