// Register bitmap rows: one warp per row for rows with at most 16 stored A
// entries whose B rows each fit in one group of lanes (uniformly sparse
// products such as random matrices and stencils).  Every lane keeps its
// products (column, and in the numeric pass the scaled value) in registers.
//
// Symbolic pass.  The row's workspace is a bitmap with one bit per column of
// the row's range -- the sparse byte-map workspace of Gustavson's SpGEMM
// (Sec. 5.1) with a bit in place of a byte.  The warp sets the bit of every
// product column, ranks the bitmap (prefix sums of bit counts: the total is
// nnz of the row, and the rank of a column is its position in the sorted
// output row) and stores, for every product, the rank of its column in the
// plan (uint16, kBmrSlots slots per row).
// Numeric pass.  No workspace search is left: the first product of every
// column stores its column and value at its stored rank in a compact staging
// array, the products that repeat a column then add theirs (a shared-memory
// atomic, the atomic level of Sec. 4), and the sorted row leaves the staging
// for C (a bulk copy for long rows, coalesced lane stores otherwise).  One
// warp owns the row (shard pattern, Sec. 4).
//
// Lanes are split into groups of G lanes; the group of lane l takes stored A
// entries j = l / G, l / G + 32/G, ...; lane l takes element l % G of B[k_j,:].
// The ranks of a lane's steps s and s + steps/2 share one 32-bit slot.
//
// Bitmap layout.  With WPL = words / 32 words per lane, word w is stored at
// (w % WPL) * 32 + w / WPL: lane l owns the contiguous words [l*WPL, (l+1)*WPL)
// and they sit in bank l.  The ranking pass reads 32 consecutive words per
// step, and the 32 sorted columns of one B row mostly fall in different
// banks.  After use, a row clears only the words it set.
//
// Planning.  When B has at most 65,536 columns every row fits a bitmap over
// all columns (lo = 0), and bmr_plan_kernel ranks every eligible row of A in
// the first pass over A, a CTA of two warps per row (no separate analysis
// pass for those rows); the rows it does not take are queued for the
// analysis kernel.  Its numeric pass is bmr_numeric_kernel, as for the
// binned rows.
#include <climits>
#include <type_traits>

#include "ws_internal.cuh"

namespace wsk {

namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr int kRowsPerCta = 4;

template <int LOGW>
struct BmrShape {
  static constexpr int kWords = 1 << LOGW;
  static constexpr int kWPL = kWords >= 32 ? kWords / 32 : 1;  // words per lane
  static constexpr int kLogWPL = LOGW >= 5 ? LOGW - 5 : 0;
  static constexpr int kPhysWords = kWPL * 32;
  static constexpr int kSPL = kWPL >= 32 ? kWPL / 32 : 1;  // summary words per lane
  // bitmap + per-word rank prefix + per-lane base + summary
  static constexpr size_t bytes() {
    return static_cast<size_t>(kPhysWords) * 6 + 32 * 4 + static_cast<size_t>(kSPL) * 32 * 4;
  }
};

template <class S>
__device__ __forceinline__ uint32_t phys_word(uint32_t w) {
  return ((w & (S::kWPL - 1)) << 5) | (w >> S::kLogWPL);
}

// Rank slots.  In the one-warp kernels lane `lane` holds, at step st of
// kSteps, the product of stored A entry st * (32 / G) + lane / G.  Steps q and
// q + kSteps / 2 of a lane (A entries j and j + 8) share the 32-bit word
// (q * 32 + lane): low half step q, high half step q + kSteps / 2, so the
// numeric pass fetches two ranks per load and the symbolic passes write whole
// words.
template <int kSteps>
__device__ __forceinline__ int rank_word(int st, int lane) { return ((st % (kSteps / 2)) << 5) | lane; }
__device__ __forceinline__ uint32_t rank_pack(int lo_rank, int hi_rank) {
  return static_cast<uint32_t>(lo_rank & 0xffff) | (static_cast<uint32_t>(hi_rank & 0xffff) << 16);
}

// Loads the row's products into registers: lane j < na first loads stored A
// entry j (its B row start, length and value), then every lane loads its
// elements of the B rows of its group.
template <typename T, int G, bool NUMERIC, int kSteps>
__device__ __forceinline__ void load_products(const RowPlan<T>& p, int64_t ra, int na, int lane, int* col, T* val) {
  constexpr int kGroups = 32 / G;
  const int grp = lane / G, gl = lane % G;
  long long my_b0 = 0;
  int my_len = 0;
  T my_a = T(0);
  if (lane < na) {
    const int k = p.A.colidx[ra + lane];
    my_b0 = p.B.rowptr[k];
    my_len = static_cast<int>(p.B.rowptr[k + 1] - my_b0);
    if constexpr (NUMERIC) my_a = p.A.vals[ra + lane];
  }
#pragma unroll
  for (int s = 0; s < kSteps; ++s) {
    const int j = s * kGroups + grp;
    const long long b0 = __shfl_sync(kFull, my_b0, j & 31);
    const int len = __shfl_sync(kFull, my_len, j & 31);
    T a = T(0);
    if constexpr (NUMERIC) a = __shfl_sync(kFull, my_a, j & 31);
    col[s] = -1;
    val[s] = T(0);
    if (j < na && gl < len) {
      col[s] = p.B.colidx[b0 + gl];
      if constexpr (NUMERIC) val[s] = a * p.B.vals[b0 + gl];
    }
  }
}

template <class S, int kSteps>
__device__ __forceinline__ void clear_bits(uint32_t* bm, const int* col, int lo) {
#pragma unroll
  for (int s = 0; s < kSteps; ++s) {
    if (col[s] >= 0) bm[phys_word<S>(static_cast<uint32_t>(col[s] - lo) >> 5)] = 0u;
  }
}

// Ranks the row's bitmap and stores the rank of every product column at
// its rank slot, with bit 15 set when another product of the row
// already claimed that column (so exactly one product per column has it
// clear); clears the words it set; returns nnz of the row.
// A summary bitmap (one bit per bitmap word, lane l's summary words at
// h * 32 + l) lets each lane visit only the non-zero words it owns.
template <class S, int kSteps>
__device__ __forceinline__ int rank_products(uint32_t* bm, uint32_t* sm, uint16_t* pre, int* base, const int* col,
                                             int lo, int lane, uint16_t* ranks) {
  uint32_t dup = 0;  // bit s: product s found its column's bit already set
#pragma unroll
  for (int s = 0; s < kSteps; ++s) {
    if (col[s] >= 0) {
      const uint32_t off = static_cast<uint32_t>(col[s] - lo);
      const uint32_t w = off >> 5;
      const uint32_t j = w & (S::kWPL - 1);  // word index inside the owner's range
      const uint32_t bit = 1u << (off & 31u);
      if (atomicOr(bm + phys_word<S>(w), bit) & bit) dup |= 1u << s;
      atomicOr(sm + (((j >> 5) << 5) | (w >> S::kLogWPL)), 1u << (j & 31u));
    }
  }
  __syncwarp();
  int run = 0;
#pragma unroll
  for (int h = 0; h < S::kSPL; ++h) {
    uint32_t m = sm[(h << 5) | lane];
    sm[(h << 5) | lane] = 0u;  // only this lane reads it
    while (m) {
      const int b = __ffs(m) - 1;
      m &= m - 1u;
      const int ph = (((h << 5) | b) << 5) | lane;
      pre[ph] = static_cast<uint16_t>(run);
      run += __popc(bm[ph]);
    }
  }
  int incl = run;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(kFull, incl, o);
    if (lane >= o) incl += y;
  }
  base[lane] = incl - run;
  const int total = __shfl_sync(kFull, incl, 31);
  __syncwarp();
  int rk[kSteps];
#pragma unroll
  for (int s = 0; s < kSteps; ++s) {
    rk[s] = 0;
    if (col[s] >= 0) {
      const uint32_t off = static_cast<uint32_t>(col[s] - lo);
      const uint32_t w = off >> 5;
      const uint32_t ph = phys_word<S>(w);
      const int pos = base[w >> S::kLogWPL] + pre[ph] + __popc(bm[ph] & ((1u << (off & 31u)) - 1u));
      rk[s] = pos | static_cast<int>(((dup >> s) & 1u) << 15);
    }
  }
  uint32_t* ranks32 = reinterpret_cast<uint32_t*>(ranks);
#pragma unroll
  for (int q = 0; q < kSteps / 2; ++q) {
    if (col[q] >= 0 || col[q + kSteps / 2] >= 0) ranks32[rank_word<kSteps>(q, lane)] = rank_pack(rk[q], rk[q + kSteps / 2]);
  }
  __syncwarp();
  clear_bits<S, kSteps>(bm, col, lo);
  __syncwarp();
  return total;
}

// Symbolic pass of the binned register bitmap rows.  Like the numeric pass
// below, a warp takes kHdrRows rows of its share at a time: the lanes first
// fetch, for all of them together, the row bounds, the row's first column and
// every stored A entry with its B row extent (the chain of dependent loads is
// paid once per batch), then rank the rows one by one, each with one round of
// independent loads of its products.
constexpr int kHdrRows = 8;

template <int LOGW>
constexpr size_t symbolic_warp_bytes() {
  return BmrShape<LOGW>::bytes() + static_cast<size_t>(kHdrRows) * kBmrMaxA * (sizeof(long long) + sizeof(int)) +
         static_cast<size_t>(kHdrRows) * 2 * sizeof(int);
}

template <typename T, int LOGW, int G>
__global__ void __launch_bounds__(32 * kRowsPerCta, 6) bmr_symbolic_kernel(const RowPlan<T> p, int hb) {
  using S = BmrShape<LOGW>;
  constexpr int kGroups = 32 / G;
  constexpr int kSteps = kBmrMaxA / kGroups;
  constexpr int kEnt = kHdrRows * kBmrMaxA;
  extern __shared__ __align__(16) unsigned char smem_raw[];
  const int sub = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int grp = lane / G, gl = lane % G;
  unsigned char* ws = smem_raw + static_cast<size_t>(sub) * symbolic_warp_bytes<LOGW>();
  uint32_t* bm = reinterpret_cast<uint32_t*>(ws);
  uint16_t* pre = reinterpret_cast<uint16_t*>(ws + static_cast<size_t>(S::kPhysWords) * 4);
  int* base = reinterpret_cast<int*>(ws + static_cast<size_t>(S::kPhysWords) * 6);
  uint32_t* sm = reinterpret_cast<uint32_t*>(base + 32);
  long long* h_b0 = reinterpret_cast<long long*>(ws + S::bytes());
  int* h_len = reinterpret_cast<int*>(h_b0 + kEnt);
  int* h_row = h_len + kEnt;
  int* h_lo = h_row + kHdrRows;
  for (int s2 = lane; s2 < S::kPhysWords; s2 += 32) bm[s2] = 0u;
  for (int s2 = lane; s2 < S::kSPL * 32; s2 += 32) sm[s2] = 0u;
  __syncwarp();

  // hb (1..kHdrRows) rows per batch: fewer when the segment is too short to
  // give every warp of the grid a full batch.
  const int64_t warps = static_cast<int64_t>(gridDim.x) * kRowsPerCta;
  for (int64_t r0 = (static_cast<int64_t>(blockIdx.x) * kRowsPerCta + sub) * hb; r0 < p.seg_len; r0 += warps * hb) {
    // Batch header: lane i < hb fetches row r0 + i.
    int na_l = 0;
    long long ra_l = 0;
    if (lane < kHdrRows) {
      int row_l = -1;
      if (lane < hb && r0 + lane < p.seg_len) {
        row_l = p.perm[p.seg_begin + r0 + lane];
        ra_l = p.A.rowptr[row_l];
        const long long na = p.A.rowptr[row_l + 1] - ra_l;
        na_l = static_cast<int>(na < kBmrMaxA ? (na > 0 ? na : 0) : kBmrMaxA);
        h_lo[lane] = p.lo[row_l];
      }
      h_row[lane] = row_l;
    }
#pragma unroll
    for (int q = 0; q < kEnt / 32; ++q) {
      const int e = q * 32 + lane;
      const int i = e / kBmrMaxA, j = e % kBmrMaxA;
      const long long ra = __shfl_sync(kFull, ra_l, i);
      const int na = __shfl_sync(kFull, na_l, i);
      int len = 0;
      if (j < na) {
        const int k = p.A.colidx[ra + j];
        const long long b0 = p.B.rowptr[k];
        len = static_cast<int>(p.B.rowptr[k + 1] - b0);
        h_b0[e] = b0;
      }
      h_len[e] = len;
    }
    __syncwarp();
    for (int i = 0; i < kHdrRows; ++i) {
      const int row = h_row[i];
      if (row < 0) break;
      int col[kSteps];
#pragma unroll
      for (int st = 0; st < kSteps; ++st) {
        const int e = i * kBmrMaxA + st * kGroups + grp;
        col[st] = -1;
        if (gl < h_len[e]) col[st] = p.B.colidx[h_b0[e] + gl];
      }
      const int total = rank_products<S, kSteps>(bm, sm, pre, base, col, h_lo[i], lane,
                                                 p.ranks + static_cast<int64_t>(row) * kBmrSlots);
      if (lane == 0) p.c_rowptr[row + 1] = total;
    }
    __syncwarp();  // the next batch rewrites the headers
  }
}

// Numeric pass of the register bitmap rows.  A warp takes kHdrRows rows of
// its share at a time: first the lanes fetch, for all of them together, the
// row bounds, C's row offsets and every stored A entry with its B row extent
// (a chain of dependent loads, paid once per batch instead of once per row);
// then, row by row, every lane loads its products and their stored ranks in
// one round of independent loads, the first product of every column stores
// its column and value at its rank in a compact staging array, the products
// that repeat a column add theirs (a shared-memory atomic, the atomic level
// of Sec. 4), and the warp copies the sorted row to C with coalesced stores.

// Staging slots of one warp: a row has at most kBmrMaxA * G products (the
// lane groups of G lanes take kBmrMaxA stored A entries), so at most that
// many entries; smaller groups need less shared memory and fit more warps.
// Bulk asynchronous copy of a staged output segment from shared memory to C
// (the copy engine of cp.async.bulk; addresses 16-byte aligned, size a
// multiple of 16).  The issuing thread tracks its copies in bulk groups.
__device__ __forceinline__ void bulk_store(void* gdst, const void* ssrc, uint32_t bytes) {
  asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(gdst),
               "r"(static_cast<uint32_t>(__cvta_generic_to_shared(ssrc))), "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
// Waits until every committed copy of this thread has read its source.
__device__ __forceinline__ void bulk_wait_read() { asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory"); }
// Waits until every committed copy of this thread is complete.
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }
// Orders this thread's earlier shared-memory writes before later bulk copies.
__device__ __forceinline__ void fence_async_shared() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

// Writes the staged row (entries 0..cnt-1 at stage[pad + s]) to out[0..cnt-1]:
// the 16-byte aligned middle by one bulk copy issued by lane 0, the up to
// 16 / sizeof(V) - 1 entries on either side by single lanes.  `pad` is the
// element offset of out within its 16-byte block, so stage[pad + s] and
// out[s] share their alignment.
// Rows shorter than kBulkMinEntries are copied by the lanes alone: there the
// copy engine's latency, paid before the staging is reused, costs more than
// the stores it saves.
constexpr int kBulkMinEntries = 128;
template <typename V>
__device__ __forceinline__ void store_row(V* out, const V* stage, int pad, int cnt, int lane) {
  constexpr int kPer = 16 / static_cast<int>(sizeof(V));
  const int a = (kPer - pad) & (kPer - 1);        // first entry on a 16-byte boundary of out
  const int b = ((pad + cnt) & ~(kPer - 1)) - pad;  // end of the last whole 16-byte block
  if (cnt >= kBulkMinEntries && b > a) {
    if (lane == 0) bulk_store(out + a, stage + pad + a, static_cast<uint32_t>((b - a) * sizeof(V)));
    if (lane < a) out[lane] = stage[pad + lane];
    const int t = lane - kPer;
    if (t >= 0 && b + t < cnt) out[b + t] = stage[pad + b + t];
  } else {
    for (int s2 = lane; s2 < cnt; s2 += 32) out[s2] = stage[pad + s2];
  }
}

template <int G>
constexpr int numeric_cap() { return kBmrMaxA * G; }

template <typename T, int G>
constexpr size_t numeric_warp_bytes() {
  return (static_cast<size_t>(numeric_cap<G>()) + 4) * 4 + (static_cast<size_t>(numeric_cap<G>()) + 16 / sizeof(T)) * sizeof(T) +
         static_cast<size_t>(kHdrRows) * kBmrMaxA * (sizeof(long long) + sizeof(int) + sizeof(T)) +
         static_cast<size_t>(kHdrRows) * (2 * sizeof(long long) + 2 * sizeof(int));
}

template <typename T, int G>
__global__ void __launch_bounds__(32 * kRowsPerCta, sizeof(T) == 8 ? 5 : 7) bmr_numeric_kernel(const RowPlan<T> p, int hb) {
  constexpr int kGroups = 32 / G;
  constexpr int kSteps = kBmrMaxA / kGroups;
  constexpr int kEnt = kHdrRows * kBmrMaxA;
  static_assert(kSteps % 2 == 0, "ranks are fetched in pairs of steps");
  extern __shared__ __align__(16) unsigned char smem_raw[];
  const int sub = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int grp = lane / G, gl = lane % G;
  constexpr int kCap = numeric_cap<G>();
  static_assert(kCap <= kBmrCap, "ranks fit the plan's 15 bits");
  unsigned char* ws = smem_raw + static_cast<size_t>(sub) * numeric_warp_bytes<T, G>();
  // Staging of the sorted row, each array one 16-byte block longer so that
  // entry s sits at pad + s with the alignment of C's entry.
  constexpr int kValPer = 16 / static_cast<int>(sizeof(T));
  static_assert(numeric_warp_bytes<T, G>() % 16 == 0, "every warp's staging starts on a 16-byte boundary");
  int* st_key = reinterpret_cast<int*>(ws);
  T* st_val = reinterpret_cast<T*>(ws + (static_cast<size_t>(kCap) + 4) * 4);
  long long* h_b0 = reinterpret_cast<long long*>(ws + (static_cast<size_t>(kCap) + 4) * 4 +
                                                 (static_cast<size_t>(kCap) + kValPer) * sizeof(T));
  T* h_a = reinterpret_cast<T*>(h_b0 + kEnt);
  int* h_len = reinterpret_cast<int*>(h_a + kEnt);
  long long* h_cbase = reinterpret_cast<long long*>(h_len + kEnt);  // C offset and nnz of each batch row
  long long* h_cnt = h_cbase + kHdrRows;
  int* h_row = reinterpret_cast<int*>(h_cnt + kHdrRows);
  int* h_full = h_row + kHdrRows;  // 1: the row has kBmrMaxA stored entries whose B rows hold G entries each

  // hb (1..kHdrRows) rows per batch: fewer when the segment is too short to
  // give every warp of the grid a full batch.
  const int64_t warps = static_cast<int64_t>(gridDim.x) * kRowsPerCta;
  bool bulk_pending = false;  // lane 0 has a bulk copy of the staging in flight
  for (int64_t r0 = (static_cast<int64_t>(blockIdx.x) * kRowsPerCta + sub) * hb; r0 < p.seg_len; r0 += warps * hb) {
    // Batch header: lane i < hb fetches row r0 + i.
    int na_l = 0;
    long long ra_l = 0;
    if (lane < kHdrRows) {
      int row_l = -1;
      if (lane < hb && r0 + lane < p.seg_len) {
        row_l = p.perm ? p.perm[p.seg_begin + r0 + lane] : static_cast<int>(p.seg_begin + r0 + lane);
        ra_l = p.A.rowptr[row_l];
        const long long na = p.A.rowptr[row_l + 1] - ra_l;
        na_l = static_cast<int>(na < kBmrMaxA ? (na > 0 ? na : 0) : kBmrMaxA);
        const long long cb = p.c_rowptr[row_l];
        h_cbase[lane] = cb;
        h_cnt[lane] = p.c_rowptr[row_l + 1] - cb;
      }
      h_row[lane] = row_l;
    }
#pragma unroll
    for (int q = 0; q < kEnt / 32; ++q) {
      const int e = q * 32 + lane;
      const int i = e / kBmrMaxA, j = e % kBmrMaxA;
      const long long ra = __shfl_sync(kFull, ra_l, i);
      const int na = __shfl_sync(kFull, na_l, i);
      int len = 0;
      if (j < na) {
        const int k = p.A.colidx[ra + j];
        const long long b0 = p.B.rowptr[k];
        len = static_cast<int>(p.B.rowptr[k + 1] - b0);
        h_b0[e] = b0;
        h_a[e] = p.A.vals[ra + j];
      }
      h_len[e] = len;
      // rows 2q (lanes 0..15) and 2q + 1 (lanes 16..31) of the batch
      static_assert(kBmrMaxA == 16, "a batch row is a half warp here");
      const unsigned fm = __ballot_sync(kFull, na == kBmrMaxA && len == G);
      if (j == 0) h_full[i] = ((fm >> (lane & 16)) & 0xffffu) == 0xffffu;
    }
    __syncwarp();
    for (int i = 0; i < kHdrRows; ++i) {
      const int row = h_row[i];
      if (row < 0) break;
      const long long cbase = h_cbase[i];
      const long long want = h_cnt[i];
      const int cnt = static_cast<int>(want < kCap ? want : kCap);  // staging bounds every access
      if (lane == 0 && want > kCap) atomicOr(&p.sum->status, kErrCount);
      int* out_key = p.c_colidx + cbase;
      T* out_val = p.c_vals + cbase;
      const int pk = static_cast<int>((reinterpret_cast<uintptr_t>(out_key) >> 2) & 3);
      const int pv = static_cast<int>((reinterpret_cast<uintptr_t>(out_val) / sizeof(T)) & (kValPer - 1));
      const uint32_t* ranks2 = reinterpret_cast<const uint32_t*>(p.ranks + static_cast<int64_t>(row) * kBmrSlots);
      // The row's products, their ranks, and the scatter into the staging.
      // A full row (every step of every lane has a product) takes the same
      // steps without the per-product tests.
      auto scatter = [&](auto full_tag) {
        constexpr bool kFullRow = decltype(full_tag)::value;
        int col[kSteps];
        uint32_t rk2[kSteps / 2];  // ranks of steps q (low half) and q + kSteps / 2 (high half)
        T val[kSteps];
        uint32_t has_lo = 0;  // bit q: step q has a product
#pragma unroll
        for (int st = 0; st < kSteps; ++st) {
          const int e = i * kBmrMaxA + st * kGroups + grp;
          const bool has = kFullRow || gl < h_len[e];
          col[st] = -1;
          val[st] = T(0);
          if (has) {
            const long long b = h_b0[e] + gl;
            col[st] = p.B.colidx[b];
            val[st] = p.B.vals[b];  // scaled by the A value at the scatter
          }
          if (st < kSteps / 2) {
            has_lo |= static_cast<uint32_t>(has) << st;
          } else {
            const int q = st - kSteps / 2;
            rk2[q] = (kFullRow || ((has_lo >> q) & 1u) || has) ? ranks2[rank_word<kSteps>(q, lane)] : 0u;
          }
        }
        // The previous row's bulk copies must have read the staging.
        if (lane == 0 && bulk_pending) bulk_wait_read();
        __syncwarp();
        // Common case: rank below cnt with the repeat bit clear; the rest
        // (repeated columns, and ranks out of range) after the first stores.
        uint32_t rest = 0;
#pragma unroll
        for (int st = 0; st < kSteps; ++st) {
          const uint32_t rk = st < kSteps / 2 ? rk2[st] & 0xffffu : rk2[st - kSteps / 2] >> 16;
          val[st] *= h_a[i * kBmrMaxA + st * kGroups + grp];
          if (kFullRow || col[st] >= 0) {
            if (rk < static_cast<uint32_t>(cnt)) {
              st_key[pk + rk] = col[st];
              st_val[pv + rk] = val[st];
            } else {
              rest |= 1u << st;
            }
          }
        }
        if (__any_sync(kFull, rest != 0)) {
          __syncwarp();
          bool bad = false;
#pragma unroll
          for (int st = 0; st < kSteps; ++st) {
            if ((rest >> st) & 1u) {
              const uint32_t rk = st < kSteps / 2 ? rk2[st] & 0xffffu : rk2[st - kSteps / 2] >> 16;
              const uint32_t r = rk & 0x7fffu;
              if ((rk & 0x8000u) && r < static_cast<uint32_t>(cnt)) {
                atomicAdd(&st_val[pv + r], val[st]);
              } else {
                bad = true;
              }
            }
          }
          if (__any_sync(kFull, bad) && lane == 0) atomicOr(&p.sum->status, kErrCount);
        }
      };
      if (h_full[i]) {
        scatter(std::true_type{});
      } else {
        scatter(std::false_type{});
      }
      fence_async_shared();
      __syncwarp();
      store_row(out_key, st_key, pk, cnt, lane);
      store_row(out_val, st_val, pv, cnt, lane);
      bulk_pending = cnt >= kBulkMinEntries;
      if (lane == 0 && bulk_pending) bulk_commit();
    }
    __syncwarp();  // the next batch rewrites the headers
  }
  if (lane == 0) bulk_wait_all();
}

// Grouped register bitmap rows: bin 0 (column range of at most kGrpWords * 32
// columns) when B's rows fit groups of G <= 8 lanes.  A row of a few short B
// rows (a stencil row: 5 stored entries of 5 products each) leaves most of a
// warp idle and pays the warp's fixed per-row work (headers, scan, sweep,
// copy-out) for a handful of products, so here each group of G lanes owns a
// row and a warp ranks 32 / G rows at once.  Lane gl of group g takes element
// gl of every B row of the group's row (step st = stored A entry st).
//
// Bitmap: the row of group g has kGrpWords words; lane g*G + i owns words
// [i * WPL, (i + 1) * WPL) (WPL = kGrpWords / G <= 32), and word w sits at
// (w % WPL) * 32 + owner lane, so each lane's words are in its own bank and
// one summary word per lane marks which of them are non-zero.  The ranks of
// a row are stored as uint16 at slot st * G + gl.
constexpr int kGrpLogW = 7;
constexpr int kGrpWords = 1 << kGrpLogW;
constexpr int kGrpChunk = 4;  // steps per warp-uniform branch
static_assert(32 << kGrpLogW == 32 << bmr_log_words(0), "grouped rows are the rows of bin 0");

// The per-group arrays (entry headers, staging) are padded so that the same
// index of different groups falls in different banks: neighbouring rows of a
// stencil hit the same ranks and steps at the same time.
template <int G>
struct GrpShape {
  static constexpr int kRows = 32 / G;          // rows per warp
  static constexpr int kWPL = kGrpWords / G;    // bitmap words per lane
  static constexpr int kPhys = kWPL * 32;       // bitmap words per warp
  static_assert(kWPL <= 32, "one summary word per lane");
  static constexpr int kHdr = kBmrMaxA + 1;     // entry-header stride of a group
  static constexpr int kEnt = kRows * kHdr;     // entry-header slots per warp
  static constexpr int kCap = kBmrMaxA * G;     // products (so entries) of a row at most
  static constexpr int kPadBytes = 128 / kRows;  // staging stride beyond kCap entries, in bytes
};

template <int G>
constexpr size_t grp_symbolic_warp_bytes() {
  using S = GrpShape<G>;
  return static_cast<size_t>(S::kPhys) * 6 + 32 * 4 * 2 + static_cast<size_t>(S::kEnt) * (sizeof(long long) + sizeof(int));
}

template <typename T, int G>
__global__ void __launch_bounds__(32 * kRowsPerCta, 8) bmr_group_symbolic_kernel(const RowPlan<T> p) {
  using S = GrpShape<G>;
  extern __shared__ __align__(16) unsigned char smem_raw[];
  const int sub = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int g = lane / G, gl = lane % G;
  unsigned char* ws = smem_raw + static_cast<size_t>(sub) * grp_symbolic_warp_bytes<G>();
  uint32_t* bm = reinterpret_cast<uint32_t*>(ws);
  uint16_t* pre = reinterpret_cast<uint16_t*>(bm + S::kPhys);
  uint32_t* sm = reinterpret_cast<uint32_t*>(pre + S::kPhys);
  int* base = reinterpret_cast<int*>(sm + 32);
  long long* h_b0 = reinterpret_cast<long long*>(base + 32) + g * S::kHdr;
  int* h_len = reinterpret_cast<int*>(reinterpret_cast<long long*>(base + 32) + S::kEnt) + g * S::kHdr;
  for (int i = lane; i < S::kPhys; i += 32) bm[i] = 0u;
  sm[lane] = 0u;
  __syncwarp();

  const int64_t warps = static_cast<int64_t>(gridDim.x) * kRowsPerCta;
  for (int64_t r0 = (static_cast<int64_t>(blockIdx.x) * kRowsPerCta + sub) * S::kRows; r0 < p.seg_len;
       r0 += warps * S::kRows) {
    const int64_t r = r0 + g;
    int row = -1, na = 0, lo = 0;
    long long ra = 0;
    if (r < p.seg_len) {
      row = p.perm[p.seg_begin + r];
      ra = p.A.rowptr[row];
      const long long n = p.A.rowptr[row + 1] - ra;
      na = static_cast<int>(n < kBmrMaxA ? n : kBmrMaxA);
      lo = p.lo[row];
    }
#pragma unroll
    for (int jj = 0; jj < kBmrMaxA / G; ++jj) {
      const int j = jj * G + gl;
      int len = 0;
      if (j < na) {
        const int k = p.A.colidx[ra + j];
        const long long b0 = p.B.rowptr[k];
        len = static_cast<int>(p.B.rowptr[k + 1] - b0);
        h_b0[j] = b0;
      }
      h_len[j] = len;
    }
    int nmax = na;
#pragma unroll
    for (int o = 16; o >= G; o >>= 1) nmax = max(nmax, __shfl_xor_sync(kFull, nmax, o));
    __syncwarp();
    // Steps in chunks of kGrpChunk behind warp-uniform branches: a stencil
    // row has 5 stored entries, so most of the 16 steps are skipped.
    int col[kBmrMaxA];
#pragma unroll
    for (int st = 0; st < kBmrMaxA; ++st) col[st] = -1;
    uint32_t dup = 0;
#pragma unroll
    for (int c = 0; c < kBmrMaxA / kGrpChunk; ++c) {
      if (c * kGrpChunk < nmax) {
#pragma unroll
        for (int u = 0; u < kGrpChunk; ++u) {
          const int st = c * kGrpChunk + u;
          if (st < na && gl < h_len[st]) col[st] = p.B.colidx[h_b0[st] + gl];
        }
#pragma unroll
        for (int u = 0; u < kGrpChunk; ++u) {
          const int st = c * kGrpChunk + u;
          if (col[st] >= 0) {
            const uint32_t w = static_cast<uint32_t>(col[st] - lo) >> 5;
            const uint32_t owner = static_cast<uint32_t>(g * G) + w / S::kWPL;
            const uint32_t j = w % S::kWPL;
            const uint32_t bit = 1u << ((col[st] - lo) & 31);
            if (atomicOr(bm + ((j << 5) | owner), bit) & bit) dup |= 1u << st;
            atomicOr(sm + owner, 1u << j);
          }
          // Steps in order: the product that keeps its column is the one of
          // the lowest step (a group's lanes hold distinct columns within a step).
          __syncwarp();
        }
      }
    }
    __syncwarp();
    // Rank of the first column of each non-zero word this lane owns.
    const uint32_t touched = sm[lane];
    uint32_t m = touched;
    sm[lane] = 0u;
    int run = 0;
    while (m) {
      const int b = __ffs(m) - 1;
      m &= m - 1u;
      const int ph = (b << 5) | lane;
      pre[ph] = static_cast<uint16_t>(run);
      run += __popc(bm[ph]);
    }
    // Exclusive scan over the G lanes of the group (word order = lane order).
    int incl = run;
#pragma unroll
    for (int o = 1; o < G; o <<= 1) {
      const int y = __shfl_up_sync(kFull, incl, o, G);
      if (gl >= o) incl += y;
    }
    base[lane] = incl - run;
    const int total = __shfl_sync(kFull, incl, G - 1, G);
    __syncwarp();
    uint16_t* ranks = p.ranks + static_cast<int64_t>(row) * kBmrSlots;
#pragma unroll
    for (int c = 0; c < kBmrMaxA / kGrpChunk; ++c) {
      if (c * kGrpChunk < nmax) {
#pragma unroll
        for (int u = 0; u < kGrpChunk; ++u) {
          const int st = c * kGrpChunk + u;
          if (col[st] >= 0) {
            const uint32_t off = static_cast<uint32_t>(col[st] - lo);
            const uint32_t w = off >> 5;
            const uint32_t owner = static_cast<uint32_t>(g * G) + w / S::kWPL;
            const uint32_t ph = ((w % S::kWPL) << 5) | owner;
            const int pos = base[owner] + pre[ph] + __popc(bm[ph] & ((1u << (off & 31u)) - 1u));
            ranks[st * G + gl] = static_cast<uint16_t>(pos | static_cast<int>(((dup >> st) & 1u) << 15));
          }
        }
      }
    }
    __syncwarp();
    // Clear the non-zero words this lane owns.
    for (uint32_t t2 = touched; t2; t2 &= t2 - 1u) bm[((__ffs(t2) - 1) << 5) | lane] = 0u;
    if (gl == 0 && row >= 0) p.c_rowptr[row + 1] = total;
    __syncwarp();
  }
}

// Numeric pass of the grouped rows: group g places its row's products at
// their stored ranks in its own staging array and copies the sorted row to C.
// Steps are placed in order, so the product that stores a column (the one of
// the lowest step) comes before every product that adds to it, and within a
// step the lanes of a group write distinct slots: plain shared-memory adds, no
// atomics (a Laplacian row repeats 12 of its 25 product columns).
template <typename T, int G>
struct GrpNumLayout {
  using S = GrpShape<G>;
  static constexpr int kValStride = S::kCap + S::kPadBytes / static_cast<int>(sizeof(T));
  static constexpr int kKeyStride = S::kCap + S::kPadBytes / 4;
  static constexpr size_t kKeyOff = static_cast<size_t>(S::kRows) * kValStride * sizeof(T);
  static constexpr size_t kB0Off = kKeyOff + static_cast<size_t>(S::kRows) * kKeyStride * 4;
  static constexpr size_t kAOff = kB0Off + static_cast<size_t>(S::kEnt) * sizeof(long long);
  static constexpr size_t kLenOff = kAOff + static_cast<size_t>(S::kEnt) * sizeof(T);
  static constexpr size_t kBytes = kLenOff + static_cast<size_t>(S::kEnt) * sizeof(int);
  static_assert(kB0Off % 8 == 0 && kAOff % sizeof(T) == 0 && kBytes % 8 == 0, "aligned arrays");
};

template <typename T, int G>
constexpr size_t grp_numeric_warp_bytes() {
  return GrpNumLayout<T, G>::kBytes;
}

template <typename T, int G>
__global__ void __launch_bounds__(32 * kRowsPerCta, 6) bmr_group_numeric_kernel(const RowPlan<T> p) {
  using S = GrpShape<G>;
  constexpr int kCap = S::kCap;
  extern __shared__ __align__(16) unsigned char smem_raw[];
  const int sub = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int g = lane / G, gl = lane % G;
  // Per warp: staging values and columns of every group, then the stored A
  // entries of every group (B row start, A value, B row length).
  using L = GrpNumLayout<T, G>;
  unsigned char* ws = smem_raw + static_cast<size_t>(sub) * grp_numeric_warp_bytes<T, G>();
  T* st_val = reinterpret_cast<T*>(ws) + g * L::kValStride;
  int* st_key = reinterpret_cast<int*>(ws + L::kKeyOff) + g * L::kKeyStride;
  long long* h_b0 = reinterpret_cast<long long*>(ws + L::kB0Off) + g * S::kHdr;
  T* h_a = reinterpret_cast<T*>(ws + L::kAOff) + g * S::kHdr;
  int* h_len = reinterpret_cast<int*>(ws + L::kLenOff) + g * S::kHdr;

  const int64_t warps = static_cast<int64_t>(gridDim.x) * kRowsPerCta;
  for (int64_t r0 = (static_cast<int64_t>(blockIdx.x) * kRowsPerCta + sub) * S::kRows; r0 < p.seg_len;
       r0 += warps * S::kRows) {
    const int64_t r = r0 + g;
    int row = -1, na = 0;
    long long ra = 0, cbase = 0, want = 0;
    if (r < p.seg_len) {
      row = p.perm[p.seg_begin + r];
      ra = p.A.rowptr[row];
      const long long n = p.A.rowptr[row + 1] - ra;
      na = static_cast<int>(n < kBmrMaxA ? n : kBmrMaxA);
      cbase = p.c_rowptr[row];
      want = p.c_rowptr[row + 1] - cbase;
    }
    const int cnt = static_cast<int>(want < kCap ? want : kCap);  // staging bounds every access
    bool bad = want > kCap;
#pragma unroll
    for (int jj = 0; jj < kBmrMaxA / G; ++jj) {
      const int j = jj * G + gl;
      int len = 0;
      if (j < na) {
        const int k = p.A.colidx[ra + j];
        const long long b0 = p.B.rowptr[k];
        len = static_cast<int>(p.B.rowptr[k + 1] - b0);
        h_b0[j] = b0;
        h_a[j] = p.A.vals[ra + j];
      }
      h_len[j] = len;
    }
    int nmax = na;
#pragma unroll
    for (int o = 16; o >= G; o >>= 1) nmax = max(nmax, __shfl_xor_sync(kFull, nmax, o));
    __syncwarp();
    const uint16_t* ranks = p.ranks + static_cast<int64_t>(row) * kBmrSlots;
    // Chunks of kGrpChunk steps behind warp-uniform branches: all loads of a
    // chunk are in flight before its products are placed.
#pragma unroll
    for (int c = 0; c < kBmrMaxA / kGrpChunk; ++c) {
      if (c * kGrpChunk < nmax) {
        int col[kGrpChunk], rk[kGrpChunk];
        T val[kGrpChunk];
#pragma unroll
        for (int u = 0; u < kGrpChunk; ++u) {
          const int st = c * kGrpChunk + u;
          col[u] = -1;
          rk[u] = 0;
          val[u] = T(0);
          if (st < na && gl < h_len[st]) {
            const long long q = h_b0[st] + gl;
            col[u] = p.B.colidx[q];
            val[u] = p.B.vals[q];
            rk[u] = ranks[st * G + gl];
          }
        }
#pragma unroll
        for (int u = 0; u < kGrpChunk; ++u) {
          if (col[u] >= 0) {
            const int st = c * kGrpChunk + u;
            const int rr = rk[u] & 0x7fff;
            if (rr >= cnt) {
              bad = true;
            } else if (rk[u] & 0x8000) {
              st_val[rr] += h_a[st] * val[u];
            } else {
              st_key[rr] = col[u];
              st_val[rr] = h_a[st] * val[u];
            }
          }
          __syncwarp();
        }
      }
    }
    if (__any_sync(kFull, bad) && lane == 0) atomicOr(&p.sum->status, kErrCount);
    __syncwarp();
    for (int s2 = gl; s2 < cnt; s2 += G) {
      p.c_colidx[cbase + s2] = st_key[s2];
      p.c_vals[cbase + s2] = st_val[s2];
    }
    __syncwarp();
  }
}

// First pass over A when B has at most 65,536 columns: every row with
// 2..bmr_max_a stored entries, a non-empty product, B rows that fit one group
// and a bitmap of at most kPlanWordsPerProduct words per product is ranked right here (class
// kClsBmrWide, lo = 0); every other row goes to `pending` for the analysis
// kernel.  Counts per class are added to the summary.
//
// One CTA of two warps works on one row at a time.  The products are split
// by the steps of the one-warp numeric kernel (lane l, step s: element l % G
// of the B row of stored A entry s * (32 / G) + l / G): warp w takes the
// steps s = w, w + 2, ..., so every thread stores the ranks of products that
// the same lane of the numeric kernel reads back.  The row's bitmap covers
// all columns: thread t owns the contiguous words [t * WPT, (t + 1) * WPT)
// (bits of columns [32 t WPT, 32 (t + 1) WPT)).  After the product bits are
// set, every thread counts the bits of its own words in one branch-free
// sweep of 16-byte chunks, each warp scans its counts, and every thread
// stores the rank (within its warp's half of the columns) of the first
// column of each of its words.  A product's rank is then that word rank,
// plus warp 0's count for a column of warp 1's half, plus the bits below it
// in its word.  The bitmap is cleared for the next row by a bulk copy of a
// zero block (the copy engine, tracked by an mbarrier), so the shared-memory
// pipe the rest of the row is bound by does no clearing stores.
//
// Row headers (the B row extent of every stored A entry) are fetched for
// kPlanHdrRows rows at a time.
constexpr int kPlanThreads = 64;
constexpr int kPlanHdrRows = 4;
static_assert(kPlanHdrRows * kBmrMaxA == kPlanThreads, "one header entry per thread");
// Sparsest row the planning pass takes: its sweep and clear cost the same for
// every row of a launch (the whole bitmap), so rows with fewer products go to
// the hash bins, whose cost follows the product count.  At 16 words per
// product a 65,536-column bitmap takes rows of 124 products and more.
constexpr long long kPlanWordsPerProduct = 16;

template <int LOGW>
struct PlanShape {
  static_assert(LOGW >= 7 && LOGW <= 11, "two to thirty-two words per thread");
  static constexpr int kWords = 1 << LOGW;
  static constexpr int kWPT = kWords / kPlanThreads;  // words per thread
  // bitmap, uint16 word ranks, per header entry {length, B position}, per header row {na, ub, taken}
  static constexpr size_t kBytes = static_cast<size_t>(kWords) * 6 + kPlanThreads * 8 + kPlanHdrRows * 16;
};

// Position of bitmap word w: for 32 words per thread (eight 16-byte chunks),
// chunk c of thread t sits at t * 8 + (c ^ (t % 8)), so the eight threads of
// a quarter warp that read their chunk c together hit eight different groups
// of four banks; for 8 words per thread (two chunks) chunk c sits at
// t * 2 + (c ^ ((t / 4) % 2)); for 2 words per thread, in order.
template <class S>
__device__ __forceinline__ uint32_t plan_bm(uint32_t w) {
  if constexpr (S::kWPT == 32) {
    return w ^ ((w >> 3) & 0x1cu);
  } else if constexpr (S::kWPT == 8) {
    return w ^ ((w >> 3) & 0x4u);
  } else {
    return w;
  }
}
// Position of word w's rank in the uint16 rank array: for 32 words per
// thread (four chunks of eight ranks), chunk q of thread t at
// t * 4 + (q ^ ((t / 2) % 4)); fewer words, in order (one 16-byte or 4-byte
// store per thread).
template <class S>
__device__ __forceinline__ uint32_t plan_pre(uint32_t w) {
  if constexpr (S::kWPT == 32) {
    return w ^ ((w >> 3) & 0x18u);
  } else {
    return w;
  }
}

// Zero block the planning pass copies over its bitmap after each row.
static __device__ __align__(128) uint4 g_plan_zero[2048 / 4];
__device__ __forceinline__ uint32_t smem_u32(const void* ptr) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(ptr));
}
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_expect_copy(uint64_t* bar, void* dst, const void* src, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes) : "memory");
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
               ::"r"(smem_u32(dst)), "l"(src), "r"(bytes), "r"(smem_u32(bar))
               : "memory");
}
// Waits (bounded) for the phase `parity` of the barrier; false if it gave up.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity) {
  for (int it = 0; it < (1 << 20); ++it) {
    uint32_t done;
    asm volatile("{ .reg .pred p; mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2; selp.u32 %0, 1, 0, p; }"
                 : "=r"(done) : "r"(smem_u32(bar)), "r"(parity) : "memory");
    if (done) return true;
  }
  return false;
}

template <typename T, int LOGW, int G>
__global__ void __launch_bounds__(kPlanThreads, 16) bmr_plan_kernel(const RowPlan<T> p, const AnalyzeParams ap,
                                                                    int64_t ncols, int32_t* pending, int hb) {
  using S = PlanShape<LOGW>;
  constexpr int kGroups = 32 / G;
  constexpr int kSteps = kBmrMaxA / kGroups;  // steps of the one-warp numeric layout
  constexpr int kHalf = kSteps / 2;          // steps q and q + kHalf share one rank word
  constexpr int kMy = kSteps / 2;            // steps of this warp: s = 2 * st + warp
  constexpr int kLenShift = 58;              // header entry: length in bits 58..63, B position below
  constexpr unsigned long long kPosMask = (1ull << kLenShift) - 1;
  static_assert(kSteps % 2 == 0, "two warps share the steps");
  extern __shared__ __align__(16) unsigned char smem_raw[];
  uint32_t* bm = reinterpret_cast<uint32_t*>(smem_raw);
  uint16_t* pre = reinterpret_cast<uint16_t*>(smem_raw + static_cast<size_t>(S::kWords) * 4);
  unsigned long long* h_ent = reinterpret_cast<unsigned long long*>(smem_raw + static_cast<size_t>(S::kWords) * 6);
  int4* h_row = reinterpret_cast<int4*>(h_ent + kPlanThreads);
  __shared__ int s_cnt[2];
  __shared__ __align__(8) uint64_t s_mbar;
  const int t = threadIdx.x, warp = t >> 5, lane = t & 31;
  const int grp = lane / G, gl = lane % G;
  for (int i = t; i < S::kWords / 4; i += kPlanThreads) reinterpret_cast<uint4*>(bm)[i] = make_uint4(0u, 0u, 0u, 0u);
  if (t == 0) {
    mbar_init(&s_mbar, 1);
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  uint32_t mphase = 0;
  bool clr_pending = false;
  const long long words = (ncols + 31) >> 5;
  int taken = 0;
  unsigned long long prod = 0;

  // hb (1..kPlanHdrRows) rows per batch: fewer when A has too few rows to
  // give every CTA of one wave a full batch.
  for (int64_t r0 = static_cast<int64_t>(blockIdx.x) * hb; r0 < ap.m; r0 += static_cast<int64_t>(gridDim.x) * hb) {
    __syncthreads();  // previous batch done with the header arrays (and the first bitmap clear)
    // Batch header: thread t reads stored A entry j = t % 16 of row r0 + t / 16
    // and the extent of its B row (rows with more than bmr_max_a entries are not read).
    {
      const int i = t / kBmrMaxA, j = t % kBmrMaxA;
      long long ra_l = 0;
      int na_l = 0;
      if (lane < 2 && 2 * warp + lane < hb && r0 + 2 * warp + lane < ap.m) {  // lanes 0, 1: the two rows of this warp
        const int64_t r = r0 + 2 * warp + lane;
        ra_l = p.A.rowptr[r];
        const long long n = p.A.rowptr[r + 1] - ra_l;
        na_l = static_cast<int>(n < kBmrMaxA + 1 ? n : kBmrMaxA + 1);
      }
      const long long ra = __shfl_sync(kFull, ra_l, lane / kBmrMaxA);
      const int na = __shfl_sync(kFull, na_l, lane / kBmrMaxA);
      long long b0 = 0;
      int len = 0;
      if (j < na && na <= ap.bmr_max_a) {
        const int k = p.A.colidx[ra + j];
        b0 = p.B.rowptr[k];
        const long long n = p.B.rowptr[k + 1] - b0;
        len = static_cast<int>(n < G + 1 ? n : G + 1);  // a longer B row only has to fail the fit test
      }
      h_ent[t] = (static_cast<unsigned long long>(len) << kLenShift) | static_cast<unsigned long long>(b0);
      int ub = len, mx = len;
#pragma unroll
      for (int o = kBmrMaxA / 2; o > 0; o >>= 1) {
        ub += __shfl_xor_sync(kFull, ub, o);
        mx = max(mx, __shfl_xor_sync(kFull, mx, o));
      }
      if (j == 0) {
        const bool ok = na >= 2 && na <= ap.bmr_max_a && ub > 0 && mx <= G &&
                        words <= kPlanWordsPerProduct * static_cast<long long>(ub) + 64;
        h_row[i] = make_int4(na, ub, ok ? 1 : 0, 0);
      }
    }
    __syncthreads();
    const int nrows = static_cast<int>(ap.m - r0 < hb ? ap.m - r0 : hb);
#pragma unroll 1
    for (int i = 0; i < nrows; ++i) {
      const int64_t row = r0 + i;
      const int4 hr = h_row[i];
      if (!hr.z) {
        if (t == 0) pending[atomicAdd(&p.sum->n_pending, 1)] = static_cast<int32_t>(row);
        continue;
      }
      // A full row (kBmrMaxA stored entries, B rows of G entries each) takes
      // the same steps without the per-product tests.
      auto rank_row = [&](auto full_tag) {
        constexpr bool kFullRow = decltype(full_tag)::value;
        // Products of this thread: step st is numeric step s = 2 * st + warp.
        int col[kMy];
  #pragma unroll
        for (int st = 0; st < kMy; ++st) {
          const unsigned long long h = h_ent[i * kBmrMaxA + (2 * st + warp) * kGroups + grp];
          col[st] = (kFullRow || gl < static_cast<int>(h >> kLenShift)) ? p.B.colidx[(h & kPosMask) + gl] : -1;
        }
        if (clr_pending) {  // the previous row's clear is complete
        if (!mbar_wait(&s_mbar, mphase) && t == 0) atomicOr(&p.sum->status, kErrCount);
        mphase ^= 1u;
        clr_pending = false;
      }
        // Set the product bits; a product that finds its bit set repeats a column.
        uint32_t dup = 0;
  #pragma unroll
        for (int st = 0; st < kMy; ++st) {
          if (kFullRow || col[st] >= 0) {
            const uint32_t off = static_cast<uint32_t>(col[st]);
            const uint32_t bit = 1u << (off & 31u);
            if (atomicOr(bm + plan_bm<S>(off >> 5), bit) & bit) dup |= 1u << st;
          }
        }
        __syncthreads();
        // Sweep: local rank of the first column of each of this thread's words,
        // two per register (word 2k low half, 2k + 1 high half).
        uint32_t loc[(S::kWPT + 1) / 2];
        uint32_t run = 0;
        if constexpr (S::kWPT >= 4) {
          const uint4* mine = reinterpret_cast<const uint4*>(bm) + t * (S::kWPT / 4);
  #pragma unroll
          for (int c = 0; c < S::kWPT / 4; ++c) {
            const uint4 v = mine[S::kWPT == 32 ? (c ^ (t & 7)) : S::kWPT == 8 ? (c ^ ((t >> 2) & 1)) : c];
            const uint32_t r1 = run + __popc(v.x);
            const uint32_t r2 = r1 + __popc(v.y);
            const uint32_t r3 = r2 + __popc(v.z);
            loc[2 * c] = run | (r1 << 16);
            loc[2 * c + 1] = r2 | (r3 << 16);
            run = r3 + __popc(v.w);
          }
        } else {
          const uint2 v = reinterpret_cast<const uint2*>(bm)[t];
          loc[0] = __popc(v.x) << 16;
          run = __popc(v.x) + __popc(v.y);
        }
        uint32_t incl = run;
  #pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const uint32_t y = __shfl_up_sync(kFull, incl, o);
          if (lane >= o) incl += y;
        }
        if (lane == 31) s_cnt[warp] = static_cast<int>(incl);
        // Word ranks within this warp's half (both halves of a register: no carry, every rank <= kBmrCap).
        const uint32_t base = incl - run;
        const uint32_t base2 = base | (base << 16);
        if constexpr (S::kWPT == 32) {
          uint4* pm = reinterpret_cast<uint4*>(pre) + t * 4;
  #pragma unroll
          for (int q = 0; q < 4; ++q)
            pm[q ^ ((t >> 1) & 3)] = make_uint4(loc[4 * q] + base2, loc[4 * q + 1] + base2, loc[4 * q + 2] + base2,
                                                loc[4 * q + 3] + base2);
        } else if constexpr (S::kWPT == 8) {
          reinterpret_cast<uint4*>(pre)[t] = make_uint4(loc[0] + base2, loc[1] + base2, loc[2] + base2, loc[3] + base2);
        } else {
          reinterpret_cast<uint32_t*>(pre)[t] = loc[0] + base2;
        }
        __syncthreads();
        const uint32_t lower = static_cast<uint32_t>(s_cnt[0]);  // entries in warp 0's half of the columns
        // Rank of this thread's step st product: its word's rank within its
        // half, warp 0's count for a column of warp 1's half, and the bits below
        // it in its word.
        auto rank_of = [&](int st) -> uint32_t {
          if (!kFullRow && col[st] < 0) return 0u;
          const uint32_t off = static_cast<uint32_t>(col[st]);
          const uint32_t w = off >> 5;
          const uint32_t half = (w >> (LOGW - 1)) & 1u;
          return (pre[plan_pre<S>(w)] + (half ? lower : 0u) +
                  __popc(bm[plan_bm<S>(w)] & ((1u << (off & 31u)) - 1u))) |
                 ((dup << (15 - st)) & 0x8000u);
        };
        uint32_t* ranks32 = reinterpret_cast<uint32_t*>(p.ranks + row * kBmrSlots);
        if constexpr (kHalf % 2 == 0) {
          // numeric steps s and s + kHalf (st and st + kHalf / 2 here) share a rank word
  #pragma unroll
          for (int st = 0; st < kHalf / 2; ++st)
            ranks32[((2 * st + warp) << 5) | lane] = rank_of(st) | (rank_of(st + kHalf / 2) << 16);
        } else {
          // one step per warp (G = 4): warp w fills half w of rank word 0
          p.ranks[row * kBmrSlots + 2 * lane + warp] = static_cast<uint16_t>(rank_of(0));
        }
      };
      if (hr.x == kBmrMaxA && hr.y == kBmrMaxA * G) {
        rank_row(std::true_type{});
      } else {
        rank_row(std::false_type{});
      }
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");  // the bitmap reads before the copy over it
      __syncthreads();
      if (t == 0) mbar_expect_copy(&s_mbar, bm, g_plan_zero, static_cast<uint32_t>(S::kWords * 4));
      clr_pending = true;
      if (t == 0) {
        p.c_rowptr[row + 1] = s_cnt[0] + s_cnt[1];
        p.cls[row] = kClsBmrWide;
        p.lo[row] = 0;
        p.hi[row] = static_cast<int32_t>(ncols - 1);
      }
      ++taken;
      prod += static_cast<unsigned long long>(hr.y);
    }
  }
  if (clr_pending && !mbar_wait(&s_mbar, mphase) && t == 0) atomicOr(&p.sum->status, kErrCount);
  if (t == 0) {
    if (taken) atomicAdd(&p.sum->seg_count[kSegBmrWide], taken);
    if (prod) atomicAdd(reinterpret_cast<unsigned long long*>(&p.sum->products), prod);
  }
}

template <typename K>
int occupancy(K kern, int threads, size_t smem) {
  cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  int n = 0;
  cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, kern, threads, smem);
  return n > 0 ? n : 1;
}

int64_t clamp_grid(int64_t want, int num_sms, int per_sm) {
  const int64_t cap = static_cast<int64_t>(num_sms) * per_sm;
  return want > cap ? cap : (want < 1 ? 1 : want);
}

template <typename T, int LOGW, int G>
void launch_bmr_g(const RowPlan<T>& p, bool numeric, int num_sms, cudaStream_t s) {
  if (numeric) {
    const size_t smem = static_cast<size_t>(kRowsPerCta) * numeric_warp_bytes<T, G>();
    static int per_sm = 0;
    if (per_sm == 0) per_sm = occupancy(bmr_numeric_kernel<T, G>, 32 * kRowsPerCta, smem);
    // Rows per warp batch: kHdrRows, unless that leaves warps of one full
    // wave idle (a short segment), then as few as one.
    const int64_t wave_warps = static_cast<int64_t>(num_sms) * per_sm * kRowsPerCta;
    int64_t hb = (p.seg_len + wave_warps - 1) / wave_warps;
    hb = hb < 1 ? 1 : (hb > kHdrRows ? kHdrRows : hb);
    const int64_t per_cta = static_cast<int64_t>(kRowsPerCta) * hb;
    const int64_t grid = clamp_grid((p.seg_len + per_cta - 1) / per_cta, num_sms, per_sm);
    bmr_numeric_kernel<T, G><<<static_cast<int>(grid), 32 * kRowsPerCta, smem, s>>>(p, static_cast<int>(hb));
    return;
  }
  const size_t smem = static_cast<size_t>(kRowsPerCta) * symbolic_warp_bytes<LOGW>();
  static int per_sm = 0;
  if (per_sm == 0) per_sm = occupancy(bmr_symbolic_kernel<T, LOGW, G>, 32 * kRowsPerCta, smem);
  const int64_t wave_warps = static_cast<int64_t>(num_sms) * per_sm * kRowsPerCta;
  int64_t hb = (p.seg_len + wave_warps - 1) / wave_warps;
  hb = hb < 1 ? 1 : (hb > kHdrRows ? kHdrRows : hb);
  const int64_t per_cta = static_cast<int64_t>(kRowsPerCta) * hb;
  const int64_t grid = clamp_grid((p.seg_len + per_cta - 1) / per_cta, num_sms, per_sm);
  bmr_symbolic_kernel<T, LOGW, G><<<static_cast<int>(grid), 32 * kRowsPerCta, smem, s>>>(p, static_cast<int>(hb));
}

template <typename T, int LOGW>
void launch_bmr_w(const RowPlan<T>& p, bool numeric, int num_sms, cudaStream_t s) {
  switch (p.log2_group) {
    case 2: launch_bmr_g<T, LOGW, 4>(p, numeric, num_sms, s); break;
    case 3: launch_bmr_g<T, LOGW, 8>(p, numeric, num_sms, s); break;
    case 4: launch_bmr_g<T, LOGW, 16>(p, numeric, num_sms, s); break;
    default: launch_bmr_g<T, LOGW, 32>(p, numeric, num_sms, s); break;
  }
}

template <typename T, int LOGW, int G>
void launch_plan_g(const RowPlan<T>& p, const AnalyzeParams& ap, int64_t ncols, int32_t* pending, int num_sms,
                   cudaStream_t s) {
  const size_t smem = PlanShape<LOGW>::kBytes;
  static int per_sm = 0;
  if (per_sm == 0) per_sm = occupancy(bmr_plan_kernel<T, LOGW, G>, kPlanThreads, smem);
  const int64_t wave = static_cast<int64_t>(num_sms) * per_sm;
  int64_t hb = (ap.m + wave - 1) / wave;
  hb = hb < 1 ? 1 : (hb > kPlanHdrRows ? kPlanHdrRows : hb);
  const int64_t grid = clamp_grid((ap.m + hb - 1) / hb, num_sms, per_sm);
  bmr_plan_kernel<T, LOGW, G><<<static_cast<int>(grid), kPlanThreads, smem, s>>>(p, ap, ncols, pending,
                                                                                 static_cast<int>(hb));
}

template <typename T, int G>
void launch_grp(const RowPlan<T>& p, bool numeric, int num_sms, cudaStream_t s) {
  constexpr int64_t kPerCta = static_cast<int64_t>(kRowsPerCta) * GrpShape<G>::kRows;
  const int64_t want = (p.seg_len + kPerCta - 1) / kPerCta;
  if (numeric) {
    const size_t smem = static_cast<size_t>(kRowsPerCta) * grp_numeric_warp_bytes<T, G>();
    static int per_sm = 0;
    if (per_sm == 0) per_sm = occupancy(bmr_group_numeric_kernel<T, G>, 32 * kRowsPerCta, smem);
    bmr_group_numeric_kernel<T, G>
        <<<static_cast<int>(clamp_grid(want, num_sms, per_sm)), 32 * kRowsPerCta, smem, s>>>(p);
  } else {
    const size_t smem = static_cast<size_t>(kRowsPerCta) * grp_symbolic_warp_bytes<G>();
    static int per_sm = 0;
    if (per_sm == 0) per_sm = occupancy(bmr_group_symbolic_kernel<T, G>, 32 * kRowsPerCta, smem);
    bmr_group_symbolic_kernel<T, G>
        <<<static_cast<int>(clamp_grid(want, num_sms, per_sm)), 32 * kRowsPerCta, smem, s>>>(p);
  }
}

}  // namespace

template <typename T>
void launch_bmr(const RowPlan<T>& p, int bin, bool numeric, int num_sms, cudaStream_t s, int* launches) {
  if (bin == 0 && p.log2_group <= 3) {  // B rows of at most 8 entries: a group of lanes per row
    if (p.log2_group == 2) {
      launch_grp<T, 4>(p, numeric, num_sms, s);
    } else {
      launch_grp<T, 8>(p, numeric, num_sms, s);
    }
    *launches += 1;
    return;
  }
  switch (bin) {
    case 0: launch_bmr_w<T, bmr_log_words(0)>(p, numeric, num_sms, s); break;
    case 1: launch_bmr_w<T, bmr_log_words(1)>(p, numeric, num_sms, s); break;
    case 2: launch_bmr_w<T, bmr_log_words(2)>(p, numeric, num_sms, s); break;
    case kBmrPlannedBin:  // ranked by the planning pass in the one-warp layout
      if (numeric) launch_bmr_w<T, bmr_log_words(0)>(p, true, num_sms, s);
      break;
    default: return;
  }
  *launches += 1;
}

template <typename T>
void launch_bmr_plan(const RowPlan<T>& p, const AnalyzeParams& ap, int64_t ncols, int32_t* pending, int num_sms,
                     cudaStream_t s, int* launches) {
  // The planning pass uses the smallest register-bitmap bin that covers all columns of B.
  const int bin = bmr_bin_for_span(ncols);
#define WS_PLAN(LW)                                                                         \
  switch (p.log2_group) {                                                                  \
    case 2: launch_plan_g<T, LW, 4>(p, ap, ncols, pending, num_sms, s); break;             \
    case 3: launch_plan_g<T, LW, 8>(p, ap, ncols, pending, num_sms, s); break;             \
    case 4: launch_plan_g<T, LW, 16>(p, ap, ncols, pending, num_sms, s); break;            \
    default: launch_plan_g<T, LW, 32>(p, ap, ncols, pending, num_sms, s); break;           \
  }
  if (bin == 0) {
    WS_PLAN(bmr_log_words(0))
  } else if (bin == 1) {
    WS_PLAN(bmr_log_words(1))
  } else {
    WS_PLAN(bmr_log_words(2))
  }
#undef WS_PLAN
  *launches += 1;
}

template void launch_bmr<float>(const RowPlan<float>&, int, bool, int, cudaStream_t, int*);
template void launch_bmr<double>(const RowPlan<double>&, int, bool, int, cudaStream_t, int*);
template void launch_bmr_plan<float>(const RowPlan<float>&, const AnalyzeParams&, int64_t, int32_t*, int,
                                     cudaStream_t, int*);
template void launch_bmr_plan<double>(const RowPlan<double>&, const AnalyzeParams&, int64_t, int32_t*, int,
                                      cudaStream_t, int*);

}  // namespace wsk
