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
// atomic, the atomic level of Sec. 4), and the warp copies the sorted row to
// C with coalesced stores.  One warp owns the row (shard pattern, Sec. 4).
//
// Lanes are split into groups of G lanes; the group of lane l takes stored A
// entries j = l / G, l / G + 32/G, ...; lane l takes element l % G of B[k_j,:].
// Product (step s, lane l) has slot s * 32 + l.
//
// Bitmap layout.  With WPL = words / 32 words per lane, word w is stored at
// (w % WPL) * 32 + w / WPL: lane l owns the contiguous words [l*WPL, (l+1)*WPL)
// and they sit in bank l.  The ranking pass reads 32 consecutive words per
// step, and the 32 sorted columns of one B row mostly fall in different
// banks.  After use, a row clears only the words it set.
//
// Planning.  When B has at most 65,536 columns every row fits a bitmap over
// all columns (lo = 0), and bmr_plan_kernel ranks every eligible row of A in
// the first pass over A, two warps per row (no separate analysis pass for
// those rows); the rows it does not take are queued for the analysis kernel.
#include <climits>

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
  // symbolic: bitmap + per-word rank prefix + per-lane base + summary; numeric: staging
  template <typename T>
  static constexpr size_t warp_bytes(bool numeric) {
    return numeric ? static_cast<size_t>(kBmrCap) * (4 + sizeof(T))
                   : static_cast<size_t>(kPhysWords) * 6 + 32 * 4 + static_cast<size_t>(kSPL) * 32 * 4;
  }
};

template <class S>
__device__ __forceinline__ uint32_t phys_word(uint32_t w) {
  return ((w & (S::kWPL - 1)) << 5) | (w >> S::kLogWPL);
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

// Sets the bit of every product column; returns how many bits were 0 before
// (when COUNT).  The caller clears the words after its last use.
template <class S, bool COUNT, int kSteps>
__device__ __forceinline__ int set_bits(uint32_t* bm, const int* col, int lo) {
  int fresh = 0;
#pragma unroll
  for (int s = 0; s < kSteps; ++s) {
    if (col[s] >= 0) {
      const uint32_t off = static_cast<uint32_t>(col[s] - lo);
      const uint32_t bit = 1u << (off & 31u);
      uint32_t* word = bm + phys_word<S>(off >> 5);
      if constexpr (COUNT) {
        fresh += (atomicOr(word, bit) & bit) == 0u;
      } else {
        atomicOr(word, bit);
      }
    }
  }
  return fresh;
}

template <class S, int kSteps>
__device__ __forceinline__ void clear_bits(uint32_t* bm, const int* col, int lo) {
#pragma unroll
  for (int s = 0; s < kSteps; ++s) {
    if (col[s] >= 0) bm[phys_word<S>(static_cast<uint32_t>(col[s] - lo) >> 5)] = 0u;
  }
}

// Ranks the row's bitmap and stores the rank of every product column at
// ranks[s * 32 + lane], with bit 15 set when another product of the row
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
#pragma unroll
  for (int s = 0; s < kSteps; ++s) {
    if (col[s] >= 0) {
      const uint32_t off = static_cast<uint32_t>(col[s] - lo);
      const uint32_t w = off >> 5;
      const uint32_t ph = phys_word<S>(w);
      const int pos = base[w >> S::kLogWPL] + pre[ph] + __popc(bm[ph] & ((1u << (off & 31u)) - 1u));
      ranks[(s << 5) | lane] = static_cast<uint16_t>(pos | (((dup >> s) & 1u) << 15));
    }
  }
  __syncwarp();
  clear_bits<S, kSteps>(bm, col, lo);
  __syncwarp();
  return total;
}

template <typename T, int LOGW, int G, bool NUMERIC>
__global__ void __launch_bounds__(32 * kRowsPerCta, NUMERIC ? (sizeof(T) == 8 ? 5 : 7) : 6) bmr_rows_kernel(const RowPlan<T> p) {
  using S = BmrShape<LOGW>;
  constexpr int kSteps = kBmrMaxA / (32 / G);
  extern __shared__ __align__(16) unsigned char smem_raw[];
  const int sub = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  unsigned char* ws = smem_raw + static_cast<size_t>(sub) * S::template warp_bytes<T>(NUMERIC);
  // symbolic workspace
  uint32_t* bm = reinterpret_cast<uint32_t*>(ws);
  uint16_t* pre = reinterpret_cast<uint16_t*>(ws + static_cast<size_t>(S::kPhysWords) * 4);
  int* base = reinterpret_cast<int*>(ws + static_cast<size_t>(S::kPhysWords) * 6);
  uint32_t* sm = reinterpret_cast<uint32_t*>(base + 32);
  // numeric workspace
  int* st_key = reinterpret_cast<int*>(ws);
  T* st_val = reinterpret_cast<T*>(ws + static_cast<size_t>(kBmrCap) * 4);

  if constexpr (!NUMERIC) {
    for (int s2 = lane; s2 < S::kPhysWords; s2 += 32) bm[s2] = 0u;
    for (int s2 = lane; s2 < S::kSPL * 32; s2 += 32) sm[s2] = 0u;
    __syncwarp();
  }

  for (int64_t r = static_cast<int64_t>(blockIdx.x) * kRowsPerCta + sub; r < p.seg_len;
       r += static_cast<int64_t>(gridDim.x) * kRowsPerCta) {
    const int32_t row = p.perm[p.seg_begin + r];
    const int64_t ra = p.A.rowptr[row];
    const int na = static_cast<int>(p.A.rowptr[row + 1] - ra);
    uint16_t* ranks = p.ranks + static_cast<int64_t>(row) * kBmrSlots;
    int col[kSteps];
    T val[kSteps];
    load_products<T, G, NUMERIC, kSteps>(p, ra, na, lane, col, val);

    if constexpr (!NUMERIC) {
      const int total = rank_products<S, kSteps>(bm, sm, pre, base, col, p.lo[row], lane, ranks);
      if (lane == 0) p.c_rowptr[row + 1] = total;
    } else {
      int rk[kSteps];
#pragma unroll
      for (int s = 0; s < kSteps; ++s) rk[s] = col[s] >= 0 ? ranks[(s << 5) | lane] : 0;
      const int64_t cbase = p.c_rowptr[row];
      const int64_t want = p.c_rowptr[row + 1] - cbase;
      const int cnt = static_cast<int>(want < kBmrCap ? want : kBmrCap);  // staging bounds every access
      if (lane == 0 && want > kBmrCap) atomicOr(&p.sum->status, kErrCount);
      // The first product of every column stores its value; the rare repeats add theirs after.
      bool bad = false, repeats = false;
#pragma unroll
      for (int s = 0; s < kSteps; ++s) {
        if (col[s] >= 0) {
          const int r = rk[s] & 0x7fff;
          if (r >= cnt) {
            bad = true;
          } else if (rk[s] & 0x8000) {
            repeats = true;
          } else {
            st_key[r] = col[s];
            st_val[r] = val[s];
          }
        }
      }
      if (__any_sync(kFull, bad) && lane == 0) atomicOr(&p.sum->status, kErrCount);
      __syncwarp();
      if (__any_sync(kFull, repeats)) {
#pragma unroll
        for (int s = 0; s < kSteps; ++s) {
          const int r = rk[s] & 0x7fff;
          if (col[s] >= 0 && (rk[s] & 0x8000) && r < cnt) atomicAdd(&st_val[r], val[s]);
        }
        __syncwarp();
      }
      for (int s2 = lane; s2 < cnt; s2 += 32) {
        p.c_colidx[cbase + s2] = st_key[s2];
        p.c_vals[cbase + s2] = st_val[s2];
      }
      __syncwarp();
    }
  }
}

// First pass over A when B has at most 65,536 columns: every row with
// 2..bmr_max_a stored entries, a non-empty product, B rows that fit one group
// and a bitmap of at most 8 words per product is ranked right here (class
// kClsBmrWide, lo = 0); every other row goes to `pending` for the analysis
// kernel.  Counts per class are added to the summary.
//
// One CTA of kPlanThreads threads (two warps) works on one row, so the
// bitmap of a row is shared by all of them: thread t owns the contiguous
// words [t * WPT, (t + 1) * WPT), stored at (w % WPT) * kPlanThreads + w / WPT.  Product
// (stored A entry j, element e of B[k_j,:]) keeps the slot j * G + e, the
// same slot the one-warp numeric kernel uses.
#ifndef WS_PLAN_THREADS
#define WS_PLAN_THREADS 64
#endif
constexpr int kPlanThreads = WS_PLAN_THREADS;

template <int LOGW>
struct PlanShape {
  static constexpr int kWords = 1 << LOGW;
  static constexpr int kWPT = kWords >= kPlanThreads ? kWords / kPlanThreads : 1;  // words per thread
  static constexpr int kLogThreads = kPlanThreads == 64 ? 6 : kPlanThreads == 128 ? 7 : 8;
  static constexpr int kLogWPT = LOGW >= kLogThreads ? LOGW - kLogThreads : 0;
  static constexpr int kPhysWords = kWPT * kPlanThreads;
  static constexpr int kSPT = kWPT >= 32 ? kWPT / 32 : 1;  // summary words per thread
  static constexpr size_t bytes() {
    return static_cast<size_t>(kPhysWords) * 6 + kPlanThreads * 4 + static_cast<size_t>(kSPT) * kPlanThreads * 4;
  }
};

template <class S>
__device__ __forceinline__ uint32_t plan_phys(uint32_t w) {
  return (w & (S::kWPT - 1)) * kPlanThreads + (w >> S::kLogWPT);
}

template <typename T, int LOGW, int G>
__global__ void __launch_bounds__(kPlanThreads, 1024 / kPlanThreads) bmr_plan_kernel(const RowPlan<T> p, const AnalyzeParams ap,
                                                                int64_t ncols, int32_t* pending) {
  using S = PlanShape<LOGW>;
  constexpr int kGroups = kPlanThreads / G;   // A entries per step
  constexpr int kSteps = (kBmrMaxA + kGroups - 1) / kGroups;  // steps covering kBmrMaxA entries
  extern __shared__ __align__(16) unsigned char smem_raw[];
  uint32_t* bm = reinterpret_cast<uint32_t*>(smem_raw);
  uint16_t* pre = reinterpret_cast<uint16_t*>(smem_raw + static_cast<size_t>(S::kPhysWords) * 4);
  int* base = reinterpret_cast<int*>(smem_raw + static_cast<size_t>(S::kPhysWords) * 6);
  uint32_t* sm = reinterpret_cast<uint32_t*>(base + kPlanThreads);
  __shared__ long long s_b0[kBmrMaxA];
  __shared__ int s_len[kBmrMaxA];
  __shared__ int s_red[2 * (kPlanThreads / 32)];
  __shared__ long long s_scan[32];
  const int t = threadIdx.x;
  const int lane = t & 31, warp = t >> 5;
  const int grp = t / G, gl = t % G;
  for (int i = t; i < S::kPhysWords; i += kPlanThreads) bm[i] = 0u;
  for (int i = t; i < S::kSPT * kPlanThreads; i += kPlanThreads) sm[i] = 0u;
  __syncthreads();
  const long long words = (ncols + 31) >> 5;
  int taken = 0;
  unsigned long long prod = 0;

  for (int64_t row = blockIdx.x; row < ap.m; row += gridDim.x) {
    const int64_t ra = p.A.rowptr[row];
    const int64_t na64 = p.A.rowptr[row + 1] - ra;
    bool ok = na64 >= 2 && na64 <= ap.bmr_max_a;
    const int na = static_cast<int>(ok ? na64 : 0);
    if (ok) {
      int my_len = 0;
      if (t < na) {
        const int k = p.A.colidx[ra + t];
        const long long b0 = p.B.rowptr[k];
        my_len = static_cast<int>(p.B.rowptr[k + 1] - b0);
        s_b0[t] = b0;
        s_len[t] = my_len;
      }
      int ub = my_len, mx = my_len;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        ub += __shfl_xor_sync(kFull, ub, o);
        mx = max(mx, __shfl_xor_sync(kFull, mx, o));
      }
      constexpr int kW = kPlanThreads / 32;
      if (lane == 0) {
        s_red[warp] = ub;
        s_red[kW + warp] = mx;
      }
      __syncthreads();
      ub = 0;
      mx = 0;
#pragma unroll
      for (int w2 = 0; w2 < kW; ++w2) {
        ub += s_red[w2];
        mx = max(mx, s_red[kW + w2]);
      }
      ok = ub > 0 && mx <= G && words <= 8ll * ub + 64;
      if (ok) {
        // products of this thread: step s covers A entry j = s * kGroups + grp
        int col[kSteps];
#pragma unroll
        for (int st = 0; st < kSteps; ++st) {
          const int j = st * kGroups + grp;
          col[st] = -1;
          if (j < na && gl < s_len[j]) col[st] = p.B.colidx[s_b0[j] + gl];
        }
        uint32_t dup = 0;
#pragma unroll
        for (int st = 0; st < kSteps; ++st) {
          if (col[st] >= 0) {
            const uint32_t off = static_cast<uint32_t>(col[st]);
            const uint32_t w = off >> 5;
            const uint32_t jw = w & (S::kWPT - 1);
            const uint32_t bit = 1u << (off & 31u);
            if (atomicOr(bm + plan_phys<S>(w), bit) & bit) dup |= 1u << st;
            atomicOr(sm + (jw >> 5) * kPlanThreads + (w >> S::kLogWPT), 1u << (jw & 31u));
          }
        }
        __syncthreads();
        int run = 0;
#pragma unroll
        for (int h = 0; h < S::kSPT; ++h) {
          uint32_t m = sm[h * kPlanThreads + t];
          sm[h * kPlanThreads + t] = 0u;  // only this thread reads it
          while (m) {
            const int b = __ffs(m) - 1;
            m &= m - 1u;
            const int ph = ((h << 5) | b) * kPlanThreads + t;
            pre[ph] = static_cast<uint16_t>(run);
            run += __popc(bm[ph]);
          }
        }
        long long total;
        base[t] = static_cast<int>(block_exclusive_scan(static_cast<long long>(run), s_scan, &total));
        __syncthreads();
        uint16_t* ranks = p.ranks + row * kBmrSlots;
#pragma unroll
        for (int st = 0; st < kSteps; ++st) {
          if (col[st] >= 0) {
            const uint32_t off = static_cast<uint32_t>(col[st]);
            const uint32_t w = off >> 5;
            const uint32_t ph = plan_phys<S>(w);
            const int pos = base[w >> S::kLogWPT] + pre[ph] + __popc(bm[ph] & ((1u << (off & 31u)) - 1u));
            const int j = st * kGroups + grp;
            ranks[j * G + gl] = static_cast<uint16_t>(pos | (((dup >> st) & 1u) << 15));
          }
        }
        __syncthreads();
#pragma unroll
        for (int st = 0; st < kSteps; ++st) {
          if (col[st] >= 0) bm[plan_phys<S>(static_cast<uint32_t>(col[st]) >> 5)] = 0u;
        }
        if (t == 0) {
          p.c_rowptr[row + 1] = total;
          p.cls[row] = kClsBmrWide;
          p.lo[row] = 0;
          p.hi[row] = static_cast<int32_t>(ncols - 1);
          ++taken;
          prod += static_cast<unsigned long long>(ub);
        }
      }
      __syncthreads();  // bitmap clear and s_b0/s_len reuse
    }
    if (!ok && t == 0) pending[atomicAdd(&p.sum->n_pending, 1)] = static_cast<int32_t>(row);
  }
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
  using S = BmrShape<LOGW>;
  const size_t smem = static_cast<size_t>(kRowsPerCta) * S::template warp_bytes<T>(numeric);
  auto kern = numeric ? bmr_rows_kernel<T, LOGW, G, true> : bmr_rows_kernel<T, LOGW, G, false>;
  static int per_sm[2] = {0, 0};
  if (per_sm[numeric] == 0) per_sm[numeric] = occupancy(kern, 32 * kRowsPerCta, smem);
  const int64_t grid = clamp_grid((p.seg_len + kRowsPerCta - 1) / kRowsPerCta, num_sms, per_sm[numeric]);
  kern<<<static_cast<int>(grid), 32 * kRowsPerCta, smem, s>>>(p);
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
  const size_t smem = PlanShape<LOGW>::bytes();
  static int per_sm = 0;
  if (per_sm == 0) per_sm = occupancy(bmr_plan_kernel<T, LOGW, G>, kPlanThreads, smem);
  const int64_t grid = clamp_grid(ap.m, num_sms, per_sm);
  bmr_plan_kernel<T, LOGW, G><<<static_cast<int>(grid), kPlanThreads, smem, s>>>(p, ap, ncols, pending);
}

}  // namespace

template <typename T>
void launch_bmr(const RowPlan<T>& p, int bin, bool numeric, int num_sms, cudaStream_t s, int* launches) {
  switch (bin) {
    case 0: launch_bmr_w<T, bmr_log_words(0)>(p, numeric, num_sms, s); break;
    case 1: launch_bmr_w<T, bmr_log_words(1)>(p, numeric, num_sms, s); break;
    case 2: launch_bmr_w<T, bmr_log_words(2)>(p, numeric, num_sms, s); break;
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
