// Bitmap rows: rows whose product columns span at most 65,536 columns.
//
// Workspace.  The row's private workspace w of Gustavson's algorithm
// (Sec. 5.1) is a bitmap with one bit per column of the row's range [lo, hi]
// -- the sparse byte-map workspace of the paper's SpGEMM with a bit in place
// of a byte -- plus a compact value array of exactly nnz(C[i,:]) entries:
//   symbolic:  set the bit of every product column; the number of bits that
//              were 0 before the atomicOr is nnz(C[i,:]) (no probing).
//   numeric:   1. set the bits again;
//              2. prefix sums of the bit counts give every set column its
//                 rank, which is its position in the sorted output row;
//              3. every product adds its value at the rank of its column
//                 (a shared-memory atomic, the atomic level of Sec. 4);
//              4. the team copies the compact row to C with coalesced stores.
// The output is sorted by construction, so no sort is needed, and one team
// owns the row (shard pattern, Sec. 4).
//
// Layout.  The bitmap is read in the rank pass as 128-bit chunks; thread t of
// the team owns chunks [t*IPT, (t+1)*IPT) (IPT chunks per thread) and the
// chunk it reads in step j is stored at position j*NT + t, so a step's reads
// of all threads are contiguous in shared memory (no bank conflicts).
#include "ws_internal.cuh"

namespace wsk {

namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr int kUnroll = 4;

template <int WPR>
__device__ __forceinline__ void team_sync() {
  if constexpr (WPR == 1) {
    __syncwarp();
  } else {
    __syncthreads();
  }
}

// LOGW: log2 of bitmap words (span <= 32 << LOGW columns); CAP: entries the
// staging array holds; WPR: warps per row team; RPC: row teams per CTA.
template <int LOGW, int CAP, int WPR>
struct BitmapShape {
  static constexpr int kNT = 32 * WPR;
  static constexpr int kChunks = (1 << LOGW) / 4;                     // 128-bit chunks of the bitmap
  static constexpr int kIPT = kChunks > kNT ? kChunks / kNT : 1;      // chunks per thread
  static constexpr int kLogIPT = kIPT == 1 ? 0 : (kIPT == 2 ? 1 : kIPT == 4 ? 2 : kIPT == 8 ? 3 : kIPT == 16 ? 4 : kIPT == 32 ? 5 : 6);
  static constexpr int kPhysChunks = kIPT * kNT;
  static_assert((1 << kLogIPT) == kIPT, "chunks per thread must be a power of two <= 64");
  // bytes per team
  template <typename T>
  static constexpr size_t team_bytes(bool numeric) {
    return static_cast<size_t>(kPhysChunks) * 16 +
           (numeric ? static_cast<size_t>(kPhysChunks) * 2 + kNT * 4 + static_cast<size_t>(CAP) * (4 + sizeof(T)) : 0);
  }
};

// Physical 32-bit word index of bitmap word w.
template <class S>
__device__ __forceinline__ uint32_t phys_word(uint32_t w) {
  const uint32_t chunk = w >> 2;
  const uint32_t owner = chunk >> S::kLogIPT;
  const uint32_t step = chunk & (S::kIPT - 1);
  return ((step * S::kNT + owner) << 2) | (w & 3u);
}

template <typename T, int LOGW, int CAP, int WPR, int RPC, bool NUMERIC>
__global__ void __launch_bounds__(32 * WPR * RPC, 1024 / (32 * WPR * RPC))
    bitmap_rows_kernel(const RowPlan<T> p) {
  static_assert(WPR == 1 || RPC == 1, "multi-warp row teams use the whole CTA");
  using S = BitmapShape<LOGW, CAP, WPR>;
  constexpr int kNT = S::kNT;
  extern __shared__ __align__(16) unsigned char smem_raw[];
  __shared__ long long s_b0[kNT * RPC], s_b1[kNT * RPC];  // staged B-row bounds of A entries
  __shared__ T s_a[kNT * RPC];                             // staged A values
  __shared__ int s_cnt[RPC];
  __shared__ long long s_scan[32];

  const int sub = threadIdx.x / kNT;
  const int t = threadIdx.x % kNT;
  const int lane = threadIdx.x & 31;
  unsigned char* team = smem_raw + static_cast<size_t>(sub) * S::template team_bytes<T>(NUMERIC);
  uint32_t* bm = reinterpret_cast<uint32_t*>(team);
  uint4* bm4 = reinterpret_cast<uint4*>(team);
  uint16_t* pre = reinterpret_cast<uint16_t*>(team + static_cast<size_t>(S::kPhysChunks) * 16);
  int* base = reinterpret_cast<int*>(team + static_cast<size_t>(S::kPhysChunks) * 18);
  int* st_key = base + kNT;
  T* st_val = reinterpret_cast<T*>(st_key + CAP);

  const int lg = p.log2_group;
  const int gsize = 1 << lg;
  const int grp = t >> lg;
  const int gl = t & (gsize - 1);
  const int ngrp = kNT >> lg;
  long long* sb0 = s_b0 + sub * kNT;
  long long* sb1 = s_b1 + sub * kNT;
  T* sa = s_a + sub * kNT;

  for (int64_t r = static_cast<int64_t>(blockIdx.x) * RPC + sub; r < p.seg_len;
       r += static_cast<int64_t>(gridDim.x) * RPC) {
    const int32_t row = p.perm[p.seg_begin + r];
    const int lo = p.lo[row];
    int64_t cbase = 0, cnt = 0;
    if constexpr (NUMERIC) {
      cbase = p.c_rowptr[row];
      const int64_t want = p.c_rowptr[row + 1] - cbase;
      cnt = want < CAP ? want : CAP;  // the staging array bounds every access
      if (t == 0 && want > CAP) atomicOr(&p.sum->status, kErrCount);
    }
    // Clear the workspace.
    for (int s = t; s < S::kPhysChunks; s += kNT) bm4[s] = make_uint4(0u, 0u, 0u, 0u);
    if constexpr (NUMERIC) {
      for (int s = t; s < cnt; s += kNT) st_val[s] = T(0);
    }
    int my_new = 0;
    const int64_t ra = p.A.rowptr[row], re = p.A.rowptr[row + 1];

    // Phase 1: set the bit of every product column.
    // (for the numeric pass phase 3 walks the same products again)
#pragma unroll 1
    for (int phase = 0; phase < (NUMERIC ? 2 : 1); ++phase) {
      if (phase == 1) {
        // Phase 2: rank of every 128-bit chunk inside the row (numeric only).
        team_sync<WPR>();
        int run = 0;
#pragma unroll 4
        for (int j = 0; j < S::kIPT; ++j) {
          const int ph = j * kNT + t;
          const uint4 v = bm4[ph];
          pre[ph] = static_cast<uint16_t>(run);
          run += __popc(v.x) + __popc(v.y) + __popc(v.z) + __popc(v.w);
        }
        int total;
        if constexpr (WPR == 1) {
          int incl = run;
#pragma unroll
          for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(kFull, incl, o);
            if (lane >= o) incl += y;
          }
          base[t] = incl - run;
          total = __shfl_sync(kFull, incl, 31);
        } else {
          long long tot;
          base[t] = static_cast<int>(block_exclusive_scan(static_cast<long long>(run), s_scan, &tot));
          total = static_cast<int>(tot);
        }
        if (t == 0 && total != cnt) atomicOr(&p.sum->status, kErrCount);
      }
      team_sync<WPR>();
      for (int64_t cb = ra; cb < re; cb += kNT) {
        const int n = static_cast<int>(min(static_cast<int64_t>(kNT), re - cb));
        if (t < n) {
          const int k = p.A.colidx[cb + t];
          sb0[t] = p.B.rowptr[k];
          sb1[t] = p.B.rowptr[k + 1];
          if constexpr (NUMERIC) sa[t] = p.A.vals[cb + t];
        }
        team_sync<WPR>();
        for (int j0 = grp; j0 < n; j0 += ngrp * kUnroll) {
          int cc[kUnroll];
          T vv[kUnroll];
#pragma unroll
          for (int u = 0; u < kUnroll; ++u) {
            const int j = j0 + u * ngrp;
            cc[u] = -1;
            vv[u] = T(0);
            if (j < n) {
              const long long q = sb0[j] + gl;
              if (q < sb1[j]) {
                cc[u] = p.B.colidx[q];
                if (NUMERIC && phase == 1) vv[u] = sa[j] * p.B.vals[q];
              }
            }
          }
#define WS_BITMAP_VISIT(c_, v_)                                                                   \
  do {                                                                                          \
    const uint32_t off_ = static_cast<uint32_t>((c_) - lo);                                     \
    const uint32_t w_ = off_ >> 5;                                                              \
    const uint32_t bit_ = 1u << (off_ & 31u);                                                   \
    if (phase == 0) {                                                                           \
      if constexpr (NUMERIC) {                                                                  \
        atomicOr(&bm[phys_word<S>(w_)], bit_);                                                  \
      } else {                                                                                  \
        const uint32_t old_ = atomicOr(&bm[phys_word<S>(w_)], bit_);                            \
        my_new += (old_ & bit_) == 0u;                                                          \
      }                                                                                         \
    } else {                                                                                    \
      const uint32_t chunk_ = w_ >> 2;                                                          \
      const uint32_t ph_ = (chunk_ & (S::kIPT - 1)) * kNT + (chunk_ >> S::kLogIPT);             \
      const uint4 x_ = bm4[ph_];                                                                \
      const uint32_t s_ = w_ & 3u;                                                              \
      const uint32_t word_ = s_ == 0 ? x_.x : s_ == 1 ? x_.y : s_ == 2 ? x_.z : x_.w;            \
      const int pos_ = base[chunk_ >> S::kLogIPT] + pre[ph_] + (s_ > 0 ? __popc(x_.x) : 0) +     \
                       (s_ > 1 ? __popc(x_.y) : 0) + (s_ > 2 ? __popc(x_.z) : 0) +              \
                       __popc(word_ & (bit_ - 1u));                                             \
      if (pos_ < cnt) {                                                                         \
        st_key[pos_] = (c_);                                                                    \
        atomicAdd(&st_val[pos_], (v_));                                                         \
      }                                                                                         \
    }                                                                                           \
  } while (0)
#pragma unroll
          for (int u = 0; u < kUnroll; ++u) {
            if (cc[u] >= 0) WS_BITMAP_VISIT(cc[u], vv[u]);
          }
          // B rows longer than the group: the rest of each row.
#pragma unroll 1
          for (int u = 0; u < kUnroll; ++u) {
            const int j = j0 + u * ngrp;
            if (j >= n) break;
            const long long qe = sb1[j];
            for (long long q = sb0[j] + gl + gsize; q < qe; q += gsize) {
              T v = T(0);
              if (NUMERIC && phase == 1) v = sa[j] * p.B.vals[q];
              WS_BITMAP_VISIT(p.B.colidx[q], v);
            }
          }
#undef WS_BITMAP_VISIT
        }
        team_sync<WPR>();
      }
    }

    if constexpr (!NUMERIC) {
      int c = my_new;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) c += __shfl_xor_sync(kFull, c, o);
      if constexpr (WPR > 1) {
        if (t == 0) s_cnt[sub] = 0;
        team_sync<WPR>();
        if (lane == 0) atomicAdd(&s_cnt[sub], c);
        team_sync<WPR>();
        c = s_cnt[sub];
      }
      if (t == 0) p.c_rowptr[row + 1] = c;
    } else {
      // Phase 4: copy the compact, sorted row to C.
      for (int s = t; s < cnt; s += kNT) {
        p.c_colidx[cbase + s] = st_key[s];
        p.c_vals[cbase + s] = st_val[s];
      }
    }
    team_sync<WPR>();
  }
}

template <typename T, int LOGW, int CAP, int WPR, int RPC>
void launch_bm(const RowPlan<T>& p, bool numeric, int num_sms, cudaStream_t s) {
  using S = BitmapShape<LOGW, CAP, WPR>;
  const size_t smem = static_cast<size_t>(RPC) * S::template team_bytes<T>(numeric);
  const int threads = 32 * WPR * RPC;
  auto kern = numeric ? bitmap_rows_kernel<T, LOGW, CAP, WPR, RPC, true>
                      : bitmap_rows_kernel<T, LOGW, CAP, WPR, RPC, false>;
  static int per_sm[2] = {0, 0};
  if (per_sm[numeric] == 0) {
    cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
    int n = 0;
    cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, kern, threads, smem);
    per_sm[numeric] = n > 0 ? n : 1;
  }
  int64_t grid = (p.seg_len + RPC - 1) / RPC;
  const int64_t cap = static_cast<int64_t>(num_sms) * per_sm[numeric];
  if (grid > cap) grid = cap;
  if (grid < 1) grid = 1;
  kern<<<static_cast<int>(grid), threads, smem, s>>>(p);
}

}  // namespace

template <typename T>
void launch_bitmap(const RowPlan<T>& p, int bin, bool numeric, int num_sms, cudaStream_t s, int* launches) {
  switch (bin) {
    case 0: launch_bm<T, kBitmapBins[0].log_words, kBitmapBins[0].cap, 1, 8>(p, numeric, num_sms, s); break;
    case 1: launch_bm<T, kBitmapBins[1].log_words, kBitmapBins[1].cap, 1, 4>(p, numeric, num_sms, s); break;
    case 2: launch_bm<T, kBitmapBins[2].log_words, kBitmapBins[2].cap, 1, 4>(p, numeric, num_sms, s); break;
    case 3: launch_bm<T, kBitmapBins[3].log_words, kBitmapBins[3].cap, 1, 2>(p, numeric, num_sms, s); break;
    case 4: launch_bm<T, kBitmapBins[4].log_words, kBitmapBins[4].cap, 8, 1>(p, numeric, num_sms, s); break;
    default: return;
  }
  *launches += 1;
}

template void launch_bitmap<float>(const RowPlan<float>&, int, bool, int, cudaStream_t, int*);
template void launch_bitmap<double>(const RowPlan<double>&, int, bool, int, cudaStream_t, int*);

}  // namespace wsk
