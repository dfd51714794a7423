// Register bitmap rows: one warp per row for rows with at most 16 stored A
// entries whose B rows each fit in one group of lanes (uniformly sparse
// products such as random matrices and stencils).
//
// The workspace is the bitmap + rank scheme of the bitmap rows (one bit per
// column of the row's range, the sparse byte-map workspace of Gustavson's
// SpGEMM, Sec. 5.1), but every lane keeps its products (column and scaled
// value) in registers, so B is walked once per pass:
//   symbolic:  atomicOr every product column into the bitmap and count the
//              bits that were 0 (nnz of the row);
//   numeric:   set the bits, rank every 128-bit chunk of the bitmap (prefix
//              of bit counts), add each product's value at the rank of its
//              column in a compact staging array, copy the sorted row to C.
// Lanes are split into groups of G lanes; the group of lane l takes stored A
// entries j = l / G, l / G + 32/G, ...; lane l takes element l % G of B[k_j,:].
//
// Bitmap layout: chunk i (128 bits) belongs to lane i / IPT in the rank pass
// and is stored at i ^ ((i / IPT) & 7), so the 8 lanes of a quarter warp read
// 8 different bank quads in every step.
#include "ws_internal.cuh"

namespace wsk {

namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr int kRowsPerCta = 4;

template <int LOGW>
struct BmrShape {
  static constexpr int kWords = 1 << LOGW;
  static constexpr int kChunks = kWords / 4 < 32 ? 32 : kWords / 4;
  static constexpr int kIPT = kChunks / 32;
  static constexpr int kLogIPT = kIPT == 1 ? 0 : kIPT == 2 ? 1 : kIPT == 4 ? 2 : kIPT == 8 ? 3 : 4;
  static constexpr int kSwz = kIPT >= 8 ? 7 : kIPT - 1;
  static_assert((1 << kLogIPT) == kIPT, "chunks per lane must be a power of two <= 16");
  template <typename T>
  static constexpr size_t warp_bytes(bool numeric) {
    return static_cast<size_t>(kChunks) * 16 +
           (numeric ? static_cast<size_t>(kChunks) * 2 + 32 * 4 + static_cast<size_t>(kBmrCap) * (4 + sizeof(T)) : 0);
  }
};

template <class S>
__device__ __forceinline__ uint32_t phys_chunk(uint32_t i) {
  return i ^ ((i >> S::kLogIPT) & S::kSwz);
}

template <typename T, int LOGW, int G, bool NUMERIC>
__global__ void __launch_bounds__(32 * kRowsPerCta, NUMERIC ? 3 : 6) bmr_rows_kernel(const RowPlan<T> p) {
  using S = BmrShape<LOGW>;
  constexpr int kGroups = 32 / G;                 // A entries per step
  constexpr int kSteps = kBmrMaxA / kGroups;       // steps that cover kBmrMaxA entries
  extern __shared__ __align__(16) unsigned char smem_raw[];
  const int sub = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  unsigned char* ws = smem_raw + static_cast<size_t>(sub) * S::template warp_bytes<T>(NUMERIC);
  uint32_t* bm = reinterpret_cast<uint32_t*>(ws);
  uint4* bm4 = reinterpret_cast<uint4*>(ws);
  uint16_t* pre = reinterpret_cast<uint16_t*>(ws + static_cast<size_t>(S::kChunks) * 16);
  int* base = reinterpret_cast<int*>(ws + static_cast<size_t>(S::kChunks) * 18);
  int* st_key = base + 32;
  T* st_val = reinterpret_cast<T*>(st_key + kBmrCap);
  const int grp = lane / G, gl = lane % G;

  for (int64_t r = static_cast<int64_t>(blockIdx.x) * kRowsPerCta + sub; r < p.seg_len;
       r += static_cast<int64_t>(gridDim.x) * kRowsPerCta) {
    const int32_t row = p.perm[p.seg_begin + r];
    const int lo = p.lo[row];
    const int64_t ra = p.A.rowptr[row];
    const int na = static_cast<int>(p.A.rowptr[row + 1] - ra);
    // Lane j < na holds stored A entry j: its B row start, length and value.
    long long my_b0 = 0;
    int my_len = 0;
    T my_a = T(0);
    if (lane < na) {
      const int k = p.A.colidx[ra + lane];
      my_b0 = p.B.rowptr[k];
      my_len = static_cast<int>(p.B.rowptr[k + 1] - my_b0);
      if constexpr (NUMERIC) my_a = p.A.vals[ra + lane];
    }
    // This lane's products: step s covers A entry s * kGroups + grp.
    int col[kSteps];
    T val[kSteps];
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
    int64_t cbase = 0;
    int cnt = 0;
    if constexpr (NUMERIC) {
      cbase = p.c_rowptr[row];
      const int64_t want = p.c_rowptr[row + 1] - cbase;
      cnt = static_cast<int>(want < kBmrCap ? want : kBmrCap);
      if (lane == 0 && want > kBmrCap) atomicOr(&p.sum->status, kErrCount);
      for (int s2 = lane; s2 < cnt; s2 += 32) st_val[s2] = T(0);
    }
    for (int s2 = lane; s2 < S::kChunks; s2 += 32) bm4[s2] = make_uint4(0u, 0u, 0u, 0u);
    __syncwarp();

    int my_new = 0;
#pragma unroll
    for (int s = 0; s < kSteps; ++s) {
      if (col[s] >= 0) {
        const uint32_t off = static_cast<uint32_t>(col[s] - lo);
        const uint32_t w = off >> 5;
        const uint32_t bit = 1u << (off & 31u);
        uint32_t* word = bm + ((phys_chunk<S>(w >> 2) << 2) | (w & 3u));
        if constexpr (NUMERIC) {
          atomicOr(word, bit);
        } else {
          my_new += (atomicOr(word, bit) & bit) == 0u;
        }
      }
    }

    if constexpr (!NUMERIC) {
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) my_new += __shfl_xor_sync(kFull, my_new, o);
      if (lane == 0) p.c_rowptr[row + 1] = my_new;
      __syncwarp();
    } else {
      __syncwarp();
      // Rank of every chunk: lane l owns chunks [l * IPT, (l + 1) * IPT).
      int run = 0;
#pragma unroll
      for (int j = 0; j < S::kIPT; ++j) {
        const uint32_t ph = phys_chunk<S>(static_cast<uint32_t>(lane * S::kIPT + j));
        const uint4 x = bm4[ph];
        pre[ph] = static_cast<uint16_t>(run);
        run += __popc(x.x) + __popc(x.y) + __popc(x.z) + __popc(x.w);
      }
      int incl = run;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(kFull, incl, o);
        if (lane >= o) incl += y;
      }
      base[lane] = incl - run;
      const int total = __shfl_sync(kFull, incl, 31);
      if (lane == 0 && total != cnt) atomicOr(&p.sum->status, kErrCount);
      __syncwarp();
#pragma unroll
      for (int s = 0; s < kSteps; ++s) {
        if (col[s] >= 0) {
          const uint32_t off = static_cast<uint32_t>(col[s] - lo);
          const uint32_t w = off >> 5;
          const uint32_t i = w >> 2;
          const uint32_t ph = phys_chunk<S>(i);
          const uint4 x = bm4[ph];
          const uint32_t q = w & 3u;
          const uint32_t wd = q == 0 ? x.x : q == 1 ? x.y : q == 2 ? x.z : x.w;
          const int pos = base[i >> S::kLogIPT] + pre[ph] + (q > 0 ? __popc(x.x) : 0) + (q > 1 ? __popc(x.y) : 0) +
                          (q > 2 ? __popc(x.z) : 0) + __popc(wd & ((1u << (off & 31u)) - 1u));
          if (pos < cnt) {
            st_key[pos] = col[s];
            atomicAdd(&st_val[pos], val[s]);
          }
        }
      }
      __syncwarp();
      for (int s2 = lane; s2 < cnt; s2 += 32) {
        p.c_colidx[cbase + s2] = st_key[s2];
        p.c_vals[cbase + s2] = st_val[s2];
      }
      __syncwarp();
    }
  }
}

template <typename T, int LOGW, int G>
void launch_bmr_g(const RowPlan<T>& p, bool numeric, int num_sms, cudaStream_t s) {
  using S = BmrShape<LOGW>;
  const size_t smem = static_cast<size_t>(kRowsPerCta) * S::template warp_bytes<T>(numeric);
  auto kern = numeric ? bmr_rows_kernel<T, LOGW, G, true> : bmr_rows_kernel<T, LOGW, G, false>;
  static int per_sm[2] = {0, 0};
  if (per_sm[numeric] == 0) {
    cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
    int n = 0;
    cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, kern, 32 * kRowsPerCta, smem);
    per_sm[numeric] = n > 0 ? n : 1;
  }
  int64_t grid = (p.seg_len + kRowsPerCta - 1) / kRowsPerCta;
  const int64_t cap = static_cast<int64_t>(num_sms) * per_sm[numeric];
  if (grid > cap) grid = cap;
  if (grid < 1) grid = 1;
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

template void launch_bmr<float>(const RowPlan<float>&, int, bool, int, cudaStream_t, int*);
template void launch_bmr<double>(const RowPlan<double>&, int, bool, int, cudaStream_t, int*);

}  // namespace wsk
