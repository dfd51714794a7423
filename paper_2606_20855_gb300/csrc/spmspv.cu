// Sparse matrix - sparse vector product y = A x (Sec. 5.2, "Sparse Linear
// Algebra": SpMSpV).  The paper's formulation walks the stored entries of x
// and accumulates the matching columns of A into a sparse byte-map over y,
// wrapped in a merge level because different columns hit the same positions
// of y.  Here A is given by columns (the CSR of A^T), and the merge level is
// the L2: every product is added into one dense accumulator of length m with
// a global atomic add, and its position is marked in a byte-map (a plain
// store of 1: idempotent, so positions that many columns hit need no atomic).
// The coalesce step is a compaction of the byte-map in index order.
//
//   1. product offsets: off[k + 1] = length of column x_idx[k] of A, and the
//      column's first entry; scan -> off[k] = first product of x entry k
//   2. scatter: tiles of consecutive products (balanced over the GPU) find
//      the x entries they span, and every product finds its entry by binary
//      search in those offsets, then acc[i] += A[i,j] x[j] and mark[i] = 1
//   3. compaction: marks per tile of 4096 positions -> scan -> every tile
//      writes its positions (ascending) and accumulated values to y
#include "ws_internal.cuh"

namespace wsk {

namespace {

constexpr int kSvThreads = 256;
constexpr int kSvTile = 4096;  // positions of y per compaction tile (4 KB of the byte-map)

// Counts the non-zero bytes of 16 bytes.
__device__ __forceinline__ int marked(const uint4 v) {
  return __popc(__vcmpne4(v.x, 0u) & 0x01010101u) + __popc(__vcmpne4(v.y, 0u) & 0x01010101u) +
         __popc(__vcmpne4(v.z, 0u) & 0x01010101u) + __popc(__vcmpne4(v.w, 0u) & 0x01010101u);
}

template <typename T>
__global__ void __launch_bounds__(kSvThreads) sv_offsets_kernel(const SpmspvPlan<T> p) {
  for (int64_t k = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; k < p.nx;
       k += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t j = p.x_idx[k];
    int64_t len = 0, first = 0;
    if (j >= 0 && j < p.n) {
      first = p.At.rowptr[j];
      len = p.At.rowptr[j + 1] - first;
    } else {
      atomicOr(&p.sum->status, kErrCount);  // index outside A's columns: skipped
    }
    p.off[k + 1] = len;
    p.first[k] = first;
  }
}

// Largest k in [lo, hi] with off[k] <= q, given off[lo] <= q; a 32-way search
// by one warp (every lane probes one point per level).  O(log_32 (hi - lo)) levels.
__device__ __forceinline__ int64_t warp_last_le(const int64_t* off, int64_t lo, int64_t hi, int64_t q) {
  const int lane = threadIdx.x & 31;
  for (int level = 0; level < 16 && hi > lo; ++level) {
    const int64_t step = (hi - lo + 32) / 32;
    const int64_t pos = lo + lane * step;
    const unsigned m = __ballot_sync(0xffffffffu, pos <= hi && off[pos] <= q);
    lo += static_cast<int64_t>(31 - __clz(m)) * step;  // lane 0 always qualifies
    hi = hi < lo + step - 1 ? hi : lo + step - 1;
  }
  return lo;
}

// Load-balanced scatter: a CTA takes kScatterTile consecutive products, two
// warps find the x entries holding the first and the last, the offsets of
// that range go to shared memory (when it fits), and every thread finds the
// entry of each of its products by binary search there.
// Positions of y below kPrivRows are summed in a CTA-private copy in shared
// memory and added to y once per CTA at the end: adds to one address of y
// serialise in L2, and a power-law matrix concentrates its products on a few
// rows (an R-MAT matrix without vertex permutation on its first rows).  The
// result is the same for any input; only the speed depends on where the
// heavy rows lie.
constexpr int kPerThread = 8;
constexpr int kScatterTile = kSvThreads * kPerThread;
constexpr int kScatterSpan = 2048;  // x entries of one tile kept in shared memory
constexpr int kPrivRows = 4096;     // positions of y summed per CTA in shared memory first

template <typename T>
__global__ void __launch_bounds__(kSvThreads) sv_scatter_kernel(const SpmspvPlan<T> p) {
  __shared__ long long s_off[kScatterSpan + 1];
  __shared__ long long s_k[2];
  __shared__ T s_acc[kPrivRows];
  __shared__ uint8_t s_hit[kPrivRows];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t total = p.off[p.nx];
  const int priv = static_cast<int>(p.m < kPrivRows ? p.m : kPrivRows);
  for (int i = threadIdx.x; i < kPrivRows; i += blockDim.x) {
    s_acc[i] = T(0);
    s_hit[i] = 0;
  }
  __syncthreads();
  bool bad = false;
  for (int64_t t0 = static_cast<int64_t>(blockIdx.x) * kScatterTile; t0 < total;
       t0 += static_cast<int64_t>(gridDim.x) * kScatterTile) {
    const int64_t t1 = t0 + kScatterTile < total ? t0 + kScatterTile : total;
    if (warp < 2) {
      const int64_t k = warp_last_le(p.off, 0, p.nx - 1, warp == 0 ? t0 : t1 - 1);
      if (lane == 0) s_k[warp] = k;
    }
    __syncthreads();
    const int64_t k0 = s_k[0], k1 = s_k[1];
    const bool in_smem = k1 - k0 + 1 <= kScatterSpan;
    if (in_smem) {
      for (int64_t i = threadIdx.x; i <= k1 - k0 + 1; i += blockDim.x) s_off[i] = p.off[k0 + i];
    }
    __syncthreads();
    // Each thread takes kPerThread products of the tile; the lookups come
    // first, then every load is issued before the first add, so the loads of
    // all its products are in flight together.
    int64_t kk[kPerThread], bb[kPerThread];
#pragma unroll
    for (int r = 0; r < kPerThread; ++r) {
      const int64_t q = t0 + threadIdx.x + static_cast<int64_t>(r) * kSvThreads;
      kk[r] = -1;
      bb[r] = 0;
      if (q < t1) {
        int64_t k;
        if (in_smem) {  // largest local index with s_off <= q
          int lo = 0, hi = static_cast<int>(k1 - k0);
          while (lo < hi) {
            const int mid = (lo + hi + 1) >> 1;
            if (s_off[mid] <= q) {
              lo = mid;
            } else {
              hi = mid - 1;
            }
          }
          k = k0 + lo;
          bb[r] = q - s_off[lo];
        } else {
          int64_t lo = k0, hi = k1;
          while (lo < hi) {
            const int64_t mid = (lo + hi + 1) >> 1;
            if (p.off[mid] <= q) {
              lo = mid;
            } else {
              hi = mid - 1;
            }
          }
          k = lo;
          bb[r] = q - p.off[lo];
        }
        kk[r] = k;
      }
    }
#pragma unroll
    for (int r = 0; r < kPerThread; ++r) {
      if (kk[r] >= 0) bb[r] += p.first[kk[r]];
    }
    int32_t ii[kPerThread];
    T vv[kPerThread];
#pragma unroll
    for (int r = 0; r < kPerThread; ++r) {
      ii[r] = -1;
      vv[r] = T(0);
      if (kk[r] >= 0) {
        ii[r] = p.At.colidx[bb[r]];
        vv[r] = p.At.vals[bb[r]] * p.x_vals[kk[r]];
      }
    }
#pragma unroll
    for (int r = 0; r < kPerThread; ++r) {
      if (kk[r] < 0) continue;
      const int32_t i = ii[r];
      if (i < 0 || i >= p.m) {
        bad = true;
        continue;
      }
      if (i < priv) {
        atomicAdd(s_acc + i, vv[r]);
        s_hit[i] = 1;
      } else {
        atomicAdd(p.acc + i, vv[r]);
        p.mark[i] = 1;
      }
    }
    __syncthreads();  // s_off and s_k are reused by the next tile
  }
  // The CTA's private sums: one add per position it hit.
  for (int i = threadIdx.x; i < priv; i += blockDim.x) {
    if (s_hit[i]) {
      atomicAdd(p.acc + i, s_acc[i]);
      p.mark[i] = 1;
    }
  }
  if (bad) atomicOr(&p.sum->status, kErrCount);
}

// Marked positions of every compaction tile: cnt[t + 1].  One thread reads 16
// bytes (the byte-map is padded to whole tiles with zeros).
__global__ void __launch_bounds__(kSvThreads) sv_tile_count_kernel(const uint8_t* mark, int64_t m, int64_t* cnt) {
  static_assert(kSvTile == kSvThreads * 16, "one 16-byte load per thread and tile");
  __shared__ int s_red[kSvThreads / 32];
  const int64_t tiles = (m + kSvTile - 1) / kSvTile;
  for (int64_t t = blockIdx.x; t < tiles; t += gridDim.x) {
    int c = marked(reinterpret_cast<const uint4*>(mark + t * kSvTile)[threadIdx.x]);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) c += __shfl_xor_sync(0xffffffffu, c, o);
    if ((threadIdx.x & 31) == 0) s_red[threadIdx.x >> 5] = c;
    __syncthreads();
    if (threadIdx.x == 0) {
      int s = 0;
      for (int w = 0; w < kSvThreads / 32; ++w) s += s_red[w];
      cnt[t + 1] = s;
    }
    __syncthreads();
  }
}

// Tile t writes its marked positions in ascending order from y offset
// cnt[t]: warp w takes the tile's positions [512 w, 512 w + 512) in 16 rounds
// of 32, and ballots give the order.
template <typename T>
__global__ void __launch_bounds__(kSvThreads) sv_write_kernel(const SpmspvPlan<T> p) {
  constexpr int kPerWarp = kSvTile / (kSvThreads / 32);  // 512
  __shared__ long long s_base[kSvThreads / 32 + 1];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int64_t tiles = (p.m + kSvTile - 1) / kSvTile;
  for (int64_t t = blockIdx.x; t < tiles; t += gridDim.x) {
    const int64_t i0 = t * kSvTile + static_cast<int64_t>(warp) * kPerWarp;
    int c = marked(reinterpret_cast<const uint4*>(p.mark + i0)[lane]);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) c += __shfl_xor_sync(0xffffffffu, c, o);
    if (lane == 0) s_base[warp + 1] = c;
    __syncthreads();
    if (threadIdx.x == 0) {
      s_base[0] = p.cnt[t];
      for (int w = 0; w < kSvThreads / 32; ++w) s_base[w + 1] += s_base[w];
    }
    __syncthreads();
    long long pos = s_base[warp];
    const long long end = p.cnt[t + 1];
    for (int q = 0; q < kPerWarp / 32; ++q) {
      const int64_t i = i0 + q * 32 + lane;
      const bool set = p.mark[i] != 0;
      const unsigned bal = __ballot_sync(0xffffffffu, set);
      if (set) {
        const long long at = pos + __popc(bal & ((1u << lane) - 1u));
        if (at < end && at < p.cap && i < p.m) {
          p.y_idx[at] = static_cast<int32_t>(i);
          p.y_vals[at] = p.acc[i];
        } else {
          atomicOr(&p.sum->status, kErrCount);
        }
      }
      pos += __popc(bal);
    }
    __syncthreads();
  }
}

int grid_for(int64_t work, int per_block, int num_sms, int per_sm) {
  const int64_t want = (work + per_block - 1) / per_block;
  const int64_t cap = static_cast<int64_t>(num_sms) * per_sm;
  return static_cast<int>(want < 1 ? 1 : (want > cap ? cap : want));
}

}  // namespace

int64_t spmspv_tiles(int64_t m) { return (m + kSvTile - 1) / kSvTile; }

template <typename T>
void launch_spmspv(const SpmspvPlan<T>& p, int num_sms, cudaStream_t s, int* launches) {
  if (p.nx > 0) {
    sv_offsets_kernel<T><<<grid_for(p.nx, kSvThreads, num_sms, 8), kSvThreads, 0, s>>>(p);
    launch_scan(p.off, p.nx, p.partials, p.sum, s, launches);
    // products are at most nnz(A); the kernel stops at the scanned total
    sv_scatter_kernel<T><<<grid_for(p.nnz_a, kScatterTile, num_sms, 8), kSvThreads, 0, s>>>(p);
    *launches += 2;
  }
  const int64_t tiles = spmspv_tiles(p.m);
  sv_tile_count_kernel<<<grid_for(tiles, 1, num_sms, 8), kSvThreads, 0, s>>>(p.mark, p.m, p.cnt);
  launch_scan(p.cnt, tiles, p.partials, p.sum, s, launches);
  sv_write_kernel<T><<<grid_for(tiles, 1, num_sms, 8), kSvThreads, 0, s>>>(p);
  *launches += 2;
}

template void launch_spmspv<float>(const SpmspvPlan<float>&, int, cudaStream_t, int*);
template void launch_spmspv<double>(const SpmspvPlan<double>&, int, cudaStream_t, int*);

}  // namespace wsk
