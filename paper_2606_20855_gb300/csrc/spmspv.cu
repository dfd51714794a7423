// Sparse matrix - sparse vector product y = A x (Sec. 5.2, "Sparse Linear
// Algebra": SpMSpV).  The paper's formulation walks the stored entries of x
// and accumulates the matching columns of A into a sparse byte-map over y,
// wrapped in a merge level because different columns hit the same positions
// of y.  Here A is given by columns (the CSR of A^T), and the merge level is
// the L2: every product is added into one dense accumulator of length m with
// a global atomic add, and its position is marked in a bitmap (the byte-map
// with a bit per position).  The coalesce step is a compaction of the bitmap
// in index order.
//
//   1. product offsets: off[k + 1] = length of column x_idx[k] of A, and the
//      column's first entry; scan -> off[k] = first product of x entry k
//   2. scatter: product p (balanced over the GPU: every thread takes products
//      p, p + stride, ...) finds its x entry by binary search in off, then
//      acc[i] += A[i,j] x[j] and sets bit i
//   3. compaction: set bits per tile of 4096 positions -> scan -> every tile
//      writes its positions (ascending) and accumulated values to y
#include "ws_internal.cuh"

namespace wsk {

namespace {

constexpr int kSvThreads = 256;
constexpr int kSvTile = 4096;  // positions of y per compaction tile (128 bitmap words)

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

template <typename T>
__global__ void __launch_bounds__(kSvThreads) sv_scatter_kernel(const SpmspvPlan<T> p) {
  const int64_t total = p.off[p.nx];
  for (int64_t q = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; q < total;
       q += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    // x entry k with off[k] <= q < off[k + 1] (off is non-decreasing; the last k wins for empty columns)
    int64_t lo = 0, hi = p.nx - 1;
    while (lo < hi) {  // O(log nx) probes
      const int64_t mid = (lo + hi + 1) >> 1;
      if (p.off[mid] <= q) {
        lo = mid;
      } else {
        hi = mid - 1;
      }
    }
    const int64_t b = p.first[lo] + (q - p.off[lo]);
    const int32_t i = p.At.colidx[b];
    if (i < 0 || i >= p.m) {
      atomicOr(&p.sum->status, kErrCount);
      continue;
    }
    atomicAdd(p.acc + i, p.At.vals[b] * p.x_vals[lo]);
    atomicOr(p.bits + (i >> 5), 1u << (i & 31));
  }
}

// Set bits of every compaction tile: cnt[t + 1].
__global__ void __launch_bounds__(kSvThreads) sv_tile_count_kernel(const uint32_t* bits, int64_t m, int64_t* cnt) {
  __shared__ int s_red[kSvThreads / 32];
  const int64_t words = (m + 31) >> 5;
  const int64_t tiles = (m + kSvTile - 1) / kSvTile;
  for (int64_t t = blockIdx.x; t < tiles; t += gridDim.x) {
    const int64_t w0 = t * (kSvTile / 32);
    int c = 0;
    for (int64_t w = w0 + threadIdx.x; w < w0 + kSvTile / 32 && w < words; w += blockDim.x) c += __popc(bits[w]);
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

// Tile t writes its set positions in ascending order from y offset cnt[t]:
// one warp per 32-word slice of the tile, ballots give the order.
template <typename T>
__global__ void __launch_bounds__(kSvThreads) sv_write_kernel(const SpmspvPlan<T> p) {
  __shared__ long long s_base[kSvThreads / 32 + 1];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int64_t words = (p.m + 31) >> 5;
  const int64_t tiles = (p.m + kSvTile - 1) / kSvTile;
  for (int64_t t = blockIdx.x; t < tiles; t += gridDim.x) {
    // the tile's 128 words: warp w takes words [w0 + 16w, w0 + 16w + 16)
    constexpr int kWordsPerWarp = kSvTile / 32 / (kSvThreads / 32);
    const int64_t w0 = t * (kSvTile / 32) + static_cast<int64_t>(warp) * kWordsPerWarp;
    int c = 0;
    if (lane < kWordsPerWarp && w0 + lane < words) c = __popc(p.bits[w0 + lane]);
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
    for (int q = 0; q < kWordsPerWarp; ++q) {
      const int64_t w = w0 + q;
      const uint32_t word = w < words ? p.bits[w] : 0u;  // same word for every lane
      const bool set = (word >> lane) & 1u;
      if (set) {
        const long long at = pos + __popc(word & ((1u << lane) - 1u));
        const int64_t i = (w << 5) + lane;
        if (at < end && at < p.cap) {
          p.y_idx[at] = static_cast<int32_t>(i);
          p.y_vals[at] = p.acc[i];
        } else {
          atomicOr(&p.sum->status, kErrCount);
        }
      }
      pos += __popc(word);
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
    sv_scatter_kernel<T><<<grid_for(p.nnz_a, kSvThreads, num_sms, 8), kSvThreads, 0, s>>>(p);
    *launches += 2;
  }
  const int64_t tiles = spmspv_tiles(p.m);
  sv_tile_count_kernel<<<grid_for(tiles, 1, num_sms, 8), kSvThreads, 0, s>>>(p.bits, p.m, p.cnt);
  launch_scan(p.cnt, tiles, p.partials, p.sum, s, launches);
  sv_write_kernel<T><<<grid_for(tiles, 1, num_sms, 8), kSvThreads, 0, s>>>(p);
  *launches += 2;
}

template void launch_spmspv<float>(const SpmspvPlan<float>&, int, cudaStream_t, int*);
template void launch_spmspv<double>(const SpmspvPlan<double>&, int, cudaStream_t, int*);

}  // namespace wsk
