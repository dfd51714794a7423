// Direct rows: a row of A with exactly one stored entry A[i,k] gives
// C[i,:] = A[i,k] * B[k,:] (Gustavson's accumulation with a single term, Sec. 5.1).
// B[k,:] is already sorted and duplicate-free, so the row is a scaled copy
// and needs no workspace.  A group of 2^log2_group lanes copies one row with
// coalesced loads and stores (a whole warp for a long row).
#include "ws_internal.cuh"

namespace wsk {

namespace {

// Short rows are copied by their group, four loads in flight per lane; a row
// longer than kDirectLong entries (a hub row of B) is copied by the whole
// warp after its group's turn, so it does not hold a group of a few lanes
// for hundreds of rounds.
constexpr int kDirectLong = 512;

template <typename T>
__device__ __forceinline__ void direct_copy(const RowPlan<T>& p, int64_t qb, int64_t len, int64_t base, T a, int lane,
                                            int width) {
  for (int64_t t0 = lane; t0 < len; t0 += 4 * width) {
    int32_t c[4];
    T v[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int64_t t = t0 + static_cast<int64_t>(u) * width;
      c[u] = t < len ? p.B.colidx[qb + t] : 0;
      v[u] = t < len ? p.B.vals[qb + t] : T(0);
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int64_t t = t0 + static_cast<int64_t>(u) * width;
      if (t < len) {
        p.c_colidx[base + t] = c[u];
        p.c_vals[base + t] = a * v[u];
      }
    }
  }
}

template <typename T>
__global__ void __launch_bounds__(256) direct_rows_kernel(const RowPlan<T> p) {
  const int lg = p.log2_group;
  const int gsize = 1 << lg;
  const int lane = threadIdx.x & 31;
  const int gl = lane & (gsize - 1);
  const int per_warp = 32 >> lg;  // rows a warp takes per round
  const int64_t warps = (static_cast<int64_t>(gridDim.x) * blockDim.x) >> 5;
  for (int64_t r0 = ((static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5) * per_warp; r0 < p.seg_len;
       r0 += warps * per_warp) {  // warp-uniform loop: the ballot below needs every lane
    const int64_t r = r0 + (lane >> lg);
    int64_t qb = 0, len = 0, base = 0;
    T a = T(0);
    if (r < p.seg_len) {
      const int32_t row = p.perm[p.seg_begin + r];
      const int64_t pa = p.A.rowptr[row];
      const int k = p.A.colidx[pa];
      a = p.A.vals[pa];
      qb = p.B.rowptr[k];
      len = p.B.rowptr[k + 1] - qb;
      base = p.c_rowptr[row];
      if (len != p.c_rowptr[row + 1] - base) {
        if (gl == 0) atomicOr(&p.sum->status, kErrCount);
        len = 0;
      }
    }
    const bool lng = len > kDirectLong;
    if (!lng) direct_copy(p, qb, len, base, a, gl, gsize);
    for (unsigned m = __ballot_sync(0xffffffffu, lng && gl == 0); m; m &= m - 1u) {
      const int src = __ffs(m) - 1;
      direct_copy(p, __shfl_sync(0xffffffffu, qb, src), __shfl_sync(0xffffffffu, len, src),
                  __shfl_sync(0xffffffffu, base, src), __shfl_sync(0xffffffffu, a, src), lane, 32);
    }
  }
}

}  // namespace

template <typename T>
void launch_direct(const RowPlan<T>& p, int num_sms, cudaStream_t s, int* launches) {
  const int64_t threads_needed = p.seg_len << p.log2_group;
  int64_t grid = (threads_needed + 255) / 256;
  const int64_t cap = static_cast<int64_t>(num_sms) * 8;
  if (grid > cap) grid = cap;
  if (grid < 1) grid = 1;
  direct_rows_kernel<T><<<static_cast<int>(grid), 256, 0, s>>>(p);
  *launches += 1;
}

template void launch_direct<float>(const RowPlan<float>&, int, cudaStream_t, int*);
template void launch_direct<double>(const RowPlan<double>&, int, cudaStream_t, int*);

}  // namespace wsk
