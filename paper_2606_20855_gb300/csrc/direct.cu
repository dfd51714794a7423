// Direct rows: a row of A with exactly one stored entry A[i,k] gives
// C[i,:] = A[i,k] * B[k,:] (Gustavson's accumulation with a single term, Sec. 5.1).
// B[k,:] is already sorted and duplicate-free, so the row is a scaled copy
// and needs no workspace.  A group of 2^log2_group lanes copies one row with
// coalesced loads and stores.
#include "ws_internal.cuh"

namespace wsk {

namespace {

template <typename T>
__global__ void __launch_bounds__(256) direct_rows_kernel(const RowPlan<T> p) {
  const int lg = p.log2_group;
  const int gsize = 1 << lg;
  const int gl = threadIdx.x & (gsize - 1);
  const int64_t groups = (static_cast<int64_t>(gridDim.x) * blockDim.x) >> lg;
  for (int64_t r = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> lg; r < p.seg_len;
       r += groups) {
    const int32_t row = p.perm[p.seg_begin + r];
    const int64_t pa = p.A.rowptr[row];
    const int k = p.A.colidx[pa];
    const T a = p.A.vals[pa];
    const int64_t qb = p.B.rowptr[k];
    const int64_t len = p.B.rowptr[k + 1] - qb;
    const int64_t base = p.c_rowptr[row];
    if (len != p.c_rowptr[row + 1] - base) {
      if (gl == 0) atomicOr(&p.sum->status, kErrCount);
      continue;
    }
    for (int64_t t = gl; t < len; t += gsize) {
      p.c_colidx[base + t] = p.B.colidx[qb + t];
      p.c_vals[base + t] = a * p.B.vals[qb + t];
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
