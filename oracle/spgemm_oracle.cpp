// CPU oracle for sparse x sparse -> sparse matrix multiply (C = A*B, CSR).
//
// TEST INFRASTRUCTURE ONLY.  This file is the plain, slow, obviously correct
// reference that the CUDA path is checked against.  Only the test suite, the
// smoke check and the benchmark's CPU-baseline leg may load it.  It shares no
// code, header or constant with the CUDA library and includes nothing from it.
//
// What it computes (the definition of the product):
//   C[i, j] = sum over stored A[i, k] with (k, j) stored in B of A[i, k] * B[k, j]
// with the *structural* pattern {(i, j) : some stored A[i, k] meets a stored
// B[k, j]}.  An entry whose sum is exactly 0.0 is kept; stored zeros in A or B
// are structural.
//
// How (Gustavson's algorithm, Sec. 5.1, Fig. "SpGEMM implemented in
// WingSpan", written for rows of CSR instead of columns of CSC -- the
// row-wise product C[i,:] = sum_k A[i,k] B[k,:] is the same algorithm applied
// to C^T = B^T A^T):
//   for each output row i (the parallel loop; each row owns its fiber of C,
//   the shard argument of Sec. 5.1):
//       w := empty ordered map                       -- the workspace w .= 0
//       for each stored A[i, k] in ascending position:
//           for each stored B[k, j] in ascending position:
//               w[j] += A[i, k] * B[k, j]             -- first touch starts at 0
//       C[i, :] := w in ascending j                   -- C[i,j] = w[i] step
//   rowptr := exclusive prefix sum of |w| per row   -- CSR position invariant
//                                                      (Sec. 1, monotone prefix sums)
// Rows are split over threads in contiguous blocks following the static
// schedule rule of Sec. 4 (worker q of n takes a + floor((q-1)(b-a+1)/n) ..).
//
// Arithmetic: every value is widened to double and accumulated in double
// (the paper's element type is Float64).  The file must be compiled with
// -ffp-contract=off so the sums follow the sequential order above exactly.
//
// Besides C the oracle returns, per output entry, absmass = sum |A[i,k]*B[k,j]|,
// the magnitude against which summation-order differences are judged.

#include <cstdint>
#include <cstdlib>
#include <cmath>
#include <map>
#include <new>
#include <thread>
#include <vector>

namespace {

struct Entry {
  double val;
  double absmass;
};

struct RowResult {
  std::vector<int32_t> col;
  std::vector<double> val;
  std::vector<double> absmass;
};

struct OracleResult {
  int64_t nrows = 0;
  std::vector<int64_t> rowptr;
  std::vector<RowResult> rows;
};

void one_row(int64_t i, const int64_t* rpA, const int32_t* ciA, const double* vA,
             const int64_t* rpB, const int32_t* ciB, const double* vB, RowResult& out) {
  std::map<int32_t, Entry> w;
  for (int64_t p = rpA[i]; p < rpA[i + 1]; ++p) {
    const int32_t k = ciA[p];
    const double a = vA[p];
    for (int64_t q = rpB[k]; q < rpB[k + 1]; ++q) {
      const double prod = a * vB[q];
      Entry& e = w[ciB[q]];  // value-initialised to {0, 0} on first touch
      e.val = e.val + prod;
      e.absmass = e.absmass + std::fabs(prod);
    }
  }
  out.col.reserve(w.size());
  out.val.reserve(w.size());
  out.absmass.reserve(w.size());
  for (const auto& kv : w) {
    out.col.push_back(kv.first);
    out.val.push_back(kv.second.val);
    out.absmass.push_back(kv.second.absmass);
  }
}

}  // namespace

extern "C" {

// Computes rows `rows[0..nsel)` of C = A*B (all m rows when rows == NULL).
// A is m x k and B is k x n, both CSR with int64 row pointers, int32 column
// indices and double values.  Returns an opaque result (NULL on allocation
// failure) and stores the number of output entries in *nnz_out.
// The caller releases the result with oracle_result_free.
void* oracle_spgemm(int64_t m, int64_t k, int64_t n, const int64_t* rpA, const int32_t* ciA,
                    const double* vA, const int64_t* rpB, const int32_t* ciB, const double* vB,
                    const int64_t* rows, int64_t nsel, int nthreads, int64_t* nnz_out) {
  (void)k;
  (void)n;
  OracleResult* res = new (std::nothrow) OracleResult;
  if (!res) return nullptr;
  const int64_t nr = rows ? nsel : m;
  res->nrows = nr;
  try {
    res->rows.resize(static_cast<size_t>(nr));
    res->rowptr.assign(static_cast<size_t>(nr) + 1, 0);
  } catch (...) {
    delete res;
    return nullptr;
  }
  int nt = nthreads > 0 ? nthreads : 1;
  if (nr < nt) nt = nr > 0 ? static_cast<int>(nr) : 1;
  auto work = [&](int q) {  // static schedule: contiguous block per worker
    const int64_t lo = (static_cast<int64_t>(q) * nr) / nt;
    const int64_t hi = (static_cast<int64_t>(q + 1) * nr) / nt;
    for (int64_t t = lo; t < hi; ++t) {
      const int64_t i = rows ? rows[t] : t;
      one_row(i, rpA, ciA, vA, rpB, ciB, vB, res->rows[static_cast<size_t>(t)]);
    }
  };
  if (nt == 1) {
    work(0);
  } else {
    std::vector<std::thread> pool;
    pool.reserve(static_cast<size_t>(nt));
    for (int q = 0; q < nt; ++q) pool.emplace_back(work, q);
    for (auto& th : pool) th.join();
  }
  // Exclusive prefix sum of the per-row counts, serially.
  for (int64_t t = 0; t < nr; ++t)
    res->rowptr[static_cast<size_t>(t) + 1] =
        res->rowptr[static_cast<size_t>(t)] + static_cast<int64_t>(res->rows[static_cast<size_t>(t)].col.size());
  *nnz_out = res->rowptr[static_cast<size_t>(nr)];
  return res;
}

// Copies the result into caller-owned arrays: rowptr[nrows+1], colidx[nnz],
// vals[nnz], absmass[nnz] (any of the last three may be NULL).  Returns 0.
int oracle_result_copy(void* handle, int64_t* rowptr, int32_t* colidx, double* vals, double* absmass) {
  const OracleResult* res = static_cast<const OracleResult*>(handle);
  if (!res) return -1;
  for (size_t t = 0; t < res->rowptr.size(); ++t) rowptr[t] = res->rowptr[t];
  for (int64_t t = 0; t < res->nrows; ++t) {
    const RowResult& r = res->rows[static_cast<size_t>(t)];
    const int64_t base = res->rowptr[static_cast<size_t>(t)];
    for (size_t e = 0; e < r.col.size(); ++e) {
      if (colidx) colidx[base + static_cast<int64_t>(e)] = r.col[e];
      if (vals) vals[base + static_cast<int64_t>(e)] = r.val[e];
      if (absmass) absmass[base + static_cast<int64_t>(e)] = r.absmass[e];
    }
  }
  return 0;
}

void oracle_result_free(void* handle) { delete static_cast<OracleResult*>(handle); }

}  // extern "C"
