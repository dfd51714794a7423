// Hash-bin rows: per-row shared-memory hash workspace with a monotone hash and
// sort-free ranking.
//
// Workspace.  Row i of C = A*B is the sum of the scaled rows A[i,k] * B[k,:]
// (Gustavson's algorithm, Sec. 5.1).  One thread team (one or more warps)
// owns the row, so the team's table is the private workspace w of the paper
// and the row's output segment is written by nobody else.  Inside the team,
// concurrent updates of one workspace entry use shared-memory atomics (the
// atomic-level protection of Sec. 4).
//
// Monotone hash.  Every product column of the row lies in [lo, hi] (B's rows
// are sorted).  The home slot of column c is
//     h(c) = floor((c - lo) * T / span),  span = hi - lo + 1,
// (h(c) = c - lo when span <= T), which never decreases as c grows.
// Symbolic pass: plain linear probing counts the distinct columns.  The set
// of occupied slots of a linear-probing table depends only on the keys'
// home slots, not on the insertion order or on which key of a run sits
// where, so the pass also checks the run structure the numeric pass will
// meet: a row whose probes wrap around the table (or, as a tuning limit,
// whose table holds a long run) is re-routed to the sorting path.
// Numeric pass: ordered linear probing -- an inserted key moves on past
// smaller keys and takes the place of the first larger one, which then moves
// on in its turn (a compare-and-swap per exchange, no wrap-around).  Keys
// only move forward and a slot's key only ever shrinks, so every run of
// occupied slots ends sorted and, with the monotone hash, so does the whole
// table: the output position of the key in slot s is the number of occupied
// slots before s, and the row is written in column order without a sort.
// Once every key is in place, each product finds its key's slot and adds
// its value there.
// Table sizes: bin b holds rows with at most 32 << b products whose home
// slots span 64 << b slots, so the load factor is at most 1/2.  The table
// has tail_slots() extra slots past the home range, so a run of keys that reaches
// the end of the home range continues upward instead of wrapping to slot 0.
// Teams: both passes use the same home range per bin; the numeric pass gives
// each (larger) pair table a team of more warps than the symbolic pass gives
// a key table (launch_bin).  A team fetches the headers of its next 32 rows
// (row, column range, A extent, and in the numeric pass C's extent) with one
// load per lane and hands them out by shuffles, so the per-row chain of
// dependent loads starts at the row's A entries.
#include <climits>
#include <type_traits>

#include "ws_internal.cuh"

namespace wsk {

namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr int kUnroll = 4;  // B entries a lane loads before inserting them
constexpr int kEmptyKey = -1;
// Slots past the home range: at least 64, and a multiple of 32 per warp so
// every warp of a row team ranks a whole number of 32-slot chunks.
__host__ __device__ constexpr int tail_slots(int wpr) { return 32 * (wpr > 2 ? wpr : 2); }

template <int WPR>
__device__ __forceinline__ void team_sync() {
  if constexpr (WPR == 1) {
    __syncwarp();
  } else {
    __syncthreads();
  }
}

// Inserts key c into the symbolic pass's key table.  Returns a bit set:
// kInsNew if the key was new, kInsWrapped if the probe wrapped from the last
// slot to slot 0, kInsFailed if every slot was probed.
constexpr int kInsNew = 1, kInsWrapped = 2, kInsFailed = 4;
__device__ __forceinline__ int probe_insert(int* keys, uint32_t h, uint32_t nslots, int c) {
  volatile int* vk = keys;
  int wrapped = 0;
  for (uint32_t n = 0; n < nslots; ++n) {
    int cur = vk[h];
    if (cur == kEmptyKey) {
      cur = atomicCAS(&keys[h], kEmptyKey, c);
      if (cur == kEmptyKey) return kInsNew | wrapped;
    }
    if (cur == c) return wrapped;
    if (++h == nslots) {
      h = 0;
      wrapped = kInsWrapped;
    }
  }
  return kInsFailed | wrapped;
}

// Numeric-pass slot: a column and its accumulated value in one word that a
// single compare-and-swap replaces (8 bytes for float, 16 for double).  The
// key sits in the low 32 bits; an empty slot has key -1 and value 0.
template <typename T>
struct PairSlot;
template <>
struct PairSlot<float> {
  using W = unsigned long long;
  static __device__ __forceinline__ W make(int c, float v) {
    return static_cast<W>(static_cast<uint32_t>(c)) | (static_cast<W>(__float_as_uint(v)) << 32);
  }
  static __device__ __forceinline__ int key(W w) { return static_cast<int>(static_cast<uint32_t>(w)); }
  static __device__ __forceinline__ float val(W w) { return __uint_as_float(static_cast<uint32_t>(w >> 32)); }
};
template <>
struct PairSlot<double> {
  using W = unsigned __int128;
  static __device__ __forceinline__ W make(int c, double v) {
    return static_cast<W>(static_cast<uint32_t>(c)) |
           (static_cast<W>(static_cast<unsigned long long>(__double_as_longlong(v))) << 64);
  }
  static __device__ __forceinline__ int key(W w) { return static_cast<int>(static_cast<uint32_t>(w)); }
  static __device__ __forceinline__ double val(W w) {
    return __longlong_as_double(static_cast<long long>(static_cast<unsigned long long>(w >> 64)));
  }
};

// Ordered insert of product (c, v) into the numeric pass's pair table:
// returns 0, or kInsFailed if a pair would move past the last slot.  The
// pair moves on past smaller keys; at the first larger key it takes that
// slot and carries the displaced pair (key and value together) on; at an
// empty slot it settles; at an equal key it adds its value there.  A slot's
// key only ever shrinks and keys only move forward, so every run of
// occupied slots stays sorted and no value is lost: a pair is either in the
// table or carried by exactly one thread, and a carried pair that meets its
// own key merges into it.  No wrap-around.
template <typename T>
__device__ __forceinline__ int ordered_insert_pair(typename PairSlot<T>::W* slots, uint32_t h, uint32_t nslots, int c, T v) {
  using P = PairSlot<T>;
  using W = typename P::W;
  W carry = P::make(c, v);
  // Every failed compare-and-swap follows a successful change of the slot by
  // another insert; the guard only bounds the loop for a broken table.
  for (uint32_t guard = 0; h < nslots && guard < 16u * nslots; ++guard) {
    const W cur = slots[h];
    const int kc = P::key(cur);
    const int kn = P::key(carry);
    W next;
    if (kc == kEmptyKey || kc > kn) {
      next = carry;
    } else if (kc == kn) {
      next = P::make(kn, P::val(cur) + P::val(carry));
    } else {
      ++h;
      continue;
    }
    if (atomicCAS(slots + h, cur, next) != cur) continue;  // the slot changed: look again
    if (kc == kEmptyKey || kc == kn) return 0;
    carry = cur;  // carry the displaced larger pair on
    ++h;
  }
  return kInsFailed;
}

// True if the table holds a run of more than `limit` occupied slots.  Called
// by one full warp; every lane returns the same value.
__device__ __forceinline__ bool has_long_run(const int* keys, int nslots, int limit, int lane) {
  int carry = 0;
  bool bad = false;
  for (int base = 0; base < nslots; base += 32) {
    const unsigned m = __ballot_sync(kFull, keys[base + lane] != kEmptyKey);
    if (m == kFull) {
      carry += 32;
      bad |= carry > limit;
    } else {
      bad |= carry + (__ffs(~m) - 1) > limit;
      if (limit < 31) {
        unsigned x = m;
        for (int j = 0; j < limit; ++j) x &= x >> 1;
        bad |= x != 0;
      }
      carry = __clz(~m);
    }
  }
  return bad;
}


// LOGT: log2 of table slots; WPR: warps per row team; RPC: row teams per CTA.
// The launch bounds let the compiler use up to 64 registers per thread.
template <typename T, int LOGT, int WPR, int RPC, bool NUMERIC>
__global__ void __launch_bounds__(32 * WPR * RPC, 1024 / (32 * WPR * RPC)) hash_rows_kernel(const RowPlan<T> p, const uint8_t my_cls) {
  static_assert(WPR == 1 || RPC == 1, "multi-warp row teams use the whole CTA");
  constexpr int kT = 1 << LOGT;        // home range
  constexpr int kS = kT + tail_slots(WPR);  // slots
  constexpr int kNT = 32 * WPR;
  extern __shared__ __align__(16) unsigned char smem_raw[];
  __shared__ int s_warp[WPR > 1 ? WPR : 1];
  __shared__ int s_flags;
  __shared__ long long s_b0[kNT * RPC], s_b1[kNT * RPC];  // staged B-row bounds of A entries
  __shared__ T s_a[kNT * RPC];                             // staged A values

  const int sub = threadIdx.x / kNT;
  const int t = threadIdx.x % kNT;
  const int lane = threadIdx.x & 31;
  const int warp = t >> 5;
  using PW = typename PairSlot<T>::W;
  // symbolic pass: keys; numeric pass: (key, value) pairs
  int* keys = reinterpret_cast<int*>(smem_raw) + sub * kS;
  PW* pairs = reinterpret_cast<PW*>(smem_raw) + sub * kS;

  const int lg = p.log2_group;
  const int gsize = 1 << lg;
  const int grp = t >> lg;
  const int gl = t & (gsize - 1);
  const int ngrp = kNT >> lg;

  const int64_t stride = static_cast<int64_t>(gridDim.x) * RPC;
  for (int64_t rb = static_cast<int64_t>(blockIdx.x) * RPC + sub; rb < p.seg_len; rb += 32 * stride) {
    // Row headers of a batch of 32 rows: lane l of every warp of the team
    // fetches row rb + l * stride, so the chain perm -> row bounds (and, in
    // the numeric pass, C's row extent) is waited for once per batch, not
    // once per row.  A row the symbolic pass re-routed to the sorting path
    // gets row -1 here.
    int32_t b_row = -1;
    int b_lo = 0, b_hi = 0, b_cnt = 0;
    long long b_ra = 0, b_re = 0, b_cb = 0;
    {
      const int64_t rr = rb + lane * stride;
      if (rr < p.seg_len) {
        const int32_t row = p.perm[p.seg_begin + rr];
        bool take = true;
        if constexpr (NUMERIC) take = p.cls[row] == my_cls;
        if (take) {
          b_row = row;
          b_lo = p.lo[row];
          b_hi = p.hi[row];
          b_ra = p.A.rowptr[row];
          b_re = p.A.rowptr[row + 1];
          if constexpr (NUMERIC) {
            b_cb = p.c_rowptr[row];
            const long long n = p.c_rowptr[row + 1] - b_cb;
            b_cnt = static_cast<int>(n < INT_MAX ? (n > 0 ? n : 0) : INT_MAX);  // a bad count fails the write check
          }
        }
      }
    }
    const int64_t left = (p.seg_len - rb + stride - 1) / stride;
    const int nb = left < 32 ? static_cast<int>(left) : 32;
    for (int jb = 0; jb < nb; ++jb) {
      const int32_t row = __shfl_sync(kFull, b_row, jb);
      if (row < 0) continue;  // the same rows in every warp of the team
      const int lo = __shfl_sync(kFull, b_lo, jb);
      const uint32_t span = static_cast<uint32_t>(__shfl_sync(kFull, b_hi, jb) - lo) + 1u;
      const int64_t ra = __shfl_sync(kFull, b_ra, jb), re = __shfl_sync(kFull, b_re, jb);
      const int64_t c_base = __shfl_sync(kFull, b_cb, jb);
      const int64_t c_cnt = __shfl_sync(kFull, b_cnt, jb);
      const bool ident = span <= static_cast<uint32_t>(kT);
      const unsigned long long mul = ident ? 0ull : ((static_cast<unsigned long long>(kT) << 32) / span);

      // Clear the workspace (w .= 0).
      {
        if constexpr (NUMERIC) {
          const PW empty = PairSlot<T>::make(kEmptyKey, T(0));
          for (int s = t; s < kS; s += kNT) pairs[s] = empty;
        } else {
          int4* k4 = reinterpret_cast<int4*>(keys);
          for (int s = t; s < kS / 4; s += kNT) k4[s] = make_int4(kEmptyKey, kEmptyKey, kEmptyKey, kEmptyKey);
        }
        if constexpr (WPR > 1) {
          if (t < WPR) s_warp[t] = 0;
          if (t == 0) s_flags = 0;
        }
      }
      team_sync<WPR>();

      // Accumulate: w[j] += A[i,k] * B[k,j] for every stored A[i,k], B[k,j].
      // The team first stages a chunk of the row's A entries (B-row bounds and
      // A values) in shared memory, then every group of gsize lanes walks B
      // rows, loading kUnroll B entries before it handles any of them.
      // Symbolic pass: one walk, plain probing.  Numeric pass: a walk that
      // places the keys (ordered probing), then a walk that adds the values.
      int my_new = 0, my_flags = 0;
      long long* st_b0 = s_b0 + sub * kNT;
      long long* st_b1 = s_b1 + sub * kNT;
      T* st_a = s_a + sub * kNT;
      auto home = [&](int c) -> uint32_t {
        const uint32_t d = static_cast<uint32_t>(c - lo);
        return ident ? d : static_cast<uint32_t>((static_cast<unsigned long long>(d) * mul) >> 32);
      };
      // Calls f(column, scaled value) for every product of the row this lane
      // owns (with_vals false: the value is not loaded and f gets 0).
      auto for_products = [&](auto with_vals, auto&& f) {
        constexpr bool kVals = NUMERIC && decltype(with_vals)::value;
        for (int64_t cb = ra; cb < re; cb += kNT) {
          const int n = static_cast<int>(min(static_cast<int64_t>(kNT), re - cb));
          if (t < n) {
            const int k = p.A.colidx[cb + t];
            st_b0[t] = p.B.rowptr[k];
            st_b1[t] = p.B.rowptr[k + 1];
            if constexpr (kVals) st_a[t] = p.A.vals[cb + t];
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
                const long long q = st_b0[j] + gl;
                if (q < st_b1[j]) {
                  cc[u] = p.B.colidx[q];
                  if constexpr (kVals) vv[u] = st_a[j] * p.B.vals[q];
                }
              }
            }
  #pragma unroll
            for (int u = 0; u < kUnroll; ++u) {
              if (cc[u] >= 0) f(cc[u], vv[u]);
            }
            // B rows longer than the group: the rest of each row.
  #pragma unroll 1
            for (int u = 0; u < kUnroll; ++u) {
              const int j = j0 + u * ngrp;
              if (j >= n) break;
              const long long qe = st_b1[j];
              for (long long q = st_b0[j] + gl + gsize; q < qe; q += gsize) {
                T v = T(0);
                if constexpr (kVals) v = st_a[j] * p.B.vals[q];
                f(p.B.colidx[q], v);
              }
            }
          }
          team_sync<WPR>();
        }
      };
      if constexpr (!NUMERIC) {
        for_products(std::false_type{}, [&](int c, T) {
          const int r = probe_insert(keys, home(c), kS, c);
          my_new += r & kInsNew;
          my_flags |= r;
        });
      } else {
        for_products(std::true_type{},
                     [&](int c, T v) { my_flags |= ordered_insert_pair<T>(pairs, home(c), kS, c, v); });
      }
      const bool wrapped = (my_flags & kInsWrapped) != 0;
      const bool failed = (my_flags & kInsFailed) != 0;

      if constexpr (!NUMERIC) {
        // Count the distinct columns, check the table for the ranking condition.
        int cnt = my_new;
  #pragma unroll
        for (int o = 16; o > 0; o >>= 1) cnt += __shfl_xor_sync(kFull, cnt, o);
        const int flags = (__any_sync(kFull, wrapped) ? 1 : 0) | (__any_sync(kFull, failed) ? 2 : 0);
        if constexpr (WPR > 1) {
          if (lane == 0) {
            atomicAdd(&s_warp[0], cnt);
            atomicOr(&s_flags, flags);
          }
        }
        team_sync<WPR>();
        if (warp == 0) {
          int total = cnt, fl = flags;
          if constexpr (WPR > 1) {
            total = s_warp[0];
            fl = s_flags;
          }
          const bool long_run = has_long_run(keys, kS, p.run_limit, lane);
          if (lane == 0) {
            p.c_rowptr[row + 1] = total;
            if (fl & 2) atomicOr(&p.sum->status, kErrProbe);
            if ((fl & 1) || long_run) {
              p.cls[row] = kClsSort;
              p.sort_list[atomicAdd(&p.sum->n_sort, 1)] = row;
            }
          }
        }
        team_sync<WPR>();
      } else {
        team_sync<WPR>();
        // Rank and write: each warp ranks a contiguous range of slots.
        constexpr int kPerWarp = kS / WPR;
        static_assert(kPerWarp % 32 == 0 && kPerWarp * WPR == kS, "whole chunks per warp");
        const int s_begin = warp * kPerWarp;
        int carry = 0;
        if constexpr (WPR > 1) {
          int occ = 0;
          for (int s = s_begin + lane; s < s_begin + kPerWarp; s += 32) occ += PairSlot<T>::key(pairs[s]) != kEmptyKey;
  #pragma unroll
          for (int o = 16; o > 0; o >>= 1) occ += __shfl_xor_sync(kFull, occ, o);
          if (lane == 0) s_warp[warp] = occ;
          team_sync<WPR>();
          for (int w = 0; w < warp; ++w) carry += s_warp[w];
        }
        const int64_t base = c_base;
        const int64_t cnt = c_cnt;
        bool count_err = false;
        for (int c0 = s_begin; c0 < s_begin + kPerWarp; c0 += 32) {
          const int s = c0 + lane;
          const PW pr = pairs[s];
          const int key = PairSlot<T>::key(pr);
          const bool occ = key != kEmptyKey;
          const unsigned m = __ballot_sync(kFull, occ);
          if (occ) {
            // The table is sorted: the key's position is the count of occupied slots before it.
            const int64_t pos = static_cast<int64_t>(carry) + __popc(m & ((1u << lane) - 1u));
            if (pos < cnt) {
              p.c_colidx[base + pos] = key;
              p.c_vals[base + pos] = PairSlot<T>::val(pr);
            } else {
              count_err = true;
            }
          }
          carry += __popc(m);
        }
        if (WPR == 1 || warp == WPR - 1) {
          if (carry != cnt) count_err = true;
        }
        if (__any_sync(kFull, count_err) && lane == 0) atomicOr(&p.sum->status, kErrCount);
        if (__any_sync(kFull, failed) && lane == 0) atomicOr(&p.sum->status, kErrProbe);
        team_sync<WPR>();
      }
    }
  }
}

template <typename T, int LOGT, int WPR, int RPC, bool NUMERIC>
void launch_pass(const RowPlan<T>& p, int bin, int num_sms, cudaStream_t s) {
  constexpr int kS = (1 << LOGT) + tail_slots(WPR);
  const size_t smem = static_cast<size_t>(RPC) * kS * (NUMERIC ? sizeof(typename PairSlot<T>::W) : sizeof(int));
  const int threads = 32 * WPR * RPC;
  auto kern = hash_rows_kernel<T, LOGT, WPR, RPC, NUMERIC>;
  static bool configured = false;
  if (!configured) {
    cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
    configured = true;
  }
  int per_sm = 0;
  cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, threads, smem);
  if (per_sm < 1) per_sm = 1;
  int64_t grid = (p.seg_len + RPC - 1) / RPC;
  const int64_t cap = static_cast<int64_t>(num_sms) * per_sm;
  if (grid > cap) grid = cap;
  if (grid < 1) grid = 1;
  kern<<<static_cast<int>(grid), threads, smem, s>>>(p, static_cast<uint8_t>(kClsHash0 + bin));
}

// Team shapes of a bin: the symbolic pass runs RPC_S teams of WPR_S warps
// per CTA over 4-byte key tables; the numeric pass's pair tables (8 or 16
// bytes a slot) leave room for only a few tables per SM, so there one table
// gets a team of WPR_N warps (one team per CTA): more loads in flight per
// row at the same shared memory.  The numeric table must have at least the
// symbolic table's slots: the symbolic pass vouches that no run of the row
// reaches past its last slot.
template <typename T, int LOGT, int WPR_S, int RPC_S, int WPR_N>
void launch_bin(const RowPlan<T>& p, bool numeric, int bin, int num_sms, cudaStream_t s) {
  static_assert(tail_slots(WPR_N) >= tail_slots(WPR_S), "numeric table smaller than the symbolic one");
  if (numeric) {
    launch_pass<T, LOGT, WPR_N, WPR_N == 1 ? RPC_S : 1, true>(p, bin, num_sms, s);
  } else {
    launch_pass<T, LOGT, WPR_S, RPC_S, false>(p, bin, num_sms, s);
  }
}

}  // namespace

template <typename T>
void launch_hash(const RowPlan<T>& p, int bin, bool numeric, int num_sms, cudaStream_t s, int* launches) {
  switch (bin) {
    case 0: launch_bin<T, 6, 1, 8, 1>(p, numeric, bin, num_sms, s); break;
    case 1: launch_bin<T, 7, 1, 8, 1>(p, numeric, bin, num_sms, s); break;
    case 2: launch_bin<T, 8, 1, 8, 1>(p, numeric, bin, num_sms, s); break;
    case 3: launch_bin<T, 9, 1, 8, 2>(p, numeric, bin, num_sms, s); break;
    case 4: launch_bin<T, 10, 1, 4, 2>(p, numeric, bin, num_sms, s); break;
    case 5: launch_bin<T, 11, 2, 1, 4>(p, numeric, bin, num_sms, s); break;
    case 6: launch_bin<T, 12, 4, 1, 8>(p, numeric, bin, num_sms, s); break;
    case 7: launch_bin<T, 13, 8, 1, 16>(p, numeric, bin, num_sms, s); break;
    default: return;
  }
  *launches += 1;
}

template void launch_hash<float>(const RowPlan<float>&, int, bool, int, cudaStream_t, int*);
template void launch_hash<double>(const RowPlan<double>&, int, bool, int, cudaStream_t, int*);

}  // namespace wsk
