// Sorting networks over a register array, for one thread that holds one
// vector's 128 magnitude keys (the per-vector top-k of Section 3.2, taken in
// bulk).  Every index is a template argument, so the array stays in registers
// and each compare-exchange is one max and one min.
//
//   sort_oe<LO, N, DESC>  Batcher's odd-even merge sort of v[LO .. LO+N)
//                         (N a power of two), decreasing if DESC
//   top_half_desc         v[0..64) := the 64 largest of v[0..128), decreasing,
//                         given v[0..64) decreasing and v[64..128) increasing
//   merge_desc<LO, N>     bitonic merge of the bitonic run v[LO .. LO+N) into
//                         decreasing order
//
// The header compiles as plain C++ too (the host test of the networks).
#pragma once

#include <stdint.h>

#if defined(__CUDACC__)
#define SWAN_SORT_FN __host__ __device__ __forceinline__
#else
#define SWAN_SORT_FN inline
#endif

namespace swan {
namespace sortnet {

SWAN_SORT_FN uint32_t umax(uint32_t a, uint32_t b) { return a > b ? a : b; }
SWAN_SORT_FN uint32_t umin(uint32_t a, uint32_t b) { return a > b ? b : a; }

// the larger key to position A if DESC, else to position B
template <int A, int B, bool DESC, int M>
SWAN_SORT_FN void cx(uint32_t (&v)[M]) {
  static_assert(0 <= A && A < B && B < M, "compare-exchange out of range");
  const uint32_t hi = umax(v[A], v[B]), lo = umin(v[A], v[B]);
  v[A] = DESC ? hi : lo;
  v[B] = DESC ? lo : hi;
}

// compare-exchange (I, I+R) for I = FIRST, FIRST+STEP, ... while I+R < END
template <int I, int END, int R, int STEP, bool DESC, int M>
SWAN_SORT_FN void cx_run(uint32_t (&v)[M]) {
  if constexpr (I + R < END) {
    cx<I, I + R, DESC>(v);
    cx_run<I + STEP, END, R, STEP, DESC>(v);
  }
}

// Odd-even merge of the elements LO, LO+R, LO+2R, ... below LO+N, whose two
// halves (by position in that subsequence) are each sorted.
template <int LO, int N, int R, bool DESC, int M>
SWAN_SORT_FN void merge_oe(uint32_t (&v)[M]) {
  constexpr int step = 2 * R;
  if constexpr (step < N) {
    merge_oe<LO, N, step, DESC>(v);      // even-position subsequence
    merge_oe<LO + R, N, step, DESC>(v);  // odd-position subsequence
    cx_run<LO + R, LO + N, R, step, DESC>(v);
  } else {
    cx<LO, LO + R, DESC>(v);
  }
}

template <int LO, int N, bool DESC, int M>
SWAN_SORT_FN void sort_oe(uint32_t (&v)[M]) {
  if constexpr (N > 1) {
    sort_oe<LO, N / 2, DESC>(v);
    sort_oe<LO + N / 2, N / 2, DESC>(v);
    merge_oe<LO, N, 1, DESC>(v);
  }
}

// one half-cleaner step of a bitonic merge: (I, I+J) for the I in
// [LO, LO+N) with bit J clear, larger key to I
template <int I, int LO, int N, int J, int M>
SWAN_SORT_FN void half_clean(uint32_t (&v)[M]) {
  if constexpr (I < LO + N) {
    if constexpr (((I - LO) & J) == 0) cx<I, I + J, true>(v);
    half_clean<I + 1, LO, N, J, M>(v);
  }
}

template <int LO, int N, int J, int M>
SWAN_SORT_FN void merge_steps(uint32_t (&v)[M]) {
  if constexpr (J >= 1) {
    half_clean<LO, LO, N, J, M>(v);
    merge_steps<LO, N, J / 2>(v);
  }
}

template <int LO, int N, int M>
SWAN_SORT_FN void merge_desc(uint32_t (&v)[M]) {
  merge_steps<LO, N, N / 2>(v);
}

// v[0..64) decreasing and v[64..128) increasing form one bitonic run; its
// first half-cleaner leaves the 64 largest in v[0..64), a bitonic run again
template <int I = 0>
SWAN_SORT_FN void top_half_desc(uint32_t (&v)[128]) {
  if constexpr (I < 64) {
    v[I] = umax(v[I], v[I + 64]);
    top_half_desc<I + 1>(v);
  } else {
    merge_desc<0, 64>(v);
  }
}

// All 128 keys, decreasing.
SWAN_SORT_FN void sort128_desc_full(uint32_t (&v)[128]) {
  sort_oe<0, 64, true>(v);
  sort_oe<64, 64, false>(v);
  merge_desc<0, 128>(v);
}

// The 64 largest of 128 keys, decreasing, in v[0..64) (v[64..128) undefined).
SWAN_SORT_FN void top64_of128_desc(uint32_t (&v)[128]) {
  sort_oe<0, 64, true>(v);
  sort_oe<64, 64, false>(v);
  top_half_desc(v);
}

}  // namespace sortnet
}  // namespace swan
