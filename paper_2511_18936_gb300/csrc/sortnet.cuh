// Sorting networks over a register array, for one thread that holds one
// vector's magnitude keys (the per-vector top-k of Section 3.2, taken in
// bulk).  Every index is a template argument, so the array stays in registers.
//
//   sort_oe<LO, N, DESC>  Batcher's odd-even merge sort of v[LO .. LO+N)
//                         (N a power of two), decreasing if DESC
//   top_half_desc         v[0..64) := the 64 largest of v[0..128), decreasing,
//                         given v[0..64) decreasing and v[64..128) increasing
//   merge_desc<LO, N>     bitonic merge of the bitonic run v[LO .. LO+N) into
//                         decreasing order
//   top64_of128_desc,     the same top-64 and full sort of 128 keys in one
//   sort128_desc_full     thread.  The bulk append splits a vector over a lane
//                         pair instead (append.cu), built from sort_oe and
//                         merge_desc; the host test checks these one-thread
//                         forms, and with them those building blocks.
//
// A compare-exchange takes the larger key with one max.  The smaller is
// either one min or, for three comparators in five, (a + b) - max: exact in
// 32-bit modular arithmetic, and written as two multiply-adds by `one` (the
// value 1, supplied at run time so that the compiler cannot fold the
// multiplications away).  Min and max share one integer pipe, the
// multiply-adds use another, and the mix raises the rate of compare-exchanges
// on sm_103a by about a third.
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

// the smaller of a and b, given hi = max(a, b)
template <bool SUM>
SWAN_SORT_FN uint32_t lower_of(uint32_t a, uint32_t b, uint32_t hi, uint32_t one) {
  if constexpr (SUM) return (a * one + b) - hi * one;
  else return umin(a, b);
}

// the larger key to position A if DESC, else to position B
template <int A, int B, bool DESC, int M>
SWAN_SORT_FN void cx(uint32_t (&v)[M], uint32_t one) {
  static_assert(0 <= A && A < B && B < M, "compare-exchange out of range");
  const uint32_t hi = umax(v[A], v[B]);
  const uint32_t lo = lower_of<(A % 5) >= 2>(v[A], v[B], hi, one);
  v[A] = DESC ? hi : lo;
  v[B] = DESC ? lo : hi;
}

// compare-exchange (I, I+R) for I = FIRST, FIRST+STEP, ... while I+R < END
template <int I, int END, int R, int STEP, bool DESC, int M>
SWAN_SORT_FN void cx_run(uint32_t (&v)[M], uint32_t one) {
  if constexpr (I + R < END) {
    cx<I, I + R, DESC>(v, one);
    cx_run<I + STEP, END, R, STEP, DESC>(v, one);
  }
}

// Odd-even merge of the elements LO, LO+R, LO+2R, ... below LO+N, whose two
// halves (by position in that subsequence) are each sorted.
template <int LO, int N, int R, bool DESC, int M>
SWAN_SORT_FN void merge_oe(uint32_t (&v)[M], uint32_t one) {
  constexpr int step = 2 * R;
  if constexpr (step < N) {
    merge_oe<LO, N, step, DESC>(v, one);      // even-position subsequence
    merge_oe<LO + R, N, step, DESC>(v, one);  // odd-position subsequence
    cx_run<LO + R, LO + N, R, step, DESC>(v, one);
  } else {
    cx<LO, LO + R, DESC>(v, one);
  }
}

template <int LO, int N, bool DESC, int M>
SWAN_SORT_FN void sort_oe(uint32_t (&v)[M], uint32_t one) {
  if constexpr (N > 1) {
    sort_oe<LO, N / 2, DESC>(v, one);
    sort_oe<LO + N / 2, N / 2, DESC>(v, one);
    merge_oe<LO, N, 1, DESC>(v, one);
  }
}

// one half-cleaner step of a bitonic merge: (I, I+J) for the I in
// [LO, LO+N) with bit J clear, larger key to I
template <int I, int LO, int N, int J, int M>
SWAN_SORT_FN void half_clean(uint32_t (&v)[M], uint32_t one) {
  if constexpr (I < LO + N) {
    if constexpr (((I - LO) & J) == 0) cx<I, I + J, true>(v, one);
    half_clean<I + 1, LO, N, J, M>(v, one);
  }
}

template <int LO, int N, int J, int M>
SWAN_SORT_FN void merge_steps(uint32_t (&v)[M], uint32_t one) {
  if constexpr (J >= 1) {
    half_clean<LO, LO, N, J, M>(v, one);
    merge_steps<LO, N, J / 2>(v, one);
  }
}

template <int LO, int N, int M>
SWAN_SORT_FN void merge_desc(uint32_t (&v)[M], uint32_t one) {
  merge_steps<LO, N, N / 2>(v, one);
}

// v[0..64) decreasing and v[64..128) increasing form one bitonic run; its
// first half-cleaner leaves the 64 largest in v[0..64), a bitonic run again
template <int I = 0>
SWAN_SORT_FN void top_half_desc(uint32_t (&v)[128], uint32_t one) {
  if constexpr (I < 64) {
    v[I] = umax(v[I], v[I + 64]);
    top_half_desc<I + 1>(v, one);
  } else {
    merge_desc<0, 64>(v, one);
  }
}

// All 128 keys, decreasing.
SWAN_SORT_FN void sort128_desc_full(uint32_t (&v)[128], uint32_t one) {
  sort_oe<0, 64, true>(v, one);
  sort_oe<64, 64, false>(v, one);
  merge_desc<0, 128>(v, one);
}

// The 64 largest of 128 keys, decreasing, in v[0..64) (v[64..128) undefined).
SWAN_SORT_FN void top64_of128_desc(uint32_t (&v)[128], uint32_t one) {
  sort_oe<0, 64, true>(v, one);
  sort_oe<64, 64, false>(v, one);
  top_half_desc(v, one);
}

}  // namespace sortnet
}  // namespace swan
