// Device code of the decode kernels (Algorithm 1, attention part; Section
// 4.3): the split decode with the fused combine and rotate-back (Appendix
// A.1, Lemma 2) for one query head per kv head, and the helpers the
// grouped-query kernel (decode_mma.cuh) shares.  Included through
// decode_mma.cuh by decode.cu, which holds the query rotation, the
// empty-cache combine and the host launchers; the committed profiles name
// the hash of every kernel file their kernel is built from.
#pragma once

#include <cuda_fp8.h>

#include <type_traits>

#include "swan_internal.h"

namespace swan {
namespace {

// Streaming loads of cache records.  With one query head per kv head nothing
// is re-read, so the records bypass L1; with head pairs split over two lanes
// the two lanes of a token read the same record in one instruction.
template <bool kL1>
__device__ __forceinline__ uint4 ld_rec16(const void* ptr) {
  uint4 r;
  if (kL1)
    asm("ld.global.nc.v4.u32 {%0,%1,%2,%3}, [%4];"
        : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w) : "l"(ptr));
  else
    asm("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
        : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w) : "l"(ptr));
  return r;
}
template <bool kL1>
__device__ __forceinline__ uint2 ld_rec8(const void* ptr) {
  uint2 r;
  if (kL1)
    asm("ld.global.nc.v2.u32 {%0,%1}, [%2];" : "=r"(r.x), "=r"(r.y) : "l"(ptr));
  else
    asm("ld.global.nc.L1::no_allocate.v2.u32 {%0,%1}, [%2];" : "=r"(r.x), "=r"(r.y) : "l"(ptr));
  return r;
}

__device__ __forceinline__ float2 h2f(uint32_t w) {
  return __half22float2(*reinterpret_cast<const __half2*>(&w));
}

// Two E4M3 values (low 16 bits of w, or the high 16 bits) to fp32.
__device__ __forceinline__ float2 e4m3x2_to_f2(uint32_t w, bool hi) {
  const __nv_fp8x2_storage_t pair = (__nv_fp8x2_storage_t)(hi ? (w >> 16) : (w & 0xffffu));
  const __half2_raw h = __nv_cvt_fp8x2_to_halfraw2(pair, __NV_E4M3);
  return __half22float2(*reinterpret_cast<const __half2*>(&h));
}

// ---------------------------------------------------------------------------
// One 8-entry chunk of a cached vector, per value format:
//   fp16: a 16-byte record of 8 fp16 values and an 8-byte record of indices;
//   fp8:  one 16-byte record: 8 E4M3 values, then 8 indices.
// ---------------------------------------------------------------------------
template <int FMT>
struct Chunk;
template <>
struct Chunk<kFmtFp16> {
  uint4 v;
  uint2 i;
};
template <>
struct Chunk<kFmtFp8> {
  uint4 r;
};

// vb: this lane's 16-byte record run, ib: its 8-byte index run (fp16 only)
template <int FMT, bool kL1>
__device__ __forceinline__ Chunk<FMT> load_chunk(const uint8_t* vb, const uint8_t* ib, int c) {
  Chunk<FMT> ch;
  if constexpr (FMT == kFmtFp16) {
    ch.v = ld_rec16<kL1>(vb + c * 512);
    ch.i = ld_rec8<kL1>(ib + c * 256);
  } else {
    ch.r = ld_rec16<kL1>(vb + c * 512);
  }
  return ch;
}
template <int FMT>
__device__ __forceinline__ uint2 chunk_idx(const Chunk<FMT>& ch) {
  if constexpr (FMT == kFmtFp16)
    return ch.i;
  else
    return make_uint2(ch.r.z, ch.r.w);
}
template <int FMT>
__device__ __forceinline__ void chunk_vals(const Chunk<FMT>& ch, float (&f)[8]) {
  float2 a, b, c, d;
  if constexpr (FMT == kFmtFp16) {
    a = h2f(ch.v.x), b = h2f(ch.v.y), c = h2f(ch.v.z), d = h2f(ch.v.w);
  } else {
    a = e4m3x2_to_f2(ch.r.x, false), b = e4m3x2_to_f2(ch.r.x, true);
    c = e4m3x2_to_f2(ch.r.y, false), d = e4m3x2_to_f2(ch.r.y, true);
  }
  f[0] = a.x, f[1] = a.y, f[2] = b.x, f[3] = b.y, f[4] = c.x, f[5] = c.y, f[6] = d.x, f[7] = d.y;
}
__device__ __forceinline__ void keep_first(float (&f)[8], int n) {
#pragma unroll
  for (int e = 0; e < 8; ++e) f[e] = (e < n) ? f[e] : 0.f;
}

// Exact maximum over the warp in one reduction: floats compare as their
// bits for v >= 0 and as bits ^ 0x7fffffff below zero (an order-preserving
// map to int32 that is its own inverse).
__device__ __forceinline__ float warp_max(float v) {
  const int i = __float_as_int(v);
  const int m = __reduce_max_sync(0xffffffffu, i >= 0 ? i : (i ^ 0x7fffffff));
  return __int_as_float(m >= 0 ? m : (m ^ 0x7fffffff));
}
// 2^x by the hardware approximation (relative error ~2^-22; results below
// 2^-126 flush to zero, negligible next to the running maximum's 1).
__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Shared-memory accesses by 32-bit shared-window address.  They are volatile
// so that they keep their program order among themselves: each chunk's eight
// loads are issued back to back, then its eight stores (the indices of one
// vector are distinct, so the batch never aliases).
__device__ __forceinline__ float lds(uint32_t a) {
  float v;
  asm volatile("ld.shared.f32 %0, [%1];" : "=f"(v) : "r"(a));
  return v;
}
__device__ __forceinline__ void sts(uint32_t a, float v) {
  asm volatile("st.shared.f32 [%0], %1;" ::"r"(a), "f"(v));
}
__device__ __forceinline__ float2 lds2(uint32_t a) {
  float2 v;
  asm volatile("ld.shared.v2.f32 {%0,%1}, [%2];" : "=f"(v.x), "=f"(v.y) : "r"(a));
  return v;
}

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_group 0;" ::: "memory"); }

// Ask the memory system to bring `bytes` (a multiple of 16, 16-byte aligned)
// into L2 ahead of the loads that will read them.
__device__ __forceinline__ void prefetch_l2(const void* ptr, uint32_t bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(ptr), "r"(bytes) : "memory");
}

// ---------------------------------------------------------------------------
// One query head per kv head: lane = token, lane-private accumulators.
// ---------------------------------------------------------------------------

// Address of coordinate idx (byte e of the index word w) in a [128][R]
// lane-interleaved fp32 array (R = 32 for the accumulators, 16 for q'), row
// 2^SH = 4R bytes, base aligned to 128 rows: base | (idx & 127) << SH |
// (lane % R) << 2.  One shift and one LOP3.  With R = 32 the 32 lanes
// gathering arbitrary coordinates hit 32 distinct banks; with R = 16 lanes
// l and l + 16 share a copy (two wavefronts when their coordinates differ
// but have the same parity).  Any index byte stays inside the array.
template <int E, int SH = 7>
__device__ __forceinline__ uint32_t addr_of(uint32_t w, uint32_t base) {
  constexpr uint32_t mask = 0x7fu << SH;
  constexpr int sh = SH - 8 * E;  // where byte e's low bit goes
  if constexpr (sh >= 0) return ((w << sh) & mask) | base;
  else return ((w >> -sh) & mask) | base;
}

// q' of the one-head kernel: 2^QS / 4 copies of each coordinate, rows of
// 2^QS bytes, aligned to their 128-row size: 16 copies (8 KB) where two CTAs
// share an SM, 32 (16 KB, conflict-free) where one CTA has the SM.

// Two fp32 fused multiply-adds in one instruction (d = a * b + c per half).
__device__ __forceinline__ float2 ffma2(float2 a, float2 b, float2 c) {
  unsigned long long ra, rb, rc, rd;
  asm("mov.b64 %0, {%1,%2};" : "=l"(ra) : "f"(a.x), "f"(a.y));
  asm("mov.b64 %0, {%1,%2};" : "=l"(rb) : "f"(b.x), "f"(b.y));
  asm("mov.b64 %0, {%1,%2};" : "=l"(rc) : "f"(c.x), "f"(c.y));
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(rd) : "l"(ra), "l"(rb), "l"(rc));
  float2 d;
  asm("mov.b64 {%0,%1}, %2;" : "=f"(d.x), "=f"(d.y) : "l"(rd));
  return d;
}

// Score contribution of one chunk into four partial sums.
template <int QS>
__device__ __forceinline__ void score_chunk(uint32_t qb, const float (&f)[8], uint2 ix, float (&s)[4]) {
  constexpr int Q = QS;
  const float q0 = lds(addr_of<0, Q>(ix.x, qb)), q1 = lds(addr_of<1, Q>(ix.x, qb));
  const float q2 = lds(addr_of<2, Q>(ix.x, qb)), q3 = lds(addr_of<3, Q>(ix.x, qb));
  const float q4 = lds(addr_of<0, Q>(ix.y, qb)), q5 = lds(addr_of<1, Q>(ix.y, qb));
  const float q6 = lds(addr_of<2, Q>(ix.y, qb)), q7 = lds(addr_of<3, Q>(ix.y, qb));
  float2 s01 = make_float2(s[0], s[1]), s23 = make_float2(s[2], s[3]);
  s01 = ffma2(make_float2(q0, q1), make_float2(f[0], f[1]), s01);
  s23 = ffma2(make_float2(q2, q3), make_float2(f[2], f[3]), s23);
  s01 = ffma2(make_float2(q4, q5), make_float2(f[4], f[5]), s01);
  s23 = ffma2(make_float2(q6, q7), make_float2(f[6], f[7]), s23);
  s[0] = s01.x, s[1] = s01.y, s[2] = s23.x, s[3] = s23.y;
}

// acc[idx_e] += p * val_e for one full chunk (distinct indices): eight loads,
// eight FMAs, eight stores.
__device__ __forceinline__ void value_chunk(uint32_t ab, float p, const float (&f)[8], uint2 ix) {
  const uint32_t a0 = addr_of<0>(ix.x, ab), a1 = addr_of<1>(ix.x, ab);
  const uint32_t a2 = addr_of<2>(ix.x, ab), a3 = addr_of<3>(ix.x, ab);
  const uint32_t a4 = addr_of<0>(ix.y, ab), a5 = addr_of<1>(ix.y, ab);
  const uint32_t a6 = addr_of<2>(ix.y, ab), a7 = addr_of<3>(ix.y, ab);
  const float o0 = lds(a0), o1 = lds(a1), o2 = lds(a2), o3 = lds(a3);
  const float o4 = lds(a4), o5 = lds(a5), o6 = lds(a6), o7 = lds(a7);
  const float2 pp = make_float2(p, p);
  const float2 r01 = ffma2(pp, make_float2(f[0], f[1]), make_float2(o0, o1));
  const float2 r23 = ffma2(pp, make_float2(f[2], f[3]), make_float2(o2, o3));
  const float2 r45 = ffma2(pp, make_float2(f[4], f[5]), make_float2(o4, o5));
  const float2 r67 = ffma2(pp, make_float2(f[6], f[7]), make_float2(o6, o7));
  sts(a0, r01.x);
  sts(a1, r01.y);
  sts(a2, r23.x);
  sts(a3, r23.y);
  sts(a4, r45.x);
  sts(a5, r45.y);
  sts(a6, r67.x);
  sts(a7, r67.y);
}

// The first `n` (< 8) entries of a chunk, one read-modify-write at a time
// (the tail of a runtime keep count that is not a multiple of 8).
__device__ __forceinline__ void value_chunk_partial(uint32_t ab, float p, const float (&f)[8], uint2 ix,
                                                    int n) {
#pragma unroll
  for (int e = 0; e < 7; ++e) {
    if (e < n) {
      const uint32_t w = e < 4 ? ix.x : ix.y;
      const uint32_t a = ((w >> (8u * (e & 3))) & 0x7fu) << 7 | ab;
      sts(a, fmaf(p, f[e], lds(a)));
    }
  }
}

constexpr uint32_t kRegionBytes = kHeadDim * 32 * sizeof(float);  // 16 KB

// Geometry of unit u's groups in the flat split: its first group `goff`,
// its group count and lengths; uniform rows read the scalars, ragged rows
// their SeqInfo entry.
struct UnitView {
  int64_t goff, N_g, sparse_len;
  int n_sg, n_b, buf_start;
};
__device__ __forceinline__ UnitView unit_view(const DecodeParams& p, int64_t u) {
  UnitView v;
  if (p.seq == nullptr) {
    v.goff = u * p.N_g;
    v.N_g = p.N_g;
    v.sparse_len = p.sparse_len;
    v.n_sg = (int)p.n_sg;
    v.n_b = p.n_b;
    v.buf_start = p.buf_start;
  } else {
    const int64_t b = u / p.H_kv, h = u - b * p.H_kv;
    const SeqInfo& q = p.seq[b];
    v.sparse_len = q.sparse_len;
    v.n_sg = (int)((q.sparse_len + 31) >> 5);
    v.n_b = q.n_b;
    v.buf_start = q.buf_start;
    v.N_g = row_groups(q.sparse_len, q.n_b);
    v.goff = q.group_prefix * p.H_kv + h * v.N_g;
  }
  return v;
}
// The unit that holds flat group g (0 <= g < total_groups).
__device__ __forceinline__ int64_t unit_of(const DecodeParams& p, int64_t g) {
  if (p.seq == nullptr) return g / p.N_g;
  int lo = 0, hi = p.B - 1;  // the last row whose first group is <= g
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (p.seq[mid].group_prefix * p.H_kv <= g) lo = mid;
    else hi = mid - 1;
  }
  const SeqInfo& q = p.seq[lo];
  const int64_t ng = row_groups(q.sparse_len, q.n_b);
  const int64_t h = min((int64_t)p.H_kv - 1, (g - q.group_prefix * p.H_kv) / ng);
  return (int64_t)lo * p.H_kv + h;
}
// Split of a segment [s0, s1) of a unit's groups (the first n_sg sparse,
// the rest dense-buffer groups, which cost about kBufferGroupCost sparse
// groups: 512 instead of 384 bytes and twice the shared-memory work per
// token, set by measurement) into `parts` contiguous runs of equal cost;
// returns where run
// `part` starts (part == parts gives s1).
constexpr int kBufferGroupCost = 3;
__device__ __forceinline__ int split_at(int s0, int s1, int n_sg, int part, int parts) {
  const int sp_in = max(0, min(s1, n_sg) - s0);
  const int bf_in = (s1 - s0) - sp_in;
  const int cost = sp_in + kBufferGroupCost * bf_in;
  const int c = (int)(((int64_t)cost * part) / parts);
  return c <= sp_in ? s0 + c : s0 + sp_in + (c - sp_in + kBufferGroupCost - 1) / kBufferGroupCost;
}

// First group of CTA c (c <= gridDim.x) and the CTA that holds group g.
// Ragged rows: the host's table.  Uniform rows: unit u's groups take cost
// positions [u U, u U + N_g) with U = N_g + V, and V positions follow each
// unit but the last (the extra visit a CTA crossing into the next unit
// pays); CTA c starts at cost x_c = floor(c T / grid), T = units U - V, at
// the first group at or after x_c.  Group g (unit u, offset o) sits at
// y = u U + o, and cta_begin(c) <= g exactly when x_c <= y, so the CTA
// holding g is the last c with x_c <= y: floor(((y + 1) grid - 1) / T).
__device__ __forceinline__ int64_t cta_begin(const DecodeParams& p, int64_t c) {
  if (p.cta_start != nullptr) return p.cta_start[c];
  const int64_t U = p.N_g + p.visit_cost;
  const int64_t T = (p.total_groups / p.N_g) * U - p.visit_cost;
  const int64_t x = c * T / (int64_t)gridDim.x;
  const int64_t u = x / U;
  return u * p.N_g + min(x - u * U, p.N_g);
}
__device__ __forceinline__ int64_t cta_of(const DecodeParams& p, int64_t g) {
  if (p.cta_start == nullptr) {
    const int64_t U = p.N_g + p.visit_cost;
    const int64_t u = g / p.N_g;
    const int64_t y = u * U + (g - u * p.N_g);
    const int64_t T = (p.total_groups / p.N_g) * U - p.visit_cost;
    return min((int64_t)gridDim.x - 1, ((y + 1) * (int64_t)gridDim.x - 1) / T);
  }
  int lo = 0, hi = (int)gridDim.x - 1;  // the last CTA whose first group is <= g
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (p.cta_start[mid] <= g) lo = mid;
    else hi = mid - 1;
  }
  return lo;
}

// out = o_hat R_vo^T for the G query heads of unit (b, h); o_hat in shared
// memory [G][128].  Thread t takes outputs 4q..4q+3 (q = t % 32) of every
// head over rows j of slice t / 32 (S = NT / 32 slices of the 128 rows): its
// float4 loads of R_vo^T are independent, eight in flight at a time, and
// each element serves all G heads.  The slices' partial sums meet in
// `part` (S * G * 128 floats of shared memory, which may overlap o_hat) and
// are added in slice order.
template <int G, int NT>
__device__ __forceinline__ void rotate_back_out(const DecodeParams& p, int64_t b, int64_t h, const float* o_hat,
                                                float* part) {
  constexpr int S = NT / 32;
  constexpr int RS = (kHeadDim + S - 1) / S;  // rows per slice (the last may have fewer)
  static_assert(NT % 32 == 0 && S >= 1, "whole warps");
  const int q = threadIdx.x & 31, sl = threadIdx.x >> 5;
  const float4* RT4 = reinterpret_cast<const float4*>(p.R_voT + (size_t)h * kHeadDim * kHeadDim);
  float acc[G][4];
#pragma unroll
  for (int gh = 0; gh < G; ++gh) acc[gh][0] = acc[gh][1] = acc[gh][2] = acc[gh][3] = 0.f;
  // eight rows in flight at a time
#pragma unroll 1
  for (int kb = 0; kb < RS; kb += 8) {
    float4 r[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      const int j = sl * RS + kb + k;
      r[k] = (kb + k < RS && j < kHeadDim) ? __ldg(RT4 + j * (kHeadDim / 4) + q) : make_float4(0.f, 0.f, 0.f, 0.f);
    }
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      const int j = sl * RS + kb + k;
      if (kb + k < RS && j < kHeadDim) {
#pragma unroll
        for (int gh = 0; gh < G; ++gh) {
          const float o = o_hat[gh * kHeadDim + j];
          acc[gh][0] = fmaf(o, r[k].x, acc[gh][0]);
          acc[gh][1] = fmaf(o, r[k].y, acc[gh][1]);
          acc[gh][2] = fmaf(o, r[k].z, acc[gh][2]);
          acc[gh][3] = fmaf(o, r[k].w, acc[gh][3]);
        }
      }
    }
  }
  __syncthreads();  // o_hat is read; part may reuse it
#pragma unroll
  for (int gh = 0; gh < G; ++gh)
    reinterpret_cast<float4*>(part + (sl * G + gh) * kHeadDim)[q] =
        make_float4(acc[gh][0], acc[gh][1], acc[gh][2], acc[gh][3]);
  __syncthreads();
  for (int o = threadIdx.x; o < G * kHeadDim; o += NT) {
    const int gh = o / kHeadDim, i = o % kHeadDim;
    float a = 0.f;
#pragma unroll
    for (int k = 0; k < S; ++k) a += part[(k * G + gh) * kHeadDim + i];
    p.out[((b * p.H_q) + h * G + gh) * kHeadDim + i] = __float2half_rn(a);
  }
}

// The last CTA to finish a segment of unit u merges the unit's partials,
// normalises, rotates back (o = o_hat R_vo^T) and writes the output.  The
// arrival counter resets itself for the next decode; nothing waits.
// `scratch` holds NT / 32 * G * 128 floats (free at this point); `flag` one
// float.  Every thread's partial writes are ordered before thread 0's fence
// by the barrier, and the fence before the arrival (the release pattern of a
// grid-wide barrier).  Each thread merges its outputs' n = c1 - c0 + 1
// partials eight at a time with all their loads issued together (an online
// max over the batches), so a merge costs one round trip per batch.
// (A unit that one CTA holds entirely never comes here: it is finished from
// shared memory by that CTA.)
template <int G, int NT>
__device__ __forceinline__ void finish_unit(const DecodeParams& p, int64_t c0, int64_t c1, int64_t u, int64_t b,
                                            int64_t h, float* scratch, float* flag) {
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    const int old = atomicAdd(p.counters + u, 1);
    const bool last = old == (int)(c1 - c0);
    if (last) {
      p.counters[u] = 0;
      __threadfence();
    }
    flag[0] = last ? 1.f : 0.f;
  }
  __syncthreads();
  if (flag[0] == 0.f) return;
  const int n = (int)(c1 - c0 + 1);
  float* o_hat = scratch;  // [G][128]
  for (int o = threadIdx.x; o < G * kHeadDim; o += NT) {
    const int gh = o / kHeadDim, dd = o % kHeadDim;
    float M = -INFINITY, L = 0.f, A = 0.f;
    for (int cb = 0; cb < n; cb += 8) {
      float mc[8], lc[8], ac[8];
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        mc[k] = -INFINITY, lc[k] = 0.f, ac[k] = 0.f;
        if (cb + k < n) {
          const float* part = p.partials + ((size_t)(c0 + cb + k + u) * G + gh) * (kHeadDim + 2);
          mc[k] = __ldcg(part);
          lc[k] = __ldcg(part + 1);
          ac[k] = __ldcg(part + 2 + dd);
        }
      }
      float Mn = M;
#pragma unroll
      for (int k = 0; k < 8; ++k) Mn = fmaxf(Mn, mc[k]);
      if (Mn == -INFINITY) continue;  // nothing attended so far
      const float f = (M == -INFINITY) ? 0.f : exp2f(M - Mn);
      L *= f;
      A *= f;
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const float w = (mc[k] == -INFINITY) ? 0.f : exp2f(mc[k] - Mn);
        L = fmaf(w, lc[k], L);
        A = fmaf(w, ac[k], A);
      }
      M = Mn;
    }
    o_hat[o] = (L > 0.f) ? A / L : 0.f;
  }
  __syncthreads();
  rotate_back_out<G, NT>(p, b, h, o_hat, scratch);
}

// Variants of the one-head kernel by the chunks read per vector (MAXC):
//   4:  one slot of 4 chunks for keys and one for values (up to 32 entries:
//       half the guarded chunk iterations of the 8-chunk form; k 32 on the
//       32k layer 0.587 -> 0.548 ms, k 16 0.464 -> 0.403 ms);
//   8:  one slot of 8 chunks for keys and one for values;
//   12: two slots, X (8 chunks) and Y (4), each loaded one phase ahead;
//   16: one slot of 16 chunks each (the registers allow 8 warps).
// The two-slot form keeps the 12-warp layout for up to 96 entries; at 128
// it was slower than the 16-chunk slots (2.65 against 2.31 ms on the 32k
// layer, while at 96 it took 1.72 against 1.99 ms).
template <int MAXC>
__host__ __device__ constexpr bool decode_two_slot() { return MAXC == 12; }
// How many blocks ahead of use a warp asks L2 for a block's records.  Over
// all resident warps the records in flight must stay well inside L2: at 96
// entries read (1824 warps x 2 blocks x 18 KB = 66 MB) two blocks ahead
// thrashed it (k 96 on the 32k layer: 1.52 ms at 2 blocks, 1.35-1.37 ms at
// 1; k 128 1.853 -> 1.833 ms), while up to 64 entries (44 MB) two stay best
// (k 32, 48: 1 % slower at one block).
template <int MAXC>
__host__ __device__ constexpr int decode_prefetch_ahead() { return MAXC > 8 ? 1 : 2; }
// Warps per CTA of the one-head kernel: one lane-private accumulator each
// (16 KB); for 16 chunks as many as the registers allow.
template <int MAXC>
__host__ __device__ constexpr int decode_warps() { return MAXC <= 12 ? 6 : 8; }
// CTAs of the one-head kernel per SM (registers and shared memory allow two
// of 6 warps; one CTA's barriers, merges and finishes then overlap the
// other's streaming)
template <int MAXC>
__host__ __device__ constexpr int decode_min_ctas() { return MAXC <= 12 ? 2 : 1; }
// q' row shift of the one-head kernel (16 or 32 copies per coordinate)
template <int MAXC>
__host__ __device__ constexpr int decode_q_shift() { return MAXC <= 12 ? 6 : 7; }

// Split decode kernel, one query head per kv head.
//   The flat list of 32-token blocks of all units is cut into ranges of
//   equal cost (cta_begin), one per CTA.  Shared memory (dynamic, laid out
//   from its actual start):
//   one lane-private rotated-space accumulator per warp ([128][32] fp32,
//   16 KB-aligned regions) and q' with 16 or 32 copies per coordinate
//   ([128][16 | 32] fp32, aligned to its size), in the gap before the first
//   aligned region when it fits there, else after the accumulators.
//   Lane = token; each warp walks a contiguous run of blocks.  While block g
//   is processed, the key records of block g+1 are in flight to registers
//   and block g+2 (g+1 for the variants that read more than 64 entries) is
//   being prefetched into L2.
template <int MAXC, int FMT>
__global__ void __launch_bounds__(decode_warps<MAXC>() * 32, decode_min_ctas<MAXC>())
    decode_kernel(DecodeParams p) {
  constexpr int NW = decode_warps<MAXC>();
  constexpr int NT = NW * 32;
  constexpr int QS = decode_q_shift<MAXC>();
  constexpr bool kTwoSlot = decode_two_slot<MAXC>();
  constexpr int KS = kTwoSlot ? 8 : MAXC;  // chunks of slot X (kc: keys, then values)
  constexpr int KY = MAXC - 8;             // chunks of slot Y (two-slot form)
  constexpr int QREP = (1 << QS) / 4;                       // copies per coordinate
  constexpr uint32_t kQBytes = kHeadDim << QS;              // 8 or 16 KB
  extern __shared__ __align__(16) unsigned char smem_dyn[];
  __shared__ float red_m[NW], red_l[NW];
  __shared__ __align__(16) float q_stage[kHeadDim];  // q' of the next unit, before replication
  pdl_trigger();

  const uint32_t raw = (uint32_t)__cvta_generic_to_shared(smem_dyn);
  const uint32_t base = (raw + kRegionBytes - 1) & ~(kRegionBytes - 1);
  uint32_t qbase = (raw + kQBytes - 1) & ~(kQBytes - 1);
  if (qbase + kQBytes > base) qbase = base + NW * kRegionBytes;
  {
    uint32_t dyn_bytes;
    asm("mov.u32 %0, %%dynamic_smem_size;" : "=r"(dyn_bytes));
    if (max(base + NW * kRegionBytes, qbase + kQBytes) > raw + dyn_bytes) {
      if (threadIdx.x == 0) atomicOr(p.status, kStatusLayout);
      return;  // the launch gave too little shared memory for this layout
    }
  }
  float* accs = reinterpret_cast<float*>(smem_dyn + (base - raw));  // [NW][128][32]
  float* qrep = reinterpret_cast<float*>(smem_dyn + (qbase - raw)); // [128][16]

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t qb = qbase + ((lane & (QREP - 1)) << 2);
  const uint32_t ab = base + warp * kRegionBytes + (lane << 2);

  const CacheGeom& g = p.geom;
  const int kfull = p.k_full_chunks, krem = p.k_rem;          // keys
  const int nchunks = kfull + (krem ? 1 : 0);
  const int kfull_v = p.k_full_chunks_v, krem_v = p.k_rem_v;  // values
  const int nchunks_v = kfull_v + (krem_v ? 1 : 0);
  // this lane's record runs inside a block
  const int o_kv = lane * 16, o_ki = g.kidx_off() + lane * 8;
  const int o_vv = g.vval_off() + lane * 16, o_vi = g.vidx_off() + lane * 8;
  const bool whole_block = nchunks * 8 == g.k_slots && nchunks_v * 8 == g.k_slots_v;
  const int bsh = p.blocks_per_page_log2, bmask = (1 << bsh) - 1;

  const int64_t g_begin = cta_begin(p, blockIdx.x);
  const int64_t g_end = min(p.total_groups, cta_begin(p, blockIdx.x + 1));
  // Before waiting for the previous launch (the step's append), ask L2 for
  // this warp's first two blocks, so their first reads overlap that launch:
  // only where finding them reads nothing that launch writes (computed page
  // ids, equal rows; a block it is still writing to stays coherent in L2),
  // and only for CTAs with a long range (32-layer stack step 4.42 -> 4.37
  // ms, 32k layer 0.925 -> 0.920 ms; at a few groups per CTA the extra
  // prologue showed in the kernel's own time and the step gained nothing).
  if (g.identity && p.seq == nullptr && g_end - g_begin >= 16 && lane == 0) {
    const int64_t u0 = unit_of(p, g_begin);
    const UnitView v0 = unit_view(p, u0);
    const int s0 = (int)(g_begin - v0.goff), s1 = (int)(min(g_end, v0.goff + v0.N_g) - v0.goff);
    const int lo = split_at(s0, s1, v0.n_sg, warp, NW);
    const int hi = min(split_at(s0, s1, v0.n_sg, warp + 1, NW), v0.n_sg);
    for (int j = 0; j < 2 && lo + j < hi; ++j) {
      const int gi = lo + j;
      prefetch_l2(g.pool + (g.identity_base + u0 * g.pages_per_unit + (gi >> bsh)) * g.page_bytes +
                      (int64_t)(gi & bmask) * g.block_bytes(),
                  (uint32_t)g.block_bytes());
    }
  }
  pdl_wait();
  if (g_begin >= g_end) return;
  const int64_t u_first = unit_of(p, g_begin), u_last = unit_of(p, g_end - 1);
  // q' of the unit the next segment starts, copied into q_stage by
  // cp.async a segment ahead (the first one here): no registers held
  const uint32_t q_stage_s = (uint32_t)__cvta_generic_to_shared(q_stage);
  auto stage_q = [&](int64_t un) {
    if (threadIdx.x < kHeadDim / 4) {
      const int64_t bn = un / p.H_kv, hn = un - bn * p.H_kv;
      cp_async16(q_stage_s + threadIdx.x * 16, p.qprime + (bn * p.H_q + hn) * kHeadDim + threadIdx.x * 4);
    }
    cp_async_commit();
  };
  stage_q(u_first);

  for (int64_t u = u_first; u <= u_last; ++u) {
    const UnitView uv = unit_view(p, u);
    const int n_sg = uv.n_sg;
    const int s0 = (int)(max(g_begin, uv.goff) - uv.goff);
    const int s1 = (int)(min(g_end, uv.goff + uv.N_g) - uv.goff);
    const int64_t b = u / p.H_kv, h = u % p.H_kv;
    // this warp's contiguous run of groups [t_lo, t_hi)
    const int t_lo = split_at(s0, s1, n_sg, warp, NW);
    const int t_hi = split_at(s0, s1, n_sg, warp + 1, NW);
    const int sp_hi = min(t_hi, n_sg);  // sparse groups of the run: [t_lo, sp_hi)
    const int32_t* ptab = g.page_table + u * g.pages_per_unit;

    cp_async_wait_all();
    __syncthreads();  // the previous segment is done with shared memory; q_stage has landed
    // q' copies (float4 f of the [128][QREP] layout holds row f / (QREP / 4))
    for (int f = threadIdx.x; f < kHeadDim * QREP / 4; f += NT) {
      const float v = q_stage[f / (QREP / 4)];
      reinterpret_cast<float4*>(qrep)[f] = make_float4(v, v, v, v);
    }
    {
      float4* az = reinterpret_cast<float4*>(accs + warp * kHeadDim * 32);
#pragma unroll 8
      for (int f = lane; f < kHeadDim * 8; f += 32) az[f] = make_float4(0.f, 0.f, 0.f, 0.f);
    }
    __syncthreads();
    if (u < u_last) stage_q(u + 1);
    // into L2 ahead of use: R_vo^T of this head (64 KB, for the rotate-back)
    // and the dense-buffer rows of this warp's run (read without a pipeline)
    if (threadIdx.x == 0) prefetch_l2(p.R_voT + (size_t)h * kHeadDim * kHeadDim, kHeadDim * kHeadDim * 4);
    for (int gi = max(t_lo, n_sg); gi < t_hi; ++gi) {
      const int64_t i = (int64_t)(gi - n_sg) * 32 + lane;
      if (i < uv.n_b) {
        const size_t row = ((size_t)u * p.cap + (int)((uv.buf_start + i) % p.cap)) * kHeadDim;
        prefetch_l2(p.ring_k + row, kHeadDim * 2);
        prefetch_l2(p.ring_v + row, kHeadDim * 2);
      }
    }

    float m_w = -INFINITY;  // running max (log2 domain), uniform in the warp
    float l_sum = 0.f;      // this lane's sum of exp2(s - m_w)

    // block of sparse group gi (nullptr past the run or on a bad page)
    auto block_of = [&](int gi) -> const uint8_t* {
      if (gi >= sp_hi) return nullptr;
      const int64_t ph = g.identity ? g.identity_base + u * g.pages_per_unit + (gi >> bsh)
                                    : (int64_t)__ldg(ptab + (gi >> bsh));
      if (ph < 0 || ph >= g.num_pages) {
        atomicOr(p.status, kStatusPageRange);
        return nullptr;
      }
      return g.pool + (int64_t)ph * g.page_bytes + (int64_t)(gi & bmask) * g.block_bytes();
    };
    auto prefetch_block = [&](const uint8_t* blk) {
      if (blk == nullptr || lane != 0) return;
      if (whole_block) {
        prefetch_l2(blk, (uint32_t)g.block_bytes());
      } else if constexpr (FMT == kFmtFp16) {
        prefetch_l2(blk, nchunks * 512u);
        prefetch_l2(blk + g.kidx_off(), nchunks * 256u);
        prefetch_l2(blk + g.vval_off(), nchunks_v * 512u);
        prefetch_l2(blk + g.vidx_off(), nchunks_v * 256u);
      } else {
        prefetch_l2(blk, nchunks * 512u);
        prefetch_l2(blk + g.vval_off(), nchunks_v * 512u);
      }
    };

    // key chunks 0 .. KS - 1 of the next block (two-slot form: the rest
    // are loaded while these are scored)
    Chunk<FMT> kc[KS];
    auto load_k = [&](const uint8_t* blk) {
      const uint8_t* src = blk ? blk : g.pool;
#pragma unroll
      for (int c = 0; c < KS; ++c)
        if (c < nchunks) kc[c] = load_chunk<FMT, false>(src + o_kv, src + o_ki, c);
    };

    const uint8_t* b_cur = block_of(t_lo);
    const uint8_t* b_n1 = block_of(t_lo + 1);
    prefetch_block(b_n1);
    if (t_lo < sp_hi) load_k(b_cur);

    for (int gi = t_lo; gi < t_hi; ++gi) {
      float s2, pr;
      if (gi < n_sg) {
        // ---- sparse group: tokens 32*gi .. 32*gi+31 of the sparse history
        const int64_t t0 = (int64_t)gi * 32;
        const bool ok = b_cur != nullptr;
        const bool valid = ok && t0 + lane < uv.sparse_len;
        const uint8_t* src = ok ? b_cur : g.pool;
        float s[4] = {0.f, 0.f, 0.f, 0.f};
        // scores of the key chunks c0 .. c0 + N - 1 held in cs[N] (a lane
        // past the end of the history scores its unwritten records: any
        // index byte addresses inside q', and the score is replaced by
        // -inf below)
        auto score_slot = [&](const auto& cs, int c0) {
          constexpr int N = std::extent<std::remove_reference_t<decltype(cs)>>::value;
#pragma unroll
          for (int c = 0; c < N; ++c)
            if (c0 + c < nchunks) {
              float f[8];
              chunk_vals<FMT>(cs[c], f);
              if (krem && c0 + c == nchunks - 1) keep_first(f, krem);
              score_chunk<QS>(qb, f, chunk_idx<FMT>(cs[c]), s);
            }
        };
        // key or value chunks c0 .. c0 + N - 1 of this block into cs[N]
        auto load_slot = [&](auto& cs, int c0, int n, int o_val, int o_idx) {
          constexpr int N = std::extent<std::remove_reference_t<decltype(cs)>>::value;
#pragma unroll
          for (int c = 0; c < N; ++c)
            if (c0 + c < n) cs[c] = load_chunk<FMT, false>(src + o_val, src + o_idx, c0 + c);
        };
        // the online softmax step of this lane's token: returns its weight
        auto softmax_step = [&]() -> float {
          const float gmax = warp_max(s2);
          if (gmax > m_w + kLazyRescale) {
            if (m_w != -INFINITY) {
              const float fs = exp2f(m_w - gmax);
              l_sum *= fs;
#pragma unroll 8
              for (int dd = 0; dd < kHeadDim; ++dd) sts(ab + dd * 128, lds(ab + dd * 128) * fs);
            }
            m_w = gmax;
          }
          const float w = valid ? exp2f(s2 - m_w) : 0.f;
          l_sum += w;
          return w;
        };
        // acc[idx] += pr * val for the value chunks c0 .. c0 + N - 1 in cs[N]
        // (lanes past the end of the history skip: their records are
        // unwritten, and 0 * inf would not be 0)
        auto value_slot = [&](const auto& cs, int c0) {
          constexpr int N = std::extent<std::remove_reference_t<decltype(cs)>>::value;
          if (!valid) return;
#pragma unroll
          for (int c = 0; c < N; ++c)
            if (c0 + c < kfull_v) {
              float f[8];
              chunk_vals<FMT>(cs[c], f);
              value_chunk(ab, pr, f, chunk_idx<FMT>(cs[c]));
            }
          if (krem_v) {
#pragma unroll
            for (int c = 0; c < N; ++c)
              if (c0 + c == kfull_v) {
                float f[8];
                chunk_vals<FMT>(cs[c], f);
                value_chunk_partial(ab, pr, f, chunk_idx<FMT>(cs[c]), krem_v);
              }
          }
        };
        if constexpr (!kTwoSlot) {
          // the value records in flight while the keys (loaded during the
          // previous block) are scored
          Chunk<FMT> vc[KS];
          load_slot(vc, 0, nchunks_v, o_vv, o_vi);
          // one or two blocks ahead: into L2
          const uint8_t* b_n2 = block_of(gi + 2);
          prefetch_block(decode_prefetch_ahead<MAXC>() == 2 ? b_n2 : b_n1);
          score_slot(kc, 0);
          s2 = valid ? ((s[0] + s[1]) + (s[2] + s[3])) * p.scale_log2 : -INFINITY;
          // the next block's key records into registers while this block's
          // values are accumulated
          if (gi + 1 < sp_hi) load_k(b_n1);
          b_cur = b_n1;
          b_n1 = b_n2;
          pr = softmax_step();
          value_slot(vc, 0);
        } else {
          // two register slots, X (kc, 8 chunks) and Y (KY chunks), each
          // loaded one phase ahead of its use: key chunks 8.. into Y while
          // keys 0..7 are scored, values 0..7 into X while keys 8.. are
          // scored, values 8.. into Y during the softmax and values 0..7,
          // the next block's keys 0..7 into X during values 8..
          Chunk<FMT> cy[KY];
          load_slot(cy, KS, nchunks, o_kv, o_ki);
          const uint8_t* b_n2 = block_of(gi + 2);
          prefetch_block(decode_prefetch_ahead<MAXC>() == 2 ? b_n2 : b_n1);
          score_slot(kc, 0);
          load_slot(kc, 0, nchunks_v, o_vv, o_vi);
          score_slot(cy, KS);
          load_slot(cy, KS, nchunks_v, o_vv, o_vi);
          s2 = valid ? ((s[0] + s[1]) + (s[2] + s[3])) * p.scale_log2 : -INFINITY;
          const uint8_t* b_next = b_n1;
          b_cur = b_n1;
          b_n1 = b_n2;
          pr = softmax_step();
          value_slot(kc, 0);
          if (gi + 1 < sp_hi) load_k(b_next);
          value_slot(cy, KS);
        }
      } else {
        // ---- buffer group: dense rotated fp16 vectors of the ring buffer
        const int64_t i = (int64_t)(gi - n_sg) * 32 + lane;
        const bool valid = i < uv.n_b;
        const int slot = valid ? (int)((uv.buf_start + i) % p.cap) : 0;
        const size_t row = ((size_t)u * p.cap + slot) * kHeadDim;
        const uint4* kr = reinterpret_cast<const uint4*>(p.ring_k + row);
        const uint4* vr = reinterpret_cast<const uint4*>(p.ring_v + row);
        float s[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll 4
        for (int c = 0; c < 16; ++c) {
          const uint4 w = __ldg(kr + c);
          const float2 a = h2f(w.x), bb = h2f(w.y), cc = h2f(w.z), d = h2f(w.w);
          constexpr uint32_t QR = 1u << QS;
          const uint32_t q = qb + c * 8 * QR;
          s[0] = fmaf(lds(q + 0 * QR), a.x, s[0]);
          s[1] = fmaf(lds(q + 1 * QR), a.y, s[1]);
          s[2] = fmaf(lds(q + 2 * QR), bb.x, s[2]);
          s[3] = fmaf(lds(q + 3 * QR), bb.y, s[3]);
          s[0] = fmaf(lds(q + 4 * QR), cc.x, s[0]);
          s[1] = fmaf(lds(q + 5 * QR), cc.y, s[1]);
          s[2] = fmaf(lds(q + 6 * QR), d.x, s[2]);
          s[3] = fmaf(lds(q + 7 * QR), d.y, s[3]);
        }
        s2 = valid ? ((s[0] + s[1]) + (s[2] + s[3])) * p.scale_log2 : -INFINITY;
        const float gmax = warp_max(s2);
        if (gmax > m_w + kLazyRescale) {
          if (m_w != -INFINITY) {
            const float fs = exp2f(m_w - gmax);
            l_sum *= fs;
#pragma unroll 8
            for (int dd = 0; dd < kHeadDim; ++dd) sts(ab + dd * 128, lds(ab + dd * 128) * fs);
          }
          m_w = gmax;
        }
        pr = valid ? exp2f(s2 - m_w) : 0.f;
        l_sum += pr;
        if (valid) {
#pragma unroll 2
          for (int c = 0; c < 16; ++c) {
            const uint4 w = __ldg(vr + c);
            const float2 a = h2f(w.x), bb = h2f(w.y), cc = h2f(w.z), d = h2f(w.w);
            const uint32_t t = ab + c * 8 * 128;
            const float o0 = lds(t + 0 * 128), o1 = lds(t + 1 * 128), o2 = lds(t + 2 * 128),
                        o3 = lds(t + 3 * 128), o4 = lds(t + 4 * 128), o5 = lds(t + 5 * 128),
                        o6 = lds(t + 6 * 128), o7 = lds(t + 7 * 128);
            sts(t + 0 * 128, fmaf(pr, a.x, o0));
            sts(t + 1 * 128, fmaf(pr, a.y, o1));
            sts(t + 2 * 128, fmaf(pr, bb.x, o2));
            sts(t + 3 * 128, fmaf(pr, bb.y, o3));
            sts(t + 4 * 128, fmaf(pr, cc.x, o4));
            sts(t + 5 * 128, fmaf(pr, cc.y, o5));
            sts(t + 6 * 128, fmaf(pr, d.x, o6));
            sts(t + 7 * 128, fmaf(pr, d.y, o7));
          }
        }
      }
    }

    // ---- merge the lanes and warps into one partial: each warp sums its
    // lanes' accumulators (lane l coordinates l, l+32, l+64, l+96, reading
    // the columns in rotated order: conflict-free) into the first 128 floats
    // of its region, then one thread per coordinate combines the warps
    l_sum = warp_sum(l_sum);
    {
      float* a = accs + warp * kHeadDim * 32;
      float sum[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll 8
      for (int jj = 0; jj < 32; ++jj) {
        const int col = (jj + lane) & 31;
#pragma unroll
        for (int k = 0; k < 4; ++k) sum[k] += a[(lane + 32 * k) * 32 + col];
      }
      __syncwarp();
#pragma unroll
      for (int k = 0; k < 4; ++k) a[lane + 32 * k] = sum[k];
    }
    if (lane == 0) {
      red_m[warp] = m_w;
      red_l[warp] = l_sum;
    }
    __syncthreads();
    const int64_t c0 = cta_of(p, uv.goff), c1 = cta_of(p, uv.goff + uv.N_g - 1);
    const bool solo = c0 == c1;  // this CTA holds the whole unit
    for (int dd = threadIdx.x; dd < kHeadDim; dd += NT) {
      float M = -INFINITY;
#pragma unroll
      for (int w = 0; w < NW; ++w) M = fmaxf(M, red_m[w]);
      float tot = 0.f, L = 0.f;
#pragma unroll
      for (int w = 0; w < NW; ++w) {
        const float mw = red_m[w];
        const float f = (mw == -INFINITY) ? 0.f : exp2f(mw - M);
        tot = fmaf(f, accs[w * kHeadDim * 32 + dd], tot);
        L = fmaf(f, red_l[w], L);
      }
      if (solo) {
        qrep[dd] = (L > 0.f) ? tot / L : 0.f;  // q' is no longer needed
        continue;
      }
      float* dst = p.partials + ((size_t)(blockIdx.x + u)) * (kHeadDim + 2);
      dst[2 + dd] = tot;
      if (dd == 0) {
        dst[0] = M;
        dst[1] = L;
      }
    }
    if (solo) {
      __syncthreads();
      rotate_back_out<1, NT>(p, b, h, qrep, qrep);
    } else {
      finish_unit<1, NT>(p, c0, c1, u, b, h, qrep, red_m);
    }
  }
}

}  // namespace
}  // namespace swan
