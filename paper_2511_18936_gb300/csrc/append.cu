// Compress-on-append: rotation of new keys/values, dense ring-buffer insert,
// and magnitude top-k pruning into the paged sparse cache (Algorithm 1;
// Section 4.3; Section 5.1).
#include <cuda_fp8.h>

#include "sm100.h"
#include "sortnet.cuh"
#include "swan_internal.h"

namespace swan {
namespace {

// Sort 128 unique 32-bit keys held by one warp (lane l holds elements
// 4l..4l+3) into decreasing order with a bitonic network: the element of
// rank r ends up in lane r/4, slot r%4.
__device__ __forceinline__ void sort128_desc(uint32_t (&v)[4], int lane) {
#pragma unroll
  for (int k = 2; k <= 128; k <<= 1) {
#pragma unroll
    for (int j = k >> 1; j > 0; j >>= 1) {
      uint32_t nv[4];
#pragma unroll
      for (int s = 0; s < 4; ++s) {
        const int i = 4 * lane + s;
        const uint32_t other = (j >= 4) ? __shfl_xor_sync(0xffffffffu, v[s], j >> 2) : v[s ^ j];
        const bool desc = (i & k) == 0;   // direction of this bitonic run
        const bool lower = (i & j) == 0;  // lower element of the pair
        const uint32_t hi = max(v[s], other), lo = min(v[s], other);
        nv[s] = (lower == desc) ? hi : lo;
      }
#pragma unroll
      for (int s = 0; s < 4; ++s) v[s] = nv[s];
    }
  }
}

// Prune one rotated fp16 vector (lane l holds coordinates 4l..4l+3 as raw
// bits) to its k_store largest-magnitude coordinates, ties to the lower
// index, and store them in decreasing order at sparse position `sp` of
// `unit`.  The sort key is (|x| as fp16 bits, 127 - j, sign): unique, and its
// order is magnitude first, then lower index first.
__device__ __forceinline__ void warp_prune_store(uint2 raw, int lane, int kind, int64_t unit,
                                                 int64_t sp, const CacheGeom& g,
                                                 unsigned* status) {
  uint32_t key[4];
  const uint32_t h16[4] = {raw.x & 0xffffu, raw.x >> 16, raw.y & 0xffffu, raw.y >> 16};
#pragma unroll
  for (int s = 0; s < 4; ++s) {
    const uint32_t j = 4u * lane + s;
    key[s] = ((h16[s] & 0x7fffu) << 16) | ((127u - j) << 1) | (h16[s] >> 15);
  }
  sort128_desc(key, lane);

  const int64_t page = sp / g.P;
  const int slot = (int)(sp % g.P);
  if (page >= g.pages_per_unit) {
    if (lane == 0) atomicOr(status, kStatusPageRange);
    return;
  }
  const int32_t phys = g.page_table[unit * g.pages_per_unit + page];
  if (phys < 0 || phys >= g.num_pages) {
    if (lane == 0) atomicOr(status, kStatusPageRange);
    return;
  }
  uint8_t* blk = g.pool + (int64_t)phys * g.page_bytes + (int64_t)(slot >> 5) * g.block_bytes();
  const int t = slot & 31;
  const int slots = kind ? g.k_slots_v : g.k_slots;
  const int kept = kind ? g.k_store_v : g.k_store;
  if (lane < (slots >> 2)) {
    const int c = lane >> 1, half = lane & 1;
    uint32_t vb[4], ib[4];
#pragma unroll
    for (int s = 0; s < 4; ++s) {
      const bool keep = (4 * lane + s) < kept;
      const uint32_t j = 127u - ((key[s] >> 1) & 127u);
      const uint32_t bits = ((key[s] & 1u) << 15) | (key[s] >> 16);
      vb[s] = keep ? bits : 0u;
      ib[s] = keep ? j : 0u;
    }
    const uint32_t idx = ib[0] | (ib[1] << 8) | (ib[2] << 16) | (ib[3] << 24);
    const int rec = c * 32 + t;
    if (g.fmt == kFmtFp8) {
      // one 16-byte record per chunk: 8 E4M3 values (round to nearest even,
      // saturating to +-448), then the 8 indices
      uint32_t v8 = 0;
#pragma unroll
      for (int s = 0; s < 4; ++s) {
        __half_raw hr;
        hr.x = (unsigned short)vb[s];
        v8 |= (uint32_t)__nv_cvt_halfraw_to_fp8(hr, __NV_SATFINITE, __NV_E4M3) << (8 * s);
      }
      uint8_t* r = blk + (kind ? g.vval_off() : 0) + rec * 16;
      *reinterpret_cast<uint32_t*>(r + half * 4) = v8;
      *reinterpret_cast<uint32_t*>(r + 8 + half * 4) = idx;
    } else {
      const uint2 vals = make_uint2(vb[0] | (vb[1] << 16), vb[2] | (vb[3] << 16));
      const int voff = kind ? g.vval_off() : 0;
      const int ioff = kind ? g.vidx_off() : g.kidx_off();
      *reinterpret_cast<uint2*>(blk + voff + rec * 16 + half * 8) = vals;
      *reinterpret_cast<uint32_t*>(blk + ioff + rec * 8 + half * 4) = idx;
    }
  }
}

// Lengths of row b for an append: the uniform scalars, or its SeqInfo entry.
struct RowView {
  int64_t sparse_len, evict;
  int n_b, buf_start, n_new, prune;
};
__device__ __forceinline__ RowView row_view(const AppendParams& p, int64_t b, int evict_old) {
  if (p.seq == nullptr) return RowView{p.sparse_len, p.evict, p.n_b, p.buf_start, p.T, evict_old};
  const SeqInfo& q = p.seq[b];
  return RowView{q.sparse_len, q.evict, q.n_b, q.buf_start, q.n_new, q.prune};
}


// Small appends (decode steps): one CTA per (kv head h, K or V, bpc
// sequences from bz * bpc).  Phase 1 prunes the `evict_old` oldest buffered
// vectors of every sequence out of the ring; after a barrier, phase 2 rotates
// the new vectors one per warp (lane l computes coordinates 4l..4l+3 from R
// in shared memory, Rs: 64 KB, as a sequential fp32 FMA chain over the 128
// inputs) and either prunes them or writes them to the ring.  Ring slots
// freed in phase 1 are reused in phase 2 only after the barrier.
__device__ __forceinline__ void append_small_cta(const AppendParams& p, int evict_old, int bpc, int kind,
                                                 int h, int bz, float* Rs) {
  const int b0 = bz * bpc;                         // this CTA's sequences: [b0, b0 + nb)
  const int nb = min(bpc, p.B - b0);
  const float* R = (kind ? p.R_vo : p.R_qk) + (size_t)h * kHeadDim * kHeadDim;
  const __half* X = kind ? p.v_new : p.k_new;
  __half* ring = kind ? p.ring_v : p.ring_k;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  stage_matrix(Rs, R);
  pdl_wait();

  // phase 1: evict the oldest buffered vectors (sparse positions L_s + i)
  for (int item = warp; item < nb * evict_old; item += kWarpsPerCta) {
    const int b = b0 + item / evict_old, i = item % evict_old;
    const RowView rv = row_view(p, b, evict_old);
    if (i >= rv.prune) continue;
    const int64_t unit = (int64_t)b * p.H + h;
    const int slot = (rv.buf_start + i) % p.cap;
    const uint2 raw = __ldg(reinterpret_cast<const uint2*>(ring + (unit * p.cap + slot) * kHeadDim) + lane);
    warp_prune_store(raw, lane, kind, unit, rv.sparse_len + i, p.geom, p.status);
  }
  __syncthreads();

  // phase 2: the new vectors
  for (int item = warp; item < nb * p.T; item += kWarpsPerCta) {
    const int b = b0 + item / p.T, j = item % p.T;
    const RowView rv = row_view(p, b, evict_old);
    if (j >= rv.n_new) continue;
    const int64_t unit = (int64_t)b * p.H + h;
    const uint2 xw = __ldg(reinterpret_cast<const uint2*>(X + ((unit * p.T) + j) * kHeadDim) + lane);
    const float2 x01 = __half22float2(*reinterpret_cast<const __half2*>(&xw.x));
    const float2 x23 = __half22float2(*reinterpret_cast<const __half2*>(&xw.y));
    const float xs[4] = {x01.x, x01.y, x23.x, x23.y};
    float acc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll 8
    for (int i = 0; i < kHeadDim; ++i) {
      const float xi = __shfl_sync(0xffffffffu, xs[i & 3], i >> 2);
      const float4 r = reinterpret_cast<const float4*>(Rs + i * kHeadDim)[lane];
      acc[0] = fmaf(xi, r.x, acc[0]);
      acc[1] = fmaf(xi, r.y, acc[1]);
      acc[2] = fmaf(xi, r.z, acc[2]);
      acc[3] = fmaf(xi, r.w, acc[3]);
    }
    uint2 yw;
    yw.x = (uint32_t)__half_as_ushort(__float2half_rn(acc[0])) |
           ((uint32_t)__half_as_ushort(__float2half_rn(acc[1])) << 16);
    yw.y = (uint32_t)__half_as_ushort(__float2half_rn(acc[2])) |
           ((uint32_t)__half_as_ushort(__float2half_rn(acc[3])) << 16);
    const int64_t pos = (int64_t)rv.n_b + j;
    if (pos < rv.evict) {
      warp_prune_store(yw, lane, kind, unit, rv.sparse_len + pos, p.geom, p.status);
    } else {
      const int slot = (int)((rv.buf_start + pos) % p.cap);
      reinterpret_cast<uint2*>(ring + (unit * p.cap + slot) * kHeadDim)[lane] = yw;
    }
  }
}

__global__ void __launch_bounds__(kThreads) append_small_kernel(AppendParams p, int evict_old, int bpc) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  pdl_trigger();
  append_small_cta(p, evict_old, bpc, blockIdx.y, blockIdx.x, blockIdx.z, reinterpret_cast<float*>(smem_raw));
}

// A decode step's append and query rotation in one launch (they touch
// disjoint data): blockIdx.y 0 and 1 are the append's key and value CTAs
// (blockIdx.z < append_z), 2..5 the four coordinate slices of the query
// rotation (blockIdx.z < rotate_z query chunks).  CTAs beyond either range
// exit at once.
__global__ void __launch_bounds__(kThreads) append_rotate_kernel(AppendParams p, int evict_old, int bpc,
                                                                 int append_z, RotateQParams rq, int rotate_z) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  float* Rs = reinterpret_cast<float*>(smem_raw);
  pdl_trigger();
  if (blockIdx.y < 2) {
    if ((int)blockIdx.z < append_z) append_small_cta(p, evict_old, bpc, blockIdx.y, blockIdx.x, blockIdx.z, Rs);
  } else if ((int)blockIdx.z < rotate_z) {
    rotate_q_slice(rq, p.B, blockIdx.x, blockIdx.z, blockIdx.y - 2, Rs);
  }
}

// One warp per (unit, buffered token, K or V): read the ring row and prune.
__global__ void __launch_bounds__(kThreads) prune_ring_kernel(PruneRingParams p) {
  pdl_trigger();
  pdl_wait();
  const int lane = threadIdx.x & 31;
  const int64_t gw = ((int64_t)blockIdx.x * kThreads + threadIdx.x) >> 5;
  const int64_t total = (int64_t)p.units * p.count * 2;
  if (gw >= total) return;
  const int kind = (int)(gw & 1);
  const int64_t rest = gw >> 1;
  const int64_t unit = rest / p.count;
  const int i = (int)(rest % p.count);
  int buf_start = p.buf_start;
  int64_t sparse_len = p.sparse_len;
  if (p.seq != nullptr) {
    const SeqInfo& q = p.seq[unit / p.H];
    if (i >= q.prune) return;
    buf_start = q.buf_start;
    sparse_len = q.sparse_len;
  }
  const int slot = (buf_start + i) % p.cap;
  const __half* row = (kind ? p.ring_v : p.ring_k) + ((size_t)unit * p.cap + slot) * kHeadDim;
  const uint2 raw = __ldg(reinterpret_cast<const uint2*>(row) + lane);
  warp_prune_store(raw, lane, kind, unit, sparse_len + i, p.geom, p.status);
}

__global__ void transpose_r_kernel(const float* src, float* dst, int64_t mats) {
  __shared__ float tile[32][33];
  const int64_t m = blockIdx.z;
  const int bx = blockIdx.x * 32, by = blockIdx.y * 32;
  const float* s = src + m * kHeadDim * kHeadDim;
  float* d = dst + m * kHeadDim * kHeadDim;
  for (int r = threadIdx.y; r < 32; r += blockDim.y)
    tile[r][threadIdx.x] = s[(by + r) * kHeadDim + bx + threadIdx.x];
  __syncthreads();
  for (int r = threadIdx.y; r < 32; r += blockDim.y)
    d[(bx + r) * kHeadDim + by + threadIdx.x] = tile[threadIdx.x][r];
}

// ---------------------------------------------------------------------------
// Bulk append with the rotation on the tensor cores.
//   One CTA of 256 threads: 128 new vectors of one (row, kv head, K or V).
//   TMA brings the fp16 vectors (A: 128 x 128, K-major, 128-byte swizzle) and
//   the split rotation R^T = R_hi^T + 2^-12 R_lo^T (B: two fp16 128 x 128
//   tiles); two tcgen05.mma chains (K = 16 each step) accumulate x R_hi and
//   x R_lo in two 128-column TMEM accumulators.  The rows are read back as
//   y = hi + 2^-12 lo in fp32, rounded to fp16 and turned into sort keys,
//   which pass through shared memory to their owners: lanes 2v and 2v+1 hold
//   coordinates 0..63 and 64..127 of vector v.  Each lane sorts its 64 keys
//   in registers (sortnet.cuh); the pair then merges the two sorted halves
//   with shuffles and writes its ring row or its sparse records (consecutive
//   pairs hold consecutive tokens, so the records of a chunk are contiguous).
//   The products are exact (fp16 x fp16) and summed in fp32; the split
//   leaves 2^-22 |R| per term, inside the fp32-dot bound of the CUDA-core
//   path.
// ---------------------------------------------------------------------------
constexpr int kTcThreads = 256;              // two threads per vector of the tile
constexpr uint32_t kTcTile = 128 * 128 * 2;  // 32 KB: one fp16 128 x 128 tile
constexpr size_t kTcSmem = 3 * kTcTile + 1024;
constexpr uint64_t kTcWaitNs = 2000000000ull;
// a key that decodes to value +0 at index 0 (the padding entries of a chunk)
constexpr uint32_t kPadKey = 127u << 1;

// fp16 bits of two keys, packed (first key in the low half)
__device__ __forceinline__ uint32_t key_bits2(uint32_t ka, uint32_t kb) {
  return __byte_perm(ka, kb, 0x7632) | ((ka & 1u) << 15) | (kb << 31);
}
// coordinate indices of four keys, one per byte: the low key byte is
// (127 - c) << 1 | sign, and (~byte >> 1) & 127 = c
__device__ __forceinline__ uint32_t key_idx4(uint32_t k0, uint32_t k1, uint32_t k2, uint32_t k3) {
  const uint32_t w = __byte_perm(__byte_perm(k0, k1, 0x0040), __byte_perm(k2, k3, 0x0040), 0x5410);
  return (~w >> 1) & 0x7f7f7f7fu;
}

// r ? x : y for r in {0, 1}, as multiply-adds (off the integer min/max pipe)
__device__ __forceinline__ uint32_t pick(uint32_t r, uint32_t x, uint32_t y, uint32_t one) {
  return r * (x - y * one) + y;
}

// The 64 largest keys of a vector whose halves A (lane r = 0) and B (r = 1)
// are each sorted decreasing in a[]: A followed by B reversed is a bitonic
// run whose first half-cleaner keeps C[i] = max(A[i], B[63 - i]), the 64
// largest, again bitonic; its merge starts with a half-cleaner across the
// pair.  Afterwards lane r holds ranks 32 r .. 32 r + 31 in c[].
__device__ __forceinline__ void pair_top64(const uint32_t (&a)[64], uint32_t (&c)[32], uint32_t r,
                                           uint32_t one) {
#pragma unroll
  for (int m = 0; m < 32; ++m) {  // lane r computes C[32 r + m]
    const uint32_t send = pick(r, a[63 - m], a[32 + m], one);
    const uint32_t own = pick(r, a[31 - m], a[m], one);
    c[m] = sortnet::umax(own, __shfl_xor_sync(0xffffffffu, send, 1));
  }
#pragma unroll
  for (int m = 0; m < 32; ++m) {  // larger to lane 0, smaller to lane 1
    const uint32_t o = __shfl_xor_sync(0xffffffffu, c[m], 1);
    const uint32_t hi = sortnet::umax(c[m], o);
    c[m] = pick(r, (c[m] * one + o) - hi * one, hi, one);
  }
  sortnet::merge_desc<0, 32>(c, one);
}

// All 128 keys: the first half-cleaner of the same bitonic run crosses the
// pair (A[i] against B[63 - i]); afterwards lane r holds ranks 64 r ..
// 64 r + 63 in a[].
__device__ __forceinline__ void pair_sort128(uint32_t (&a)[64], uint32_t r, uint32_t one) {
  uint32_t s[64];
#pragma unroll
  for (int i = 0; i < 64; ++i) {
    const uint32_t own = pick(r, a[63 - i], a[i], one);
    const uint32_t o = __shfl_xor_sync(0xffffffffu, own, 1);
    const uint32_t hi = sortnet::umax(own, o);
    s[i] = pick(r, (own * one + o) - hi * one, hi, one);
  }
#pragma unroll
  for (int i = 0; i < 64; ++i) a[i] = s[i];
  sortnet::merge_desc<0, 64>(a, one);
}

// Write sorted keys of ranks rank0 .. rank0 + N - 1 of one vector (ranks at
// or beyond `kept` as padding, none at or beyond `slots`) to its records:
// the chunk of ranks 8c .. 8c + 7 at record c * 32 + t of the block.
template <int N>
__device__ __forceinline__ void store_sorted(const uint32_t (&key)[N], int rank0, int slots, int kept,
                                             uint8_t* vals, uint8_t* idx, int t, bool fp8) {
#pragma unroll
  for (int cc = 0; cc < N / 8; ++cc) {
    const int c = rank0 / 8 + cc;
    if (8 * c >= slots) break;
    uint32_t k[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) k[e] = key[8 * cc + e];
    if (8 * c + 8 > kept) {  // the last kept chunk (uniform in the CTA)
#pragma unroll
      for (int e = 0; e < 8; ++e) k[e] = (8 * c + e < kept) ? k[e] : kPadKey;
    }
    const int rec = c * 32 + t;
    const uint32_t i0 = key_idx4(k[0], k[1], k[2], k[3]), i1 = key_idx4(k[4], k[5], k[6], k[7]);
    if (fp8) {
      // one 16-byte record: 8 E4M3 values (round to nearest even, saturating
      // to +-448), then the 8 indices
      uint32_t v8[2];
#pragma unroll
      for (int w = 0; w < 2; ++w) {
        uint32_t pair[2];
#pragma unroll
        for (int q = 0; q < 2; ++q) {
          const uint32_t b2 = key_bits2(k[4 * w + 2 * q], k[4 * w + 2 * q + 1]);
          __half2_raw hr;
          hr.x = (unsigned short)(b2 & 0xffffu);
          hr.y = (unsigned short)(b2 >> 16);
          pair[q] = __nv_cvt_halfraw2_to_fp8x2(hr, __NV_SATFINITE, __NV_E4M3);
        }
        v8[w] = pair[0] | (pair[1] << 16);
      }
      *reinterpret_cast<uint4*>(vals + rec * 16) = make_uint4(v8[0], v8[1], i0, i1);
    } else {
      *reinterpret_cast<uint4*>(vals + rec * 16) =
          make_uint4(key_bits2(k[0], k[1]), key_bits2(k[2], k[3]), key_bits2(k[4], k[5]), key_bits2(k[6], k[7]));
      *reinterpret_cast<uint2*>(idx + rec * 8) = make_uint2(i0, i1);
    }
  }
}

__global__ void __launch_bounds__(kTcThreads, 2) append_tc_kernel(const __grid_constant__ CUtensorMap xk,
                                                                   const __grid_constant__ CUtensorMap xv,
                                                                   const __grid_constant__ CUtensorMap rhi,
                                                                   const __grid_constant__ CUtensorMap rlo,
                                                                   AppendParams p, int r_slice0, uint32_t one) {
  using namespace sm100;
  extern __shared__ __align__(1024) unsigned char smem_tc[];
  __shared__ __align__(8) uint64_t bars[2];
  __shared__ uint32_t tmem_slot;
  __shared__ int failed;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int kind = blockIdx.z, h = blockIdx.y;
  const int tiles_per_row = (p.T + 127) / 128;
  const int b = blockIdx.x / tiles_per_row, j0 = (blockIdx.x % tiles_per_row) * 128;
  const RowView rv = row_view(p, b, 0);
  pdl_trigger();
  if (j0 >= rv.n_new) return;  // no new token of this row in the tile (uniform in the CTA)

  const uint32_t raw = smem_u32(smem_tc);
  const uint32_t ta = (raw + 1023u) & ~1023u;
  const uint32_t tb_hi = ta + kTcTile, tb_lo = tb_hi + kTcTile;
  const uint32_t full = smem_u32(&bars[0]), done = smem_u32(&bars[1]);
  if (threadIdx.x == 0) {
    mbar_init(full, 1);
    mbar_init(done, 1);
    failed = 0;
    fence_barrier_init();
  }
  if (warp == 1) tmem_alloc(smem_u32(&tmem_slot), 256);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_slot;
  const uint64_t wait_ns = p.tc_wait_ns ? p.tc_wait_ns : kTcWaitNs;
  pdl_wait();

  if (threadIdx.x == 0) {
    const CUtensorMap* xm = kind ? &xv : &xk;
    const int slice = r_slice0 + kind * p.H + h;
    if (!p.tc_starve) {  // starved (test hook): nothing arrives on `full`
      mbar_arrive_expect_tx(full, 3 * kTcTile);
      tma_load_4d(ta, xm, full, 0, j0, h, b);
      tma_load_4d(ta + kTcTile / 2, xm, full, 64, j0, h, b);
      tma_load_3d(tb_hi, &rhi, full, 0, 0, slice);
      tma_load_3d(tb_hi + kTcTile / 2, &rhi, full, 64, 0, slice);
      tma_load_3d(tb_lo, &rlo, full, 0, 0, slice);
      tma_load_3d(tb_lo + kTcTile / 2, &rlo, full, 64, 0, slice);
    }
    if (!mbar_wait(full, 0, wait_ns)) {
      atomicOr(p.status, kStatusTimeout);
      failed = 1;
    } else {
      tc_fence_after();
      constexpr uint32_t idesc = idesc_f16_f32(128, 128, 0, 0);
#pragma unroll
      for (int kk = 0; kk < 8; ++kk) {
        const uint32_t off = (uint32_t)(kk >> 2) * (kTcTile / 2) + (uint32_t)(kk & 3) * 32;
        const uint64_t da = sdesc_sw128(ta + off, 16, 1024);
        mma_f16(tmem, da, sdesc_sw128(tb_hi + off, 16, 1024), idesc, kk > 0);
        mma_f16(tmem + 128, da, sdesc_sw128(tb_lo + off, 16, 1024), idesc, kk > 0);
      }
    }
    mma_commit(done);
  }
  __syncwarp();

  // ---- TMEM -> sort keys in shared memory (the operand tiles are free once
  // the MMAs are done).  Warp w reads rows 32 (w % 4) .. + 31 (its TMEM lane
  // quarter), coordinates 64 (w / 4) .. + 63.  The key of coordinate c is
  // (|y_c| as fp16 bits, 127 - c, sign): unique, ordered by magnitude first,
  // then lower index first.  Keys 4q .. 4q + 3 of half r of vector v sit at
  // 16-byte slot 256 q + 2 v + r: each lane's later reload of its 64 keys is
  // a conflict-free 512-byte run per warp.
  if (!mbar_wait(done, 0, wait_ns)) {
    atomicOr(p.status, kStatusTimeout);
    failed = 1;
  }
  tc_fence_after();
  uint4* keys_s = reinterpret_cast<uint4*>(smem_tc + (ta - raw));
  {
    const int row = 32 * (warp & 3) + lane, half = warp >> 2;
    const uint32_t taddr = tmem + ((uint32_t)(32 * (warp & 3)) << 16) + 64 * half;
#pragma unroll 1
    for (int c = 0; c < 2; ++c) {
      uint32_t hi[32], lo[32];
      tmem_ld32(taddr + c * 32, hi);
      tmem_ld32(taddr + 128 + c * 32, lo);
      tmem_wait_ld();
      tmem_regs_ready(hi);
      tmem_regs_ready(lo);
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        uint32_t k[4];
#pragma unroll
        for (int e = 0; e < 4; e += 2) {
          const int m = 4 * q + e;
          const float y0 = fmaf(__uint_as_float(lo[m]), 1.f / 4096.f, __uint_as_float(hi[m]));
          const float y1 = fmaf(__uint_as_float(lo[m + 1]), 1.f / 4096.f, __uint_as_float(hi[m + 1]));
          const __half2 y2 = __floats2half2_rn(y0, y1);
          const uint32_t h2 = *reinterpret_cast<const uint32_t*>(&y2);
          const uint32_t j = (uint32_t)(64 * half + 32 * c + m);
          k[e] = ((h2 & 0x7fffu) << 16) | ((127u - j) << 1) | ((h2 >> 15) & 1u);
          k[e + 1] = (h2 & 0x7fff0000u) | ((126u - j) << 1) | (h2 >> 31);
        }
        keys_s[256 * (8 * c + q) + 2 * row + half] = make_uint4(k[0], k[1], k[2], k[3]);
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) tmem_dealloc(tmem, 256);
  if (failed != 0) return;  // uniform in the CTA

  // ---- lanes 2v, 2v+1: vector v (coordinates 64 r .. 64 r + 63 in a[])
  const int v = threadIdx.x >> 1, j = j0 + v;
  const uint32_t r = threadIdx.x & 1u;
  uint32_t a[64];
#pragma unroll
  for (int q = 0; q < 16; ++q) {
    const uint4 k4 = keys_s[256 * q + threadIdx.x];
    a[4 * q] = k4.x;
    a[4 * q + 1] = k4.y;
    a[4 * q + 2] = k4.z;
    a[4 * q + 3] = k4.w;
  }
  const int64_t unit = (int64_t)b * p.H + h;
  const int64_t pos = (int64_t)rv.n_b + j;
  const bool live = j < rv.n_new;  // the same for both lanes of a pair
  if (live && pos >= rv.evict) {
    const int slot = (int)((rv.buf_start + pos) % p.cap);
    uint4* row = reinterpret_cast<uint4*>((kind ? p.ring_v : p.ring_k) + (unit * p.cap + slot) * kHeadDim) + 8 * (int)r;
#pragma unroll
    for (int q = 0; q < 8; ++q)
      row[q] = make_uint4(key_bits2(a[8 * q], a[8 * q + 1]), key_bits2(a[8 * q + 2], a[8 * q + 3]),
                          key_bits2(a[8 * q + 4], a[8 * q + 5]), key_bits2(a[8 * q + 6], a[8 * q + 7]));
  }
  const bool prune = live && pos < rv.evict;
  if (!__any_sync(0xffffffffu, prune)) return;  // the pair exchanges below need the whole warp

  const CacheGeom& g = p.geom;
  const int64_t sp = rv.sparse_len + pos;
  const int64_t page = sp / g.P;
  const int slot = (int)(sp % g.P);
  int32_t phys = -1;
  if (prune) {
    if (page < g.pages_per_unit) phys = g.page_table[unit * g.pages_per_unit + page];
    if (phys < 0 || phys >= g.num_pages) {
      if (r == 0) atomicOr(p.status, kStatusPageRange);
      phys = -1;
    }
  }
  uint8_t* blk = g.pool + (int64_t)max(phys, 0) * g.page_bytes + (int64_t)(slot >> 5) * g.block_bytes();
  const bool fp8 = g.fmt == kFmtFp8;
  const int slots = kind ? g.k_slots_v : g.k_slots;
  const int kept = kind ? g.k_store_v : g.k_store;
  uint8_t* vals = blk + (kind ? g.vval_off() : 0);
  uint8_t* idx = blk + (kind ? g.vidx_off() : g.kidx_off());
  sortnet::sort_oe<0, 64, true>(a, one);
  if (slots <= 64) {  // uniform in the CTA
    uint32_t c[32];
    pair_top64(a, c, r, one);
    if (phys >= 0) store_sorted<32>(c, 32 * (int)r, slots, kept, vals, idx, slot & 31, fp8);
  } else {
    pair_sort128(a, r, one);
    if (phys >= 0) store_sorted<64>(a, 64 * (int)r, slots, kept, vals, idx, slot & 31, fp8);
  }
}

__global__ void split_r_kernel(const float* R_qk, const float* R_vo, __half* hi, __half* lo, int H) {
  // blockIdx.y: layer * 2 + kind; blockIdx.x: head; threads over (n, k)
  const int lk = blockIdx.y, kind = lk & 1, layer = lk >> 1, h = blockIdx.x;
  const float* R = (kind ? R_vo : R_qk) + ((size_t)layer * H + h) * kHeadDim * kHeadDim;
  const size_t dst = ((size_t)lk * H + h) * kHeadDim * kHeadDim;
  for (int e = threadIdx.x; e < kHeadDim * kHeadDim; e += blockDim.x) {
    const int n = e >> 7, k = e & 127;
    const float r = R[k * kHeadDim + n];
    const __half rh = __float2half_rn(r);
    hi[dst + e] = rh;
    lo[dst + e] = __float2half_rn((r - __half2float(rh)) * 4096.f);
  }
}

__global__ void scatter_pages_kernel(const int2* pairs, int n, int32_t* table) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i < n) {
    const int2 pr = pairs[i];
    table[pr.x] = pr.y;
  }
}

}  // namespace

cudaError_t launch_append_tc(const AppendParams& p, const CUtensorMap* maps, int r_slice0, cudaStream_t s) {
  cudaError_t e = ensure_smem<append_tc_kernel>(kTcSmem);
  if (e != cudaSuccess) return e;
  const int tiles = p.B * ((p.T + 127) / 128);
  // the sorting networks' multiply-adds take their factor 1 at run time
  return launch_pdl(append_tc_kernel, dim3((unsigned)tiles, (unsigned)p.H, 2), dim3(kTcThreads), kTcSmem, s,
                    maps[0], maps[1], maps[2], maps[3], p, r_slice0, 1u);
}

cudaError_t launch_split_r(const float* R_qk, const float* R_vo, __half* hi, __half* lo, int layers, int H,
                           cudaStream_t s) {
  split_r_kernel<<<dim3((unsigned)H, (unsigned)(2 * layers)), 256, 0, s>>>(R_qk, R_vo, hi, lo, H);
  return cudaGetLastError();
}

cudaError_t launch_scatter_pages(const int2* pairs, int n, int32_t* table, cudaStream_t s) {
  if (n <= 0) return cudaSuccess;
  scatter_pages_kernel<<<(n + 255) / 256, 256, 0, s>>>(pairs, n, table);
  return cudaGetLastError();
}

cudaError_t launch_append_small(const AppendParams& p, int evict_old, const RotateQParams* rq, cudaStream_t s) {
  constexpr size_t smem = 128 * 128 * sizeof(float);
  // enough sequences per CTA for one vector per warp and phase
  const int per = max(p.T, evict_old);
  const int bpc = max(1, kWarpsPerCta / max(per, 1));
  const int append_z = (p.B + bpc - 1) / bpc;
  if (rq == nullptr) {
    const cudaError_t e = ensure_smem<append_small_kernel>(smem);
    if (e != cudaSuccess) return e;
    return launch_pdl(append_small_kernel, dim3((unsigned)p.H, 2, (unsigned)append_z), dim3(kThreads), smem, s,
                      p, evict_old, bpc);
  }
  const cudaError_t e = ensure_smem<append_rotate_kernel>(smem);
  if (e != cudaSuccess) return e;
  const int rotate_z = (p.B * rq->G + kWarpsPerCta - 1) / kWarpsPerCta;
  return launch_pdl(append_rotate_kernel, dim3((unsigned)p.H, 6, (unsigned)max(append_z, rotate_z)),
                    dim3(kThreads), smem, s, p, evict_old, bpc, append_z, *rq, rotate_z);
}

cudaError_t launch_prune_ring(const PruneRingParams& p, cudaStream_t s) {
  const int64_t warps = (int64_t)p.units * p.count * 2;
  const int64_t blocks = (warps + kWarpsPerCta - 1) / kWarpsPerCta;
  return launch_pdl(prune_ring_kernel, dim3((unsigned)blocks), dim3(kThreads), 0, s, p);
}

cudaError_t launch_transpose_r(const float* src, float* dst, int64_t mats, cudaStream_t s) {
  dim3 grid(kHeadDim / 32, kHeadDim / 32, (unsigned)mats);
  transpose_r_kernel<<<grid, dim3(32, 8), 0, s>>>(src, dst, mats);
  return cudaGetLastError();
}

}  // namespace swan
