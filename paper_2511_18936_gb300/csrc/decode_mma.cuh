// Device code of the grouped-query decode kernel (Algorithm 1, attention
// part; Section 4.1.1 grouping; Section 4.3): G query heads per kv head, the
// value product (and at G = 8 the scores) on the tensor cores, with the
// split combine and rotate-back of decode_kernels.cuh.  Included by
// decode.cu.
#pragma once

#include "decode_kernels.cuh"

namespace swan {
namespace {

// ---------------------------------------------------------------------------
// Grouped-query heads with the value product on the tensor cores (G = 2, 4, 8).
//   Lane = token, as in the one-head kernel; each lane scores its token for
//   all G query heads of the kv head from q' replicated per lane
//   ([128][32 / G][G] fp32: one 8- or 16-byte conflict-free gather per entry,
//   two 16-byte gathers at G = 8).
//   The value product o_h += sum_t p_h(t) v_t is dense once the kept
//   entries are scattered into a zero-filled [32 tokens][128] fp16 tile per
//   warp, so it runs as mma.sync.m16n8k16 (k = the 32 tokens, n = the 128
//   coordinates) with the fp32 accumulators in registers; p is split into
//   fp16 hi + lo parts, rows 0..G-1 and G..2G-1 of the same product (at
//   G = 8 the eight rows take the hi parts, then the lo parts, in two
//   products into the same accumulators), so the result keeps fp32 accuracy.  No per-warp shared accumulator: the tile
//   and a [G][32] p table are all a warp holds in shared memory.
// ---------------------------------------------------------------------------
// Value tile rows: 128 fp16 (256 bytes, 256-byte aligned), the 16-byte
// chunk j of token t's row stored at chunk j ^ (t & 7), so an ldmatrix of 8
// token rows at one chunk hits 8 distinct bank groups, and the scatter
// address is (2 idx) ^ (row | (t & 7) << 4): one shift and one LOP3.
constexpr int kVRowBytes = 256;
constexpr uint32_t kVTileBytes = 32 * kVRowBytes;    // 8192
// p [max(G, 4) heads][32 tokens] fp32, rows 40 floats apart: the value
// product reads p at (row r, column 2 cq + e) for four rows at once, which
// with 32-float rows all fall in one bank (a 4-way conflict; 8 rows apart
// they are distinct).
constexpr int kPStride = 40;
template <int G>
__host__ __device__ constexpr uint32_t mma_ptile_bytes() {  // rounded up to whole 256-byte rows of the tiles
  return ((G > 4 ? G : 4) * kPStride * 4 + 255u) / 256u * 256u;
}
// Scores on the tensor cores (G = 8, up to 64 entries read): each warp also
// holds a zero-filled [32 tokens][128] fp16 key tile, laid out like the value
// tile, into which its tokens' kept key entries are scattered; the scores
// are then S = K_tile (q'_hi + q'_lo) as mma.sync.m16n8k16 products (k = the
// 128 coordinates, n = the 8 heads), in place of two 16-byte q' gathers per
// kept entry.
template <int G, int MAXC>
__host__ __device__ constexpr bool mma_scores() { return G == 8 && MAXC == 8; }
// Per warp: the value tile, the key tile (scores on the tensor cores only),
// the p table and a staging area for the value records of the next block
// (cp.async: MAXC chunks of 512 B values + 256 B indices).  A multiple of
// 256 bytes: the scatter forms a tile address by XOR of the row base with
// 2 idx (up to 0xfe) and the chunk swizzle, which needs 256-byte rows.
template <int G, int MAXC>
__host__ __device__ constexpr uint32_t mma_warp_bytes() {
  return (mma_scores<G, MAXC>() ? 2 : 1) * kVTileBytes + mma_ptile_bytes<G>() + (uint32_t)MAXC * 768;
}
// 8 warps: the kernel needs ~230-255 registers a thread; registers are
// allocated per scheduler, so 9 to 12 warps all get 168 a thread and spill
// (a sweep on the GB300 measured 8 < 10 < 12 warps in time: 0.480, 0.491,
// 0.565 ms on the GQA 131k layer).
template <int MAXC>
__host__ __device__ constexpr int mma_warps() { return 8; }
// q' replicated in 32 / G copies per coordinate: [128][32 / G][G] fp32, 16 KB.
// A G-float gather is served in phases of 32 / G lanes (16-byte loads: 8
// lanes, 8-byte loads: 16), and the lanes of a phase read distinct copies,
// so they never share a bank.  With the scores on the tensor cores the
// region holds q' as B fragments instead: [8 k-steps][hi, lo][32 lanes]
// (b0, b1) fp16 pairs, 4 KB.
constexpr uint32_t kQrepBytes = kHeadDim * 32 * 4;
template <int G, int MAXC>
__host__ __device__ constexpr size_t mma_smem() {  // + the 16 KB alignment slack
  static_assert(mma_warp_bytes<G, MAXC>() % 256 == 0, "tile rows 256-byte aligned");
  return (size_t)kQrepBytes + (size_t)mma_warps<MAXC>() * mma_warp_bytes<G, MAXC>() + 16384;
}

__device__ __forceinline__ uint4 lds_v4u(uint32_t a) {
  uint4 v;
  asm volatile("ld.shared.v4.u32 {%0,%1,%2,%3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(a)
               : "memory");
  return v;
}
__device__ __forceinline__ uint2 lds_v2u(uint32_t a) {
  uint2 v;
  asm volatile("ld.shared.v2.u32 {%0,%1}, [%2];" : "=r"(v.x), "=r"(v.y) : "r"(a) : "memory");
  return v;
}

__device__ __forceinline__ float4 lds4(uint32_t a) {
  float4 v;
  asm volatile("ld.shared.v4.f32 {%0,%1,%2,%3}, [%4];" : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w) : "r"(a));
  return v;
}
// Tile accesses carry a memory clobber: they alias the C++ accesses to the
// same tile (the p table, the o rows of the merge).
__device__ __forceinline__ void sts_u16(uint32_t a, uint32_t v) {
  asm volatile("st.shared.u16 [%0], %1;" ::"r"(a), "h"((unsigned short)v) : "memory");
}
__device__ __forceinline__ void sts_v4(uint32_t a, uint4 v) {
  asm volatile("st.shared.v4.u32 [%0], {%1,%2,%3,%4};" ::"r"(a), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w)
               : "memory");
}
__device__ __forceinline__ void ldsm_x4_trans(uint32_t a, uint32_t (&r)[4]) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(a)
               : "memory");
}
// d[0..1] += A (16 x 16, rows g and g + 8) * B (16 x 8); the rows g + 8 of A
// are zero, so their accumulators are dropped.
__device__ __forceinline__ void mma_16816(float (&d)[2], uint32_t a0, uint32_t a2, uint32_t b0, uint32_t b1) {
  asm volatile(
      "{\n\t.reg .f32 x2, x3;\n\t"
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,x2,x3}, {%2,%3,%4,%5}, {%6,%7}, "
      "{%8,%9,%10,%11};\n\t}"
      : "=f"(d[0]), "=f"(d[1])
      : "r"(a0), "r"(0u), "r"(a2), "r"(0u), "r"(b0), "r"(b1), "f"(d[0]), "f"(d[1]), "f"(0.f), "f"(0.f));
}
// d[0..3] += A (16 x 16) * B (16 x 8), all rows of A
__device__ __forceinline__ void mma_16816_full(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
__device__ __forceinline__ void ldsm_x4(uint32_t a, uint32_t (&r)[4]) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(a)
               : "memory");
}
// Two fp32 values as (hi, lo) fp16 pairs: x = hi + lo to ~2^-22 relative.
__device__ __forceinline__ void split_pair(float x0, float x1, uint32_t& hi, uint32_t& lo) {
  const __half2 h = __floats2half2_rn(x0, x1);  // x0 in the low half
  const float2 hf = __half22float2(h);
  const __half2 l = __floats2half2_rn(x0 - hf.x, x1 - hf.y);
  hi = *reinterpret_cast<const uint32_t*>(&h);
  lo = *reinterpret_cast<const uint32_t*>(&l);
}
// The 8 values of a chunk as fp16 bits, two per word.
template <int FMT>
__device__ __forceinline__ void chunk_half_words(const Chunk<FMT>& ch, uint32_t (&w)[4]) {
  if constexpr (FMT == kFmtFp16) {
    w[0] = ch.v.x, w[1] = ch.v.y, w[2] = ch.v.z, w[3] = ch.v.w;
  } else {
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const uint32_t src = q < 2 ? ch.r.x : ch.r.y;
      const __half2_raw h = __nv_cvt_fp8x2_to_halfraw2(
          (__nv_fp8x2_storage_t)((q & 1) ? (src >> 16) : (src & 0xffffu)), __NV_E4M3);
      w[q] = (uint32_t)h.x | ((uint32_t)h.y << 16);
    }
  }
}
// Scores of G heads for one chunk: q' row idx of this lane is G floats
// (128-byte rows, 16 KB-aligned base: the address is one shift and one
// LOP3).  With two partial-sum sets (NS = 2) even and odd entries go to
// separate sums (half-length FMA chains).  At G = 8 the lane reads its copy's
// two 16-byte halves in the order its qb gives (bit 4: upper half first), so
// the 8 lanes of a phase hit 8 distinct bank groups; s[.][0..3] then hold the
// heads of the first half read and s[.][4..7] the other (g8_heads_in_order
// puts them back).
template <int G, int NS>
__device__ __forceinline__ void score_g_chunk(uint32_t qb, const float (&f)[8], uint2 ix, float (&s)[NS][G]) {
#pragma unroll
  for (int e = 0; e < 8; ++e) {
    const uint32_t w = e < 4 ? ix.x : ix.y;
    const int sh = 7 - 8 * (e & 3);  // byte e & 3 of w to bits 7..13
    const uint32_t a = ((sh >= 0 ? (w << sh) : (w >> -sh)) & 0x3f80u) | qb;
    float* t = s[e % NS];
    if constexpr (G == 8) {
      const float4 q0 = lds4(a), q1 = lds4(a ^ 16u);
      t[0] = fmaf(q0.x, f[e], t[0]);
      t[1] = fmaf(q0.y, f[e], t[1]);
      t[2] = fmaf(q0.z, f[e], t[2]);
      t[3] = fmaf(q0.w, f[e], t[3]);
      t[4] = fmaf(q1.x, f[e], t[4]);
      t[5] = fmaf(q1.y, f[e], t[5]);
      t[6] = fmaf(q1.z, f[e], t[6]);
      t[7] = fmaf(q1.w, f[e], t[7]);
    } else if constexpr (G == 4) {
      const float4 q = lds4(a);
      t[0] = fmaf(q.x, f[e], t[0]);
      t[1] = fmaf(q.y, f[e], t[1]);
      t[2] = fmaf(q.z, f[e], t[2]);
      t[3] = fmaf(q.w, f[e], t[3]);
    } else {
      const float2 q = lds2(a);
      t[0] = fmaf(q.x, f[e], t[0]);
      t[1] = fmaf(q.y, f[e], t[1]);
    }
  }
}
// G = 8: a lane that read its copy's upper half first (hi) holds heads 4..7
// in s[0..3] and heads 0..3 in s[4..7]; swap them into head order.
template <int G>
__device__ __forceinline__ void g8_heads_in_order(float (&s)[G], bool hi) {
  if constexpr (G == 8) {
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float a = s[j], b = s[j + 4];
      s[j] = hi ? b : a;
      s[j + 4] = hi ? a : b;
    }
  }
}
// Scatter the first n (<= 8) entries of a chunk into this lane's tile row
// (vsw = the row's address | (lane & 7) << 4, the chunk swizzle).
__device__ __forceinline__ void scatter_chunk(uint32_t vsw, const uint32_t (&w)[4], uint2 ix, int n) {
#pragma unroll
  for (int e = 0; e < 8; ++e) {
    if (e < n) {
      const uint32_t iw = e < 4 ? ix.x : ix.y;
      const int sh = 1 - 8 * (e & 3);  // byte e & 3 of iw, times 2
      const uint32_t off = (sh >= 0 ? (iw << sh) : (iw >> -sh)) & 0xfeu;
      const uint32_t hw = w[e >> 1];
      sts_u16(off ^ vsw, (e & 1) ? (hw >> 16) : (hw & 0xffffu));
    }
  }
}

template <int G, int MAXC, int FMT>
__global__ void __launch_bounds__(mma_warps<MAXC>() * 32, 1) decode_mma_kernel(DecodeParams p) {
  constexpr int NW = mma_warps<MAXC>(), NT = NW * 32;
  constexpr uint32_t kWarpBytes = mma_warp_bytes<G, MAXC>();
  constexpr int NS = G == 8 ? 1 : 2;  // partial-sum sets of the scores
  extern __shared__ __align__(16) unsigned char smem_raw[];
  __shared__ float red_m[NW * G], red_l[NW * G];
  __shared__ float flag[1];
  __shared__ __align__(16) float q_stage[G * kHeadDim];  // q' of the next unit's G heads
  static_assert(G * kHeadDim / 4 <= NT, "one 16-byte piece of q' per thread");
  pdl_trigger();

  const uint32_t raw = (uint32_t)__cvta_generic_to_shared(smem_raw);
  const uint32_t base = (raw + 16383u) & ~16383u;  // 16 KB aligned: q' and 256-byte tile rows
  unsigned char* base_ptr = smem_raw + (base - raw);
  float* qrep = reinterpret_cast<float*>(base_ptr);                         // [128][32/G][G]
  const uint32_t wbase = base + kQrepBytes;                                 // per-warp regions
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  constexpr bool kMma = mma_scores<G, MAXC>();
  constexpr uint32_t kTiles = (kMma ? 2 : 1) * kVTileBytes;
  const uint32_t vtile = wbase + warp * kWarpBytes;                         // [32][256 B] fp16, swizzled
  const uint32_t ktile = vtile + kVTileBytes;                               // the same, keys (kMma)
  float* ptile_f = reinterpret_cast<float*>(base_ptr + (vtile + kTiles - base));  // [G][kPStride] fp32
  const uint32_t vstage = vtile + kTiles + mma_ptile_bytes<G>();            // value records, next block
  // this lane's copy (at G = 8 with the half it reads first in bit 4)
  const bool q_hi_first = G == 8 && ((lane >> 2) & 1);
  const uint32_t qb = base + (lane & (32 / G - 1)) * (G * 4) + (q_hi_first ? 16u : 0u);
  const uint32_t vrow = vtile + lane * kVRowBytes;
  const uint32_t vsw = vrow | ((uint32_t)(lane & 7) << 4);  // this row with its chunk swizzle
  const uint32_t ksw = vsw + kVTileBytes;                   // its key tile row (kMma)
  const int gq = lane >> 2, cq = lane & 3;  // mma fragment coordinates

  const CacheGeom& g = p.geom;
  const int kfull = p.k_full_chunks, krem = p.k_rem;
  const int nchunks = kfull + (krem ? 1 : 0);
  const int kfull_v = p.k_full_chunks_v, krem_v = p.k_rem_v;
  const int nchunks_v = kfull_v + (krem_v ? 1 : 0);
  const int o_kv = lane * 16, o_ki = g.kidx_off() + lane * 8;
  const int o_vv = g.vval_off() + lane * 16, o_vi = g.vidx_off() + lane * 8;
  const bool whole_block = nchunks * 8 == g.k_slots && nchunks_v * 8 == g.k_slots_v;
  const int bsh = p.blocks_per_page_log2, bmask = (1 << bsh) - 1;

  const int64_t g_begin = cta_begin(p, blockIdx.x);
  const int64_t g_end = min(p.total_groups, cta_begin(p, blockIdx.x + 1));
  pdl_wait();
  if (g_begin >= g_end) return;
  const int64_t u_first = unit_of(p, g_begin), u_last = unit_of(p, g_end - 1);
  // q' of the G heads of the unit the next segment starts (G * 128
  // consecutive floats), copied into q_stage by cp.async a segment ahead
  const uint32_t q_stage_s = (uint32_t)__cvta_generic_to_shared(q_stage);
  auto stage_q = [&](int64_t un) {
    if (threadIdx.x < G * kHeadDim / 4) {
      const int64_t bn = un / p.H_kv, hn = un - bn * p.H_kv;
      cp_async16(q_stage_s + threadIdx.x * 16, p.qprime + (bn * p.H_q + hn * G) * kHeadDim + threadIdx.x * 4);
    }
    cp_async_commit();
  };
  stage_q(u_first);

  // the tiles start zeroed; every use restores the zeros it disturbed
  auto zero_rows = [&]() {
    for (int c = 0; c < 16; ++c) {
      sts_v4(vsw ^ (uint32_t)(c << 4), make_uint4(0, 0, 0, 0));
      if constexpr (kMma) sts_v4(ksw ^ (uint32_t)(c << 4), make_uint4(0, 0, 0, 0));
    }
  };
  zero_rows();

  for (int64_t u = u_first; u <= u_last; ++u) {
    const UnitView uv = unit_view(p, u);
    const int n_sg = uv.n_sg;
    const int s0 = (int)(max(g_begin, uv.goff) - uv.goff);
    const int s1 = (int)(min(g_end, uv.goff + uv.N_g) - uv.goff);
    const int64_t b = u / p.H_kv, h = u % p.H_kv;
    const int t_lo = split_at(s0, s1, n_sg, warp, NW);
    const int t_hi = split_at(s0, s1, n_sg, warp + 1, NW);
    const int sp_hi = min(t_hi, n_sg);
    const int32_t* ptab = g.page_table + u * g.pages_per_unit;

    cp_async_wait_all();
    __syncthreads();  // the previous segment is done with q'; q_stage has landed
    if constexpr (kMma) {
      // B fragments: lane l of k-step ks holds head l / 4 (zero beyond G) at
      // coordinates 16 ks + 2 (l % 4) + {0, 1} (b0) and + {8, 9} (b1), as
      // fp16 hi parts, then lo parts
      for (int f = threadIdx.x; f < 8 * 32; f += NT) {
        const int ks = f >> 5, l = f & 31, hd = l >> 2, c = 16 * ks + 2 * (l & 3);
        const float* qh = q_stage + (hd < G ? hd : 0) * kHeadDim;
        const float z = hd < G ? 1.f : 0.f;
        uint32_t h0, l0, h1, l1;
        split_pair(z * qh[c], z * qh[c + 1], h0, l0);
        split_pair(z * qh[c + 8], z * qh[c + 9], h1, l1);
        reinterpret_cast<uint2*>(qrep)[(2 * ks) * 32 + l] = make_uint2(h0, h1);
        reinterpret_cast<uint2*>(qrep)[(2 * ks + 1) * 32 + l] = make_uint2(l0, l1);
      }
    } else {
      // 32 floats per coordinate c: 32 / G copies of its G heads (float4 f
      // holds coordinate f / 8, heads (4 (f % 8) + e) % G, e = 0..3: 0..3 at
      // G = 4, 0, 1, 0, 1 at G = 2, the lower or upper four at G = 8)
      for (int f = threadIdx.x; f < kHeadDim * 8; f += NT) {
        const int c = f >> 3, h0 = (4 * (f & 7)) % G;
        const float4 v = make_float4(q_stage[(h0 % G) * kHeadDim + c], q_stage[((h0 + 1) % G) * kHeadDim + c],
                                     q_stage[((h0 + 2) % G) * kHeadDim + c], q_stage[((h0 + 3) % G) * kHeadDim + c]);
        reinterpret_cast<float4*>(qrep)[f] = v;
      }
    }
    __syncthreads();
    if (u < u_last) stage_q(u + 1);

    float m[G], l[G];
#pragma unroll
    for (int j = 0; j < G; ++j) m[j] = -INFINITY, l[j] = 0.f;
    float acc[16][2];
#pragma unroll
    for (int nt = 0; nt < 16; ++nt) acc[nt][0] = acc[nt][1] = 0.f;

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
    Chunk<FMT> kc[MAXC];
    auto load_k = [&](const uint8_t* blk) {
      const uint8_t* src = blk ? blk : g.pool;
#pragma unroll
      for (int c = 0; c < MAXC; ++c)
        if (c < nchunks) kc[c] = load_chunk<FMT, false>(src + o_kv, src + o_ki, c);
    };
    // the value records of a block into this warp's staging area, in flight
    // while the warp works on the block before it
    auto stage_v = [&](const uint8_t* blk) {
      if (blk != nullptr) {
        const int n_val = nchunks_v * 32;  // 16-byte pieces
        for (int i = lane; i < n_val; i += 32) cp_async16(vstage + i * 16, blk + g.vval_off() + i * 16);
        if constexpr (FMT == kFmtFp16) {
          const int n_idx = nchunks_v * 16;
          for (int i = lane; i < n_idx; i += 32)
            cp_async16(vstage + nchunks_v * 512 + i * 16, blk + g.vidx_off() + i * 16);
        }
      }
      cp_async_commit();
    };

    // kMma: the scores of the warp's 32 tokens from the key tile,
    // S[t][h] = sum_c K[t][c] (q'_hi + q'_lo)[c][h] (two products into the
    // same accumulators), through the p table ([h][t]) to lane t
    auto tile_scores = [&](float (&sc)[G]) {
      float d[2][4];
#pragma unroll
      for (int mt = 0; mt < 2; ++mt) d[mt][0] = d[mt][1] = d[mt][2] = d[mt][3] = 0.f;
#pragma unroll
      for (int ks = 0; ks < 8; ++ks) {
        const uint2 bh = lds_v2u(base + (uint32_t)((2 * ks) * 32 + lane) * 8u);
        const uint2 bl = lds_v2u(base + (uint32_t)((2 * ks + 1) * 32 + lane) * 8u);
#pragma unroll
        for (int mt = 0; mt < 2; ++mt) {
          // matrix lane / 8: token rows + 8 (bit 0), coordinates + 8 (bit 1)
          const int mi = lane >> 3;
          const uint32_t row = (uint32_t)(16 * mt + (mi & 1) * 8 + (lane & 7));
          const uint32_t chunk = (uint32_t)(2 * ks + (mi >> 1));
          uint32_t a[4];
          ldsm_x4(ktile + row * kVRowBytes + ((chunk ^ (uint32_t)(lane & 7)) << 4), a);
          mma_16816_full(d[mt], a, bh.x, bh.y);
          mma_16816_full(d[mt], a, bl.x, bl.y);
        }
      }
      // d[mt]: tokens 16 mt + gq (0, 1) and + 8 (2, 3), heads 2 cq, 2 cq + 1
      if (2 * cq < G) {
#pragma unroll
        for (int mt = 0; mt < 2; ++mt) {
          float* pc = ptile_f + (2 * cq) * kPStride + 16 * mt + gq;
          pc[0] = d[mt][0];
          pc[kPStride] = d[mt][1];
          pc[8] = d[mt][2];
          pc[kPStride + 8] = d[mt][3];
        }
      }
      __syncwarp();
#pragma unroll
      for (int j = 0; j < G; ++j) sc[j] = ptile_f[j * kPStride + lane];
    };

    const uint8_t* b_cur = block_of(t_lo);
    const uint8_t* b_n1 = block_of(t_lo + 1);
    prefetch_block(b_n1);
    if (t_lo < sp_hi) {
      load_k(b_cur);
      stage_v(b_cur);
    }

    for (int gi = t_lo; gi < t_hi; ++gi) {
      float s[G];
      float s2[NS][G];
#pragma unroll
      for (int i = 0; i < NS; ++i)
#pragma unroll
        for (int j = 0; j < G; ++j) s2[i][j] = 0.f;
      bool valid;
      if (gi < n_sg) {
        // ---- sparse tokens 32 gi .. 32 gi + 31
        const int64_t t0 = (int64_t)gi * 32;
        const bool ok = b_cur != nullptr;
        valid = ok && t0 + lane < uv.sparse_len;
        const uint8_t* b_n2 = block_of(gi + 2);
        prefetch_block(b_n2);
        if constexpr (kMma) {
          // this token's kept keys into its key tile row (the first k_active
          // entries only: a padding entry would overwrite coordinate 0)
          if (valid) {
#pragma unroll
            for (int c = 0; c < MAXC; ++c)
              if (c < nchunks) {
                uint32_t w[4];
                chunk_half_words<FMT>(kc[c], w);
                scatter_chunk(ksw, w, chunk_idx<FMT>(kc[c]), (krem && c == nchunks - 1) ? krem : 8);
              }
          }
          __syncwarp();
          tile_scores(s);
        } else {
          if (valid) {
#pragma unroll
            for (int c = 0; c < MAXC; ++c)
              if (c < nchunks) {
                float f[8];
                chunk_vals<FMT>(kc[c], f);
                if (krem && c == nchunks - 1) keep_first(f, krem);
                score_g_chunk<G, NS>(qb, f, chunk_idx<FMT>(kc[c]), s2);
              }
          }
#pragma unroll
          for (int j = 0; j < G; ++j) s[j] = NS == 2 ? s2[0][j] + s2[NS - 1][j] : s2[0][j];
          g8_heads_in_order<G>(s, q_hi_first);
        }
        // this token's kept values (staged by cp.async) into its tile row;
        // each staged chunk is read before the previous one is stored
        cp_async_wait_all();
        __syncwarp();
        if (valid) {
          auto staged = [&](int c) {
            Chunk<FMT> vc;
            if constexpr (FMT == kFmtFp16) {
              vc.v = lds_v4u(vstage + c * 512 + lane * 16);
              vc.i = lds_v2u(vstage + nchunks_v * 512 + c * 256 + lane * 8);
            } else {
              vc.r = lds_v4u(vstage + c * 512 + lane * 16);
            }
            return vc;
          };
          Chunk<FMT> vc = staged(0);
#pragma unroll
          for (int c = 0; c < MAXC; ++c)
            if (c < nchunks_v) {
              Chunk<FMT> vn = vc;
              if (c + 1 < nchunks_v) vn = staged(c + 1);
              uint32_t w[4];
              chunk_half_words<FMT>(vc, w);
              scatter_chunk(vsw, w, chunk_idx<FMT>(vc), (krem_v && c == nchunks_v - 1) ? krem_v : 8);
              vc = vn;
            }
        }
        __syncwarp();
        if (gi + 1 < sp_hi) {
          load_k(b_n1);
          stage_v(b_n1);
        }
        b_cur = b_n1;
        b_n1 = b_n2;
      } else {
        // ---- dense buffer tokens: scores over all 128 coordinates, the
        // value row copied into the tile
        const int64_t i = (int64_t)(gi - n_sg) * 32 + lane;
        valid = i < uv.n_b;
#pragma unroll
        for (int j = 0; j < G; ++j) s[j] = 0.f;
        if (valid) {
          const int slot = (int)((uv.buf_start + i) % p.cap);
          const size_t row = ((size_t)u * p.cap + slot) * kHeadDim;
          const uint4* kr = reinterpret_cast<const uint4*>(p.ring_k + row);
          const uint4* vr = reinterpret_cast<const uint4*>(p.ring_v + row);
          if constexpr (kMma) {
#pragma unroll 1
            for (int cb = 0; cb < 16; cb += 8) {
              uint4 wk[8];
#pragma unroll
              for (int k = 0; k < 8; ++k) wk[k] = __ldg(kr + cb + k);
#pragma unroll
              for (int k = 0; k < 8; ++k) sts_v4(ksw ^ (uint32_t)((cb + k) << 4), wk[k]);
            }
          } else {
#pragma unroll 1
            for (int cb = 0; cb < 16; cb += 8) {
              uint4 wk[8];
#pragma unroll
              for (int k = 0; k < 8; ++k) wk[k] = __ldg(kr + cb + k);
#pragma unroll
              for (int k = 0; k < 8; ++k) {
                const int c = cb + k;
                const uint4 w = wk[k];
                const float2 a = h2f(w.x), bb = h2f(w.y), cc = h2f(w.z), d = h2f(w.w);
                const float f[8] = {a.x, a.y, bb.x, bb.y, cc.x, cc.y, d.x, d.y};
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                  const uint32_t qa = qb + (uint32_t)(c * 8 + e) * 128u;
                  float* t = s2[e % NS];
                  if constexpr (G == 8) {
                    const float4 q0 = lds4(qa), q1 = lds4(qa ^ 16u);
                    t[0] = fmaf(q0.x, f[e], t[0]);
                    t[1] = fmaf(q0.y, f[e], t[1]);
                    t[2] = fmaf(q0.z, f[e], t[2]);
                    t[3] = fmaf(q0.w, f[e], t[3]);
                    t[4] = fmaf(q1.x, f[e], t[4]);
                    t[5] = fmaf(q1.y, f[e], t[5]);
                    t[6] = fmaf(q1.z, f[e], t[6]);
                    t[7] = fmaf(q1.w, f[e], t[7]);
                  } else if constexpr (G == 4) {
                    const float4 q = lds4(qa);
                    t[0] = fmaf(q.x, f[e], t[0]);
                    t[1] = fmaf(q.y, f[e], t[1]);
                    t[2] = fmaf(q.z, f[e], t[2]);
                    t[3] = fmaf(q.w, f[e], t[3]);
                  } else {
                    const float2 q = lds2(qa);
                    t[0] = fmaf(q.x, f[e], t[0]);
                    t[1] = fmaf(q.y, f[e], t[1]);
                  }
                }
              }
            }
#pragma unroll
            for (int j = 0; j < G; ++j) s[j] = NS == 2 ? s2[0][j] + s2[NS - 1][j] : s2[0][j];
            g8_heads_in_order<G>(s, q_hi_first);
          }
#pragma unroll 1
          for (int cb = 0; cb < 16; cb += 8) {
            uint4 wv[8];
#pragma unroll
            for (int k = 0; k < 8; ++k) wv[k] = __ldg(vr + cb + k);
#pragma unroll
            for (int k = 0; k < 8; ++k) sts_v4(vsw ^ (uint32_t)((cb + k) << 4), wv[k]);
          }
        }
        if constexpr (kMma) {
          __syncwarp();
          tile_scores(s);
        }
      }

      // ---- online softmax per head (lazy rescale of the register accumulators)
      float pj[G];
#pragma unroll
      for (int j = 0; j < G; ++j) {
        const float sj = valid ? s[j] * p.scale_log2 : -INFINITY;
        const float gmax = warp_max(sj);
        if (gmax > m[j] + kLazyRescale) {
          if (m[j] != -INFINITY) {
            const float fs = ex2(m[j] - gmax);
            l[j] *= fs;
            if (gq == j || gq == j + G) {  // the head's hi and lo rows
#pragma unroll
              for (int nt = 0; nt < 16; ++nt) acc[nt][0] *= fs, acc[nt][1] *= fs;
            }
          }
          m[j] = gmax;
        }
        pj[j] = valid ? ex2(sj - m[j]) : 0.f;
        l[j] += pj[j];
        ptile_f[j * kPStride + lane] = pj[j];
      }
      __syncwarp();

      // ---- o[head][:] += p[head][tokens] * tile[tokens][:] on the tensor cores:
      // A rows 0..G-1 hold the fp16 hi parts of p, rows G..2G-1 the lo
      // parts, so one product covers both (the two row sets are added at
      // the merge)
#pragma unroll
      for (int ks = 0; ks < 2; ++ks) {
        if constexpr (G == 8) {
          // rows 0..7: the heads' hi parts, then their lo parts, into the
          // same accumulators
          const float* pr = ptile_f + gq * kPStride + ks * 16 + 2 * cq;
          uint32_t hi0, lo0, hi2, lo2;
          split_pair(pr[0], pr[1], hi0, lo0);
          split_pair(pr[8], pr[9], hi2, lo2);
#pragma unroll
          for (int np = 0; np < 8; ++np) {
            const int mi = lane >> 3;
            const uint32_t chunk = 2 * np + (mi >> 1);
            const uint32_t addr = vtile + (uint32_t)(ks * 16 + (mi & 1) * 8 + (lane & 7)) * kVRowBytes +
                                  ((chunk ^ (uint32_t)(lane & 7)) << 4);
            uint32_t bf[4];
            ldsm_x4_trans(addr, bf);
            mma_16816(acc[2 * np], hi0, hi2, bf[0], bf[1]);
            mma_16816(acc[2 * np], lo0, lo2, bf[0], bf[1]);
            mma_16816(acc[2 * np + 1], hi0, hi2, bf[2], bf[3]);
            mma_16816(acc[2 * np + 1], lo0, lo2, bf[2], bf[3]);
          }
          continue;
        }
        uint32_t a0 = 0, a2 = 0;
        if (gq < 2 * G) {
          const bool hi_row = gq < G;
          const float* pr = ptile_f + (hi_row ? gq : gq - G) * kPStride + ks * 16 + 2 * cq;
          uint32_t hi0, lo0, hi2, lo2;
          split_pair(pr[0], pr[1], hi0, lo0);
          split_pair(pr[8], pr[9], hi2, lo2);
          a0 = hi_row ? hi0 : lo0;
          a2 = hi_row ? hi2 : lo2;
        }
#pragma unroll
        for (int np = 0; np < 8; ++np) {
          const int mi = lane >> 3;
          const uint32_t chunk = 2 * np + (mi >> 1);  // of 8 coordinates; rows of tokens, row & 7 = lane & 7
          const uint32_t addr = vtile + (uint32_t)(ks * 16 + (mi & 1) * 8 + (lane & 7)) * kVRowBytes +
                                ((chunk ^ (uint32_t)(lane & 7)) << 4);
          uint32_t bf[4];
          ldsm_x4_trans(addr, bf);
          mma_16816(acc[2 * np], a0, a2, bf[0], bf[1]);
          mma_16816(acc[2 * np + 1], a0, a2, bf[2], bf[3]);
        }
      }
      __syncwarp();
      // restore the zeros of this lane's tile rows
      if (valid) zero_rows();
    }

    // ---- merge lanes and warps per query head into one partial
#pragma unroll
    for (int j = 0; j < G; ++j) l[j] = warp_sum(l[j]);
    if (lane == 0) {
#pragma unroll
      for (int j = 0; j < G; ++j) {
        red_m[warp * G + j] = m[j];
        red_l[warp * G + j] = l[j];
      }
    }
    // the lo rows (G..2G-1, lanes 4G above) onto the hi rows (at G = 8 the
    // products already summed them), then this warp's o rows into its tile
    // region ([G][128] fp32)
    if constexpr (G < 8) {
#pragma unroll
      for (int nt = 0; nt < 16; ++nt) {
        acc[nt][0] += __shfl_down_sync(0xffffffffu, acc[nt][0], 4 * G);
        acc[nt][1] += __shfl_down_sync(0xffffffffu, acc[nt][1], 4 * G);
      }
    }
    __syncwarp();
    float* obuf = reinterpret_cast<float*>(base_ptr + (vtile - base));
    if (gq < G) {
#pragma unroll
      for (int nt = 0; nt < 16; ++nt) {
        obuf[gq * kHeadDim + nt * 8 + 2 * cq] = acc[nt][0];
        obuf[gq * kHeadDim + nt * 8 + 2 * cq + 1] = acc[nt][1];
      }
    }
    __syncthreads();
    const int64_t c0 = cta_of(p, uv.goff), c1 = cta_of(p, uv.goff + uv.N_g - 1);
    const bool solo = c0 == c1;
    for (int o = threadIdx.x; o < G * kHeadDim; o += NT) {
      const int hd = o / kHeadDim, dd = o % kHeadDim;
      float M = -INFINITY;
#pragma unroll
      for (int w = 0; w < NW; ++w) M = fmaxf(M, red_m[w * G + hd]);
      float tot = 0.f, L = 0.f;
#pragma unroll
      for (int w = 0; w < NW; ++w) {
        const float mw = red_m[w * G + hd];
        const float f = (mw == -INFINITY) ? 0.f : exp2f(mw - M);
        const float* ob = reinterpret_cast<const float*>(base_ptr + (wbase - base) + w * kWarpBytes);
        tot = fmaf(f, ob[hd * kHeadDim + dd], tot);
        L = fmaf(f, red_l[w * G + hd], L);
      }
      if (solo) {
        qrep[o] = (L > 0.f) ? tot / L : 0.f;  // q' is no longer needed
        continue;
      }
      float* dst = p.partials + ((size_t)(blockIdx.x + u) * G + hd) * (kHeadDim + 2);
      dst[2 + dd] = tot;
      if (dd == 0) {
        dst[0] = M;
        dst[1] = L;
      }
    }
    __syncthreads();
    if (solo) {
      rotate_back_out<G, NT>(p, b, h, qrep, qrep);
    } else {
      finish_unit<G, NT>(p, c0, c1, u, b, h, qrep, flag);
    }
    // the o rows overwrote part of the tiles, and the rotate-back's slices
    // (NT / 32 * G * 128 floats: past q' into the first warps' regions at
    // G = 8) more: zero them again once every thread is done with them
    __syncthreads();
    zero_rows();
  }
}

}  // namespace
}  // namespace swan
