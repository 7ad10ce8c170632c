// Decode attention on the packed sparse cache (Algorithm 1, attention part;
// Section 4.3), split over the SMs, then the split combine and the
// rotate-back o = o_hat R_vo^T (Appendix A.1, Lemma 2).
#include "swan_internal.h"

namespace swan {
namespace {

// Streaming loads of cache records.  With one query head per kv head nothing
// is re-read, so the records bypass L1; with several heads the warps of a
// team read the same records and L1 serves the repeats.
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

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Shared-memory address (in floats, relative to a lane's column) of
// coordinate `i` in a [128][32] lane-interleaved array: element (i, lane) at
// i*32 + lane, so 32 lanes gathering arbitrary coordinates hit 32 distinct
// banks.
__device__ __forceinline__ int col(uint32_t i) { return (int)((i & 0x7fu) << 5); }

// Score contribution of one 8-entry chunk: sum_e q'[idx_e] * val_e.
__device__ __forceinline__ void score_chunk(const float* qc, uint4 v, uint2 ix, float& s0, float& s1) {
  const float2 a = h2f(v.x), b = h2f(v.y), c = h2f(v.z), d = h2f(v.w);
  s0 = fmaf(qc[col(ix.x)], a.x, s0);
  s1 = fmaf(qc[col(ix.x >> 8)], a.y, s1);
  s0 = fmaf(qc[col(ix.x >> 16)], b.x, s0);
  s1 = fmaf(qc[col(ix.x >> 24)], b.y, s1);
  s0 = fmaf(qc[col(ix.y)], c.x, s0);
  s1 = fmaf(qc[col(ix.y >> 8)], c.y, s1);
  s0 = fmaf(qc[col(ix.y >> 16)], d.x, s0);
  s1 = fmaf(qc[col(ix.y >> 24)], d.y, s1);
}

// Scatter-accumulate one 8-entry chunk: acc[idx_e] += p * val_e.
__device__ __forceinline__ void value_chunk(float* ac, float p, uint4 v, uint2 ix) {
  const float2 a = h2f(v.x), b = h2f(v.y), c = h2f(v.z), d = h2f(v.w);
  float* t;
  t = ac + col(ix.x);        *t = fmaf(p, a.x, *t);
  t = ac + col(ix.x >> 8);   *t = fmaf(p, a.y, *t);
  t = ac + col(ix.x >> 16);  *t = fmaf(p, b.x, *t);
  t = ac + col(ix.x >> 24);  *t = fmaf(p, b.y, *t);
  t = ac + col(ix.y);        *t = fmaf(p, c.x, *t);
  t = ac + col(ix.y >> 8);   *t = fmaf(p, c.y, *t);
  t = ac + col(ix.y >> 16);  *t = fmaf(p, d.x, *t);
  t = ac + col(ix.y >> 24);  *t = fmaf(p, d.y, *t);
}

__device__ __forceinline__ uint4 and4(uint4 a, uint4 m) {
  return make_uint4(a.x & m.x, a.y & m.y, a.z & m.z, a.w & m.w);
}

// Split decode kernel.
//   Shared memory: q' of the unit's G query heads replicated per lane
//   ([G][128][32] fp32) and one lane-private rotated-space accumulator per
//   warp ([8][128][32] fp32).  Both are indexed (coordinate, lane), so the
//   random gathers and scatters of 32 lanes never share a bank.
//   Warp w serves query head w % G; the G warps of a team walk the same
//   32-token groups.  Lane = token.
template <int G, int MAXC>
__global__ void __launch_bounds__(kThreads, 1) decode_kernel(DecodeParams p) {
  constexpr int TEAMS = kWarpsPerCta / G;
  constexpr bool kL1 = G > 1;
  constexpr bool kPreloadV = MAXC <= 8;
  extern __shared__ __align__(16) float smem[];
  float* qrep = smem;                          // [G][128][32]
  float* accs = smem + G * kHeadDim * 32;      // [8][128][32]
  __shared__ float red_m[kWarpsPerCta], red_l[kWarpsPerCta];

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int hh = warp % G, team = warp / G;
  float* my_acc = accs + warp * kHeadDim * 32 + lane;
  const float* my_q = qrep + hh * kHeadDim * 32 + lane;

  const CacheGeom& g = p.geom;
  const int P = g.P;
  const int nchunks = p.k_full_chunks + (p.k_rem ? 1 : 0);
  uint4 remmask = make_uint4(0, 0, 0, 0);
  {
    uint32_t w[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const uint32_t lo = (2 * e < p.k_rem) ? 0xffffu : 0u;
      const uint32_t hi = (2 * e + 1 < p.k_rem) ? 0xffff0000u : 0u;
      w[e] = lo | hi;
    }
    remmask = make_uint4(w[0], w[1], w[2], w[3]);
  }

  const int64_t g_begin = (int64_t)blockIdx.x * p.range;
  const int64_t g_end = min(p.total_groups, g_begin + p.range);
  if (g_begin >= g_end) return;
  const int64_t u_first = g_begin / p.N_g, u_last = (g_end - 1) / p.N_g;

  for (int64_t u = u_first; u <= u_last; ++u) {
    const int64_t s0 = max(g_begin, u * p.N_g) - u * p.N_g;
    const int64_t s1 = min(g_end, (u + 1) * p.N_g) - u * p.N_g;
    const int64_t b = u / p.H_kv, h = u % p.H_kv;

    __syncthreads();  // the previous segment's reduction is done with smem
    for (int i = threadIdx.x; i < G * kHeadDim * 32; i += kThreads) {
      const int gh = i >> 12, dd = (i >> 5) & (kHeadDim - 1);
      qrep[i] = __ldg(p.qprime + ((b * p.H_q + h * G + gh) * kHeadDim + dd));
    }
#pragma unroll 8
    for (int dd = 0; dd < kHeadDim; ++dd) my_acc[dd * 32] = 0.f;
    __syncthreads();

    float m_w = -INFINITY;  // running max (log2 domain), uniform in the warp
    float l_sum = 0.f;      // this lane's sum of exp2(s - m_w)

    for (int64_t gi = s0 + team; gi < s1; gi += TEAMS) {
      float s2;
      bool valid;
      if (gi < p.n_sg) {
        // ---- sparse group: tokens 32*gi .. 32*gi+31 of the sparse history
        const int64_t t0 = gi * 32;
        valid = t0 + lane < p.sparse_len;
        const int64_t page = t0 / P;
        const int slot = (int)(t0 % P) + lane;
        int32_t phys = g.page_table[u * g.pages_per_unit + page];
        if (phys < 0 || phys >= g.num_pages) {
          if (lane == 0) atomicOr(p.status, kStatusPageRange);
          phys = 0;
          valid = false;
        }
        const uint8_t* pg = g.pool + (int64_t)phys * g.page_bytes;
        const uint4* kv = reinterpret_cast<const uint4*>(pg) + slot;
        const uint2* ki = reinterpret_cast<const uint2*>(pg + g.kidx_off()) + slot;
        const uint4* vv = reinterpret_cast<const uint4*>(pg + g.vval_off()) + slot;
        const uint2* vi = reinterpret_cast<const uint2*>(pg + g.vidx_off()) + slot;
        const bool tail = t0 + 32 > p.sparse_len;  // warp-uniform
        const uint4 lanemask = valid ? make_uint4(~0u, ~0u, ~0u, ~0u) : make_uint4(0, 0, 0, 0);

        uint4 kvr[MAXC];
        uint2 kir[MAXC];
        uint4 vvr[kPreloadV ? MAXC : 1];
        uint2 vir[kPreloadV ? MAXC : 1];
#pragma unroll
        for (int c = 0; c < MAXC; ++c) {
          if (c < nchunks) {
            kvr[c] = ld_rec16<kL1>(kv + (int64_t)c * P);
            kir[c] = ld_rec8<kL1>(ki + (int64_t)c * P);
          }
        }
        if constexpr (kPreloadV) {
#pragma unroll
          for (int c = 0; c < MAXC; ++c) {
            if (c < nchunks) {
              vvr[c] = ld_rec16<kL1>(vv + (int64_t)c * P);
              vir[c] = ld_rec8<kL1>(vi + (int64_t)c * P);
            }
          }
        }
        float sa = 0.f, sb = 0.f;
#pragma unroll
        for (int c = 0; c < MAXC; ++c) {
          if (c < nchunks) {
            uint4 v = kvr[c];
            if (p.k_rem && c == nchunks - 1) v = and4(v, remmask);
            if (tail) v = and4(v, lanemask);
            score_chunk(my_q, v, kir[c], sa, sb);
          }
        }
        s2 = valid ? (sa + sb) * p.scale_log2 : -INFINITY;

        const float gmax = warp_max(s2);
        if (gmax > m_w + kLazyRescale) {
          if (m_w != -INFINITY) {
            const float f = exp2f(m_w - gmax);
            l_sum *= f;
#pragma unroll 8
            for (int dd = 0; dd < kHeadDim; ++dd) my_acc[dd * 32] *= f;
          }
          m_w = gmax;
        }
        const float pr = valid ? exp2f(s2 - m_w) : 0.f;
        l_sum += pr;

#pragma unroll
        for (int c = 0; c < MAXC; ++c) {
          if (c < nchunks) {
            uint4 v;
            uint2 ix;
            if constexpr (kPreloadV) {
              v = vvr[c];
              ix = vir[c];
            } else {
              v = ld_rec16<kL1>(vv + (int64_t)c * P);
              ix = ld_rec8<kL1>(vi + (int64_t)c * P);
            }
            if (p.k_rem && c == nchunks - 1) v = and4(v, remmask);
            if (tail) v = and4(v, lanemask);
            value_chunk(my_acc, pr, v, ix);
          }
        }
      } else {
        // ---- buffer group: dense rotated fp16 vectors of the ring buffer
        const int64_t i = (gi - p.n_sg) * 32 + lane;
        valid = i < p.n_b;
        const int slot = valid ? (int)((p.buf_start + i) % p.cap) : 0;
        const size_t row = ((size_t)u * p.cap + slot) * kHeadDim;
        const uint4* kr = reinterpret_cast<const uint4*>(p.ring_k + row);
        const uint4* vr = reinterpret_cast<const uint4*>(p.ring_v + row);
        float sa = 0.f, sb = 0.f;
#pragma unroll 4
        for (int c = 0; c < 16; ++c) {
          const uint4 w = __ldg(kr + c);
          const float2 a = h2f(w.x), bb = h2f(w.y), cc = h2f(w.z), d = h2f(w.w);
          const float* q = my_q + c * 8 * 32;
          sa = fmaf(q[0 * 32], a.x, sa);
          sb = fmaf(q[1 * 32], a.y, sb);
          sa = fmaf(q[2 * 32], bb.x, sa);
          sb = fmaf(q[3 * 32], bb.y, sb);
          sa = fmaf(q[4 * 32], cc.x, sa);
          sb = fmaf(q[5 * 32], cc.y, sb);
          sa = fmaf(q[6 * 32], d.x, sa);
          sb = fmaf(q[7 * 32], d.y, sb);
        }
        s2 = valid ? (sa + sb) * p.scale_log2 : -INFINITY;
        const float gmax = warp_max(s2);
        if (gmax > m_w + kLazyRescale) {
          if (m_w != -INFINITY) {
            const float f = exp2f(m_w - gmax);
            l_sum *= f;
#pragma unroll 8
            for (int dd = 0; dd < kHeadDim; ++dd) my_acc[dd * 32] *= f;
          }
          m_w = gmax;
        }
        const float pr = valid ? exp2f(s2 - m_w) : 0.f;
        l_sum += pr;
        if (valid) {
#pragma unroll 4
          for (int c = 0; c < 16; ++c) {
            const uint4 w = __ldg(vr + c);
            const float2 a = h2f(w.x), bb = h2f(w.y), cc = h2f(w.z), d = h2f(w.w);
            float* t = my_acc + c * 8 * 32;
            t[0 * 32] = fmaf(pr, a.x, t[0 * 32]);
            t[1 * 32] = fmaf(pr, a.y, t[1 * 32]);
            t[2 * 32] = fmaf(pr, bb.x, t[2 * 32]);
            t[3 * 32] = fmaf(pr, bb.y, t[3 * 32]);
            t[4 * 32] = fmaf(pr, cc.x, t[4 * 32]);
            t[5 * 32] = fmaf(pr, cc.y, t[5 * 32]);
            t[6 * 32] = fmaf(pr, d.x, t[6 * 32]);
            t[7 * 32] = fmaf(pr, d.y, t[7 * 32]);
          }
        }
      }
    }

    // ---- merge the lanes and warps of each head into one partial
    l_sum = warp_sum(l_sum);
    if (lane == 0) {
      red_m[warp] = m_w;
      red_l[warp] = l_sum;
    }
    __syncthreads();
    for (int o = threadIdx.x; o < G * kHeadDim; o += kThreads) {
      const int gh = o / kHeadDim, dd = o % kHeadDim;
      float M = -INFINITY;
#pragma unroll
      for (int t = 0; t < TEAMS; ++t) M = fmaxf(M, red_m[t * G + gh]);
      float tot = 0.f, L = 0.f;
#pragma unroll
      for (int t = 0; t < TEAMS; ++t) {
        const int w = t * G + gh;
        const float mw = red_m[w];
        const float f = (mw == -INFINITY) ? 0.f : exp2f(mw - M);
        const float* a = accs + w * kHeadDim * 32 + dd * 32;
        float sum = 0.f;
#pragma unroll 8
        for (int jj = 0; jj < 32; ++jj) sum += a[(jj + dd) & 31];
        tot = fmaf(f, sum, tot);
        L = fmaf(f, red_l[w], L);
      }
      float* dst = p.partials + ((size_t)(blockIdx.x + u) * G + gh) * (kHeadDim + 2);
      dst[2 + dd] = tot;
      if (dd == 0) {
        dst[0] = M;
        dst[1] = L;
      }
    }
  }
}

// q' = q R_qk for every (batch, query head): one CTA per vector, thread j
// computes coordinate j (coalesced rows of R).
__global__ void __launch_bounds__(kHeadDim) rotate_q_kernel(RotateQParams p) {
  __shared__ float qs[kHeadDim];
  const int64_t bq = blockIdx.x;
  const int hq = (int)(bq % p.H_q);
  const int h = hq / p.G;
  const int t = threadIdx.x;
  qs[t] = __half2float(p.q[bq * kHeadDim + t]);
  __syncthreads();
  const float* R = p.R_qk + (size_t)h * kHeadDim * kHeadDim;
  float a0 = 0.f, a1 = 0.f;
#pragma unroll 8
  for (int i = 0; i < kHeadDim; i += 2) {
    a0 = fmaf(qs[i], __ldg(R + i * kHeadDim + t), a0);
    a1 = fmaf(qs[i + 1], __ldg(R + (i + 1) * kHeadDim + t), a1);
  }
  p.qprime[bq * kHeadDim + t] = a0 + a1;
}

// Merge the partials of one (batch, query head), normalise, rotate back by
// R_vo^T and round to fp16.
__global__ void __launch_bounds__(kHeadDim) combine_kernel(CombineParams p) {
  __shared__ float o_hat[kHeadDim];
  const int64_t bq = blockIdx.x;
  const int64_t b = bq / p.H_q;
  const int hq = (int)(bq % p.H_q);
  const int h = hq / p.G, gh = hq % p.G;
  const int64_t u = b * p.H_kv + h;
  const int dd = threadIdx.x;
  float val = 0.f;
  if (p.total_groups > 0) {
    const int64_t c0 = (u * p.N_g) / p.range;
    const int64_t c1 = ((u + 1) * p.N_g - 1) / p.range;
    float M = -INFINITY;
    for (int64_t c = c0; c <= c1; ++c)
      M = fmaxf(M, p.partials[((size_t)(c + u) * p.G + gh) * (kHeadDim + 2)]);
    float L = 0.f, A = 0.f;
    for (int64_t c = c0; c <= c1; ++c) {
      const float* part = p.partials + ((size_t)(c + u) * p.G + gh) * (kHeadDim + 2);
      const float w = (part[0] == -INFINITY) ? 0.f : exp2f(part[0] - M);
      L = fmaf(w, part[1], L);
      A = fmaf(w, part[2 + dd], A);
    }
    val = (L > 0.f) ? A / L : 0.f;
  }
  o_hat[dd] = val;
  __syncthreads();
  const float* RT = p.R_voT + (size_t)h * kHeadDim * kHeadDim;
  float a0 = 0.f, a1 = 0.f;
#pragma unroll 8
  for (int j = 0; j < kHeadDim; j += 2) {
    a0 = fmaf(o_hat[j], __ldg(RT + j * kHeadDim + dd), a0);
    a1 = fmaf(o_hat[j + 1], __ldg(RT + (j + 1) * kHeadDim + dd), a1);
  }
  p.out[bq * kHeadDim + dd] = __float2half_rn(a0 + a1);
}

template <int G, int MAXC>
cudaError_t launch_decode_t(const DecodeParams& p, int grid, cudaStream_t s) {
  static bool attr_set = false;
  const size_t smem = decode_smem_bytes(G);
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(decode_kernel<G, MAXC>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  decode_kernel<G, MAXC><<<grid, kThreads, smem, s>>>(p);
  return cudaGetLastError();
}

template <int G, int MAXC>
int ctas_per_sm_t() {
  const size_t smem = decode_smem_bytes(G);
  if (cudaFuncSetAttribute(decode_kernel<G, MAXC>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)smem) != cudaSuccess)
    return 0;
  int n = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, decode_kernel<G, MAXC>, kThreads, smem) !=
      cudaSuccess)
    return 0;
  return n;
}

}  // namespace

size_t decode_smem_bytes(int G) { return (size_t)(G + kWarpsPerCta) * kHeadDim * 32 * sizeof(float); }

int decode_ctas_per_sm(int G, int k_slots) {
  const bool big = k_slots > 64;
  switch (G) {
    case 1: return big ? ctas_per_sm_t<1, 16>() : ctas_per_sm_t<1, 8>();
    case 2: return big ? ctas_per_sm_t<2, 16>() : ctas_per_sm_t<2, 8>();
    case 4: return big ? ctas_per_sm_t<4, 16>() : ctas_per_sm_t<4, 8>();
    default: return 0;
  }
}

cudaError_t launch_decode(const DecodeParams& p, int G, int k_slots, int grid, cudaStream_t s) {
  const bool big = k_slots > 64;
  switch (G) {
    case 1: return big ? launch_decode_t<1, 16>(p, grid, s) : launch_decode_t<1, 8>(p, grid, s);
    case 2: return big ? launch_decode_t<2, 16>(p, grid, s) : launch_decode_t<2, 8>(p, grid, s);
    case 4: return big ? launch_decode_t<4, 16>(p, grid, s) : launch_decode_t<4, 8>(p, grid, s);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t launch_rotate_q(const RotateQParams& p, int B, cudaStream_t s) {
  rotate_q_kernel<<<(unsigned)((int64_t)B * p.H_q), kHeadDim, 0, s>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_combine(const CombineParams& p, int B, cudaStream_t s) {
  combine_kernel<<<(unsigned)((int64_t)B * p.H_q), kHeadDim, 0, s>>>(p);
  return cudaGetLastError();
}

}  // namespace swan
