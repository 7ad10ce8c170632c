// Offline basis construction (Section 4.1): the Gram matrices S^T S of the
// joint matrices S_QK = Concat(Q_grouped, K) and S_VO = Concat(V, W_O^T)
// on the tensor cores (tcgen05.mma, operands staged by TMA, accumulators in
// tensor memory), their eigenvectors (= the right singular vectors of S) by
// parallel cyclic Jacobi, and the energy that per-vector top-k pruning
// (Algorithm 1) keeps in a given basis.
#include <cuda.h>

#include <algorithm>

#include "basis_internal.h"
#include "sm100.h"

namespace swan {
namespace {

using namespace sm100;

constexpr int kGramStages = 6;
constexpr uint32_t kStageBytes = 16384;  // 64 positions x 128 coordinates fp16
constexpr uint64_t kWaitLimitNs = 2000000000ull;  // 2 s per barrier wait

// ---------------------------------------------------------------------------
// Gram partials: CTA (split s, matrix m) accumulates sum_v v v^T over its
// range of 64-vector items into TMEM (128 x 128 fp32) and writes the partial.
//   ROWS (kMnMajor): a vector is 128 contiguous fp16; a stage holds
//     [2 coordinate halves][64 vectors][64 coordinates], rows of 128 B with
//     the 128-byte swizzle: A = X^T and B = X are both MN-major.
//   COLS: a vector is a column of a [128][count] block; a stage holds
//     [128 coordinates][64 positions]: A = B^T... both operands K-major.
// 4 warps: warp 0 lane 0 issues TMA, warp 1 owns TMEM and lane 0 issues the
// MMAs, all four drain TMEM (warp w: rows 32w .. 32w + 31).
// ---------------------------------------------------------------------------
template <bool kMnMajor>
__global__ void __launch_bounds__(128, 1) gram_kernel(const __grid_constant__ CUtensorMap tmap, GramParams p) {
  extern __shared__ __align__(1024) unsigned char smem_tc[];
  __shared__ __align__(8) uint64_t bars[2 * kGramStages + 1];
  __shared__ uint32_t tmem_base_slot;
  __shared__ int abort_flag;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t raw = smem_u32(smem_tc);
  const uint32_t tiles = (raw + 1023u) & ~1023u;
  const uint32_t full0 = smem_u32(&bars[0]), empty0 = smem_u32(&bars[kGramStages]);
  const uint32_t done = smem_u32(&bars[2 * kGramStages]);

  const int m = blockIdx.y, split = blockIdx.x;
  const int64_t items = (int64_t)p.group * p.chunks;
  const int64_t it0 = items * split / p.splits, it1 = items * (split + 1) / p.splits;
  const int n = (int)(it1 - it0);

  if (threadIdx.x == 0) {
    for (int s = 0; s < kGramStages; ++s) {
      mbar_init(full0 + 8 * s, 1);
      mbar_init(empty0 + 8 * s, 1);
    }
    mbar_init(done, 1);
    abort_flag = 0;
    fence_barrier_init();
    prefetch_tmap(&tmap);
  }
  if (warp == 1) tmem_alloc(smem_u32(&tmem_base_slot), 128);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_base_slot;
  const uint64_t wait_ns = p.wait_ns ? p.wait_ns : kWaitLimitNs;

  if (warp == 0 && lane == 0 && n > 0 && !p.starve) {
    // ---- producer
    int issued = 0;
    for (int i = 0; i < n; ++i) {
      const int s = i % kGramStages, round = i / kGramStages;
      if (round > 0 && !mbar_wait(empty0 + 8 * s, (round - 1) & 1, wait_ns)) {
        atomicOr(p.status, kBasisStatusTimeout);
        abort_flag = 1;
        break;
      }
      if (*(volatile int*)&abort_flag) break;
      const int64_t it = it0 + i;
      const int g = (int)(it / p.chunks);
      const int pos = (int)((it % p.chunks) * 64);
      const uint32_t dst = tiles + s * kStageBytes;
      mbar_arrive_expect_tx(full0 + 8 * s, kStageBytes);
      if (kMnMajor) {
        if (p.group > 1) {
          tma_load_4d(dst, &tmap, full0 + 8 * s, 0, g, pos, m);
          tma_load_4d(dst + kStageBytes / 2, &tmap, full0 + 8 * s, 64, g, pos, m);
        } else {
          tma_load_3d(dst, &tmap, full0 + 8 * s, 0, pos, m);
          tma_load_3d(dst + kStageBytes / 2, &tmap, full0 + 8 * s, 64, pos, m);
        }
      } else {
        if (p.group > 1)
          tma_load_4d(dst, &tmap, full0 + 8 * s, pos, 0, g, m);
        else
          tma_load_3d(dst, &tmap, full0 + 8 * s, pos, 0, m);
      }
      ++issued;
    }
    // copies still in flight must land before the CTA can exit
    for (int i = max(0, issued - kGramStages); i < issued; ++i)
      mbar_wait(full0 + 8 * (i % kGramStages), (i / kGramStages) & 1, wait_ns);
  } else if (warp == 1 && lane == 0 && n > 0) {
    // ---- MMA issuer
    constexpr uint32_t idesc = idesc_f16_f32(128, 128, kMnMajor ? 1 : 0, kMnMajor ? 1 : 0);
    bool ok = true;
    for (int i = 0; i < n && ok; ++i) {
      const int s = i % kGramStages, round = i / kGramStages;
      if (!mbar_wait(full0 + 8 * s, round & 1, wait_ns)) {
        atomicOr(p.status, kBasisStatusTimeout);
        abort_flag = 1;
        ok = false;
        break;
      }
      tc_fence_after();
      const uint32_t base = tiles + s * kStageBytes;
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) {
        // K = 16 vectors per instruction
        const uint64_t desc = kMnMajor ? sdesc_sw128(base + kk * 2048, kStageBytes / 2, 1024)
                                       : sdesc_sw128(base + kk * 32, 16, 1024);
        mma_f16(tmem, desc, desc, idesc, (i | kk) != 0);
      }
      mma_commit(empty0 + 8 * s);
    }
    mma_commit(done);
  }
  __syncwarp();

  // ---- epilogue: TMEM row (32 warp + lane) -> partial row
  const int row = 32 * warp + lane;
  float* dst = p.partials + (((size_t)m * p.splits + split) * 128 + row) * 128;
  if (n > 0 && !mbar_wait(done, 0, wait_ns)) {
    atomicOr(p.status, kBasisStatusTimeout);
    abort_flag = 1;
  }
  tc_fence_after();
  __syncthreads();
  const bool have = n > 0 && *(volatile int*)&abort_flag == 0;  // uniform in the CTA
  if (have) {
#pragma unroll 1
    for (int c = 0; c < 4; ++c) {
      uint32_t r[32];
      tmem_ld32(tmem + ((uint32_t)(32 * warp) << 16) + c * 32, r);
      tmem_wait_ld();
#pragma unroll
      for (int q = 0; q < 8; ++q)
        reinterpret_cast<float4*>(dst + c * 32)[q] =
            make_float4(__uint_as_float(r[4 * q]), __uint_as_float(r[4 * q + 1]),
                        __uint_as_float(r[4 * q + 2]), __uint_as_float(r[4 * q + 3]));
    }
  } else {
    for (int c = 0; c < 32; ++c) reinterpret_cast<float4*>(dst)[c] = make_float4(0.f, 0.f, 0.f, 0.f);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) tmem_dealloc(tmem, 128);
}

// gram[m] = (accumulate ? gram[m] : 0) + sum over splits in a fixed order.
// A block takes 32 consecutive entries; its 8 warps take the splits
// s = w, w + 8, ... (many independent loads in flight), then warp 0 adds
// the 8 warp sums in order.  fp32 throughout (fp64 arithmetic is slow on
// this part); each entry sees at most splits / 8 + 9 additions.
constexpr int kReduceGroups = 8;
__global__ void __launch_bounds__(32 * kReduceGroups) gram_reduce_kernel(const float* partials, float* gram,
                                                                         int splits, int accumulate) {
  __shared__ float part[kReduceGroups][32];
  const int m = blockIdx.y;
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int e = blockIdx.x * 32 + lane;  // < 16384
  const float* src = partials + (size_t)m * splits * 16384 + e;
  float acc = 0.f;
#pragma unroll 4
  for (int s = w; s < splits; s += kReduceGroups) acc += __ldg(src + (size_t)s * 16384);
  part[w][lane] = acc;
  __syncthreads();
  if (w == 0) {
    float tot = accumulate ? gram[(size_t)m * 16384 + e] : 0.f;
#pragma unroll
    for (int g = 0; g < kReduceGroups; ++g) tot += part[g][lane];
    gram[(size_t)m * 16384 + e] = tot;
  }
}

// ---------------------------------------------------------------------------
// Symmetric eigensolver: one CTA per 128 x 128 matrix, parallel cyclic Jacobi
// (round-robin ordering: 64 disjoint rotations per round, 127 rounds per
// sweep), fp32 in shared memory.  Rotation of pair (p, q): Golub and Van
// Loan's symmetric 2 x 2 Schur decomposition; A <- J^T A J, V <- V J.
// Output: eigenvalues in decreasing order and R[:, r] = the matching unit
// eigenvector, sign-fixed so that its largest-magnitude coordinate is
// positive.
// ---------------------------------------------------------------------------
constexpr int kEigThreads = 1024;
constexpr int kLd = 129;  // padded row length

__device__ __forceinline__ int rr_player(int pos, int round) {
  return pos == 0 ? 0 : ((pos - 1 + round) % 127) + 1;
}

__global__ void __launch_bounds__(kEigThreads, 1) jacobi_eig_kernel(EigParams p) {
  extern __shared__ float es[];
  float* A = es;                 // [128][129]
  float* V = A + 128 * kLd;      // [128][129], then a third [128][129]
  __shared__ float cs[64], sn[64], dpp[64], dqq[64];
  __shared__ int pp[64], qq[64];
  __shared__ int rotated;
  __shared__ float lam[128];
  __shared__ int rank[128];

  const int mtx = blockIdx.x;
  const float* G = p.gram + (size_t)mtx * 16384;
  for (int e = threadIdx.x; e < 16384; e += kEigThreads) {
    const int i = e >> 7, j = e & 127;
    A[i * kLd + j] = 0.5f * (G[i * 128 + j] + G[j * 128 + i]);
    V[i * kLd + j] = (i == j) ? 1.f : 0.f;
  }
  __syncthreads();

  int sweep = 0;
  bool converged = false;
  for (; sweep < p.max_sweeps && !converged; ++sweep) {
    if (threadIdx.x == 0) rotated = 0;
    __syncthreads();
    for (int round = 0; round < 127; ++round) {
      if (threadIdx.x < 64) {
        const int i = threadIdx.x;
        int a = rr_player(i, round), b = rr_player(127 - i, round);
        if (a > b) { const int t = a; a = b; b = t; }
        const float app = A[a * kLd + a], aqq = A[b * kLd + b], apq = A[a * kLd + b];
        float c = 1.f, s = 0.f;
        float t = 0.f;
        if (apq != 0.f && fabsf(apq) > p.tol * sqrtf(fabsf(app)) * sqrtf(fabsf(aqq))) {
          const float tau = (aqq - app) / (2.f * apq);
          t = (tau >= 0.f ? 1.f : -1.f) / (fabsf(tau) + sqrtf(1.f + tau * tau));
          c = 1.f / sqrtf(1.f + t * t);
          s = t * c;
          rotated = 1;
        }
        cs[i] = c;
        sn[i] = s;
        pp[i] = a;
        qq[i] = b;
        // the rotated pair's new diagonal (the (p, q) entry becomes zero)
        dpp[i] = app - t * apq;
        dqq[i] = aqq + t * apq;
      }
      __syncthreads();
      // A <- J^T A J as 64 x 64 independent 2 x 2 blocks (rows of pair i,
      // columns of pair j), and V <- V J; one pass, no intermediate barrier.
      for (int e = threadIdx.x; e < 64 * 64; e += kEigThreads) {
        const int i = e >> 6, j = e & 63;
        const float si = sn[i], sj = sn[j];
        if (si == 0.f && sj == 0.f) continue;
        const int ai = pp[i], bi = qq[i], aj = pp[j], bj = qq[j];
        if (i == j) {
          // the rotated pair's own block becomes diagonal
          A[ai * kLd + ai] = dpp[i];
          A[bi * kLd + bi] = dqq[i];
          A[ai * kLd + bi] = 0.f;
          A[bi * kLd + ai] = 0.f;
          continue;
        }
        const float ci = cs[i], cj = cs[j];
        const float x00 = A[ai * kLd + aj], x01 = A[ai * kLd + bj];
        const float x10 = A[bi * kLd + aj], x11 = A[bi * kLd + bj];
        // rows: J_i^T X
        const float r00 = ci * x00 - si * x10, r01 = ci * x01 - si * x11;
        const float r10 = si * x00 + ci * x10, r11 = si * x01 + ci * x11;
        // columns: (J_i^T X) J_j
        A[ai * kLd + aj] = cj * r00 - sj * r01;
        A[ai * kLd + bj] = sj * r00 + cj * r01;
        A[bi * kLd + aj] = cj * r10 - sj * r11;
        A[bi * kLd + bj] = sj * r10 + cj * r11;
      }
      for (int e = threadIdx.x; e < 128 * 64; e += kEigThreads) {
        const int k = e >> 6, j = e & 63;
        const float sj = sn[j];
        if (sj == 0.f) continue;
        const int aj = pp[j], bj = qq[j];
        const float cj = cs[j];
        const float u = V[k * kLd + aj], w = V[k * kLd + bj];
        V[k * kLd + aj] = cj * u - sj * w;
        V[k * kLd + bj] = sj * u + cj * w;
      }
      __syncthreads();
    }
    converged = rotated == 0;
    __syncthreads();
  }

  // eigenvalues, then one Newton-Schulz step V <- V (3 I - V^T V) / 2 to
  // restore orthogonality lost to fp32 rounding over the rotations
  if (threadIdx.x < 128) lam[threadIdx.x] = A[threadIdx.x * kLd + threadIdx.x];
  float* T = V + 128 * kLd;  // [128][129]
  __syncthreads();
  for (int e = threadIdx.x; e < 16384; e += kEigThreads) {
    const int i = e >> 7, j = e & 127;
    float acc = 0.f;
    for (int k = 0; k < 128; ++k) acc = fmaf(V[k * kLd + i], V[k * kLd + j], acc);
    T[i * kLd + j] = acc;
  }
  __syncthreads();
  for (int e = threadIdx.x; e < 16384; e += kEigThreads) {
    const int i = e >> 7, j = e & 127;
    float acc = 0.f;
    for (int k = 0; k < 128; ++k) acc = fmaf(V[i * kLd + k], T[k * kLd + j], acc);
    A[i * kLd + j] = acc;
  }
  __syncthreads();
  for (int e = threadIdx.x; e < 16384; e += kEigThreads) {
    const int i = e >> 7, j = e & 127;
    V[i * kLd + j] = 1.5f * V[i * kLd + j] - 0.5f * A[i * kLd + j];
  }
  // sort by decreasing eigenvalue (ties: lower index first)
  __syncthreads();
  if (threadIdx.x < 128) {
    const int i = threadIdx.x;
    int r = 0;
    for (int j = 0; j < 128; ++j) r += (lam[j] > lam[i]) || (lam[j] == lam[i] && j < i);
    rank[i] = r;
  }
  __syncthreads();
  float* R = p.R + (size_t)mtx * 16384;
  if (threadIdx.x < 128) {
    const int i = threadIdx.x;
    // sign rule on column i of V
    int lead = 0;
    float best = -1.f;
    for (int k = 0; k < 128; ++k) {
      const float a = fabsf(V[k * kLd + i]);
      if (a > best) { best = a; lead = k; }
    }
    const float sg = V[lead * kLd + i] < 0.f ? -1.f : 1.f;
    const int r = rank[i];
    for (int k = 0; k < 128; ++k) R[k * 128 + r] = sg * V[k * kLd + i];
    if (p.lambda) p.lambda[(size_t)mtx * 128 + r] = lam[i];
  }
  if (threadIdx.x == 0 && p.sweeps) p.sweeps[mtx] = converged ? sweep : -1;
}

// ---------------------------------------------------------------------------
// Energy kept by top-k pruning: lane = vector; x_hat = x R (fp32, R in shared
// memory), squares staged per warp, then per vector a warp sorts the 128
// squares (bitonic, descending) and adds the prefix sums to per-lane fp64
// totals; one fp64 atomic per (CTA, k) at the end.
// ---------------------------------------------------------------------------
constexpr int kEnergyThreads = 256;

__device__ __forceinline__ void sort128_desc_u32(uint32_t (&k)[4], int lane) {
  // element index e = 4 * lane + j
#pragma unroll
  for (int size = 2; size <= 128; size <<= 1) {
#pragma unroll
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      if (stride >= 4) {
        const int lstride = stride >> 2;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const int e = 4 * lane + j;
          const uint32_t other = __shfl_xor_sync(0xffffffffu, k[j], lstride);
          const bool desc = (e & size) == 0;
          const bool lower = (e & stride) == 0;
          const bool keep_max = desc == lower;
          k[j] = keep_max ? max(k[j], other) : min(k[j], other);
        }
      } else {
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          if ((j & stride) == 0) {
            const int e = 4 * lane + j;
            const bool desc = (e & size) == 0;
            const uint32_t a = k[j], b = k[j + stride];
            k[j] = desc ? max(a, b) : min(a, b);
            k[j + stride] = desc ? min(a, b) : max(a, b);
          }
        }
      }
    }
  }
}

__global__ void __launch_bounds__(kEnergyThreads, 1) energy_kernel(EnergyParams p) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  float* Rs = reinterpret_cast<float*>(smem_raw);                      // [128][128]
  float* sq = Rs + 128 * 128;                                          // [256 vectors][129]
  const int m = blockIdx.y;
  const float* R = p.R + (size_t)m * 16384;
  for (int e = threadIdx.x; e < 16384 / 4; e += kEnergyThreads)
    reinterpret_cast<float4*>(Rs)[e] = __ldg(reinterpret_cast<const float4*>(R) + e);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  double tot[4] = {0.0, 0.0, 0.0, 0.0};
  const int64_t nvec = (int64_t)p.group * p.count;
  __syncthreads();

  for (int64_t base = (int64_t)blockIdx.x * kEnergyThreads; base < nvec;
       base += (int64_t)gridDim.x * kEnergyThreads) {
    const int64_t v = base + threadIdx.x;
    const bool valid = v < nvec;
    float x[128];
    if (valid) {
      const int64_t g = v / p.count, pos = v % p.count;
      const __half* src = p.data + m * p.s_m + g * p.s_g + pos * p.s_p;
      if (p.s_i == 1) {
#pragma unroll
        for (int c = 0; c < 16; ++c) {
          const uint4 w = __ldg(reinterpret_cast<const uint4*>(src) + c);
          const __half2* h = reinterpret_cast<const __half2*>(&w);
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const float2 f = __half22float2(h[e]);
            x[8 * c + 2 * e] = f.x;
            x[8 * c + 2 * e + 1] = f.y;
          }
        }
      } else {
#pragma unroll
        for (int i = 0; i < 128; ++i) x[i] = __half2float(src[i * p.s_i]);
      }
    } else {
#pragma unroll
      for (int i = 0; i < 128; ++i) x[i] = 0.f;
    }
    float* my = sq + threadIdx.x * 129;
#pragma unroll 1
    for (int cb = 0; cb < 4; ++cb) {
      float acc[32];
#pragma unroll
      for (int j = 0; j < 32; ++j) acc[j] = 0.f;
#pragma unroll
      for (int i = 0; i < 128; ++i) {
        const float4* Rrow = reinterpret_cast<const float4*>(Rs + i * 128 + cb * 32);
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          const float4 r = Rrow[q];
          acc[4 * q + 0] = fmaf(x[i], r.x, acc[4 * q + 0]);
          acc[4 * q + 1] = fmaf(x[i], r.y, acc[4 * q + 1]);
          acc[4 * q + 2] = fmaf(x[i], r.z, acc[4 * q + 2]);
          acc[4 * q + 3] = fmaf(x[i], r.w, acc[4 * q + 3]);
        }
      }
#pragma unroll
      for (int j = 0; j < 32; ++j) my[cb * 32 + j] = acc[j] * acc[j];
    }
    __syncwarp();
    // per vector of this warp: sort, prefix-sum, accumulate
    const int64_t wbase = base + warp * 32;
#pragma unroll 1
    for (int t = 0; t < 32; ++t) {
      if (wbase + t >= nvec) break;
      const float* row = sq + (warp * 32 + t) * 129;
      uint32_t k4[4];
#pragma unroll
      for (int j = 0; j < 4; ++j) k4[j] = __float_as_uint(row[4 * lane + j]);
      sort128_desc_u32(k4, lane);
      float run[4];
      run[0] = __uint_as_float(k4[0]);
#pragma unroll
      for (int j = 1; j < 4; ++j) run[j] = run[j - 1] + __uint_as_float(k4[j]);
      // exclusive scan of the lane totals
      float incl = run[3];
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const float y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += y;
      }
      const float excl = incl - run[3];
#pragma unroll
      for (int j = 0; j < 4; ++j) tot[j] += (double)(excl + run[j]);
    }
    __syncwarp();
  }
  // E[k] for k = 4 lane + j + 1
  double* E = p.energy + (size_t)m * 129;
#pragma unroll
  for (int j = 0; j < 4; ++j) atomicAdd(E + 4 * lane + j + 1, tot[j]);
}

}  // namespace

// ---------------------------------------------------------------------------
// Launchers
// ---------------------------------------------------------------------------

size_t gram_smem_bytes() { return (size_t)kGramStages * kStageBytes + 1024; }

cudaError_t launch_gram(const CUtensorMap& tmap, const GramParams& p, bool mn_major, cudaStream_t s) {
  const dim3 grid(p.splits, p.n_mats);
  const size_t smem = gram_smem_bytes();
  if (mn_major) {
    cudaError_t e = cudaFuncSetAttribute(gram_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    gram_kernel<true><<<grid, 128, smem, s>>>(tmap, p);
  } else {
    cudaError_t e = cudaFuncSetAttribute(gram_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    gram_kernel<false><<<grid, 128, smem, s>>>(tmap, p);
  }
  return cudaGetLastError();
}

cudaError_t launch_gram_reduce(const float* partials, float* gram, int n_mats, int splits, int accumulate,
                               cudaStream_t s) {
  gram_reduce_kernel<<<dim3(16384 / 32, n_mats), 32 * kReduceGroups, 0, s>>>(partials, gram, splits, accumulate);
  return cudaGetLastError();
}

cudaError_t launch_jacobi_eig(const EigParams& p, int n_mats, cudaStream_t s) {
  const size_t smem = 3 * 128 * kLd * sizeof(float);
  cudaError_t e = cudaFuncSetAttribute(jacobi_eig_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  jacobi_eig_kernel<<<n_mats, kEigThreads, smem, s>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_energy(const EnergyParams& p, int n_mats, int sms, cudaStream_t s) {
  const size_t smem = (128 * 128 + kEnergyThreads * 129) * sizeof(float);
  cudaError_t e = cudaFuncSetAttribute(energy_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  const int64_t nvec = (int64_t)p.group * p.count;
  const int64_t want = (nvec + kEnergyThreads - 1) / kEnergyThreads;
  const int per_mat = (int)std::max<int64_t>(1, std::min<int64_t>(want, std::max(1, sms / std::max(1, n_mats))));
  energy_kernel<<<dim3(per_mat, n_mats), kEnergyThreads, smem, s>>>(p);
  return cudaGetLastError();
}

}  // namespace swan
