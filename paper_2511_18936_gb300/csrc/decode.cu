// Decode attention on the packed sparse cache (Algorithm 1, attention part;
// Section 4.3): the query rotation q' = q R_qk, the empty-cache combine, and
// the host launchers of the kernels in decode_kernels.cuh and decode_mma.cuh.
#include "decode_mma.cuh"

namespace swan {
namespace {

// q' = q R_qk: one CTA per (kv head, up to 8 query vectors of that head,
// 32 of the 128 output coordinates); see rotate_q_slice.
__global__ void __launch_bounds__(kThreads) rotate_q_kernel(RotateQParams p, int B) {
  __shared__ __align__(16) float Rs[kHeadDim * 32];
  pdl_trigger();
  rotate_q_slice(p, B, blockIdx.x, blockIdx.y, blockIdx.z, Rs);
}

// Empty cache: the output is zero (one CTA per query vector).
__global__ void __launch_bounds__(kHeadDim) combine_kernel(CombineParams p) {
  pdl_trigger();
  pdl_wait();
  p.out[(int64_t)blockIdx.x * kHeadDim + threadIdx.x] = __float2half_rn(0.f);
}

// Dynamic shared memory of the one-head kernel: the warps' accumulators and
// one more 16 KB region for the alignment gap, which holds an 8 KB q' unless
// the allocation starts within 8 KB below a 16 KB boundary; a 16 KB q' goes
// after the accumulators.
template <int MAXC>
size_t one_head_smem() {
  const int q_regions = decode_q_shift<MAXC>() == 7 ? 1 : 0;
  return (size_t)(decode_warps<MAXC>() + 1 + q_regions) * kRegionBytes;
}

template <typename K>
int occupancy(K kernel, int threads, size_t smem) {
  if (cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess)
    return 0;
  int n = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, kernel, threads, smem) != cudaSuccess) return 0;
  return n;
}

template <int G, int MAXC, int FMT>
cudaError_t launch_t(const DecodeParams& p, int grid, cudaStream_t s) {
  if constexpr (G == 1) {
    const size_t smem = one_head_smem<MAXC>();
    const cudaError_t e = ensure_smem<decode_kernel<MAXC, FMT>>(smem);
    if (e != cudaSuccess) return e;
    return launch_pdl(decode_kernel<MAXC, FMT>, dim3(grid), dim3(decode_warps<MAXC>() * 32), smem, s, p);
  } else {
    constexpr size_t smem = mma_smem<G, MAXC>();
    const cudaError_t e = ensure_smem<decode_mma_kernel<G, MAXC, FMT>>(smem);
    if (e != cudaSuccess) return e;
    return launch_pdl(decode_mma_kernel<G, MAXC, FMT>, dim3(grid), dim3(mma_warps<MAXC>() * 32), smem, s, p);
  }
}

template <int G, int MAXC>
cudaError_t launch_fmt(const DecodeParams& p, int grid, cudaStream_t s) {
  return p.geom.fmt == kFmtFp8 ? launch_t<G, MAXC, kFmtFp8>(p, grid, s)
                               : launch_t<G, MAXC, kFmtFp16>(p, grid, s);
}

}  // namespace

int decode_ctas_per_sm(int G, int k_read) {
  const bool big = k_read > 64;
  if (G == 1) {
    if (k_read <= 32) return occupancy(decode_kernel<4, kFmtFp16>, decode_warps<4>() * 32, one_head_smem<4>());
    if (k_read <= 64) return occupancy(decode_kernel<8, kFmtFp16>, decode_warps<8>() * 32, one_head_smem<8>());
    if (k_read <= 96)
      return occupancy(decode_kernel<12, kFmtFp16>, decode_warps<12>() * 32, one_head_smem<12>());
    return occupancy(decode_kernel<16, kFmtFp16>, decode_warps<16>() * 32, one_head_smem<16>());
  }
  if (G == 2)
    return big ? occupancy(decode_mma_kernel<2, 16, kFmtFp16>, mma_warps<16>() * 32, mma_smem<2, 16>())
               : occupancy(decode_mma_kernel<2, 8, kFmtFp16>, mma_warps<8>() * 32, mma_smem<2, 8>());
  if (G == 4)
    return big ? occupancy(decode_mma_kernel<4, 16, kFmtFp16>, mma_warps<16>() * 32, mma_smem<4, 16>())
               : occupancy(decode_mma_kernel<4, 8, kFmtFp16>, mma_warps<8>() * 32, mma_smem<4, 8>());
  if (G == 8)
    return big ? occupancy(decode_mma_kernel<8, 16, kFmtFp16>, mma_warps<16>() * 32, mma_smem<8, 16>())
               : occupancy(decode_mma_kernel<8, 8, kFmtFp16>, mma_warps<8>() * 32, mma_smem<8, 8>());
  return 0;
}

cudaError_t launch_decode(const DecodeParams& p, int G, int k_read, int grid, cudaStream_t s) {
  const bool big = k_read > 64;
  switch (G) {
    case 1:
      if (k_read <= 32) return launch_fmt<1, 4>(p, grid, s);
      return k_read <= 64 ? launch_fmt<1, 8>(p, grid, s)
                          : k_read <= 96 ? launch_fmt<1, 12>(p, grid, s) : launch_fmt<1, 16>(p, grid, s);
    case 2: return big ? launch_fmt<2, 16>(p, grid, s) : launch_fmt<2, 8>(p, grid, s);
    case 4: return big ? launch_fmt<4, 16>(p, grid, s) : launch_fmt<4, 8>(p, grid, s);
    case 8: return big ? launch_fmt<8, 16>(p, grid, s) : launch_fmt<8, 8>(p, grid, s);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t launch_rotate_q(const RotateQParams& p, int B, cudaStream_t s) {
  const int vecs = B * p.G;  // query vectors per kv head
  return launch_pdl(rotate_q_kernel,
                    dim3((unsigned)(p.H_q / p.G), (unsigned)((vecs + kWarpsPerCta - 1) / kWarpsPerCta), 4),
                    dim3(kThreads), 0, s, p, B);
}

cudaError_t launch_combine(const CombineParams& p, int B, cudaStream_t s) {
  return launch_pdl(combine_kernel, dim3((unsigned)((int64_t)B * p.H_q)), dim3(kHeadDim), 0, s, p);
}

}  // namespace swan
