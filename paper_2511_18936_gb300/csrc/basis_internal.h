// Internal interfaces of the offline-basis kernels (basis.cu) and their
// host entry points (basis_api.cpp).
#pragma once

#include <cuda.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include <cstdint>

namespace swan {

constexpr uint32_t kBasisStatusTimeout = 1u << 0;  // a barrier wait gave up

// Upper bound on split CTAs per call of the Gram kernel (sets the workspace).
constexpr int kGramMaxCtas = 320;

struct GramParams {
  float* partials;   // [n_mats][splits][128][128]
  uint32_t* status;
  int n_mats, splits, group;
  int64_t chunks;    // 64-position chunks per (matrix, group member)
  // test hook (swan_debug_starve_tc): no copies are issued, so the MMA
  // warp's barrier wait runs out after wait_ns (0: the default 2 s)
  int starve;
  uint64_t wait_ns;
};

struct EigParams {
  const float* gram;  // [n][128][128]
  float* R;           // [n][128][128]
  float* lambda;      // [n][128] or null
  int* sweeps;        // [n] or null
  int max_sweeps;
  float tol;
};

struct EnergyParams {
  const __half* data;
  int64_t s_m, s_g, s_p, s_i;
  int group;
  int64_t count;
  const float* R;     // [n_mats][128][128]
  double* energy;     // [n_mats][129]
};

size_t gram_smem_bytes();
cudaError_t launch_gram(const CUtensorMap& tmap, const GramParams& p, bool mn_major, cudaStream_t s);
cudaError_t launch_gram_reduce(const float* partials, float* gram, int n_mats, int splits, int accumulate,
                               cudaStream_t s);
cudaError_t launch_jacobi_eig(const EigParams& p, int n_mats, cudaStream_t s);
cudaError_t launch_energy(const EnergyParams& p, int n_mats, int sms, cudaStream_t s);

}  // namespace swan
