// Host entry points of the offline basis construction (swan_basis.h):
// argument checks, TMA tensor maps, launches.
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cstdarg>
#include <cstdio>
#include <mutex>

#include "basis_internal.h"
#include "swan.h"
#include "swan_basis.h"
#include "swan_internal.h"

using namespace swan;

namespace {

swan_status bfail(swan_status s, const char* fmt, ...) __attribute__((format(printf, 2, 3)));
swan_status bfail(swan_status s, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  set_last_error(buf);
  return s;
}

swan_status cuda_err(cudaError_t e, const char* where) {
  return bfail(SWAN_ERR_CUDA, "%s: %s", where, cudaGetErrorString(e));
}

using EncodeTiled = EncodeTiledFn;
EncodeTiled encode_fn() { return tensor_map_encoder(); }

int sm_count() {
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
  return sms;
}

int gram_splits_max(int n_mats) { return std::max(1, kGramMaxCtas / std::max(1, n_mats)); }

bool stride_ok(int64_t s) { return s > 0 && s % 8 == 0 && s < ((int64_t)1 << 36); }

// Validate a vector set; `rows` is set to true when a vector is contiguous.
swan_status check_vectors(const swan_vectors* x, bool* rows) {
  if (!x) return bfail(SWAN_ERR_INVALID_ARG, "vectors is NULL");
  if (!x->data) return bfail(SWAN_ERR_INVALID_ARG, "vectors.data is NULL");
  if ((uintptr_t)x->data % 16) return bfail(SWAN_ERR_INVALID_ARG, "vectors.data must be 16-byte aligned");
  if (x->n_mats < 1 || x->n_mats > 65535)
    return bfail(SWAN_ERR_INVALID_ARG, "n_mats %d out of [1, 65535]", x->n_mats);
  if (x->group < 1 || x->group > 65535)
    return bfail(SWAN_ERR_INVALID_ARG, "group %d out of [1, 65535]", x->group);
  if (x->count < 1 || x->count >= ((int64_t)1 << 31))
    return bfail(SWAN_ERR_INVALID_ARG, "count %lld out of [1, 2^31)", (long long)x->count);
  if (x->stride_coord == 1) {
    *rows = true;
    if (x->count > 1 && !stride_ok(x->stride_pos))
      return bfail(SWAN_ERR_INVALID_ARG, "stride_pos must be a positive multiple of 8 below 2^36");
  } else if (x->stride_pos == 1) {
    *rows = false;
    if (!stride_ok(x->stride_coord))
      return bfail(SWAN_ERR_INVALID_ARG, "stride_coord must be a positive multiple of 8 below 2^36");
  } else {
    return bfail(SWAN_ERR_INVALID_ARG, "either stride_coord or stride_pos must be 1");
  }
  if (x->group > 1 && !stride_ok(x->stride_group))
    return bfail(SWAN_ERR_INVALID_ARG, "stride_group must be a positive multiple of 8 below 2^36");
  if (x->n_mats > 1 && !stride_ok(x->stride_mat))
    return bfail(SWAN_ERR_INVALID_ARG, "stride_mat must be a positive multiple of 8 below 2^36");
  return SWAN_OK;
}

// Stride in bytes for the tensor map of a dimension that may have size 1.
cuuint64_t map_stride(int64_t elems, int64_t size) { return size > 1 ? (cuuint64_t)elems * 2 : 16; }

swan_status make_tmap(const swan_vectors* x, bool rows, CUtensorMap* map) {
  EncodeTiled enc = encode_fn();
  if (!enc) return bfail(SWAN_ERR_CUDA, "cuTensorMapEncodeTiled is not available from the driver");
  cuuint64_t dims[4], strides[3];
  cuuint32_t box[4], estr[4] = {1, 1, 1, 1};
  cuuint32_t rank = 0;
  if (rows) {
    // (coordinate, [group], position, matrix); box 64 coordinates x 64 positions
    dims[rank] = 128, box[rank++] = 64;
    if (x->group > 1) {
      strides[rank - 1] = map_stride(x->stride_group, x->group);
      dims[rank] = (cuuint64_t)x->group, box[rank++] = 1;
    }
    strides[rank - 1] = map_stride(x->stride_pos, x->count);
    dims[rank] = (cuuint64_t)x->count, box[rank++] = 64;
    strides[rank - 1] = map_stride(x->stride_mat, x->n_mats);
    dims[rank] = (cuuint64_t)x->n_mats, box[rank++] = 1;
  } else {
    // (position, coordinate, [group], matrix); box 64 positions x 128 coordinates
    dims[rank] = (cuuint64_t)x->count, box[rank++] = 64;
    strides[rank - 1] = map_stride(x->stride_coord, 128);
    dims[rank] = 128, box[rank++] = 128;
    if (x->group > 1) {
      strides[rank - 1] = map_stride(x->stride_group, x->group);
      dims[rank] = (cuuint64_t)x->group, box[rank++] = 1;
    }
    strides[rank - 1] = map_stride(x->stride_mat, x->n_mats);
    dims[rank] = (cuuint64_t)x->n_mats, box[rank++] = 1;
  }
  const CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, rank, const_cast<void*>(x->data), dims, strides,
                         box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                         CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return bfail(SWAN_ERR_INVALID_ARG, "cuTensorMapEncodeTiled rejected the layout (%d)", (int)r);
  return SWAN_OK;
}

}  // namespace

EncodeTiledFn swan::tensor_map_encoder() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  });
  return fn;
}

extern "C" {

size_t swan_gram_workspace_bytes(int n_mats) {
  if (n_mats < 1) return 0;
  return (size_t)n_mats * gram_splits_max(n_mats) * 128 * 128 * sizeof(float) + 256;
}

swan_status swan_gram(const swan_vectors* x, float* gram, int accumulate, void* workspace,
                      size_t workspace_bytes, void* stream) {
  bool rows = false;
  swan_status st = check_vectors(x, &rows);
  if (st != SWAN_OK) return st;
  if (!gram) return bfail(SWAN_ERR_INVALID_ARG, "gram is NULL");
  if (!workspace || (uintptr_t)workspace % 256)
    return bfail(SWAN_ERR_INVALID_ARG, "workspace must be a 256-byte aligned device pointer");
  if (workspace_bytes < swan_gram_workspace_bytes(x->n_mats))
    return bfail(SWAN_ERR_INVALID_ARG, "workspace of %zu bytes is smaller than the %zu needed", workspace_bytes,
                 swan_gram_workspace_bytes(x->n_mats));
  CUtensorMap map;
  st = make_tmap(x, rows, &map);
  if (st != SWAN_OK) return st;
  const int sms = std::max(1, sm_count());
  GramParams p{};
  p.status = reinterpret_cast<uint32_t*>(workspace);
  p.partials = reinterpret_cast<float*>(static_cast<char*>(workspace) + 256);
  p.n_mats = x->n_mats;
  p.group = x->group;
  p.chunks = (x->count + 63) / 64;
  const int64_t items = p.chunks * x->group;
  // two CTAs per SM over all matrices, at most one item per CTA
  const int64_t want = std::max<int64_t>(1, (2 * sms + x->n_mats - 1) / x->n_mats);
  p.splits = (int)std::min<int64_t>({want, items, (int64_t)gram_splits_max(x->n_mats)});
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  cudaError_t e = cudaMemsetAsync(p.status, 0, sizeof(uint32_t), s);
  if (e != cudaSuccess) return cuda_err(e, "cudaMemsetAsync");
  if (const int64_t starve_ns = take_tc_starve()) {
    p.starve = 1;
    p.wait_ns = (uint64_t)starve_ns;
  }
  e = launch_gram(map, p, rows, s);
  if (e != cudaSuccess) return cuda_err(e, "gram kernel launch");
  e = launch_gram_reduce(p.partials, gram, p.n_mats, p.splits, accumulate, s);
  if (e != cudaSuccess) return cuda_err(e, "gram reduce launch");
  return SWAN_OK;
}

swan_status swan_basis_eig(const float* gram, int n_mats, float* R, float* lambda, int* sweeps, void* stream) {
  if (!gram || !R) return bfail(SWAN_ERR_INVALID_ARG, "gram and R must not be NULL");
  if (n_mats < 1 || n_mats > 65535) return bfail(SWAN_ERR_INVALID_ARG, "n_mats %d out of [1, 65535]", n_mats);
  EigParams p{};
  p.gram = gram;
  p.R = R;
  p.lambda = lambda;
  p.sweeps = sweeps;
  p.max_sweeps = 40;
  p.tol = 2e-7f;
  const cudaError_t e = launch_jacobi_eig(p, n_mats, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_err(e, "eigensolver launch");
  return SWAN_OK;
}

swan_status swan_energy(const swan_vectors* x, const float* R, double* energy, int accumulate, void* stream) {
  bool rows = false;
  swan_status st = check_vectors(x, &rows);
  if (st != SWAN_OK) return st;
  if (!R || !energy) return bfail(SWAN_ERR_INVALID_ARG, "R and energy must not be NULL");
  if (rows && (x->stride_pos % 8 && x->count > 1))
    return bfail(SWAN_ERR_INVALID_ARG, "stride_pos must be a multiple of 8");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (!accumulate) {
    const cudaError_t e = cudaMemsetAsync(energy, 0, (size_t)x->n_mats * 129 * sizeof(double), s);
    if (e != cudaSuccess) return cuda_err(e, "cudaMemsetAsync");
  }
  EnergyParams p{};
  p.data = static_cast<const __half*>(x->data);
  p.s_m = x->stride_mat;
  p.s_g = x->stride_group;
  p.s_p = x->stride_pos;
  p.s_i = x->stride_coord;
  p.group = x->group;
  p.count = x->count;
  p.R = R;
  p.energy = energy;
  const cudaError_t e = launch_energy(p, x->n_mats, std::max(1, sm_count()), s);
  if (e != cudaSuccess) return cuda_err(e, "energy kernel launch");
  return SWAN_OK;
}

swan_status swan_basis_check(void* workspace, void* stream) {
  if (!workspace) return bfail(SWAN_ERR_INVALID_ARG, "workspace is NULL");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  uint32_t status = 0;
  cudaError_t e = cudaMemcpyAsync(&status, workspace, sizeof(status), cudaMemcpyDeviceToHost, s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return cuda_err(e, "reading the workspace status");
  if (status) {
    const uint32_t zero = 0;
    e = cudaMemcpyAsync(workspace, &zero, sizeof(zero), cudaMemcpyHostToDevice, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return cuda_err(e, "clearing the workspace status");
    if (status & kBasisStatusTimeout)
      return bfail(SWAN_ERR_DEVICE_TIMEOUT, "a tensor-core pipeline wait gave up (status 0x%x)", status);
  }
  return SWAN_OK;
}

}  // extern "C"
