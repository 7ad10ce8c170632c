/*
 * swan_basis.h -- C ABI of libswan's offline basis construction (Section 4.1
 * of "SWAN: Sparse Winnowed Attention", arXiv 2511.18936).
 *
 * For each kv head j the paper forms two joint matrices by concatenating, along
 * the sequence dimension, the vectors that interact in attention:
 *   S_QK[j] = Concat(Q_grouped[j], K[j])   (query heads jG .. jG+G-1 and key
 *                                           head j, after RoPE; Section 4.1.1)
 *   S_VO[j] = Concat(V[j], W_O_grouped[j]^T) (value head j and the d_model
 *                                           columns of the [d_h][d_model]
 *                                           output-projection slices of those
 *                                           query heads)
 * and takes P = SVD(S)_V, the right singular vectors in order of decreasing
 * singular value (Section 4.1.2).  The library computes the same basis as the
 * eigenvectors of the Gram matrix S^T S:
 *
 *   swan_gram        accumulate S^T S over sets of vectors (tensor cores)
 *   swan_basis_eig   eigenvectors and eigenvalues of the Gram matrices
 *   swan_energy      energy kept by per-vector top-k pruning (Algorithm 1)
 *                    in a given basis, for every k at once
 *
 * A set of vectors is described by swan_vectors: coordinate i (0..127) of
 * vector (matrix m, group member g, position p) is the fp16 element
 *   data[m * stride_mat + g * stride_group + p * stride_pos + i * stride_coord]
 * with either stride_coord == 1 (a vector is 128 contiguous values: query,
 * key and value activations) or stride_pos == 1 (a vector is a column of a
 * [128][count] block: slices of W_O).  Examples, d = 128:
 *   Q as [N_q][n][d], grouped for kv head m: n_mats = N_kv, group = G,
 *     count = n, stride_mat = G n d, stride_group = n d, stride_pos = d,
 *     stride_coord = 1;
 *   K or V as [N_kv][n][d]: group = 1, stride_mat = n d, stride_pos = d;
 *   W_O as [N_q d][d_model] row-major: group = G, count = d_model,
 *     stride_mat = G d d_model, stride_group = d d_model, stride_pos = 1,
 *     stride_coord = d_model.
 * Requirements: data 16-byte aligned; every stride other than the unit one a
 * positive multiple of 8 elements below 2^36 (ignored for a dimension of
 * size 1); 1 <= n_mats, group <= 65535; 1 <= count < 2^31.
 *
 * Conventions: as in swan.h (device pointers on the current device, work
 * enqueued on `stream` asynchronously, host-side argument checks before any
 * launch, nothing thrown).  These calls allocate no device memory: swan_gram
 * takes a caller-provided workspace.  None of them needs a swan_ctx.
 */
#ifndef SWAN_BASIS_H
#define SWAN_BASIS_H

#include <stddef.h>
#include <stdint.h>

#include "swan.h"

#ifdef __cplusplus
extern "C" {
#endif

typedef struct {
  const void* data;       /* device, fp16 */
  int n_mats;             /* Gram matrices (kv heads) */
  int group;              /* vectors per (matrix, position) */
  int64_t count;          /* positions */
  int64_t stride_mat;     /* element strides, see above */
  int64_t stride_group;
  int64_t stride_pos;
  int64_t stride_coord;
} swan_vectors;

/* Device status bits that swan_basis_check reports. */
#define SWAN_BASIS_STATUS_TIMEOUT 1u /* a pipeline wait gave up (2 s); results invalid */

/* Bytes of workspace swan_gram needs for `n_mats` matrices (at most ~21 MB
 * plus 64 KB per matrix beyond 320). */
size_t swan_gram_workspace_bytes(int n_mats);

/*
 * Gram matrices of the vector sets (Section 4.1.2: S^T S of the joint matrix,
 * whose eigenvectors are SVD(S)_V):
 *   gram[m][i][j] (+)= sum over g, p of x[m,g,p,i] * x[m,g,p,j]
 * gram: device fp32 [n_mats][128][128] row-major; accumulate != 0 adds to its
 * contents (call once per part of a joint matrix: Q then K, or V then W_O),
 * 0 overwrites.  Products are exact (fp16 x fp16) and summed in fp32 on the
 * tensor cores (tcgen05.mma, kind::f16), each CTA over its own range of
 * vectors; the per-CTA partials are added in a fixed order, so the result is
 * deterministic.  workspace: device, >= swan_gram_workspace_bytes(n_mats),
 * 256-byte aligned, used until the work on `stream` completes (calls that
 * share a workspace must be ordered).
 * Errors: INVALID_ARG (layout, alignment, sizes, workspace), CUDA (launch or
 * tensor-map encoding).
 */
swan_status swan_gram(const swan_vectors* x, float* gram, int accumulate, void* workspace,
                      size_t workspace_bytes, void* stream);

/*
 * Eigen-decomposition of symmetric Gram matrices (the input is symmetrised as
 * (G + G^T) / 2), one CTA per matrix: parallel cyclic Jacobi in fp32 followed
 * by one Newton-Schulz orthogonality step.
 *   gram:   device fp32 [n_mats][128][128]
 *   R:      device fp32 [n_mats][128][128] out; column r is the unit
 *           eigenvector of the r-th largest eigenvalue, its largest-magnitude
 *           coordinate positive.  Use it as the rotation of swan_init:
 *           x_hat = x R (the paper's P = SVD(S)_V).
 *   lambda: device fp32 [n_mats][128] out (decreasing), or NULL
 *   sweeps: device int32 [n_mats] out, sweeps until no rotation was needed,
 *           -1 if 40 sweeps did not converge; or NULL
 * Errors: INVALID_ARG, CUDA.
 */
swan_status swan_basis_eig(const float* gram, int n_mats, float* R, float* lambda, int* sweeps,
                           void* stream);

/*
 * Energy kept by per-vector magnitude top-k pruning (Algorithm 1) after the
 * rotation x_hat = x R[m], for every k:
 *   energy[m][k] (+)= sum over the vectors of matrix m of the k largest
 *                     x_hat_j^2          (k = 0 .. 128; energy[m][128] is
 *                                         the total, R orthogonal)
 * x_hat is computed in fp32 from the fp16 vectors; sums are fp64.
 * energy: device fp64 [n_mats][129]; accumulate == 0 zeroes it first.
 * R: device fp32 [n_mats][128][128].
 * Errors: INVALID_ARG, CUDA.
 */
swan_status swan_energy(const swan_vectors* x, const float* R, double* energy, int accumulate,
                        void* stream);

/*
 * Wait for `stream` and report the device status word of a swan_gram
 * workspace (each swan_gram call clears it first, so this reports the last
 * call on that workspace): SWAN_OK, or SWAN_ERR_DEVICE_TIMEOUT if a wait gave
 * up.  Errors: INVALID_ARG, CUDA.
 */
swan_status swan_basis_check(void* workspace, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* SWAN_BASIS_H */
