// Internal definitions shared by the host library and the kernels.
//
// Sparse cache page layout (Section 5.1's values + 8-bit indices, arranged
// for 128-bit coalesced loads on sm_103a).  A page holds P tokens (P a power
// of two >= 32) of one (layer, batch, kv-head) unit, as P/32 consecutive
// blocks of 32 tokens.  Each vector's kept entries are grouped in chunks of
// 8, in stored (decreasing magnitude) order; keys keep ks_k entries (k_slots
// = ks_k rounded up to 8) and values ks_v (the two may differ).  With fp16
// values a block (96 * (ks_k + ks_v) bytes) is
//
//   [K values  : ks_k/8 chunks][32 tokens][8 x fp16]    at 0
//   [K indices : ks_k/8 chunks][32 tokens][8 x uint8]   at 64 * ks_k
//   [V values  : ks_v/8 chunks][32 tokens][8 x fp16]    at 96 * ks_k
//   [V indices : ks_v/8 chunks][32 tokens][8 x uint8]   at 96 * ks_k + 64 * ks_v
//
// and with 8-bit (E4M3) values (Section 4.3, Section 5.1) a block
// (64 * (ks_k + ks_v) bytes) is
//
//   [K records : ks_k/8 chunks][32 tokens][8 x e4m3, 8 x uint8]  at 0
//   [V records : ks_v/8 chunks][32 tokens][8 x e4m3, 8 x uint8]  at 64 * ks_k
//
// A warp that handles the 32 tokens of a block (one per lane) reads chunk c
// of all of them as one contiguous 512-byte run (values or records), at
// compile-time offsets from the region base.  A runtime keep count reads only
// the first ceil(k_active / 8) chunks: a contiguous prefix of each region.
#pragma once

#include <cuda.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>

namespace swan {

constexpr int kHeadDim = 128;
constexpr int kWarpsPerCta = 8;
constexpr int kThreads = kWarpsPerCta * 32;
// log2-domain slack before the running max of the online softmax is moved:
// scores may exceed the running max by up to 2^kLazyRescale before the
// accumulators are rescaled (exact; only the reference point changes).
constexpr float kLazyRescale = 8.0f;

// Device status word bits (set instead of faulting on inconsistent state).
constexpr unsigned kStatusPageRange = 1u;
constexpr unsigned kStatusRingRange = 2u;
constexpr unsigned kStatusTimeout = 4u;  // a bounded barrier wait gave up
constexpr unsigned kStatusLayout = 8u;   // too little shared memory for a kernel's layout (kernel skipped)

constexpr int kFmtFp16 = 0;  // fp16 values
constexpr int kFmtFp8 = 1;   // E4M3 values

struct CacheGeom {
  uint8_t* pool;             // all pages of all layers
  const int32_t* page_table; // this layer: [units][pages_per_unit] -> page id
  int pages_per_unit;
  int64_t num_pages;         // pages in the pool (bounds check)
  int P;                     // tokens per page
  int k_slots;               // key entries stored per vector, rounded up to 8
  int k_store;               // key entries kept per vector
  int k_slots_v;             // the same for values
  int k_store_v;
  int64_t page_bytes;        // P / 32 * block_bytes()
  int fmt;                   // kFmtFp16 or kFmtFp8
  // 1: the table is the identity (every unit owns its pages; never written
  // after init), so page g of unit u is identity_base + u * pages_per_unit
  // + g and the decode kernels skip the table read; 0: read the table
  int identity;
  int64_t identity_base;
  // offsets inside a 32-token block (index regions: fp16 only)
  __device__ __host__ int block_bytes() const {
    return (fmt == kFmtFp8 ? 64 : 96) * (k_slots + k_slots_v);
  }
  __device__ __host__ int kidx_off() const { return 64 * k_slots; }
  __device__ __host__ int vval_off() const { return (fmt == kFmtFp8 ? 64 : 96) * k_slots; }
  __device__ __host__ int vidx_off() const { return 96 * k_slots + 64 * k_slots_v; }
};

inline int64_t page_bytes_for(int P, int k_slots, int k_slots_v, int fmt) {
  return (int64_t)(P / 32) * (fmt == kFmtFp8 ? 64 : 96) * (k_slots + k_slots_v);
}

// Per-sequence state for batches whose sequences differ in length (one entry
// per batch row, shared by the row's kv heads).  A kernel reads it instead of
// the uniform scalars of its parameter block when the block's `seq` is set.
struct SeqInfo {
  int64_t sparse_len;    // sparse tokens (before the call; decode: current)
  int64_t group_prefix;  // decode: 32-token groups of rows 0..b-1, per kv head
  int32_t buf_start;     // ring slot of the oldest buffered token
  int32_t n_b;           // buffered tokens (before the call; decode: current)
  int32_t n_new;         // append: new tokens of this row (<= T)
  int32_t evict;         // append: logical positions < evict go to the sparse cache
  int32_t prune;         // prune_ring: buffered tokens 0..prune-1 are pruned
  int32_t pad;
};

// Groups a decode walks for a row: sparse groups, then buffer groups; at
// least one, so that an empty row still gets its (zero) output written.
__host__ __device__ inline int64_t row_groups(int64_t sparse_len, int n_b) {
  const int64_t g = (sparse_len + 31) / 32 + (n_b + 31) / 32;
  return g > 0 ? g : 1;
}

// Rotate T new tokens per unit, then either write them to the ring buffer or
// prune them straight into the sparse cache (Algorithm 1, generalised to T).
struct AppendParams {
  const __half* k_new;  // [B][H][T][d]
  const __half* v_new;
  const float* R_qk;    // this layer: [H][d][d]
  const float* R_vo;
  __half* ring_k;       // this layer: [B*H][cap][d]
  __half* ring_v;
  int B, H, T, cap;
  int buf_start;        // ring slot of the oldest buffered token
  int n_b;              // buffered tokens before the append
  int64_t evict;        // logical positions < evict go to the sparse cache
  int64_t sparse_len;   // sparse tokens before the append
  const SeqInfo* seq;   // per-row state instead of the four scalars above, or null
  CacheGeom geom;
  unsigned* status;
  // test hook (swan_debug_starve_tc): the bulk-append kernel issues no
  // copies, so its barrier wait runs out after tc_wait_ns (0: the default 2 s)
  int tc_starve;
  uint64_t tc_wait_ns;
};

// Prune `count` buffered tokens (logical positions 0..count-1) per unit from
// the ring buffer into the sparse cache (eviction and flush).
struct PruneRingParams {
  const __half* ring_k;
  const __half* ring_v;
  int units, cap, buf_start, count;  // count: the most tokens of any row
  int64_t sparse_len;
  const SeqInfo* seq;   // per-row start, count (prune) and length, or null
  int H;                // kv heads (row of a unit = unit / H)
  CacheGeom geom;
  unsigned* status;
};

struct RotateQParams {
  const __half* q;   // [B][H_q][d]
  const float* R_qk; // this layer: [H_kv][d][d]
  float* qprime;     // [B][H_q][d]
  int H_q, G;
};

// Split decode: the flat list of 32-token groups of all units is cut into
// contiguous ranges of equal cost, one per CTA, a unit costing its groups
// plus `visit_cost` groups for each CTA that works on it.  Group g of unit u
// is a sparse group for g < n_sg (tokens 32g..32g+31 of the sparse history)
// and a buffer group after that.  A CTA writes one partial (m, l, acc[d])
// per (unit, head) it touches, at pair index (cta + unit).
struct DecodeParams {
  const float* qprime;     // [B][H_q][d]
  CacheGeom geom;
  const __half* ring_k;    // this layer: [units][cap][d]
  const __half* ring_v;
  int cap, buf_start, n_b;
  int64_t sparse_len;
  int64_t n_sg, N_g;       // sparse groups per unit; groups per unit
  int64_t total_groups;
  int64_t visit_cost;      // groups a CTA's visit to a unit costs (uniform split)
  const SeqInfo* seq;      // per-row lengths (then the five scalars above are unused), or null
  const int64_t* cta_start;  // [grid + 1] first group of each CTA (ragged rows), or null: computed
  int B;                   // rows
  int H_kv, H_q;
  int blocks_per_page_log2; // log2(P / 32)
  int k_full_chunks;       // keys: k_active / 8
  int k_rem;               // keys: k_active % 8
  int k_full_chunks_v;     // values: k_active_v / 8
  int k_rem_v;             // values: k_active_v % 8
  float scale_log2;        // log2(e) / sqrt(d)
  float* partials;         // [pairs][G][d + 2]
  int* counters;           // [units] arrival counters, zero between decodes
  const float* R_voT;      // this layer: [H_kv][d][d], transposed
  __half* out;             // [B][H_q][d]
  unsigned* status;
};

// A decode over an empty cache: the output is the rotate-back of an empty
// attention, zero.
struct CombineParams {
  __half* out;             // [B][H_q][d]
  int H_q;
};

#ifdef __CUDACC__
// Programmatic dependent launch: every kernel of the library is launched so
// that it may start while the previous kernel on the stream finishes.  A
// kernel may touch only static data (R, page tables) before pdl_wait(), which
// returns once the previous kernel has completed and its writes are visible;
// pdl_trigger() lets the next kernel be scheduled early.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                       Args... args) {
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cudaError_t e = cudaLaunchKernelEx(&cfg, kernel, args...);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

// Stage a 128 x 128 fp32 matrix in shared memory with a CTA of kThreads
// threads: every thread issues its 16 loads before its first store, so all
// of them are in flight at once.
__device__ __forceinline__ void stage_matrix(float* dst, const float* src) {
  float4 r[16];
#pragma unroll
  for (int k = 0; k < 16; ++k)
    r[k] = __ldg(reinterpret_cast<const float4*>(src) + threadIdx.x + k * kThreads);
#pragma unroll
  for (int k = 0; k < 16; ++k) reinterpret_cast<float4*>(dst)[threadIdx.x + k * kThreads] = r[k];
}

// One slice of q' = q R_qk (Section 4.3: the query is rotated once, the cache
// never is): query vectors [8 chunk, 8 chunk + 8) of kv head h (row-major
// over (b, group member)), output coordinates [32 z, 32 z + 32).  Stages the
// 128 x 32 slice of R in Rs (16 KB of shared memory), waits for the previous
// kernel, then one warp per query vector: lane l computes coordinate 32 z + l
// as a sequential fp32 FMA chain over the 128 inputs.  The query-rotation
// kernel and the fused append + rotation kernel both run this, so q' has the
// same bits either way.
__device__ __forceinline__ void rotate_q_slice(const RotateQParams& p, int B, int h, int chunk, int z,
                                               float* Rs) {
  const float* R = p.R_qk + (size_t)h * kHeadDim * kHeadDim + z * 32;
  for (int e = threadIdx.x; e < kHeadDim * 8; e += kThreads) {  // 128 rows x 8 float4
    const int i = e >> 3, c = e & 7;
    reinterpret_cast<float4*>(Rs)[e] = __ldg(reinterpret_cast<const float4*>(R + i * kHeadDim) + c);
  }
  __syncthreads();
  pdl_wait();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int item = chunk * kWarpsPerCta + warp; item < min(B * p.G, (chunk + 1) * kWarpsPerCta);
       item += kWarpsPerCta) {
    const int b = item / p.G, gh = item % p.G;
    const int64_t bq = (int64_t)b * p.H_q + h * p.G + gh;
    const uint2 xw = __ldg(reinterpret_cast<const uint2*>(p.q + bq * kHeadDim) + lane);
    const float2 x01 = __half22float2(*reinterpret_cast<const __half2*>(&xw.x));
    const float2 x23 = __half22float2(*reinterpret_cast<const __half2*>(&xw.y));
    const float xs[4] = {x01.x, x01.y, x23.x, x23.y};
    float acc = 0.f;
#pragma unroll 16
    for (int i = 0; i < kHeadDim; ++i) {
      const float xi = __shfl_sync(0xffffffffu, xs[i & 3], i >> 2);
      acc = fmaf(xi, Rs[i * 32 + lane], acc);
    }
    p.qprime[bq * kHeadDim + z * 32 + lane] = acc;
  }
}
#endif

// Raise a kernel's dynamic shared-memory limit once per device (the limit
// is a per-device function attribute; thread-safe).
template <auto Kernel>
cudaError_t ensure_smem(size_t bytes) {
  static std::atomic<uint64_t> done{0};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const uint64_t bit = dev < 64 ? (uint64_t)1 << dev : 0;
  if (bit && (done.load(std::memory_order_acquire) & bit)) return cudaSuccess;
  e = cudaFuncSetAttribute(Kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
  if (e == cudaSuccess && bit) done.fetch_or(bit, std::memory_order_release);
  return e;
}

// Launchers (return the launch error, if any).
// Bulk append with the rotation on the tensor cores: maps[0..1] the new keys
// and values ([B][H][T][128] fp16, 64 x 128-vector boxes), maps[2..3] the
// split rotations (see launch_split_r), r_slice0 = layer * 2 * H.
cudaError_t launch_append_tc(const AppendParams& p, const CUtensorMap* maps, int r_slice0, cudaStream_t s);
// R_hi^T and R_lo^T (fp16, [layer][2 kinds][H][n][k]) from fp32 R: hi = fp16(R),
// lo = fp16((R - hi) * 2^12); kind 0 from R_qk, 1 from R_vo.
cudaError_t launch_split_r(const float* R_qk, const float* R_vo, __half* hi, __half* lo, int layers, int H,
                           cudaStream_t s);
// cuTensorMapEncodeTiled from the driver (null if unavailable).
using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                   const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                   CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
EncodeTiledFn tensor_map_encoder();
// Eviction of `evict_old` buffered tokens and insertion of T new ones in one
// launch; for small batch * T (decode steps).  With rq non-null the same
// launch also computes the query rotation q' = q R_qk of rq.
cudaError_t launch_append_small(const AppendParams& p, int evict_old, const RotateQParams* rq, cudaStream_t s);
cudaError_t launch_prune_ring(const PruneRingParams& p, cudaStream_t s);
cudaError_t launch_rotate_q(const RotateQParams& p, int B, cudaStream_t s);
// k_read: entries read per vector rounded up to 8 (selects the kernel variant:
// up to 32 and up to 96 (one query head per kv head only), up to 64, up to
// 128)
cudaError_t launch_decode(const DecodeParams& p, int G, int k_read, int grid, cudaStream_t s);
cudaError_t launch_combine(const CombineParams& p, int B, cudaStream_t s);
cudaError_t launch_transpose_r(const float* src, float* dst, int64_t mats, cudaStream_t s);
// table[pairs[i].x] = pairs[i].y for i < n (page-table entries of a shared pool).
cudaError_t launch_scatter_pages(const int2* pairs, int n, int32_t* table, cudaStream_t s);
// Decode CTAs of the variant launch_decode takes for k_read that fit on one
// SM together (for the grid size).
int decode_ctas_per_sm(int G, int k_read);
// The variant class of k_read: 0 (<= 32), 1 (<= 64), 2 (<= 96), 3 (<= 128).
constexpr int kDecodeVariants = 4;
inline int decode_variant(int k_read) { return k_read <= 32 ? 0 : k_read <= 64 ? 1 : k_read <= 96 ? 2 : 3; }
// Fewest 32-token groups a decode CTA takes: a small cache is split over
// fewer CTAs so that each one's fixed cost (staging q', the merge) and the
// final combine over the CTAs' partials stay small next to its groups
// (swept on the GB300 for one head at 1088 tokens, L2 flushed: decode 20.4 us
// at 2 and 4, 22.4 us at 8, 24.8 us at 16).
constexpr int64_t kMinGroupsPerCta = 4;
// What a CTA's extra visit to a unit (prologue, merge, arrival) costs in
// 32-token groups of streaming, for the cost-balanced split of the decode
// kernels: equal-length rows (computed in the kernel) and ragged rows (the
// host's table).  Set by sweeps on the GB300: ragged serving batch (32 rows,
// 1k-56k tokens) 0.914 ms at 48, 0.898 at 56, 0.883 at 64, 0.865 at 72,
// 0.864 at 80, 0.870 at 88; equal rows flat within 0.5 % from 12 to 64 for
// one head (32k layer, 32-layer stack: 48 and up 2 % slower there, k 32),
// GQA best at 40 (0.360 ms; 0.362 at 20 and 60).
inline int64_t decode_visit_cost(int G, bool ragged) {
  if (ragged) return 80;
  return G == 1 ? 12 : 40;
}
// Record the detail string that swan_last_error() returns on this thread.
void set_last_error(const char* msg);
// Test hook armed by swan_debug_starve_tc: the wait limit in nanoseconds for
// the next tensor-core launch, which then issues no copies (0: not armed).
// Disarms it.
int64_t take_tc_starve();

}  // namespace swan
