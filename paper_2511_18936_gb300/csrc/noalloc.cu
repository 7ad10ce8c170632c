// swan_decode_noalloc: one decode step over a cache held in caller-owned
// device memory, with no device allocation of any kind.
//
// For callers that may not call cudaMalloc (for example an engine whose
// device memory all comes from its own pre-reserved pool, or code running
// where an allocation would break a memory budget or a captured sequence of
// work), the per-call scratch of the decode path (rotated queries and split
// partials) lives in a file-scope static device array of a fixed size
// instead of context-owned memory.  The array exists once per device that
// loads the library and stays allocated until the process exits.
#include <algorithm>
#include <cmath>
#include <cstdio>
#include <mutex>

#include "swan.h"
#include "swan_internal.h"

namespace swan {
namespace {

constexpr int kNoallocMaxQ = 1024;         // batch * n_q_heads
constexpr int kNoallocMaxSlots = 2048;     // (decode CTAs + units) * G partials
constexpr size_t kQFloats = (size_t)kNoallocMaxQ * kHeadDim;
constexpr size_t kPartFloats = (size_t)kNoallocMaxSlots * (kHeadDim + 2);
constexpr size_t kCounterFloats = kNoallocMaxSlots;  // per-unit arrival counters (int)
constexpr size_t kStatusFloats = 64;       // 256 bytes, the status word first

// Layout: [rotated queries][split partials][counters][status word]
__device__ __align__(256) float
    g_noalloc_scratch[kQFloats + kPartFloats + kCounterFloats + kStatusFloats];

constexpr int kMaxDevices = 64;
struct DeviceSetup {
  bool ready = false;
  unsigned long long ctx_id = 0;  // driver context the address belongs to
  float* scratch = nullptr;       // device address of g_noalloc_scratch
  int sms = 0;
  int ctas_per_sm[4][kDecodeVariants] = {};  // [G = 1, 2, 4, 8][kernel variant: <= 32, 64, 96, 128 entries read]
};
DeviceSetup g_setup[kMaxDevices];
std::mutex g_setup_mutex;

// The current driver context's unique id (cuCtxGetId; 0 if the driver
// cannot say).  The static array's device address belongs to the module
// loaded in one context: after cudaDeviceReset the primary context, and
// with it the module and the array, are created anew, so the address is
// resolved again whenever the id changes.
using CtxGetCurrentFn = CUresult (*)(CUcontext*);
using CtxGetIdFn = CUresult (*)(CUcontext, unsigned long long*);
unsigned long long current_ctx_id() {
  static CtxGetCurrentFn get_current = nullptr;
  static CtxGetIdFn get_id = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess && q == cudaDriverEntryPointSuccess)
      get_current = reinterpret_cast<CtxGetCurrentFn>(p);
    p = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_id = reinterpret_cast<CtxGetIdFn>(p);
  });
  if (!get_current || !get_id) return 0;
  CUcontext c = nullptr;
  unsigned long long id = 0;
  if (get_current(&c) != CUDA_SUCCESS || !c || get_id(c, &id) != CUDA_SUCCESS) return 0;
  return id;
}

// Byte alignment the kernels' widest access to a pointer needs.
bool aligned(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) & (a - 1)) == 0; }

thread_local char g_err[256];

swan_status err(swan_status s, const char* msg) {
  snprintf(g_err, sizeof(g_err), "swan_decode_noalloc: %s", msg);
  set_last_error(g_err);
  return s;
}

int gi(int G) { return G == 1 ? 0 : G == 2 ? 1 : G == 4 ? 2 : 3; }

// Once per device (and again if the device's context was re-created), with
// that device current: resolve the device address of the static scratch
// array and the decode grid limits.
swan_status setup_device(int dev, DeviceSetup** out) {
  if (dev < 0 || dev >= kMaxDevices) return err(SWAN_ERR_UNSUPPORTED, "device index out of range");
  std::lock_guard<std::mutex> lock(g_setup_mutex);
  DeviceSetup& s = g_setup[dev];
  // id 0: no context is current yet, or the driver cannot name it; resolve
  // again (cheap host calls) rather than trust a cached address
  const unsigned long long id = current_ctx_id();
  if (!s.ready || id == 0 || s.ctx_id != id) {
    s.ready = false;
    void* p = nullptr;
    cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);  // also makes the context current
    if (e != cudaSuccess || p == nullptr) return err(SWAN_ERR_CUDA, "cudaGetSymbolAddress failed");
    e = cudaDeviceGetAttribute(&s.sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return err(SWAN_ERR_CUDA, "cudaDeviceGetAttribute failed");
    const int gs[4] = {1, 2, 4, 8};
    for (int g = 0; g < 4; ++g)
      for (int v = 0; v < kDecodeVariants; ++v) {
        s.ctas_per_sm[g][v] = decode_ctas_per_sm(gs[g], 32 + 32 * v);
        if (s.ctas_per_sm[g][v] < 1) return err(SWAN_ERR_CUDA, "decode kernel occupancy query failed");
      }
    s.scratch = static_cast<float*>(p);
    s.ctx_id = current_ctx_id();
    s.ready = true;
  }
  *out = &s;
  return SWAN_OK;
}

}  // namespace
}  // namespace swan

using namespace swan;

extern "C" swan_status swan_decode_noalloc(const swan_cache_view* v, const void* q, void* out,
                                           void* stream) {
  set_last_error("");
  if (!v || !q || !out) return err(SWAN_ERR_INVALID_ARG, "NULL view, q or out");
  if (v->head_dim != kHeadDim) return err(SWAN_ERR_UNSUPPORTED, "head_dim must be 128");
  if (v->batch < 1 || v->n_kv_heads < 1 || v->n_q_heads < 1 || v->n_q_heads % v->n_kv_heads)
    return err(SWAN_ERR_INVALID_ARG, "bad batch or head counts");
  const int G = v->n_q_heads / v->n_kv_heads;
  if (G != 1 && G != 2 && G != 4 && G != 8) return err(SWAN_ERR_UNSUPPORTED, "group size must be 1, 2, 4 or 8");
  if (v->k_slots < 8 || v->k_slots > kHeadDim || v->k_slots % 8)
    return err(SWAN_ERR_INVALID_ARG, "k_slots must be a multiple of 8 in [8, 128]");
  if (v->k_active < 1 || v->k_active > v->k_slots) return err(SWAN_ERR_INVALID_ARG, "k_active out of range");
  const int ksv = v->k_slots_v ? v->k_slots_v : v->k_slots;    // 0: as for keys
  const int kav = v->k_active_v ? v->k_active_v : v->k_active;
  if (ksv < 8 || ksv > kHeadDim || ksv % 8)
    return err(SWAN_ERR_INVALID_ARG, "k_slots_v must be a multiple of 8 in [8, 128]");
  if (kav < 1 || kav > ksv) return err(SWAN_ERR_INVALID_ARG, "k_active_v out of range");
  if (v->page_tokens < 32 || v->page_tokens > 4096 || (v->page_tokens & (v->page_tokens - 1)))
    return err(SWAN_ERR_INVALID_ARG, "page_tokens must be a power of two in [32, 4096]");
  if (v->sparse_len < 0 || v->buf_len < 0 || v->buf_len > v->buffer_cap || v->buffer_cap < 0 ||
      (v->buffer_cap > 0 && (v->buf_start < 0 || v->buf_start >= v->buffer_cap)))
    return err(SWAN_ERR_INVALID_ARG, "inconsistent buffer or sparse lengths");
  if (v->pages_per_unit < 0 || v->sparse_len > (int64_t)v->pages_per_unit * v->page_tokens)
    return err(SWAN_ERR_INVALID_ARG, "sparse_len exceeds pages_per_unit * page_tokens");
  if (v->sparse_len > 0 && (!v->pages || !v->page_table || v->num_pages < 1))
    return err(SWAN_ERR_INVALID_ARG, "NULL pages or page table");
  if (v->buf_len > 0 && (!v->buf_k || !v->buf_v)) return err(SWAN_ERR_INVALID_ARG, "NULL buffer");
  if (!v->R_qk || !v->R_vo_t) return err(SWAN_ERR_INVALID_ARG, "NULL rotation matrix");
  if (v->value_format != SWAN_VALUES_FP16 && v->value_format != SWAN_VALUES_FP8_E4M3)
    return err(SWAN_ERR_INVALID_ARG, "value_format must be fp16 (0) or fp8 e4m3 (1)");
  // the kernels read pages, buffers and R with 16-byte loads, q with 8-byte
  // loads, and write out as fp16: a misaligned address would fault the context
  if ((v->sparse_len > 0 && (!aligned(v->pages, 16) || !aligned(v->page_table, 4))) ||
      (v->buf_len > 0 && (!aligned(v->buf_k, 16) || !aligned(v->buf_v, 16))) || !aligned(v->R_qk, 16) ||
      !aligned(v->R_vo_t, 16) || !aligned(q, 8) || !aligned(out, 2))
    return err(SWAN_ERR_INVALID_ARG,
               "misaligned pointer (pages, buf_k, buf_v, R_qk, R_vo_t: 16 bytes; q: 8; page_table: 4; out: 2)");
  const int fmt = v->value_format == SWAN_VALUES_FP8_E4M3 ? kFmtFp8 : kFmtFp16;
  const int64_t nq = (int64_t)v->batch * v->n_q_heads;
  if (nq > kNoallocMaxQ) return err(SWAN_ERR_INVALID_ARG, "batch * n_q_heads exceeds 1024 (static scratch)");

  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return err(SWAN_ERR_CUDA, "cudaGetDevice failed");
  DeviceSetup* ds = nullptr;
  swan_status st = setup_device(dev, &ds);
  if (st != SWAN_OK) return st;

  const int64_t units = (int64_t)v->batch * v->n_kv_heads;
  const int64_t n_sg = (v->sparse_len + 31) / 32;
  const int64_t n_bg = ((int64_t)v->buf_len + 31) / 32;
  const int64_t N_g = n_sg + n_bg;
  const int64_t total = units * N_g;
  int64_t grid = 0;
  if (total > 0)
    grid = std::min<int64_t>(
        (int64_t)ds->sms * ds->ctas_per_sm[gi(G)][decode_variant((std::max(v->k_active, kav) + 7) / 8 * 8)],
        std::max<int64_t>(1, total / kMinGroupsPerCta));
  if ((grid + units) * G > kNoallocMaxSlots)
    return err(SWAN_ERR_INVALID_ARG, "(decode CTAs + batch * n_kv_heads) * G exceeds 2048 (static scratch)");

  cudaStream_t s = static_cast<cudaStream_t>(stream);
  float* qprime = ds->scratch;
  float* partials = ds->scratch + kQFloats;
  int* counters = reinterpret_cast<int*>(ds->scratch + kQFloats + kPartFloats);
  unsigned* status = reinterpret_cast<unsigned*>(ds->scratch + kQFloats + kPartFloats + kCounterFloats);
  // the counters and the status word must start at zero; the rest is fully
  // written before use
  if (cudaMemsetAsync(counters, 0, (size_t)units * sizeof(int), s) != cudaSuccess ||
      cudaMemsetAsync(status, 0, sizeof(unsigned), s) != cudaSuccess)
    return err(SWAN_ERR_CUDA, "cudaMemsetAsync of the counters failed");

  RotateQParams rq{};
  rq.q = static_cast<const __half*>(q);
  rq.R_qk = v->R_qk;
  rq.qprime = qprime;
  rq.H_q = v->n_q_heads;
  rq.G = G;
  if (launch_rotate_q(rq, v->batch, s) != cudaSuccess) return err(SWAN_ERR_CUDA, "rotate_q launch failed");

  if (grid > 0) {
    DecodeParams p{};
    p.qprime = qprime;
    p.geom.pool = static_cast<uint8_t*>(const_cast<void*>(v->pages));
    p.geom.page_table = v->page_table;
    p.geom.pages_per_unit = v->pages_per_unit;
    p.geom.num_pages = v->num_pages;
    p.geom.P = v->page_tokens;
    p.geom.k_slots = v->k_slots;
    p.geom.k_store = v->k_slots;
    p.geom.k_slots_v = ksv;
    p.geom.k_store_v = ksv;
    p.geom.fmt = fmt;
    p.geom.page_bytes = page_bytes_for(v->page_tokens, v->k_slots, ksv, fmt);
    p.ring_k = static_cast<const __half*>(v->buf_k);
    p.ring_v = static_cast<const __half*>(v->buf_v);
    p.cap = v->buffer_cap > 0 ? v->buffer_cap : 1;
    p.buf_start = v->buf_start;
    p.n_b = v->buf_len;
    p.sparse_len = v->sparse_len;
    p.n_sg = n_sg;
    p.N_g = N_g;
    p.total_groups = total;
    p.visit_cost = decode_visit_cost(G, false);
    p.B = v->batch;
    p.H_kv = v->n_kv_heads;
    p.H_q = v->n_q_heads;
    p.blocks_per_page_log2 = __builtin_ctz((unsigned)(v->page_tokens / 32));
    p.k_full_chunks = v->k_active / 8;
    p.k_rem = v->k_active % 8;
    p.k_full_chunks_v = kav / 8;
    p.k_rem_v = kav % 8;
    p.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)kHeadDim));
    p.partials = partials;
    p.counters = counters;
    p.R_voT = v->R_vo_t;
    p.out = static_cast<__half*>(out);
    p.status = status;
    if (launch_decode(p, G, (std::max(v->k_active, kav) + 7) / 8 * 8, (int)grid, s) != cudaSuccess)
      return err(SWAN_ERR_CUDA, "decode launch failed");
    return SWAN_OK;
  }

  CombineParams cp{};
  cp.out = static_cast<__half*>(out);
  cp.H_q = v->n_q_heads;
  if (launch_combine(cp, v->batch, s) != cudaSuccess) return err(SWAN_ERR_CUDA, "combine launch failed");
  return SWAN_OK;
}

extern "C" swan_status swan_noalloc_check(void* stream) {
  set_last_error("");
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return err(SWAN_ERR_CUDA, "cudaGetDevice failed");
  DeviceSetup* ds = nullptr;
  swan_status st = setup_device(dev, &ds);
  if (st != SWAN_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  unsigned* status = reinterpret_cast<unsigned*>(ds->scratch + kQFloats + kPartFloats + kCounterFloats);
  unsigned word = 0;
  if (cudaStreamSynchronize(s) != cudaSuccess) return err(SWAN_ERR_CUDA, "cudaStreamSynchronize failed");
  if (cudaMemcpyAsync(&word, status, sizeof(word), cudaMemcpyDeviceToHost, s) != cudaSuccess ||
      cudaStreamSynchronize(s) != cudaSuccess)
    return err(SWAN_ERR_CUDA, "reading the status word failed");
  if (!word) return SWAN_OK;
  if (cudaMemsetAsync(status, 0, sizeof(unsigned), s) != cudaSuccess ||
      cudaStreamSynchronize(s) != cudaSuccess)
    return err(SWAN_ERR_CUDA, "clearing the status word failed");
  char msg[96];
  snprintf(msg, sizeof(msg), "device status word 0x%x of the last call", word);
  return err(word & kStatusTimeout ? SWAN_ERR_DEVICE_TIMEOUT : SWAN_ERR_DEVICE_CHECK, msg);
}
