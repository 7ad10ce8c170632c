// Host side of libswan: validation, the one-time allocation of the cache,
// per-layer bookkeeping of the hybrid cache (Section 4.3), and the launch
// sequence of each entry point declared in include/swan.h.
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <new>
#include <string>
#include <vector>

#include "swan.h"
#include "swan_internal.h"

using namespace swan;

namespace {

thread_local std::string g_last_error;

swan_status fail(swan_status s, const char* fmt, ...) __attribute__((format(printf, 2, 3)));
swan_status fail(swan_status s, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  g_last_error = buf;
  return s;
}

struct LayerState {
  int64_t sparse_len = 0;
  int buf_start = 0;  // ring slot of the oldest buffered token
  int buf_count = 0;
};

struct EventPair {
  cudaEvent_t start, stop;
  int kind;
};

}  // namespace

struct swan_ctx {
  swan_config cfg{};
  int G = 1;
  int k_slots = 0;    // key entries stored per vector, rounded up to 8
  int k_active = 0;
  int k_store_v = 0;  // value entries kept per vector
  int k_slots_v = 0;
  int k_active_v = 0;
  int P = 128;
  int ppu = 0;  // pages per unit
  int64_t page_bytes = 0;
  int64_t num_pages = 0;
  int fmt = kFmtFp16;
  int64_t units = 0;  // batch * n_kv_heads (per layer)
  cudaStream_t stream = nullptr;
  int device = 0;
  int num_sms = 0;
  int decode_ctas = 0;  // max decode CTAs resident at once

  float* R_qk = nullptr;
  float* R_vo = nullptr;   // == R_qk when the caller passed NULL
  float* R_voT = nullptr;  // transposed copy for the rotate-back
  uint8_t* pool = nullptr;
  int32_t* page_table = nullptr;
  __half* ring_k = nullptr;
  __half* ring_v = nullptr;
  float* qprime = nullptr;
  float* partials = nullptr;
  int* counters = nullptr;  // per-unit arrival counters of the fused combine
  unsigned* status = nullptr;
  int64_t device_bytes = 0;

  std::vector<LayerState> layers;
  bool poisoned = false;
  int64_t launches = 0;

  bool timing = false;
  std::vector<EventPair> ev_free, ev_used;
  double ms_acc[SWAN_KERNEL_KINDS] = {};
  int64_t n_acc[SWAN_KERNEL_KINDS] = {};
};

namespace {

constexpr int kMaxBufferCap = 4096;
constexpr int64_t kSmallAppendVectors = 256;  // batch * T per kv head
constexpr size_t kMaxEventPairs = 4096;

void free_all(swan_ctx* c) {
  if (c->R_vo && c->R_vo != c->R_qk) cudaFree(c->R_vo);
  cudaFree(c->R_qk);
  cudaFree(c->R_voT);
  cudaFree(c->pool);
  cudaFree(c->page_table);
  cudaFree(c->ring_k);
  cudaFree(c->ring_v);
  cudaFree(c->qprime);
  cudaFree(c->partials);
  cudaFree(c->counters);
  cudaFree(c->status);
  for (auto& e : c->ev_free) {
    cudaEventDestroy(e.start);
    cudaEventDestroy(e.stop);
  }
  for (auto& e : c->ev_used) {
    cudaEventDestroy(e.start);
    cudaEventDestroy(e.stop);
  }
}

swan_status dev_alloc(swan_ctx* c, void** p, size_t bytes, const char* what) {
  if (bytes == 0) bytes = 256;
  cudaError_t e = cudaMalloc(p, bytes);
  if (e != cudaSuccess) {
    cudaGetLastError();
    *p = nullptr;
    return fail(SWAN_ERR_NOMEM, "cudaMalloc of %zu bytes for %s failed: %s", bytes, what,
                cudaGetErrorString(e));
  }
  c->device_bytes += (int64_t)bytes;
  return SWAN_OK;
}

swan_status cuda_fail(swan_ctx* c, cudaError_t e, const char* where) {
  c->poisoned = true;
  return fail(SWAN_ERR_CUDA, "%s: %s", where, cudaGetErrorString(e));
}

// Fold finished event pairs into the per-kind sums (synchronises).
swan_status drain_events(swan_ctx* c) {
  if (c->ev_used.empty()) return SWAN_OK;
  cudaError_t e = cudaStreamSynchronize(c->stream);
  if (e != cudaSuccess) return cuda_fail(c, e, "cudaStreamSynchronize");
  for (auto& ev : c->ev_used) {
    float ms = 0.f;
    e = cudaEventElapsedTime(&ms, ev.start, ev.stop);
    if (e != cudaSuccess) return cuda_fail(c, e, "cudaEventElapsedTime");
    c->ms_acc[ev.kind] += ms;
    c->n_acc[ev.kind] += 1;
    c->ev_free.push_back(ev);
  }
  c->ev_used.clear();
  return SWAN_OK;
}

// Launch wrapper: counts launches and, when timing is on, brackets the launch
// with an event pair on the context's stream.
template <typename F>
swan_status launch(swan_ctx* c, int kind, const char* name, F&& f) {
  EventPair ev{};
  if (c->timing) {
    if (c->ev_used.size() >= kMaxEventPairs) {
      swan_status s = drain_events(c);
      if (s != SWAN_OK) return s;
    }
    if (c->ev_free.empty()) {
      cudaError_t e1 = cudaEventCreate(&ev.start);
      cudaError_t e2 = cudaEventCreate(&ev.stop);
      if (e1 != cudaSuccess || e2 != cudaSuccess) return cuda_fail(c, cudaGetLastError(), "cudaEventCreate");
    } else {
      ev = c->ev_free.back();
      c->ev_free.pop_back();
    }
    ev.kind = kind;
    cudaEventRecord(ev.start, c->stream);
  }
  cudaError_t e = f();
  c->launches += 1;
  if (c->timing) {
    cudaEventRecord(ev.stop, c->stream);
    c->ev_used.push_back(ev);
  }
  if (e != cudaSuccess) return cuda_fail(c, e, name);
  return SWAN_OK;
}

CacheGeom geom_for(const swan_ctx* c, int layer) {
  CacheGeom g;
  g.pool = c->pool;
  g.page_table = c->page_table + (int64_t)layer * c->units * c->ppu;
  g.pages_per_unit = c->ppu;
  g.num_pages = c->num_pages;
  g.P = c->P;
  g.k_slots = c->k_slots;
  g.k_store = c->cfg.k_store;
  g.k_slots_v = c->k_slots_v;
  g.k_store_v = c->k_store_v;
  g.page_bytes = c->page_bytes;
  g.fmt = c->fmt;
  return g;
}

size_t ring_elems_per_layer(const swan_ctx* c) {
  return (size_t)c->units * (size_t)c->cfg.buffer_cap * kHeadDim;
}

swan_status usable(const swan_ctx* c) {
  if (!c) return fail(SWAN_ERR_INVALID_ARG, "NULL context");
  if (c->poisoned) return fail(SWAN_ERR_STATE, "context poisoned by an earlier CUDA error");
  return SWAN_OK;
}

swan_status check_layer(const swan_ctx* c, int layer) {
  if (layer < 0 || layer >= c->cfg.num_layers)
    return fail(SWAN_ERR_INVALID_ARG, "layer %d out of range [0, %d)", layer, c->cfg.num_layers);
  return SWAN_OK;
}

// An E4M3 byte widened to fp16 bits (exact: every E4M3 value is an fp16
// value).  E4M3: sign, 4 exponent bits (bias 7), 3 mantissa bits;
// exponent 0 holds the subnormals m * 2^-9; S.1111.111 is NaN.
uint16_t e4m3_to_half_bits(uint8_t b) {
  const uint16_t sign = (uint16_t)((b & 0x80u) << 8);
  const int e = (b >> 3) & 15, m = b & 7;
  if (e == 15 && m == 7) return sign | 0x7e00u;
  if (e == 0 && m == 0) return sign;
  double v = e == 0 ? std::ldexp((double)m, -9) : std::ldexp((double)(8 + m), e - 10);
  int ex = 0;
  const double fr = std::frexp(v, &ex);  // v = fr * 2^ex, fr in [0.5, 1)
  const int he = ex - 1 + 15;            // fp16 biased exponent (always >= 6 here)
  const int hm = (int)std::lround((fr * 2.0 - 1.0) * 1024.0);
  return sign | (uint16_t)(he << 10) | (uint16_t)hm;
}

// Prune buffered tokens 0..count-1 of a layer into the sparse cache.
swan_status prune_from_ring(swan_ctx* c, int layer, int count) {
  if (count <= 0) return SWAN_OK;
  LayerState& L = c->layers[layer];
  PruneRingParams p{};
  p.ring_k = c->ring_k + (size_t)layer * ring_elems_per_layer(c);
  p.ring_v = c->ring_v + (size_t)layer * ring_elems_per_layer(c);
  p.units = (int)c->units;
  p.cap = c->cfg.buffer_cap;
  p.buf_start = L.buf_start;
  p.count = count;
  p.sparse_len = L.sparse_len;
  p.geom = geom_for(c, layer);
  p.status = c->status;
  swan_status s = launch(c, SWAN_KERNEL_PRUNE, "prune_ring kernel",
                         [&] { return launch_prune_ring(p, c->stream); });
  if (s != SWAN_OK) return s;
  L.sparse_len += count;
  L.buf_start = c->cfg.buffer_cap ? (L.buf_start + count) % c->cfg.buffer_cap : 0;
  L.buf_count -= count;
  return SWAN_OK;
}

}  // namespace

void swan::set_last_error(const char* msg) { g_last_error = msg ? msg : ""; }

extern "C" {

const char* swan_status_string(swan_status s) {
  switch (s) {
    case SWAN_OK: return "ok";
    case SWAN_ERR_INVALID_ARG: return "invalid argument";
    case SWAN_ERR_UNSUPPORTED: return "unsupported configuration";
    case SWAN_ERR_CAPACITY: return "cache capacity exceeded";
    case SWAN_ERR_CUDA: return "CUDA error";
    case SWAN_ERR_STATE: return "context unusable after an earlier error";
    case SWAN_ERR_DEVICE_TIMEOUT: return "device wait timed out";
    case SWAN_ERR_NOMEM: return "out of memory";
    case SWAN_ERR_DEVICE_CHECK: return "device-side consistency check failed";
  }
  return "unknown status";
}

const char* swan_last_error(void) { return g_last_error.c_str(); }

swan_status swan_init(swan_ctx** out, const swan_config* cfg, const float* R_qk, const float* R_vo) {
  g_last_error.clear();
  if (!out) return fail(SWAN_ERR_INVALID_ARG, "out is NULL");
  *out = nullptr;
  if (!cfg) return fail(SWAN_ERR_INVALID_ARG, "cfg is NULL");
  if (!R_qk) return fail(SWAN_ERR_INVALID_ARG, "R_qk is NULL");
  const swan_config& C = *cfg;
  if (C.head_dim != kHeadDim)
    return fail(SWAN_ERR_UNSUPPORTED, "head_dim %d: only 128 is built", C.head_dim);
  if (C.num_layers < 1 || C.batch < 1 || C.n_kv_heads < 1 || C.n_q_heads < 1)
    return fail(SWAN_ERR_INVALID_ARG, "num_layers, batch and head counts must be >= 1");
  if (C.n_q_heads % C.n_kv_heads)
    return fail(SWAN_ERR_INVALID_ARG, "n_q_heads %d is not a multiple of n_kv_heads %d", C.n_q_heads,
                C.n_kv_heads);
  const int G = C.n_q_heads / C.n_kv_heads;
  if (G != 1 && G != 2 && G != 4)
    return fail(SWAN_ERR_UNSUPPORTED, "group size %d: only 1, 2 and 4 are built", G);
  if (C.k_store < 1 || C.k_store > C.head_dim)
    return fail(SWAN_ERR_INVALID_ARG, "k_store %d out of [1, %d]", C.k_store, C.head_dim);
  const int k_store_v = C.k_store_v ? C.k_store_v : C.k_store;
  if (k_store_v < 1 || k_store_v > C.head_dim)
    return fail(SWAN_ERR_INVALID_ARG, "k_store_v %d out of [1, %d]", C.k_store_v, C.head_dim);
  if (C.buffer_cap < 0 || C.buffer_cap > kMaxBufferCap)
    return fail(SWAN_ERR_INVALID_ARG, "buffer_cap %d out of [0, %d]", C.buffer_cap, kMaxBufferCap);
  if (C.max_seq < 1) return fail(SWAN_ERR_INVALID_ARG, "max_seq must be >= 1");
  if (C.value_format != SWAN_VALUES_FP16 && C.value_format != SWAN_VALUES_FP8_E4M3)
    return fail(SWAN_ERR_INVALID_ARG, "value_format %d is neither fp16 (0) nor fp8 e4m3 (1)", C.value_format);
  const int P = C.page_tokens ? C.page_tokens : 128;
  if (P < 32 || P > 4096 || (P & (P - 1)))
    return fail(SWAN_ERR_INVALID_ARG, "page_tokens %d must be a power of two in [32, 4096]", P);

  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return fail(SWAN_ERR_CUDA, "cudaGetDevice: %s", cudaGetErrorString(e));
  int sms = 0;
  e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return fail(SWAN_ERR_CUDA, "cudaDeviceGetAttribute: %s", cudaGetErrorString(e));

  swan_ctx* c = new (std::nothrow) swan_ctx();
  if (!c) return fail(SWAN_ERR_NOMEM, "host allocation of the context failed");
  c->cfg = C;
  c->G = G;
  c->k_slots = (C.k_store + 7) / 8 * 8;
  c->k_active = C.k_store;
  c->k_store_v = k_store_v;
  c->k_slots_v = (k_store_v + 7) / 8 * 8;
  c->k_active_v = k_store_v;
  c->P = P;
  c->ppu = (int)((C.max_seq + P - 1) / P);
  c->fmt = C.value_format == SWAN_VALUES_FP8_E4M3 ? kFmtFp8 : kFmtFp16;
  c->page_bytes = page_bytes_for(P, c->k_slots, c->k_slots_v, c->fmt);
  c->units = (int64_t)C.batch * C.n_kv_heads;
  c->num_pages = (int64_t)C.num_layers * c->units * c->ppu;
  c->stream = static_cast<cudaStream_t>(C.stream);
  c->device = dev;
  c->num_sms = sms;
  c->layers.assign(C.num_layers, LayerState{});

  const int per_sm = decode_ctas_per_sm(G, std::max(c->k_slots, c->k_slots_v));
  if (per_sm < 1) {
    delete c;
    return fail(SWAN_ERR_CUDA, "decode kernel does not fit on an SM (%s)",
                cudaGetErrorString(cudaGetLastError()));
  }
  c->decode_ctas = per_sm * sms;

  const size_t rmat = (size_t)C.num_layers * C.n_kv_heads * kHeadDim * kHeadDim;
  const size_t ring_elems = (size_t)C.num_layers * ring_elems_per_layer(c);
  const size_t q_elems = (size_t)C.batch * C.n_q_heads * kHeadDim;
  const size_t pairs = (size_t)c->decode_ctas + (size_t)c->units;
  const size_t part_elems = pairs * G * (kHeadDim + 2);
  const size_t pt_elems = (size_t)c->num_pages;
  if (c->num_pages > INT32_MAX) {
    const long long np = (long long)c->num_pages;
    delete c;
    return fail(SWAN_ERR_UNSUPPORTED, "too many pages (%lld)", np);
  }

  swan_status s = SWAN_OK;
  if (s == SWAN_OK) s = dev_alloc(c, (void**)&c->R_qk, rmat * sizeof(float), "R_qk");
  if (s == SWAN_OK && R_vo) s = dev_alloc(c, (void**)&c->R_vo, rmat * sizeof(float), "R_vo");
  if (s == SWAN_OK) s = dev_alloc(c, (void**)&c->R_voT, rmat * sizeof(float), "R_vo^T");
  if (s == SWAN_OK)
    s = dev_alloc(c, (void**)&c->pool, (size_t)c->num_pages * (size_t)c->page_bytes, "page pool");
  if (s == SWAN_OK) s = dev_alloc(c, (void**)&c->page_table, pt_elems * sizeof(int32_t), "page table");
  if (s == SWAN_OK) s = dev_alloc(c, (void**)&c->ring_k, ring_elems * sizeof(__half), "key ring");
  if (s == SWAN_OK) s = dev_alloc(c, (void**)&c->ring_v, ring_elems * sizeof(__half), "value ring");
  if (s == SWAN_OK) s = dev_alloc(c, (void**)&c->qprime, q_elems * sizeof(float), "rotated queries");
  if (s == SWAN_OK) s = dev_alloc(c, (void**)&c->partials, part_elems * sizeof(float), "split partials");
  if (s == SWAN_OK) s = dev_alloc(c, (void**)&c->counters, (size_t)c->units * sizeof(int), "counters");
  if (s == SWAN_OK) s = dev_alloc(c, (void**)&c->status, sizeof(unsigned), "status word");
  if (s != SWAN_OK) {
    free_all(c);
    delete c;
    return s;
  }
  if (!R_vo) c->R_vo = c->R_qk;

  // Contents: R copies, identity page table, zeroed pool and rings.
  std::vector<int32_t> pt(pt_elems);
  for (size_t i = 0; i < pt_elems; ++i) pt[i] = (int32_t)i;
  cudaStream_t st = c->stream;
  e = cudaMemcpyAsync(c->R_qk, R_qk, rmat * sizeof(float), cudaMemcpyDeviceToDevice, st);
  if (e == cudaSuccess && R_vo)
    e = cudaMemcpyAsync(c->R_vo, R_vo, rmat * sizeof(float), cudaMemcpyDeviceToDevice, st);
  if (e == cudaSuccess) e = launch_transpose_r(c->R_vo, c->R_voT, (int64_t)C.num_layers * C.n_kv_heads, st);
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(c->page_table, pt.data(), pt_elems * sizeof(int32_t), cudaMemcpyHostToDevice, st);
  if (e == cudaSuccess) e = cudaMemsetAsync(c->pool, 0, (size_t)c->num_pages * (size_t)c->page_bytes, st);
  if (e == cudaSuccess) e = cudaMemsetAsync(c->ring_k, 0, ring_elems * sizeof(__half), st);
  if (e == cudaSuccess) e = cudaMemsetAsync(c->ring_v, 0, ring_elems * sizeof(__half), st);
  if (e == cudaSuccess) e = cudaMemsetAsync(c->counters, 0, (size_t)c->units * sizeof(int), st);
  if (e == cudaSuccess) e = cudaMemsetAsync(c->status, 0, sizeof(unsigned), st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);  // pt is a pageable host vector
  if (e != cudaSuccess) {
    swan_status r = fail(SWAN_ERR_CUDA, "initialising the cache: %s", cudaGetErrorString(e));
    free_all(c);
    delete c;
    return r;
  }
  *out = c;
  return SWAN_OK;
}

swan_status swan_destroy(swan_ctx* c) {
  if (!c) return SWAN_OK;
  cudaStreamSynchronize(c->stream);
  cudaGetLastError();
  free_all(c);
  delete c;
  return SWAN_OK;
}

swan_status swan_set_kv(swan_ctx* c, int k_active, int k_active_v) {
  swan_status s = usable(c);
  if (s != SWAN_OK) return s;
  if (k_active < 1 || k_active > c->cfg.k_store)
    return fail(SWAN_ERR_INVALID_ARG, "k_active %d out of [1, %d]", k_active, c->cfg.k_store);
  if (k_active_v < 1 || k_active_v > c->k_store_v)
    return fail(SWAN_ERR_INVALID_ARG, "k_active_v %d out of [1, %d]", k_active_v, c->k_store_v);
  c->k_active = k_active;
  c->k_active_v = k_active_v;
  return SWAN_OK;
}

swan_status swan_set_k(swan_ctx* c, int k_active) {
  swan_status s = usable(c);
  if (s != SWAN_OK) return s;
  if (k_active < 1 || k_active > c->cfg.k_store)
    return fail(SWAN_ERR_INVALID_ARG, "k_active %d out of [1, %d]", k_active, c->cfg.k_store);
  c->k_active = k_active;
  c->k_active_v = std::min(k_active, c->k_store_v);
  return SWAN_OK;
}

swan_status swan_append(swan_ctx* c, int layer, const void* k_new, const void* v_new, int T) {
  swan_status s = usable(c);
  if (s != SWAN_OK) return s;
  if ((s = check_layer(c, layer)) != SWAN_OK) return s;
  if (T < 0) return fail(SWAN_ERR_INVALID_ARG, "T %d < 0", T);
  if (T == 0) return SWAN_OK;
  if (!k_new || !v_new) return fail(SWAN_ERR_INVALID_ARG, "k_new or v_new is NULL");
  LayerState& L = c->layers[layer];
  const int cap = c->cfg.buffer_cap;
  const int64_t total = L.sparse_len + L.buf_count + (int64_t)T;
  if (total > c->cfg.max_seq)
    return fail(SWAN_ERR_CAPACITY, "layer %d would hold %lld tokens > max_seq %d", layer, (long long)total,
                c->cfg.max_seq);
  if ((int64_t)c->cfg.batch * T > (int64_t)INT32_MAX * 128)
    return fail(SWAN_ERR_INVALID_ARG, "T too large");

  // Algorithm 1 generalised to T tokens: logical positions 0..n_b-1 are the
  // buffered tokens (oldest first), n_b..n_b+T-1 the new ones; everything
  // before `evict` goes to the sparse history, in order.
  const int64_t evict = std::max<int64_t>(0, (int64_t)L.buf_count + T - cap);
  const int old_evict = (int)std::min<int64_t>(evict, L.buf_count);

  const int64_t sparse_before = L.sparse_len;
  const int start_before = L.buf_start;
  const int count_before = L.buf_count;
  // Decode-step appends (few vectors per head) run as one launch that evicts
  // and inserts; bulk appends as a pruning launch for the evicted buffered
  // tokens followed by the rotation launch.
  const bool small = (int64_t)c->cfg.batch * T <= kSmallAppendVectors &&
                     (int64_t)c->cfg.batch * old_evict <= kSmallAppendVectors;

  // 1) prune the evicted buffered tokens (they leave the ring first, so the
  //    new tokens may reuse their slots)
  if (!small && (s = prune_from_ring(c, layer, old_evict)) != SWAN_OK) return s;

  // 2) rotate the new tokens; those before `evict` are pruned directly, the
  //    rest land in the ring after the surviving buffered tokens
  AppendParams p{};
  p.k_new = static_cast<const __half*>(k_new);
  p.v_new = static_cast<const __half*>(v_new);
  p.R_qk = c->R_qk + (size_t)layer * c->cfg.n_kv_heads * kHeadDim * kHeadDim;
  p.R_vo = c->R_vo + (size_t)layer * c->cfg.n_kv_heads * kHeadDim * kHeadDim;
  p.ring_k = c->ring_k + (size_t)layer * ring_elems_per_layer(c);
  p.ring_v = c->ring_v + (size_t)layer * ring_elems_per_layer(c);
  p.B = c->cfg.batch;
  p.H = c->cfg.n_kv_heads;
  p.T = T;
  p.cap = cap > 0 ? cap : 1;
  p.buf_start = start_before;
  p.n_b = count_before;
  p.evict = evict;
  p.sparse_len = sparse_before;
  p.geom = geom_for(c, layer);
  p.status = c->status;
  if (small)
    s = launch(c, SWAN_KERNEL_APPEND, "append_small kernel",
               [&] { return launch_append_small(p, old_evict, c->stream); });
  else
    s = launch(c, SWAN_KERNEL_APPEND, "append kernel", [&] { return launch_append(p, c->stream); });
  if (s != SWAN_OK) return s;

  L.sparse_len = sparse_before + evict;
  L.buf_count = (int)((int64_t)count_before + T - evict);
  L.buf_start = cap > 0 ? (int)((start_before + evict) % cap) : 0;
  return SWAN_OK;
}

swan_status swan_flush_buffer(swan_ctx* c, int layer) {
  swan_status s = usable(c);
  if (s != SWAN_OK) return s;
  if (layer == -1) {
    for (int l = 0; l < c->cfg.num_layers; ++l)
      if ((s = prune_from_ring(c, l, c->layers[l].buf_count)) != SWAN_OK) return s;
    return SWAN_OK;
  }
  if ((s = check_layer(c, layer)) != SWAN_OK) return s;
  return prune_from_ring(c, layer, c->layers[layer].buf_count);
}

swan_status swan_decode(swan_ctx* c, int layer, const void* q, void* out) {
  swan_status s = usable(c);
  if (s != SWAN_OK) return s;
  if ((s = check_layer(c, layer)) != SWAN_OK) return s;
  if (!q || !out) return fail(SWAN_ERR_INVALID_ARG, "q or out is NULL");
  const size_t qbytes = (size_t)c->cfg.batch * c->cfg.n_q_heads * kHeadDim * 2;
  const char* qa = static_cast<const char*>(q);
  const char* oa = static_cast<const char*>(out);
  if (qa < oa + qbytes && oa < qa + qbytes) return fail(SWAN_ERR_INVALID_ARG, "q and out overlap");
  const LayerState& L = c->layers[layer];
  const int G = c->G;
  const float* R_qk = c->R_qk + (size_t)layer * c->cfg.n_kv_heads * kHeadDim * kHeadDim;

  RotateQParams rq{};
  rq.q = static_cast<const __half*>(q);
  rq.R_qk = R_qk;
  rq.qprime = c->qprime;
  rq.H_q = c->cfg.n_q_heads;
  rq.G = G;
  s = launch(c, SWAN_KERNEL_ROTATE_Q, "rotate_q kernel",
             [&] { return launch_rotate_q(rq, c->cfg.batch, c->stream); });
  if (s != SWAN_OK) return s;

  const int64_t n_sg = (L.sparse_len + 31) / 32;
  const int64_t n_bg = (L.buf_count + 31) / 32;
  const int64_t N_g = n_sg + n_bg;
  const int64_t total = c->units * N_g;
  int64_t range = 1, grid = 0;
  if (total > 0) {
    const int64_t ctas = std::min<int64_t>(c->decode_ctas, total);
    range = (total + ctas - 1) / ctas;
    grid = (total + range - 1) / range;
  }
  if (grid > 0) {
    DecodeParams p{};
    p.qprime = c->qprime;
    p.geom = geom_for(c, layer);
    p.ring_k = c->ring_k + (size_t)layer * ring_elems_per_layer(c);
    p.ring_v = c->ring_v + (size_t)layer * ring_elems_per_layer(c);
    p.cap = c->cfg.buffer_cap > 0 ? c->cfg.buffer_cap : 1;
    p.buf_start = L.buf_start;
    p.n_b = L.buf_count;
    p.sparse_len = L.sparse_len;
    p.n_sg = n_sg;
    p.N_g = N_g;
    p.total_groups = total;
    p.range = range;
    p.H_kv = c->cfg.n_kv_heads;
    p.H_q = c->cfg.n_q_heads;
    p.blocks_per_page_log2 = __builtin_ctz((unsigned)(c->P / 32));
    p.k_full_chunks = c->k_active / 8;
    p.k_rem = c->k_active % 8;
    p.k_full_chunks_v = c->k_active_v / 8;
    p.k_rem_v = c->k_active_v % 8;
    p.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)kHeadDim));
    p.partials = c->partials;
    p.counters = c->counters;
    p.R_voT = c->R_voT + (size_t)layer * c->cfg.n_kv_heads * kHeadDim * kHeadDim;
    p.out = static_cast<__half*>(out);
    p.status = c->status;
    // the split combine and the rotate-back run inside the decode kernel
    return launch(c, SWAN_KERNEL_DECODE, "decode kernel",
                  [&] {
                    const int k_read = (std::max(c->k_active, c->k_active_v) + 7) / 8 * 8;
                    return launch_decode(p, G, k_read, (int)grid, c->stream);
                  });
  }
  // empty cache: the combine kernel writes zeros

  CombineParams cp{};
  cp.partials = c->partials;
  cp.R_voT = c->R_voT + (size_t)layer * c->cfg.n_kv_heads * kHeadDim * kHeadDim;
  cp.out = static_cast<__half*>(out);
  cp.H_kv = c->cfg.n_kv_heads;
  cp.H_q = c->cfg.n_q_heads;
  cp.G = G;
  cp.N_g = N_g > 0 ? N_g : 1;
  cp.range = range;
  cp.total_groups = total;
  return launch(c, SWAN_KERNEL_COMBINE, "combine kernel",
                [&] { return launch_combine(cp, c->cfg.batch, c->stream); });
}

swan_status swan_query(const swan_ctx* c, int layer, swan_layer_info* info) {
  swan_status s = usable(c);
  if (s != SWAN_OK) return s;
  if ((s = check_layer(c, layer)) != SWAN_OK) return s;
  if (!info) return fail(SWAN_ERR_INVALID_ARG, "info is NULL");
  info->sparse_len = c->layers[layer].sparse_len;
  info->buffer_len = c->layers[layer].buf_count;
  info->k_active = c->k_active;
  info->k_store = c->cfg.k_store;
  info->k_slots = c->k_slots;
  info->k_active_v = c->k_active_v;
  info->k_store_v = c->k_store_v;
  info->k_slots_v = c->k_slots_v;
  info->page_tokens = c->P;
  info->page_bytes = c->page_bytes;
  info->device_bytes = c->device_bytes;
  info->value_format = c->fmt == kFmtFp8 ? SWAN_VALUES_FP8_E4M3 : SWAN_VALUES_FP16;
  return SWAN_OK;
}

swan_status swan_debug_export(swan_ctx* c, int layer, int what, void* host_dst, size_t bytes) {
  swan_status s = usable(c);
  if (s != SWAN_OK) return s;
  if ((s = check_layer(c, layer)) != SWAN_OK) return s;
  if (!host_dst) return fail(SWAN_ERR_INVALID_ARG, "host_dst is NULL");
  const LayerState& L = c->layers[layer];
  const int cap = c->cfg.buffer_cap;
  cudaError_t e = cudaStreamSynchronize(c->stream);
  if (e != cudaSuccess) return cuda_fail(c, e, "cudaStreamSynchronize");

  if (what == SWAN_EXPORT_BUFFER_K || what == SWAN_EXPORT_BUFFER_V) {
    const size_t need = (size_t)c->units * L.buf_count * kHeadDim * 2;
    if (bytes != need) return fail(SWAN_ERR_INVALID_ARG, "bytes %zu != %zu", bytes, need);
    if (need == 0) return SWAN_OK;
    const __half* ring = (what == SWAN_EXPORT_BUFFER_K ? c->ring_k : c->ring_v) +
                         (size_t)layer * ring_elems_per_layer(c);
    std::vector<uint16_t> all((size_t)c->units * cap * kHeadDim);
    e = cudaMemcpy(all.data(), ring, all.size() * 2, cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_fail(c, e, "cudaMemcpy");
    uint16_t* dst = static_cast<uint16_t*>(host_dst);
    for (int64_t u = 0; u < c->units; ++u)
      for (int i = 0; i < L.buf_count; ++i) {
        const int slot = (L.buf_start + i) % cap;
        std::memcpy(dst + ((size_t)u * L.buf_count + i) * kHeadDim,
                    all.data() + ((size_t)u * cap + slot) * kHeadDim, kHeadDim * 2);
      }
    return SWAN_OK;
  }
  if (what == SWAN_EXPORT_SPARSE_K || what == SWAN_EXPORT_SPARSE_V) {
    const bool isv_ = what == SWAN_EXPORT_SPARSE_V;
    const int ks = isv_ ? c->k_store_v : c->cfg.k_store;
    const size_t n_ent = (size_t)c->units * L.sparse_len * ks;
    const size_t need = n_ent * 3;
    if (bytes != need) return fail(SWAN_ERR_INVALID_ARG, "bytes %zu != %zu", bytes, need);
    if (need == 0) return SWAN_OK;
    const bool isv = what == SWAN_EXPORT_SPARSE_V;
    const bool fp8 = c->fmt == kFmtFp8;
    const int64_t P = c->P;
    const int64_t ksk = c->k_slots, ksv = c->k_slots_v;
    const int64_t blk = (fp8 ? 64 : 96) * (ksk + ksv);
    // fp16: value records of 16 B and index records of 8 B in separate
    // regions; fp8: 16-byte records of 8 values then 8 indices
    const int64_t voff = fp8 ? (isv ? 64 * ksk : 0) : (isv ? 96 * ksk : 0);
    const int64_t ioff = fp8 ? voff + 8 : (isv ? 96 * ksk + 64 * ksv : 64 * ksk);
    std::vector<int32_t> pt((size_t)c->units * c->ppu);
    e = cudaMemcpy(pt.data(), c->page_table + (int64_t)layer * c->units * c->ppu, pt.size() * 4,
                   cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_fail(c, e, "cudaMemcpy");
    uint8_t* idx_dst = static_cast<uint8_t*>(host_dst);
    uint16_t* val_dst = reinterpret_cast<uint16_t*>(idx_dst + n_ent);
    std::vector<uint8_t> page(c->page_bytes);
    const int64_t pages_used = (L.sparse_len + P - 1) / P;
    for (int64_t u = 0; u < c->units; ++u)
      for (int64_t pg = 0; pg < pages_used; ++pg) {
        const int32_t phys = pt[(size_t)u * c->ppu + pg];
        if (phys < 0 || phys >= c->num_pages) return fail(SWAN_ERR_DEVICE_CHECK, "page table corrupt");
        e = cudaMemcpy(page.data(), c->pool + (int64_t)phys * c->page_bytes, c->page_bytes,
                       cudaMemcpyDeviceToHost);
        if (e != cudaSuccess) return cuda_fail(c, e, "cudaMemcpy");
        for (int64_t sl = 0; sl < P; ++sl) {
          const int64_t t = pg * P + sl;
          if (t >= L.sparse_len) break;
          const int64_t b0 = (sl / 32) * blk;
          for (int r = 0; r < ks; ++r) {
            const int64_t rec = (int64_t)(r / 8) * 32 + (sl % 32);
            const size_t o = ((size_t)u * L.sparse_len + t) * ks + r;
            if (fp8) {
              idx_dst[o] = page[b0 + ioff + rec * 16 + (r % 8)];
              val_dst[o] = e4m3_to_half_bits(page[b0 + voff + rec * 16 + (r % 8)]);
            } else {
              idx_dst[o] = page[b0 + ioff + rec * 8 + (r % 8)];
              uint16_t v;
              std::memcpy(&v, page.data() + b0 + voff + rec * 16 + (r % 8) * 2, 2);
              val_dst[o] = v;
            }
          }
        }
      }
    return SWAN_OK;
  }
  return fail(SWAN_ERR_INVALID_ARG, "unknown export kind %d", what);
}

swan_status swan_check(swan_ctx* c) {
  swan_status s = usable(c);
  if (s != SWAN_OK) return s;
  cudaError_t e = cudaStreamSynchronize(c->stream);
  if (e != cudaSuccess) return cuda_fail(c, e, "cudaStreamSynchronize");
  unsigned word = 0;
  e = cudaMemcpy(&word, c->status, sizeof(word), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(c, e, "cudaMemcpy");
  if (word) {
    e = cudaMemset(c->status, 0, sizeof(unsigned));
    if (e != cudaSuccess) return cuda_fail(c, e, "cudaMemset");
    return fail(SWAN_ERR_DEVICE_CHECK, "device status word 0x%x", word);
  }
  return SWAN_OK;
}

swan_status swan_timing_enable(swan_ctx* c, int enable) {
  swan_status s = usable(c);
  if (s != SWAN_OK) return s;
  if ((s = drain_events(c)) != SWAN_OK) return s;
  for (int k = 0; k < SWAN_KERNEL_KINDS; ++k) {
    c->ms_acc[k] = 0.0;
    c->n_acc[k] = 0;
  }
  c->timing = enable != 0;
  return SWAN_OK;
}

swan_status swan_timing_read(swan_ctx* c, swan_timing* out) {
  swan_status s = usable(c);
  if (s != SWAN_OK) return s;
  if (!out) return fail(SWAN_ERR_INVALID_ARG, "out is NULL");
  if ((s = drain_events(c)) != SWAN_OK) return s;
  for (int k = 0; k < SWAN_KERNEL_KINDS; ++k) {
    out->ms[k] = c->ms_acc[k];
    out->launches[k] = c->n_acc[k];
    c->ms_acc[k] = 0.0;
    c->n_acc[k] = 0;
  }
  return SWAN_OK;
}

int64_t swan_launch_count(const swan_ctx* c) { return c ? c->launches : 0; }

}  // extern "C"
