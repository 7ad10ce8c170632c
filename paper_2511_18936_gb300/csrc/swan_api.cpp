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
#include <unordered_map>
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

// One sequence (batch row) of one layer.
struct SeqState {
  int64_t sparse_len = 0;
  int buf_start = 0;  // ring slot of the oldest buffered token
  int buf_count = 0;
  bool operator==(const SeqState& o) const {
    return sparse_len == o.sparse_len && buf_start == o.buf_start && buf_count == o.buf_count;
  }
};

struct LayerState {
  std::vector<SeqState> seq;  // [batch]
  bool uniform() const {
    for (const SeqState& q : seq)
      if (!(q == seq[0])) return false;
    return true;
  }
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
  bool paged = false;               // pages handed out on demand from a shared pool
  std::vector<int32_t> free_pages;  // paged: free page ids
  std::vector<int32_t> page_refs;   // paged: rows holding each page (> 1 after swan_fork_sequence)
  std::vector<int32_t> pt_host;     // paged: host copy of the page tables, -1 = none
  int fmt = kFmtFp16;
  int64_t units = 0;  // batch * n_kv_heads (per layer)
  cudaStream_t stream = nullptr;
  int device = 0;
  int num_sms = 0;
  int decode_ctas = 0;  // max decode CTAs resident at once (either kernel variant)
  int decode_ctas_v[kDecodeVariants] = {};  // per kernel variant: <= 32, 64, 96, 128 entries read

  float* R_qk = nullptr;
  float* R_vo = nullptr;   // == R_qk when the caller passed NULL
  float* R_voT = nullptr;  // transposed copy for the rotate-back
  __half* R_hi = nullptr;  // split rotations for the tensor-core append: [layer][2][H][n][k] fp16
  __half* R_lo = nullptr;
  CUtensorMap r_maps[2];   // TMA maps over R_hi, R_lo
  uint8_t* pool = nullptr;
  int32_t* page_table = nullptr;
  __half* ring_k = nullptr;
  __half* ring_v = nullptr;
  float* qprime = nullptr;
  float* partials = nullptr;
  int* counters = nullptr;  // per-unit arrival counters of the fused combine
  unsigned* status = nullptr;
  uint8_t* seq_dev = nullptr;  // per layer: [batch] SeqInfo, then [decode_ctas + 1] CTA starts
  size_t seq_stride = 0;       // bytes per layer of seq_dev
  int2* pt_pairs = nullptr;    // paged: (entry, page) updates of one call
  int64_t device_bytes = 0;

  // every device allocation, with guard regions before and after it
  struct DevBuf {
    void* base;
    size_t bytes;  // without the guards
    const char* what;
  };
  std::vector<DevBuf> bufs;

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

// Guard regions of kGuardByte before (64 KB: the buffer keeps the 64 KB
// alignment of a large allocation, which the decode stream measurably
// prefers over a 256-byte offset) and after (256 bytes) every device buffer;
// swan_debug_check_guards reports any that a kernel overwrote.
constexpr size_t kFrontGuard = 65536;
constexpr size_t kBackGuard = 256;
constexpr unsigned char kGuardByte = 0xA5;

// Test hooks: the n-th next device allocation / kernel launch fails (n = 0:
// the next one); -1 = off.  Process-wide.
std::atomic<int64_t> g_fail_alloc{-1};
std::atomic<int64_t> g_fail_launch{-1};
bool injected(std::atomic<int64_t>& n) {
  int64_t v = n.load();
  while (v >= 0)
    if (n.compare_exchange_weak(v, v - 1)) return v == 0;
  return false;
}

void free_all(swan_ctx* c) {
  for (const auto& b : c->bufs) cudaFree(b.base);
  c->bufs.clear();
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
  *p = nullptr;
  if (injected(g_fail_alloc)) return fail(SWAN_ERR_NOMEM, "allocation for %s failed (injected)", what);
  void* base = nullptr;
  cudaError_t e = cudaMalloc(&base, kFrontGuard + bytes + kBackGuard);
  if (e != cudaSuccess) {
    cudaGetLastError();
    return fail(SWAN_ERR_NOMEM, "cudaMalloc of %zu bytes for %s failed: %s", bytes, what,
                cudaGetErrorString(e));
  }
  c->bufs.push_back({base, bytes, what});
  *p = static_cast<char*>(base) + kFrontGuard;
  c->device_bytes += (int64_t)(kFrontGuard + bytes + kBackGuard);
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
  if (injected(g_fail_launch)) return cuda_fail(c, cudaErrorLaunchFailure, name);  // nothing launched
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
  g.identity = c->paged ? 0 : 1;
  g.identity_base = (int64_t)layer * c->units * c->ppu;
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

int64_t pages_for(int64_t tokens, int P) { return (tokens + P - 1) / P; }

int32_t& pt_entry(swan_ctx* c, int layer, int64_t unit, int64_t pg) {
  return c->pt_host[((size_t)layer * c->units + unit) * c->ppu + pg];
}

// Pages a layer's rows need to reach new_len[b] sparse tokens: fresh pages
// past each row's last one, plus copies of the last, partly filled pages
// that a row will write into while other rows (forks) still hold them. A
// page that every holder writes into is copied for all but one of them.
int64_t pages_needed(swan_ctx* c, int layer, const std::vector<int64_t>& new_len) {
  const LayerState& L = c->layers[layer];
  const int H = c->cfg.n_kv_heads;
  int64_t need = 0;
  std::unordered_map<int32_t, int> writers;
  for (int b = 0; b < c->cfg.batch; ++b) {
    const int64_t len = L.seq[b].sparse_len;
    need += (int64_t)H * std::max<int64_t>(0, pages_for(new_len[b], c->P) - pages_for(len, c->P));
    if (new_len[b] > len && len % c->P != 0)
      for (int h = 0; h < H; ++h) {
        const int32_t id = pt_entry(c, layer, (int64_t)b * H + h, len / c->P);
        if (c->page_refs[(size_t)id] > 1) ++writers[id];
      }
  }
  for (const auto& w : writers) need += w.second < c->page_refs[(size_t)w.first] ? w.second : w.second - 1;
  return need;
}

// Paged pool: give every unit of each row the pages its sparse history needs
// to reach new_len[b] tokens, and write them into the device page table.
// A row about to write into a last page it shares with a fork gets its own
// copy first (copy on write: only a row's last, partly filled page is ever
// written, so full pages stay shared).  Nothing changes when the pool is too
// small.
swan_status grow_pages(swan_ctx* c, int layer, const std::vector<int64_t>& new_len) {
  if (!c->paged) return SWAN_OK;
  LayerState& L = c->layers[layer];
  const int H = c->cfg.n_kv_heads;
  const int64_t need = pages_needed(c, layer, new_len);
  if (need == 0) return SWAN_OK;
  if (need > (int64_t)c->free_pages.size())
    return fail(SWAN_ERR_CAPACITY, "layer %d needs %lld more pages, the pool has %zu free", layer, (long long)need,
                c->free_pages.size());
  std::vector<int2> pairs;
  pairs.reserve((size_t)need);
  for (int b = 0; b < c->cfg.batch; ++b) {
    const int64_t len = L.seq[b].sparse_len;
    const int64_t p0 = pages_for(len, c->P), p1 = pages_for(new_len[b], c->P);
    for (int h = 0; h < H; ++h) {
      const int64_t unit = (int64_t)b * H + h;
      if (new_len[b] > len && len % c->P != 0) {
        int32_t& slot = pt_entry(c, layer, unit, len / c->P);
        const int32_t old = slot;
        if (c->page_refs[(size_t)old] > 1) {
          const int32_t id = c->free_pages.back();
          c->free_pages.pop_back();
          const cudaError_t e = cudaMemcpyAsync(c->pool + (int64_t)id * c->page_bytes,
                                                c->pool + (int64_t)old * c->page_bytes, (size_t)c->page_bytes,
                                                cudaMemcpyDeviceToDevice, c->stream);
          if (e != cudaSuccess) return cuda_fail(c, e, "copying a shared page");
          --c->page_refs[(size_t)old];
          c->page_refs[(size_t)id] = 1;
          slot = id;
          pairs.push_back(make_int2((int)(unit * c->ppu + len / c->P), id));
        }
      }
      for (int64_t pg = p0; pg < p1; ++pg) {
        const int32_t id = c->free_pages.back();
        c->free_pages.pop_back();
        c->page_refs[(size_t)id] = 1;
        pt_entry(c, layer, unit, pg) = id;
        pairs.push_back(make_int2((int)(unit * c->ppu + pg), id));
      }
    }
  }
  cudaError_t e = cudaMemcpyAsync(c->pt_pairs, pairs.data(), pairs.size() * sizeof(int2), cudaMemcpyHostToDevice,
                                  c->stream);
  if (e != cudaSuccess) return cuda_fail(c, e, "uploading page-table entries");
  int32_t* table = c->page_table + (int64_t)layer * c->units * c->ppu;
  return launch(c, SWAN_KERNEL_PRUNE, "page-table scatter",
                [&] { return launch_scatter_pages(c->pt_pairs, (int)pairs.size(), table, c->stream); });
}

SeqInfo* rows_of(swan_ctx* c, int layer) {
  return reinterpret_cast<SeqInfo*>(c->seq_dev + (size_t)layer * c->seq_stride);
}
int64_t* cta_starts_of(swan_ctx* c, int layer) {
  return reinterpret_cast<int64_t*>(c->seq_dev + (size_t)layer * c->seq_stride + (size_t)c->cfg.batch * sizeof(SeqInfo));
}

// Upload a layer's per-row table (and, for a decode, the CTA starts right
// after it) for the next ragged launch: one copy, ordered on the stream; the
// host vectors may be reused once this returns.
swan_status upload_rows(swan_ctx* c, int layer, const std::vector<SeqInfo>& rows,
                        const std::vector<int64_t>* starts = nullptr) {
  std::vector<uint8_t> buf(rows.size() * sizeof(SeqInfo) + (starts ? starts->size() * sizeof(int64_t) : 0));
  std::memcpy(buf.data(), rows.data(), rows.size() * sizeof(SeqInfo));
  if (starts) std::memcpy(buf.data() + rows.size() * sizeof(SeqInfo), starts->data(), starts->size() * sizeof(int64_t));
  cudaError_t e = cudaMemcpyAsync(rows_of(c, layer), buf.data(), buf.size(), cudaMemcpyHostToDevice, c->stream);
  if (e != cudaSuccess) return cuda_fail(c, e, "uploading per-row lengths");
  return SWAN_OK;
}


// Work of one unit segment of a decode CTA beyond its groups (staging q',
// the merge, the rotate-back, and the pipeline start of every warp's short
// run), in 32-token groups; measured on the ragged serving batch (a sweep of
// 12 to 96 took its decode from 1.89 to 1.12 ms, level with equal rows).
// First group of each decode CTA for ragged rows: contiguous ranges of equal
// cost, a unit costing its groups plus `visit` groups for every CTA it is
// processed by, so that CTAs covering many short rows take fewer groups.
std::vector<int64_t> balanced_starts(const std::vector<int64_t>& row_groups, int H, int64_t max_ctas,
                                     int64_t visit) {
  int64_t total = 0;
  for (int64_t g : row_groups) total += g * H;
  const int64_t units = (int64_t)row_groups.size() * H;
  const int64_t ctas = std::max<int64_t>(1, std::min<int64_t>(max_ctas, total));
  const double target = ((double)total + (double)visit * units) / (double)ctas;
  std::vector<int64_t> starts{0};
  int64_t next = 1, goff = 0, u = 0;
  for (int64_t ng : row_groups)
    for (int h = 0; h < H; ++h, ++u) {
      // group goff + j costs base + j so far (this unit's overhead included)
      const double base = (double)goff + (double)visit * (double)(u + 1);
      while (next < ctas && (double)next * target <= base + (double)(ng - 1)) {
        const int64_t j = std::max<int64_t>(0, (int64_t)std::ceil((double)next * target - base));
        const int64_t g = goff + j;
        if (g > starts.back() && g < total) starts.push_back(g);
        ++next;
      }
      goff += ng;
    }
  starts.push_back(total);
  return starts;
}

// Prune buffered tokens 0..count[b]-1 of every row b of a layer into the
// sparse cache (eviction before a bulk append, and flush).
swan_status prune_from_ring(swan_ctx* c, int layer, const std::vector<int>& count) {
  LayerState& L = c->layers[layer];
  const int B = c->cfg.batch;
  int most = 0;
  bool same = L.uniform();
  for (int b = 0; b < B; ++b) {
    most = std::max(most, count[b]);
    same = same && count[b] == count[0];
  }
  if (most <= 0) return SWAN_OK;
  std::vector<int64_t> new_len(B);
  for (int b = 0; b < B; ++b) new_len[b] = L.seq[b].sparse_len + count[b];
  swan_status s = grow_pages(c, layer, new_len);
  if (s != SWAN_OK) return s;
  PruneRingParams p{};
  p.ring_k = c->ring_k + (size_t)layer * ring_elems_per_layer(c);
  p.ring_v = c->ring_v + (size_t)layer * ring_elems_per_layer(c);
  p.units = (int)c->units;
  p.cap = c->cfg.buffer_cap;
  p.buf_start = L.seq[0].buf_start;
  p.count = most;
  p.sparse_len = L.seq[0].sparse_len;
  p.H = c->cfg.n_kv_heads;
  p.geom = geom_for(c, layer);
  p.status = c->status;
  if (!same) {
    std::vector<SeqInfo> rows(B);
    for (int b = 0; b < B; ++b) {
      rows[b] = SeqInfo{};
      rows[b].sparse_len = L.seq[b].sparse_len;
      rows[b].buf_start = L.seq[b].buf_start;
      rows[b].n_b = L.seq[b].buf_count;
      rows[b].prune = count[b];
    }
    if ((s = upload_rows(c, layer, rows)) != SWAN_OK) return s;
    p.seq = rows_of(c, layer);
  }
  s = launch(c, SWAN_KERNEL_PRUNE, "prune_ring kernel", [&] { return launch_prune_ring(p, c->stream); });
  if (s != SWAN_OK) return s;
  for (int b = 0; b < B; ++b) {
    SeqState& q = L.seq[b];
    q.sparse_len += count[b];
    q.buf_start = c->cfg.buffer_cap ? (q.buf_start + count[b]) % c->cfg.buffer_cap : 0;
    q.buf_count -= count[b];
  }
  return SWAN_OK;
}

std::vector<int> buffer_counts(const LayerState& L) {
  std::vector<int> n(L.seq.size());
  for (size_t b = 0; b < L.seq.size(); ++b) n[b] = L.seq[b].buf_count;
  return n;
}

}  // namespace

void swan::set_last_error(const char* msg) { g_last_error = msg ? msg : ""; }

namespace swan {
namespace {
std::atomic<int64_t> g_tc_starve{0};
}  // namespace
int64_t take_tc_starve() {
  return g_tc_starve.load(std::memory_order_relaxed) ? g_tc_starve.exchange(0) : 0;
}
}  // namespace swan

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
  if (G != 1 && G != 2 && G != 4 && G != 8)
    return fail(SWAN_ERR_UNSUPPORTED, "group size %d: only 1, 2, 4 and 8 are built", G);
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
  if (C.pool_pages < 0) return fail(SWAN_ERR_INVALID_ARG, "pool_pages %d < 0", C.pool_pages);

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
  const int64_t full_pages = (int64_t)C.num_layers * c->units * c->ppu;
  c->paged = C.pool_pages > 0;
  c->num_pages = c->paged ? (int64_t)C.pool_pages : full_pages;
  c->stream = static_cast<cudaStream_t>(C.stream);
  c->device = dev;
  c->num_sms = sms;
  c->layers.assign(C.num_layers, LayerState{});
  for (LayerState& L : c->layers) L.seq.assign(C.batch, SeqState{});

  // resident decode CTAs of the kernel variant each runtime keep count uses
  const int slots = std::max(c->k_slots, c->k_slots_v);
  for (int v = 0; v < kDecodeVariants; ++v) {
    const int k_read = 32 + 32 * v;  // the largest keep count of the variant
    if (v > 0 && slots <= k_read - 32) {
      c->decode_ctas_v[v] = c->decode_ctas_v[v - 1];  // never launched: no larger count is stored
      continue;
    }
    const int per_sm = decode_ctas_per_sm(G, k_read);
    if (per_sm < 1) {
      delete c;
      return fail(SWAN_ERR_CUDA, "decode kernel does not fit on an SM (%s)",
                  cudaGetErrorString(cudaGetLastError()));
    }
    c->decode_ctas_v[v] = per_sm * sms;
    c->decode_ctas = std::max(c->decode_ctas, c->decode_ctas_v[v]);
  }

  const size_t rmat = (size_t)C.num_layers * C.n_kv_heads * kHeadDim * kHeadDim;
  const size_t ring_elems = (size_t)C.num_layers * ring_elems_per_layer(c);
  const size_t q_elems = (size_t)C.batch * C.n_q_heads * kHeadDim;
  const size_t pairs = (size_t)c->decode_ctas + (size_t)c->units;
  const size_t part_elems = pairs * G * (kHeadDim + 2);
  const size_t pt_elems = (size_t)full_pages;  // page-table entries: [layer][unit][page]
  if (full_pages > INT32_MAX || c->num_pages > INT32_MAX) {
    const long long np = (long long)std::max(full_pages, c->num_pages);
    delete c;
    return fail(SWAN_ERR_UNSUPPORTED, "too many pages (%lld)", np);
  }

  swan_status s = SWAN_OK;
  if (s == SWAN_OK) s = dev_alloc(c, (void**)&c->R_qk, rmat * sizeof(float), "R_qk");
  if (s == SWAN_OK && R_vo) s = dev_alloc(c, (void**)&c->R_vo, rmat * sizeof(float), "R_vo");
  if (s == SWAN_OK) s = dev_alloc(c, (void**)&c->R_voT, rmat * sizeof(float), "R_vo^T");
  if (s == SWAN_OK) s = dev_alloc(c, (void**)&c->R_hi, 2 * rmat * sizeof(__half), "split R (hi)");
  if (s == SWAN_OK) s = dev_alloc(c, (void**)&c->R_lo, 2 * rmat * sizeof(__half), "split R (lo)");
  if (s == SWAN_OK)
    s = dev_alloc(c, (void**)&c->pool, (size_t)c->num_pages * (size_t)c->page_bytes, "page pool");
  if (s == SWAN_OK) s = dev_alloc(c, (void**)&c->page_table, pt_elems * sizeof(int32_t), "page table");
  if (s == SWAN_OK) s = dev_alloc(c, (void**)&c->ring_k, ring_elems * sizeof(__half), "key ring");
  if (s == SWAN_OK) s = dev_alloc(c, (void**)&c->ring_v, ring_elems * sizeof(__half), "value ring");
  if (s == SWAN_OK) s = dev_alloc(c, (void**)&c->qprime, q_elems * sizeof(float), "rotated queries");
  if (s == SWAN_OK) s = dev_alloc(c, (void**)&c->partials, part_elems * sizeof(float), "split partials");
  if (s == SWAN_OK) s = dev_alloc(c, (void**)&c->counters, (size_t)c->units * sizeof(int), "counters");
  if (s == SWAN_OK) s = dev_alloc(c, (void**)&c->status, sizeof(unsigned), "status word");
  c->seq_stride = ((size_t)C.batch * sizeof(SeqInfo) + ((size_t)c->decode_ctas + 1) * sizeof(int64_t) + 255) / 256 * 256;
  if (s == SWAN_OK)
    s = dev_alloc(c, (void**)&c->seq_dev, (size_t)C.num_layers * c->seq_stride, "per-row lengths");
  if (s == SWAN_OK && c->paged)
    s = dev_alloc(c, (void**)&c->pt_pairs, (size_t)c->units * c->ppu * sizeof(int2), "page-table updates");
  if (s != SWAN_OK) {
    free_all(c);
    delete c;
    return s;
  }
  if (!R_vo) c->R_vo = c->R_qk;

  // Contents: R copies, identity page table, zeroed pool and rings.
  // every unit owns its pages (identity table), or none until it needs them
  std::vector<int32_t> pt(pt_elems);
  for (size_t i = 0; i < pt_elems; ++i) pt[i] = c->paged ? -1 : (int32_t)i;
  if (c->paged) {
    c->pt_host = pt;
    c->page_refs.assign((size_t)c->num_pages, 0);
    c->free_pages.resize((size_t)c->num_pages);
    for (int64_t i = 0; i < c->num_pages; ++i) c->free_pages[(size_t)i] = (int32_t)(c->num_pages - 1 - i);
  }
  cudaStream_t st = c->stream;
  e = cudaMemcpyAsync(c->R_qk, R_qk, rmat * sizeof(float), cudaMemcpyDeviceToDevice, st);
  if (e == cudaSuccess && R_vo)
    e = cudaMemcpyAsync(c->R_vo, R_vo, rmat * sizeof(float), cudaMemcpyDeviceToDevice, st);
  if (e == cudaSuccess) e = launch_transpose_r(c->R_vo, c->R_voT, (int64_t)C.num_layers * C.n_kv_heads, st);
  if (e == cudaSuccess) e = launch_split_r(c->R_qk, c->R_vo, c->R_hi, c->R_lo, C.num_layers, C.n_kv_heads, st);
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(c->page_table, pt.data(), pt_elems * sizeof(int32_t), cudaMemcpyHostToDevice, st);
  if (e == cudaSuccess) e = cudaMemsetAsync(c->pool, 0, (size_t)c->num_pages * (size_t)c->page_bytes, st);
  if (e == cudaSuccess) e = cudaMemsetAsync(c->ring_k, 0, ring_elems * sizeof(__half), st);
  if (e == cudaSuccess) e = cudaMemsetAsync(c->ring_v, 0, ring_elems * sizeof(__half), st);
  if (e == cudaSuccess) e = cudaMemsetAsync(c->counters, 0, (size_t)c->units * sizeof(int), st);
  if (e == cudaSuccess) e = cudaMemsetAsync(c->status, 0, sizeof(unsigned), st);
  for (const auto& b : c->bufs) {
    if (e == cudaSuccess) e = cudaMemsetAsync(b.base, kGuardByte, kFrontGuard, st);
    if (e == cudaSuccess)
      e = cudaMemsetAsync(static_cast<char*>(b.base) + kFrontGuard + b.bytes, kGuardByte, kBackGuard, st);
  }
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);  // pt is a pageable host vector
  if (e != cudaSuccess) {
    swan_status r = fail(SWAN_ERR_CUDA, "initialising the cache: %s", cudaGetErrorString(e));
    free_all(c);
    delete c;
    return r;
  }
  {
    EncodeTiledFn enc = tensor_map_encoder();
    CUresult r = CUDA_ERROR_NOT_FOUND;
    if (enc) {
      const cuuint64_t dims[3] = {128, 128, (cuuint64_t)2 * C.num_layers * C.n_kv_heads};
      const cuuint64_t strides[2] = {256, 128 * 256};
      const cuuint32_t box[3] = {64, 128, 1}, estr[3] = {1, 1, 1};
      r = enc(&c->r_maps[0], CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 3, c->R_hi, dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
      if (r == CUDA_SUCCESS)
        r = enc(&c->r_maps[1], CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 3, c->R_lo, dims, strides, box, estr,
                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    }
    if (r != CUDA_SUCCESS) {
      swan_status rs = fail(SWAN_ERR_CUDA, "encoding the rotation tensor maps failed (%d)", (int)r);
      free_all(c);
      delete c;
      return rs;
    }
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

namespace {

// Append T (padded) tokens per row; row b takes n_new[b] of them (all T when
// n_new is null).  Algorithm 1 generalised to T tokens, per row: logical
// positions 0..n_b-1 are the buffered tokens (oldest first), n_b..n_b+T_b-1
// the new ones; everything before evict = max(0, n_b + T_b - b_cap) goes to
// the sparse history, in order.
// Append (Algorithm 1, compression part).  rq non-null: a decode step's query
// rotation that may run in the append's own launch; *rotated says whether it
// did (only a small append takes it).
swan_status append_rows(swan_ctx* c, int layer, const void* k_new, const void* v_new, int T,
                        const int32_t* n_new, const RotateQParams* rq = nullptr, bool* rotated = nullptr) {
  if (rotated) *rotated = false;
  swan_status s = usable(c);
  if (s != SWAN_OK) return s;
  if ((s = check_layer(c, layer)) != SWAN_OK) return s;
  if (T < 0) return fail(SWAN_ERR_INVALID_ARG, "T %d < 0", T);
  if (T == 0) return SWAN_OK;
  if (!k_new || !v_new) return fail(SWAN_ERR_INVALID_ARG, "k_new or v_new is NULL");
  if ((uintptr_t)k_new % 16 || (uintptr_t)v_new % 16)
    return fail(SWAN_ERR_INVALID_ARG, "k_new and v_new must be 16-byte aligned");
  if ((int64_t)c->cfg.batch * T > (int64_t)INT32_MAX * 128) return fail(SWAN_ERR_INVALID_ARG, "T too large");
  LayerState& L = c->layers[layer];
  const int B = c->cfg.batch;
  const int cap = c->cfg.buffer_cap;
  std::vector<int> Tb(B, T);
  if (n_new) {
    for (int b = 0; b < B; ++b) {
      if (n_new[b] < 0 || n_new[b] > T)
        return fail(SWAN_ERR_INVALID_ARG, "n_new[%d] = %d out of [0, %d]", b, n_new[b], T);
      Tb[b] = n_new[b];
    }
  }
  std::vector<int64_t> evict(B), new_len(B);
  std::vector<int> old_evict(B);
  int most_tokens = 0, most_old = 0;
  bool same = L.uniform();
  for (int b = 0; b < B; ++b) {
    const SeqState& q = L.seq[b];
    const int64_t total = q.sparse_len + q.buf_count + (int64_t)Tb[b];
    if (total > c->cfg.max_seq)
      return fail(SWAN_ERR_CAPACITY, "layer %d row %d would hold %lld tokens > max_seq %d", layer, b,
                  (long long)total, c->cfg.max_seq);
    evict[b] = std::max<int64_t>(0, (int64_t)q.buf_count + Tb[b] - cap);
    old_evict[b] = (int)std::min<int64_t>(evict[b], q.buf_count);
    new_len[b] = q.sparse_len + evict[b];
    most_tokens = std::max(most_tokens, Tb[b]);
    most_old = std::max(most_old, old_evict[b]);
    same = same && Tb[b] == T;
  }
  if (most_tokens == 0) return SWAN_OK;

  // Decode-step appends (few vectors per head) run as one launch that evicts
  // and inserts; bulk appends as a pruning launch for the evicted buffered
  // tokens followed by the rotation launch (tensor cores; TMA maps of this
  // call's keys and values, encoded before anything changes).
  const bool small = (int64_t)B * T <= kSmallAppendVectors && (int64_t)B * most_old <= kSmallAppendVectors;
  CUtensorMap maps[4];
  if (!small) {
    EncodeTiledFn enc = tensor_map_encoder();
    const cuuint64_t dims[4] = {128, (cuuint64_t)T, (cuuint64_t)c->cfg.n_kv_heads, (cuuint64_t)B};
    const cuuint64_t strides[3] = {256, (cuuint64_t)T * 256, (cuuint64_t)T * 256 * c->cfg.n_kv_heads};
    const cuuint32_t box[4] = {64, 128, 1, 1}, estr[4] = {1, 1, 1, 1};
    CUresult r = enc ? CUDA_SUCCESS : CUDA_ERROR_NOT_FOUND;
    for (int kk = 0; kk < 2 && r == CUDA_SUCCESS; ++kk)
      r = enc(&maps[kk], CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 4, const_cast<void*>(kk ? v_new : k_new), dims,
              strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return fail(SWAN_ERR_INVALID_ARG, "k_new / v_new: tensor-map encoding failed (%d)", (int)r);
    maps[2] = c->r_maps[0];
    maps[3] = c->r_maps[1];
  }
  // pages for the tokens that reach the sparse history (paged pool)
  if ((s = grow_pages(c, layer, new_len)) != SWAN_OK) return s;
  const std::vector<SeqState> before = L.seq;
  const SeqInfo* rows_dev = nullptr;
  if (!same) {
    std::vector<SeqInfo> rows(B);
    for (int b = 0; b < B; ++b) {
      rows[b] = SeqInfo{};
      rows[b].sparse_len = before[b].sparse_len;
      rows[b].buf_start = before[b].buf_start;
      rows[b].n_b = before[b].buf_count;
      rows[b].n_new = Tb[b];
      rows[b].evict = (int32_t)evict[b];
      rows[b].prune = old_evict[b];
    }
    if ((s = upload_rows(c, layer, rows)) != SWAN_OK) return s;
    rows_dev = rows_of(c, layer);
  }

  // 1) prune the evicted buffered tokens (they leave the ring first, so the
  //    new tokens may reuse their slots); the table above carries the counts
  if (!small && most_old > 0) {
    PruneRingParams pr{};
    pr.ring_k = c->ring_k + (size_t)layer * ring_elems_per_layer(c);
    pr.ring_v = c->ring_v + (size_t)layer * ring_elems_per_layer(c);
    pr.units = (int)c->units;
    pr.cap = cap;
    pr.buf_start = before[0].buf_start;
    pr.count = most_old;
    pr.sparse_len = before[0].sparse_len;
    pr.seq = rows_dev;
    pr.H = c->cfg.n_kv_heads;
    pr.geom = geom_for(c, layer);
    pr.status = c->status;
    s = launch(c, SWAN_KERNEL_PRUNE, "prune_ring kernel", [&] { return launch_prune_ring(pr, c->stream); });
    if (s != SWAN_OK) return s;
  }

  // 2) rotate the new tokens; those before `evict` are pruned directly, the
  //    rest land in the ring after the surviving buffered tokens
  AppendParams p{};
  p.k_new = static_cast<const __half*>(k_new);
  p.v_new = static_cast<const __half*>(v_new);
  p.R_qk = c->R_qk + (size_t)layer * c->cfg.n_kv_heads * kHeadDim * kHeadDim;
  p.R_vo = c->R_vo + (size_t)layer * c->cfg.n_kv_heads * kHeadDim * kHeadDim;
  p.ring_k = c->ring_k + (size_t)layer * ring_elems_per_layer(c);
  p.ring_v = c->ring_v + (size_t)layer * ring_elems_per_layer(c);
  p.B = B;
  p.H = c->cfg.n_kv_heads;
  p.T = T;
  p.cap = cap > 0 ? cap : 1;
  p.buf_start = before[0].buf_start;
  p.n_b = before[0].buf_count;
  p.evict = evict[0];
  p.sparse_len = before[0].sparse_len;
  p.seq = rows_dev;
  p.geom = geom_for(c, layer);
  p.status = c->status;
  if (small)
    s = launch(c, SWAN_KERNEL_APPEND, rq ? "append_rotate kernel" : "append_small kernel",
               [&] { return launch_append_small(p, most_old, rq, c->stream); });
  else {
    if (const int64_t starve_ns = take_tc_starve()) {
      p.tc_starve = 1;
      p.tc_wait_ns = (uint64_t)starve_ns;
    }
    s = launch(c, SWAN_KERNEL_APPEND, "append kernel",
               [&] { return launch_append_tc(p, maps, layer * 2 * c->cfg.n_kv_heads, c->stream); });
  }
  if (s != SWAN_OK) return s;
  if (rotated) *rotated = small && rq != nullptr;

  for (int b = 0; b < B; ++b) {
    SeqState& q = L.seq[b];
    q.sparse_len = before[b].sparse_len + evict[b];
    q.buf_count = (int)((int64_t)before[b].buf_count + Tb[b] - evict[b]);
    q.buf_start = cap > 0 ? (int)((before[b].buf_start + evict[b]) % cap) : 0;
  }
  return SWAN_OK;
}

}  // namespace

swan_status swan_append(swan_ctx* c, int layer, const void* k_new, const void* v_new, int T) {
  return append_rows(c, layer, k_new, v_new, T, nullptr);
}

swan_status swan_append_varlen(swan_ctx* c, int layer, const void* k_new, const void* v_new, int T,
                               const int32_t* n_new) {
  if (!n_new) return fail(SWAN_ERR_INVALID_ARG, "n_new is NULL");
  return append_rows(c, layer, k_new, v_new, T, n_new);
}

swan_status swan_flush_buffer(swan_ctx* c, int layer) {
  swan_status s = usable(c);
  if (s != SWAN_OK) return s;
  if (layer == -1) {
    if (c->paged) {  // all layers or none: check the pool first
      int64_t need = 0;
      for (int l = 0; l < c->cfg.num_layers; ++l) {
        std::vector<int64_t> new_len;
        for (const SeqState& q : c->layers[l].seq) new_len.push_back(q.sparse_len + q.buf_count);
        need += pages_needed(c, l, new_len);
      }
      if (need > (int64_t)c->free_pages.size())
        return fail(SWAN_ERR_CAPACITY, "flushing every layer needs %lld more pages, the pool has %zu free",
                    (long long)need, c->free_pages.size());
    }
    for (int l = 0; l < c->cfg.num_layers; ++l)
      if ((s = prune_from_ring(c, l, buffer_counts(c->layers[l]))) != SWAN_OK) return s;
    return SWAN_OK;
  }
  if ((s = check_layer(c, layer)) != SWAN_OK) return s;
  return prune_from_ring(c, layer, buffer_counts(c->layers[layer]));
}

namespace {

// Drop row b's tokens in every layer; its pages go back to the pool once no
// fork holds them.
void reset_row(swan_ctx* c, int b) {
  for (int l = 0; l < c->cfg.num_layers; ++l) {
    SeqState& q = c->layers[l].seq[b];
    if (c->paged) {
      const int64_t used = pages_for(q.sparse_len, c->P);
      for (int h = 0; h < c->cfg.n_kv_heads; ++h) {
        const int64_t unit = (int64_t)b * c->cfg.n_kv_heads + h;
        for (int64_t pg = 0; pg < used; ++pg) {
          int32_t& id = pt_entry(c, l, unit, pg);
          if (--c->page_refs[(size_t)id] == 0) c->free_pages.push_back(id);
          id = -1;
        }
      }
    }
    q = SeqState{};
  }
}

}  // namespace

swan_status swan_reset_sequence(swan_ctx* c, int b) {
  swan_status s = usable(c);
  if (s != SWAN_OK) return s;
  if (b < 0 || b >= c->cfg.batch) return fail(SWAN_ERR_INVALID_ARG, "row %d out of [0, %d)", b, c->cfg.batch);
  reset_row(c, b);
  return SWAN_OK;
}

swan_status swan_fork_sequence(swan_ctx* c, int src, int dst) {
  swan_status s = usable(c);
  if (s != SWAN_OK) return s;
  if (!c->paged) return fail(SWAN_ERR_UNSUPPORTED, "forking a row needs a page pool (pool_pages > 0)");
  if (src < 0 || src >= c->cfg.batch || dst < 0 || dst >= c->cfg.batch || src == dst)
    return fail(SWAN_ERR_INVALID_ARG, "rows %d -> %d: two different rows of [0, %d)", src, dst, c->cfg.batch);
  reset_row(c, dst);
  const int H = c->cfg.n_kv_heads, cap = c->cfg.buffer_cap;
  for (int l = 0; l < c->cfg.num_layers; ++l) {
    LayerState& L = c->layers[l];
    const int64_t used = pages_for(L.seq[src].sparse_len, c->P);
    std::vector<int2> pairs;
    for (int h = 0; h < H; ++h) {
      const int64_t us = (int64_t)src * H + h, ud = (int64_t)dst * H + h;
      for (int64_t pg = 0; pg < used; ++pg) {
        const int32_t id = pt_entry(c, l, us, pg);
        ++c->page_refs[(size_t)id];
        pt_entry(c, l, ud, pg) = id;
        pairs.push_back(make_int2((int)(ud * c->ppu + pg), id));
      }
    }
    cudaError_t e = cudaSuccess;
    if (!pairs.empty()) {
      e = cudaMemcpyAsync(c->pt_pairs, pairs.data(), pairs.size() * sizeof(int2), cudaMemcpyHostToDevice,
                          c->stream);
      if (e != cudaSuccess) return cuda_fail(c, e, "uploading page-table entries");
      int32_t* table = c->page_table + (int64_t)l * c->units * c->ppu;
      s = launch(c, SWAN_KERNEL_PRUNE, "page-table scatter",
                 [&] { return launch_scatter_pages(c->pt_pairs, (int)pairs.size(), table, c->stream); });
      if (s != SWAN_OK) return s;
    }
    // the dense buffer is per row: copy its ring slots (all H heads of a
    // row are contiguous)
    if (cap > 0) {
      const size_t row = (size_t)H * cap * kHeadDim, off = (size_t)l * ring_elems_per_layer(c);
      for (__half* ring : {c->ring_k, c->ring_v}) {
        e = cudaMemcpyAsync(ring + off + (size_t)dst * row, ring + off + (size_t)src * row, row * sizeof(__half),
                            cudaMemcpyDeviceToDevice, c->stream);
        if (e != cudaSuccess) return cuda_fail(c, e, "copying a row's dense buffer");
      }
    }
    L.seq[dst] = L.seq[src];
  }
  return SWAN_OK;
}

namespace {

swan_status check_decode_args(const swan_ctx* c, const void* q, const void* out) {
  if (!q || !out) return fail(SWAN_ERR_INVALID_ARG, "q or out is NULL");
  const size_t qbytes = (size_t)c->cfg.batch * c->cfg.n_q_heads * kHeadDim * 2;
  const char* qa = static_cast<const char*>(q);
  const char* oa = static_cast<const char*>(out);
  if (qa < oa + qbytes && oa < qa + qbytes) return fail(SWAN_ERR_INVALID_ARG, "q and out overlap");
  return SWAN_OK;
}

// q' = q R_qk of one layer into the context's q' buffer (Section 4.3).
RotateQParams rotation_of(const swan_ctx* c, int layer, const void* q) {
  RotateQParams rq{};
  rq.q = static_cast<const __half*>(q);
  rq.R_qk = c->R_qk + (size_t)layer * c->cfg.n_kv_heads * kHeadDim * kHeadDim;
  rq.qprime = c->qprime;
  rq.H_q = c->cfg.n_q_heads;
  rq.G = c->G;
  return rq;
}

swan_status launch_rotation(swan_ctx* c, const RotateQParams& rq) {
  return launch(c, SWAN_KERNEL_ROTATE_Q, "rotate_q kernel",
                [&] { return launch_rotate_q(rq, c->cfg.batch, c->stream); });
}

// Attention of the rotated queries (already in the q' buffer) over the
// layer's cache, split-K combine and rotate-back into `out`.
swan_status decode_rotated(swan_ctx* c, int layer, void* out) {
  swan_status s = SWAN_OK;
  const LayerState& L = c->layers[layer];
  const int G = c->G;

  // Uniform rows: every unit has the same groups.  Ragged rows: each row's
  // groups (at least one, so an empty row still writes its zero output),
  // offsets in a per-row table.
  const bool same = L.uniform();
  const SeqState& q0 = L.seq[0];
  // entries read per vector, rounded up to 8: selects the kernel variant
  // and so how many of its CTAs fit at once
  const int k_read = (std::max(c->k_active, c->k_active_v) + 7) / 8 * 8;
  const int64_t max_ctas = c->decode_ctas_v[decode_variant(k_read)];
  const int64_t n_sg = (q0.sparse_len + 31) / 32;
  const int64_t n_bg = (q0.buf_count + 31) / 32;
  const int64_t N_g = n_sg + n_bg;
  int64_t total = c->units * N_g;
  const SeqInfo* rows_dev = nullptr;
  const int64_t* starts_dev = nullptr;
  int64_t ragged_grid = 0;
  if (!same) {
    std::vector<SeqInfo> rows(c->cfg.batch);
    std::vector<int64_t> groups(c->cfg.batch);
    int64_t prefix = 0;
    for (int b = 0; b < c->cfg.batch; ++b) {
      rows[b] = SeqInfo{};
      rows[b].sparse_len = L.seq[b].sparse_len;
      rows[b].buf_start = L.seq[b].buf_start;
      rows[b].n_b = L.seq[b].buf_count;
      rows[b].group_prefix = prefix;
      groups[b] = row_groups(L.seq[b].sparse_len, L.seq[b].buf_count);
      prefix += groups[b];
    }
    total = prefix * c->cfg.n_kv_heads;
    const std::vector<int64_t> starts = balanced_starts(
        groups, c->cfg.n_kv_heads, std::min<int64_t>(max_ctas, std::max<int64_t>(1, total / kMinGroupsPerCta)),
        decode_visit_cost(G, true));
    ragged_grid = (int64_t)starts.size() - 1;
    if ((s = upload_rows(c, layer, rows, &starts)) != SWAN_OK) return s;
    rows_dev = rows_of(c, layer);
    starts_dev = cta_starts_of(c, layer);
  }
  int64_t grid = 0;
  if (total > 0)
    grid = starts_dev ? ragged_grid
                      : std::min<int64_t>(max_ctas, std::max<int64_t>(1, total / kMinGroupsPerCta));
  if (grid > 0) {
    DecodeParams p{};
    p.qprime = c->qprime;
    p.geom = geom_for(c, layer);
    p.ring_k = c->ring_k + (size_t)layer * ring_elems_per_layer(c);
    p.ring_v = c->ring_v + (size_t)layer * ring_elems_per_layer(c);
    p.cap = c->cfg.buffer_cap > 0 ? c->cfg.buffer_cap : 1;
    p.buf_start = q0.buf_start;
    p.n_b = q0.buf_count;
    p.sparse_len = q0.sparse_len;
    p.n_sg = n_sg;
    p.N_g = N_g;
    p.total_groups = total;
    p.visit_cost = decode_visit_cost(G, false);
    p.seq = rows_dev;
    p.cta_start = starts_dev;
    p.B = c->cfg.batch;
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
                  [&] { return launch_decode(p, G, k_read, (int)grid, c->stream); });
  }
  // empty cache: the combine kernel writes zeros

  CombineParams cp{};
  cp.out = static_cast<__half*>(out);
  cp.H_q = c->cfg.n_q_heads;
  return launch(c, SWAN_KERNEL_COMBINE, "combine kernel",
                [&] { return launch_combine(cp, c->cfg.batch, c->stream); });
}

}  // namespace

swan_status swan_decode(swan_ctx* c, int layer, const void* q, void* out) {
  swan_status s = usable(c);
  if (s != SWAN_OK) return s;
  if ((s = check_layer(c, layer)) != SWAN_OK) return s;
  if ((s = check_decode_args(c, q, out)) != SWAN_OK) return s;
  if ((s = launch_rotation(c, rotation_of(c, layer, q))) != SWAN_OK) return s;
  return decode_rotated(c, layer, out);
}

swan_status swan_append_decode(swan_ctx* c, int layer, const void* k_new, const void* v_new, int T,
                               const int32_t* n_new, const void* q, void* out) {
  swan_status s = usable(c);
  if (s != SWAN_OK) return s;
  if ((s = check_layer(c, layer)) != SWAN_OK) return s;
  if ((s = check_decode_args(c, q, out)) != SWAN_OK) return s;
  const RotateQParams rq = rotation_of(c, layer, q);
  bool rotated = false;
  if ((s = append_rows(c, layer, k_new, v_new, T, n_new, &rq, &rotated)) != SWAN_OK) return s;
  if (!rotated && (s = launch_rotation(c, rq)) != SWAN_OK) return s;
  return decode_rotated(c, layer, out);
}

swan_status swan_query(const swan_ctx* c, int layer, swan_layer_info* info) {
  swan_status s = usable(c);
  if (s != SWAN_OK) return s;
  if ((s = check_layer(c, layer)) != SWAN_OK) return s;
  if (!info) return fail(SWAN_ERR_INVALID_ARG, "info is NULL");
  const LayerState& L = c->layers[layer];
  info->sparse_len = 0;
  info->buffer_len = 0;
  for (const SeqState& q : L.seq) {
    info->sparse_len = std::max<int64_t>(info->sparse_len, q.sparse_len);
    info->buffer_len = std::max<int64_t>(info->buffer_len, q.buf_count);
  }
  info->uniform = L.uniform() ? 1 : 0;
  info->pool_pages = c->num_pages;
  info->free_pages = c->paged ? (int64_t)c->free_pages.size() : 0;
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

namespace {

// Export the buffer or the sparse history of rows [b0, b1) of a layer (they
// must have equal lengths), in the layouts swan_debug_export documents.
swan_status export_rows(swan_ctx* c, int layer, int b0, int b1, int what, void* host_dst, size_t bytes) {
  if (!host_dst && bytes) return fail(SWAN_ERR_INVALID_ARG, "host_dst is NULL");
  const LayerState& L = c->layers[layer];
  for (int b = b0 + 1; b < b1; ++b)
    if (!(L.seq[b] == L.seq[b0]))
      return fail(SWAN_ERR_INVALID_ARG, "rows differ in length: export them one at a time (swan_debug_export_seq)");
  const SeqState& q = L.seq[b0];
  const int H = c->cfg.n_kv_heads;
  const int64_t u0 = (int64_t)b0 * H, u1 = (int64_t)b1 * H, nu = u1 - u0;
  const int cap = c->cfg.buffer_cap;
  cudaError_t e = cudaStreamSynchronize(c->stream);
  if (e != cudaSuccess) return cuda_fail(c, e, "cudaStreamSynchronize");

  if (what == SWAN_EXPORT_BUFFER_K || what == SWAN_EXPORT_BUFFER_V) {
    const size_t need = (size_t)nu * q.buf_count * kHeadDim * 2;
    if (bytes != need) return fail(SWAN_ERR_INVALID_ARG, "bytes %zu != %zu", bytes, need);
    if (need == 0) return SWAN_OK;
    const __half* ring = (what == SWAN_EXPORT_BUFFER_K ? c->ring_k : c->ring_v) +
                         (size_t)layer * ring_elems_per_layer(c) + (size_t)u0 * cap * kHeadDim;
    std::vector<uint16_t> all((size_t)nu * cap * kHeadDim);
    e = cudaMemcpy(all.data(), ring, all.size() * 2, cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_fail(c, e, "cudaMemcpy");
    uint16_t* dst = static_cast<uint16_t*>(host_dst);
    for (int64_t u = 0; u < nu; ++u)
      for (int i = 0; i < q.buf_count; ++i) {
        const int slot = (q.buf_start + i) % cap;
        std::memcpy(dst + ((size_t)u * q.buf_count + i) * kHeadDim,
                    all.data() + ((size_t)u * cap + slot) * kHeadDim, kHeadDim * 2);
      }
    return SWAN_OK;
  }
  if (what == SWAN_EXPORT_SPARSE_K || what == SWAN_EXPORT_SPARSE_V) {
    const bool isv = what == SWAN_EXPORT_SPARSE_V;
    const int ks = isv ? c->k_store_v : c->cfg.k_store;
    const int64_t Ls = q.sparse_len;
    const size_t n_ent = (size_t)nu * Ls * ks;
    const size_t need = n_ent * 3;
    if (bytes != need) return fail(SWAN_ERR_INVALID_ARG, "bytes %zu != %zu", bytes, need);
    if (need == 0) return SWAN_OK;
    const bool fp8 = c->fmt == kFmtFp8;
    const int64_t P = c->P;
    const int64_t ksk = c->k_slots, ksv = c->k_slots_v;
    const int64_t blk = (fp8 ? 64 : 96) * (ksk + ksv);
    // fp16: value records of 16 B and index records of 8 B in separate
    // regions; fp8: 16-byte records of 8 values then 8 indices
    const int64_t voff = fp8 ? (isv ? 64 * ksk : 0) : (isv ? 96 * ksk : 0);
    const int64_t ioff = fp8 ? voff + 8 : (isv ? 96 * ksk + 64 * ksv : 64 * ksk);
    std::vector<int32_t> pt((size_t)nu * c->ppu);
    e = cudaMemcpy(pt.data(), c->page_table + ((int64_t)layer * c->units + u0) * c->ppu, pt.size() * 4,
                   cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_fail(c, e, "cudaMemcpy");
    uint8_t* idx_dst = static_cast<uint8_t*>(host_dst);
    uint16_t* val_dst = reinterpret_cast<uint16_t*>(idx_dst + n_ent);
    std::vector<uint8_t> page(c->page_bytes);
    const int64_t pages_used = pages_for(Ls, (int)P);
    for (int64_t u = 0; u < nu; ++u)
      for (int64_t pg = 0; pg < pages_used; ++pg) {
        const int32_t phys = pt[(size_t)u * c->ppu + pg];
        if (phys < 0 || phys >= c->num_pages) return fail(SWAN_ERR_DEVICE_CHECK, "page table corrupt");
        e = cudaMemcpy(page.data(), c->pool + (int64_t)phys * c->page_bytes, c->page_bytes,
                       cudaMemcpyDeviceToHost);
        if (e != cudaSuccess) return cuda_fail(c, e, "cudaMemcpy");
        for (int64_t sl = 0; sl < P; ++sl) {
          const int64_t t = pg * P + sl;
          if (t >= Ls) break;
          const int64_t bo = (sl / 32) * blk;
          for (int r = 0; r < ks; ++r) {
            const int64_t rec = (int64_t)(r / 8) * 32 + (sl % 32);
            const size_t o = ((size_t)u * Ls + t) * ks + r;
            if (fp8) {
              idx_dst[o] = page[bo + ioff + rec * 16 + (r % 8)];
              val_dst[o] = e4m3_to_half_bits(page[bo + voff + rec * 16 + (r % 8)]);
            } else {
              idx_dst[o] = page[bo + ioff + rec * 8 + (r % 8)];
              uint16_t v;
              std::memcpy(&v, page.data() + bo + voff + rec * 16 + (r % 8) * 2, 2);
              val_dst[o] = v;
            }
          }
        }
      }
    return SWAN_OK;
  }
  return fail(SWAN_ERR_INVALID_ARG, "unknown export kind %d", what);
}

}  // namespace

swan_status swan_debug_export(swan_ctx* c, int layer, int what, void* host_dst, size_t bytes) {
  swan_status s = usable(c);
  if (s != SWAN_OK) return s;
  if ((s = check_layer(c, layer)) != SWAN_OK) return s;
  if (!host_dst) return fail(SWAN_ERR_INVALID_ARG, "host_dst is NULL");
  return export_rows(c, layer, 0, c->cfg.batch, what, host_dst, bytes);
}

swan_status swan_debug_export_seq(swan_ctx* c, int layer, int b, int what, void* host_dst, size_t bytes) {
  swan_status s = usable(c);
  if (s != SWAN_OK) return s;
  if ((s = check_layer(c, layer)) != SWAN_OK) return s;
  if (b < 0 || b >= c->cfg.batch) return fail(SWAN_ERR_INVALID_ARG, "row %d out of [0, %d)", b, c->cfg.batch);
  return export_rows(c, layer, b, b + 1, what, host_dst, bytes);
}

swan_status swan_query_lengths(const swan_ctx* c, int layer, int64_t* sparse_len, int32_t* buffer_len) {
  swan_status s = usable(c);
  if (s != SWAN_OK) return s;
  if ((s = check_layer(c, layer)) != SWAN_OK) return s;
  if (!sparse_len || !buffer_len) return fail(SWAN_ERR_INVALID_ARG, "output arrays must not be NULL");
  const LayerState& L = c->layers[layer];
  for (int b = 0; b < c->cfg.batch; ++b) {
    sparse_len[b] = L.seq[b].sparse_len;
    buffer_len[b] = L.seq[b].buf_count;
  }
  return SWAN_OK;
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
    if (word & kStatusTimeout)
      return fail(SWAN_ERR_DEVICE_TIMEOUT, "a tensor-core pipeline wait gave up (status word 0x%x)", word);
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

swan_status swan_debug_fail_after(int kind, int64_t n) {
  if (n < -1) return fail(SWAN_ERR_INVALID_ARG, "n = %lld < -1", (long long)n);
  if (kind == SWAN_FAULT_ALLOC) g_fail_alloc.store(n);
  else if (kind == SWAN_FAULT_LAUNCH) g_fail_launch.store(n);
  else return fail(SWAN_ERR_INVALID_ARG, "unknown fault kind %d", kind);
  return SWAN_OK;
}

swan_status swan_debug_starve_tc(int64_t limit_ns) {
  if (limit_ns != 0 && (limit_ns < 1000 || limit_ns > 2000000000))
    return fail(SWAN_ERR_INVALID_ARG, "limit_ns = %lld outside [1e3, 2e9]", (long long)limit_ns);
  g_tc_starve.store(limit_ns);
  return SWAN_OK;
}

swan_status swan_debug_check_guards(swan_ctx* c) {
  swan_status s = usable(c);
  if (s != SWAN_OK) return s;
  cudaError_t e = cudaStreamSynchronize(c->stream);
  if (e != cudaSuccess) return cuda_fail(c, e, "cudaStreamSynchronize");
  std::vector<unsigned char> g(kFrontGuard);
  for (const auto& b : c->bufs)
    for (int side = 0; side < 2; ++side) {
      const char* at = static_cast<const char*>(b.base) + (side ? kFrontGuard + b.bytes : 0);
      const size_t n = side ? kBackGuard : kFrontGuard;
      e = cudaMemcpy(g.data(), at, n, cudaMemcpyDeviceToHost);
      if (e != cudaSuccess) return cuda_fail(c, e, "cudaMemcpy");
      for (size_t i = 0; i < n; ++i)
        if (g[i] != kGuardByte)
          return fail(SWAN_ERR_DEVICE_CHECK, "the guard region %s %s was overwritten (byte %zu)",
                      side ? "after" : "before", b.what, i);
    }
  return SWAN_OK;
}

}  // extern "C"
