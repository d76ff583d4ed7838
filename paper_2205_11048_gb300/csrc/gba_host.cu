// Host side of libgba: the gradient buffer (FIFO of messages and the device
// buffers their data live in), the assembly of a global step, kernel launches
// on the handle's stream, error latching and the C ABI of include/gba.h.
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <deque>
#include <new>
#include <string>
#include <vector>

#include "gba.h"
#include "gba_internal.cuh"

using namespace gba;

namespace {

constexpr int MAX_DIM = 256;
constexpr int META_SLOTS = 4;
constexpr int MAX_PASSES = 4;
constexpr int64_t MAX_STEP_OCC = (1ll << 30) - 1;
constexpr int MAX_WTAB = 1024;  // decay weights lambda^s for s < MAX_WTAB
constexpr int EAGER_SLOTS = 8;  // pending global steps with eager dense accumulators
// Per-step buffers exist twice, so that step k + 1's message weights and sort
// run (on the sort stream) while step k's segment-sum and dense update run.
constexpr int SLOTS = 2;

struct Arena {  // contiguous-allocation ring over [0, cap) with virtual offsets
  int64_t cap = 0;
  int64_t vhead = 0, vtail = 0;
  int64_t* ids = nullptr;
  float* rows = nullptr;

  int64_t alloc(int64_t n) {
    if (n == 0) return vtail;
    int64_t v = vtail;
    if ((v % cap) + n > cap) v = (v / cap + 1) * cap;  // do not wrap inside a message
    if (v + n - vhead > cap) return -1;
    vtail = v + n;
    return v;
  }
  void release_through(int64_t v_end) { vhead = std::max(vhead, v_end); }
};

struct TableState {
  gba_table_desc desc;  // for a HASH table, rows is the current number of slots
  float* w = nullptr;
  float* s0 = nullptr;
  float* s1 = nullptr;
  int32_t* ver = nullptr;
  uint32_t key_base = 0;
  double bpow1 = 1.0, bpow2 = 1.0;  // beta^t of Adam, as successive products
  Arena arena;
  // HASH tables: slot keys, inserted-id counter, and a bound on the ids
  // inserted so far (exact at the last read plus every occurrence since)
  unsigned long long* keys = nullptr;
  unsigned long long* count = nullptr;
  int64_t id_bound = 0;
};

struct Msg {
  int64_t token;
  int32_t B;
  bool copied;
  const float* dense;
  std::vector<const int64_t*> ids;
  std::vector<const float*> rows;
  std::vector<int64_t> n;
  std::vector<int64_t> arena_v;  // virtual start in each table's arena (copied messages)
};

struct PendingTiming {
  int kind;
  cudaEvent_t a, b;
};

size_t align16(size_t x) { return (x + 15) & ~size_t(15); }

}  // namespace

#ifndef GBA_STREAM_PRIO
#define GBA_STREAM_PRIO 0
#endif

struct gba_handle {
  int device = 0;
  int num_sms = 152;
  cudaStream_t stream = nullptr;
  bool own_stream = false;
  cudaStream_t side = nullptr;   // dense update
  cudaStream_t sorts = nullptr;   // message weights, histogram, sort passes
  cudaStream_t applys = nullptr;  // segment-sum and row update
  bool overlap = false;           // consecutive steps may run concurrently
  cudaEvent_t ev_pushes = nullptr;
  cudaEvent_t ev_hist[SLOTS] = {}, ev_sorted[SLOTS] = {}, ev_applied[SLOTS] = {},
              ev_densed[SLOTS] = {};
  bool slot_busy[SLOTS] = {};

  std::vector<TableState> tables;
  int32_t T = 0;
  int64_t D = 0;
  int64_t D_pad = 0;
  gba_opt_desc dense_opt{};
  float* dw = nullptr;
  float* ds0 = nullptr;
  float* ds1 = nullptr;
  double dbpow1 = 1.0, dbpow2 = 1.0;
  int64_t G = 1;
  int32_t max_buf = 1;
  gba_staleness_desc st{};
  uint64_t seed = 0;
  int64_t k = 0;
  uint32_t total_keys_bits = 1;
  int passes = 1;

  std::deque<Msg> fifo;
  bool arenas_ready = false;
  float* dense_ring = nullptr;
  int32_t slot_head = 0, slot_count = 0;

  TableInfo* d_tinfo = nullptr;
  std::vector<TableInfo> h_tinfo;
  HashInfo* d_hinfo = nullptr;
  std::vector<HashInfo> h_hinfo;
  uint64_t seed_table = 0;

  size_t meta_bytes = 0;
  char* d_meta[SLOTS] = {};
  char* h_meta[META_SLOTS] = {};
  cudaEvent_t meta_ev[META_SLOTS] = {};
  int meta_slot = 0;

  // sort / segment scratch, grown on demand
  int64_t n_cap = 0;
  uint32_t* d_keys[SLOTS][2] = {};
  uint32_t* d_vals[SLOTS][2] = {};
  unsigned long long* d_status[SLOTS] = {};
  int64_t status_tiles = 0;
  uint32_t epoch = 0;
  char* d_step_scratch[SLOTS] = {};
  StepScratch sc[SLOTS] = {};
  // row-kernel buffers (apply stream only), grown with n_cap
  uint4* d_rr = nullptr;                   // row records, per table nbase[t] + t
  const float** d_kl = nullptr;            // kept list, per table nbase[t]
  float* d_kw = nullptr;                   // kept weights
  unsigned long long* d_scan_status = nullptr;
  uint4* d_long_rows = nullptr;
  uint4* d_small_rows = nullptr;
  uint32_t* d_long_done = nullptr;
  uint2* d_items = nullptr;
  float* d_part_hi = nullptr;
  float* d_part_lo = nullptr;
  uint32_t* d_seg_total = nullptr;         // [T] rows of each table in the last step
  int d_max = 1;

  float* d_wtab = nullptr;    // decay weights lambda^s (decay 1)
  int32_t n_wtab = 0;
  std::vector<float> h_wtab;
  bool withhold_dense = false;  // test hook of gba_debug_withhold_dense_copies

  // eager dense aggregation: one compensated accumulator (hi, lo) per pending
  // global step, filled at push time
  bool eager = false;
  struct EagerGroup {
    int64_t accB;  // local batches of the step's messages so far
    int slot;      // its accumulator
    bool has_sum;  // some message of the step was kept
  };
  std::deque<EagerGroup> egroups;
  int n_acc = 0;
  float* d_acc = nullptr;          // [n_acc][2][D_pad]
  cudaEvent_t acc_ev[EAGER_SLOTS] = {};
  bool acc_ev_set[EAGER_SLOTS] = {};
  float* d_stage_dense = nullptr;  // copying pushes stage the dense gradient here
  uint32_t* d_err = nullptr;
  uint32_t* h_err = nullptr;  // mapped pinned
  ErrSink sink{};
  DevStats* d_stats = nullptr;
  bool failed = false;
  gba_status fail_code = GBA_OK;
  std::string last_error;
  int64_t wait_ns = 2000000000ll;

  bool debug = false;
  bool timing = false;
  std::vector<PendingTiming> pending;
  std::vector<cudaEvent_t> event_pool;
  gba_kernel_times_t times{};

  // last applied step, for the debug entry points
  bool have_last = false;
  int64_t last_N = 0;
  int last_buf = 0;
  int last_slot = 0;
  int32_t last_M = 0;
  std::vector<int64_t> last_nbase;
};

namespace {

gba_status set_err(gba_handle* h, gba_status s, const std::string& msg) {
  if (h) h->last_error = msg;
  return s;
}

gba_status cuda_fail(gba_handle* h, cudaError_t e, const char* what) {
  std::string m = std::string(what) + ": " + cudaGetErrorString(e);
  if (h) h->last_error = m;
  return e == cudaErrorMemoryAllocation ? GBA_E_OOM : GBA_E_CUDA;
}

#define GBA_CUDA(h, call)                                    \
  do {                                                       \
    cudaError_t e_ = (call);                                 \
    if (e_ != cudaSuccess) return cuda_fail((h), e_, #call); \
  } while (0)

cudaEvent_t take_event(gba_handle* h) {
  if (!h->event_pool.empty()) {
    cudaEvent_t e = h->event_pool.back();
    h->event_pool.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  cudaEventCreate(&e);
  return e;
}

// Brackets one launch with events when timing is on; always counts launches.
struct Timed {
  gba_handle* h;
  int kind;
  cudaStream_t s;
  cudaEvent_t a = nullptr;
  Timed(gba_handle* h_, int kind_, cudaStream_t s_) : h(h_), kind(kind_), s(s_) {
    h->times.launches[kind]++;
    if (h->timing) {
      a = take_event(h);
      cudaEventRecord(a, s);
    }
  }
  ~Timed() {
    if (h->timing) {
      cudaEvent_t b = take_event(h);
      cudaEventRecord(b, s);
      h->pending.push_back({kind, a, b});
    }
  }
};

void collect_timing(gba_handle* h) {
  for (auto& p : h->pending) {
    float ms = 0.f;
    if (cudaEventElapsedTime(&ms, p.a, p.b) == cudaSuccess) h->times.ms[p.kind] += ms;
    h->event_pool.push_back(p.a);
    h->event_pool.push_back(p.b);
  }
  h->pending.clear();
}

gba_status validate_opt(const gba_opt_desc& o) {
  if (o.kind != GBA_ADAGRAD && o.kind != GBA_ADAM) return GBA_E_ARG;
  if (!std::isfinite(o.lr)) return GBA_E_ARG;
  if (o.kind == GBA_ADAGRAD && !(o.adagrad_init_acc > 0.f && std::isfinite(o.adagrad_init_acc)))
    return GBA_E_ARG;
  if (o.kind == GBA_ADAM && !(o.beta1 >= 0.f && o.beta1 < 1.f && o.beta2 >= 0.f &&
                              o.beta2 < 1.f && o.eps >= 0.f && std::isfinite(o.eps)))
    return GBA_E_ARG;
  return GBA_OK;
}

// Adam bias corrections and constants for the next step of one parameter group.
OptStep make_opt_step(const gba_opt_desc& o, double bpow1_next, double bpow2_next) {
  OptStep s{};
  s.kind = o.kind;
  s.lr = o.lr;
  s.b1 = o.beta1;
  s.b2 = o.beta2;
  s.eps = o.eps;
  s.c1 = 1.0f - o.beta1;
  s.c2 = 1.0f - o.beta2;
  s.bc1 = (float)(1.0 - bpow1_next);
  s.bc2 = (float)(1.0 - bpow2_next);
  return s;
}

void free_all(gba_handle* h) {
  if (!h) return;
  cudaSetDevice(h->device);
  if (h->sorts) cudaStreamSynchronize(h->sorts);
  if (h->applys) cudaStreamSynchronize(h->applys);
  if (h->side) cudaStreamSynchronize(h->side);
  if (h->stream) cudaStreamSynchronize(h->stream);
  for (auto& t : h->tables) {
    cudaFree(t.w);
    cudaFree(t.s0);
    cudaFree(t.s1);
    cudaFree(t.ver);
    cudaFree(t.keys);
    cudaFree(t.count);
    cudaFree(t.arena.ids);
    cudaFree(t.arena.rows);
  }
  cudaFree(h->d_hinfo);
  cudaFree(h->dw);
  cudaFree(h->ds0);
  cudaFree(h->ds1);
  cudaFree(h->dense_ring);
  cudaFree(h->d_tinfo);
  for (int b = 0; b < SLOTS; ++b) {
    cudaFree(h->d_meta[b]);
    cudaFree(h->d_step_scratch[b]);
    cudaFree(h->d_status[b]);
    for (int i = 0; i < 2; ++i) {
      cudaFree(h->d_keys[b][i]);
      cudaFree(h->d_vals[b][i]);
    }
    for (cudaEvent_t e : {h->ev_hist[b], h->ev_sorted[b], h->ev_applied[b], h->ev_densed[b]})
      if (e) cudaEventDestroy(e);
  }
  for (int i = 0; i < META_SLOTS; ++i) {
    if (h->h_meta[i]) cudaFreeHost(h->h_meta[i]);
    if (h->meta_ev[i]) cudaEventDestroy(h->meta_ev[i]);
  }
  for (void* p : {(void*)h->d_rr, (void*)h->d_kl, (void*)h->d_kw, (void*)h->d_scan_status,
                  (void*)h->d_long_rows, (void*)h->d_long_done, (void*)h->d_items,
                  (void*)h->d_part_hi, (void*)h->d_part_lo, (void*)h->d_seg_total,
                  (void*)h->d_small_rows})
    cudaFree(p);
  cudaFree(h->d_err);
  cudaFree(h->d_wtab);
  cudaFree(h->d_acc);
  cudaFree(h->d_stage_dense);
  for (cudaEvent_t e : h->acc_ev)
    if (e) cudaEventDestroy(e);
  if (h->h_err) cudaFreeHost(h->h_err);
  cudaFree(h->d_stats);
  for (auto& p : h->pending) {
    cudaEventDestroy(p.a);
    cudaEventDestroy(p.b);
  }
  for (auto e : h->event_pool) cudaEventDestroy(e);
  if (h->ev_pushes) cudaEventDestroy(h->ev_pushes);
  if (h->side) cudaStreamDestroy(h->side);
  if (h->sorts) cudaStreamDestroy(h->sorts);
  if (h->applys) cudaStreamDestroy(h->applys);
  if (h->own_stream && h->stream) cudaStreamDestroy(h->stream);
}

cudaError_t sync_all(gba_handle* h) {
  cudaError_t e[4] = {cudaStreamSynchronize(h->sorts), cudaStreamSynchronize(h->applys),
                      cudaStreamSynchronize(h->side), cudaStreamSynchronize(h->stream)};
  for (cudaError_t x : e)
    if (x != cudaSuccess) return x;
  return cudaSuccess;
}

// Orders the handle's stream after every step enqueued so far.
void join_steps(gba_handle* h) {
  for (int b = 0; b < SLOTS; ++b)
    if (h->slot_busy[b]) {
      cudaStreamWaitEvent(h->stream, h->ev_applied[b], 0);
      cudaStreamWaitEvent(h->stream, h->ev_densed[b], 0);
    }
}

// Device error latched by a kernel?  Polls the mapped flag without
// synchronising; if set, synchronises and turns the word into a status.
gba_status poll_device_error(gba_handle* h, bool force_sync) {
  if (!force_sync && *(volatile uint32_t*)h->h_err == 0u) return GBA_OK;
  cudaError_t e = sync_all(h);
  if (e != cudaSuccess) {
    h->failed = true;
    h->fail_code = cuda_fail(h, e, "stream synchronize");
    return h->fail_code;
  }
  uint32_t word = 0;
  e = cudaMemcpy(&word, h->d_err, sizeof word, cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) {
    h->failed = true;
    h->fail_code = cuda_fail(h, e, "read device error word");
    return h->fail_code;
  }
  if (word == 0u) return GBA_OK;
  h->failed = true;
  if (word & ERR_ID_RANGE) {
    h->fail_code = set_err(h, GBA_E_ID_RANGE, "an id outside [0, rows) in a DIRECT table");
  } else if (word & ERR_TIMEOUT) {
    h->fail_code = set_err(h, GBA_E_DEVICE_TIMEOUT, "a bounded device wait gave up");
  } else {
    h->fail_code = set_err(h, GBA_E_CUDA, "device consistency check failed");
  }
  return h->fail_code;
}

HashInfo hash_info(const gba_handle* h, int t) {
  const TableState& ts = h->tables[t];
  HashInfo hi{};
  hi.keys = ts.keys;
  hi.mask = (uint64_t)ts.desc.rows - 1;
  hi.w = ts.w;
  hi.s0 = ts.s0;
  hi.s1 = ts.s1;
  hi.ver = ts.ver;
  hi.count = ts.count;
  hi.seed = h->seed;
  hi.tag = ((uint64_t)(uint32_t)t + 1u) << 48;
  hi.d = ts.desc.dim;
  hi.kind = ts.desc.opt.kind;
  hi.init_acc = ts.desc.opt.adagrad_init_acc;
  return hi;
}

// Key bases (tables in order), key bits and sort passes from the tables' rows,
// and the device copies of the table and hash descriptions.
gba_status layout_keys(gba_handle* h) {
  uint64_t base = 0;
  for (int t = 0; t < h->T; ++t) {
    TableState& ts = h->tables[t];
    ts.key_base = (uint32_t)base;
    h->h_tinfo[t] = TableInfo{ts.desc.rows, (uint32_t)base, ts.desc.id_mode,
                              ~0ull / (uint64_t)ts.desc.rows};
    h->h_hinfo[t] = ts.desc.id_mode == GBA_ID_HASH ? hash_info(h, t) : HashInfo{};
    base += (uint64_t)ts.desc.rows;
  }
  if (base >= 0xFFFFFFFFull) return set_err(h, GBA_E_ARG, "tables hold 2^32 - 1 rows or more");
  const uint64_t kmax = base > 0 ? base - 1 : 0;
  uint32_t bits = 1;
  while (bits < 32 && (kmax >> bits) != 0) ++bits;
  h->total_keys_bits = bits;
  h->passes = (int)((bits + 7) / 8);
  if (h->T > 0) {
    GBA_CUDA(h, cudaMemcpy(h->d_tinfo, h->h_tinfo.data(), h->T * sizeof(TableInfo),
                           cudaMemcpyHostToDevice));
    GBA_CUDA(h, cudaMemcpy(h->d_hinfo, h->h_hinfo.data(), h->T * sizeof(HashInfo),
                           cudaMemcpyHostToDevice));
  }
  return GBA_OK;
}

// A HASH table's arrays for `slots` slots (keys cleared; rows are initialised
// when their id is inserted).
gba_status alloc_hash_arrays(gba_handle* h, TableState& ts, uint64_t slots) {
  const size_t n = (size_t)slots * ts.desc.dim;
  GBA_CUDA(h, cudaMalloc(&ts.w, n * 4));
  GBA_CUDA(h, cudaMalloc(&ts.s0, n * 4));
  if (ts.desc.opt.kind == GBA_ADAM) GBA_CUDA(h, cudaMalloc(&ts.s1, n * 4));
  GBA_CUDA(h, cudaMalloc(&ts.ver, (size_t)slots * 4));
  GBA_CUDA(h, cudaMalloc(&ts.keys, (size_t)slots * 8));
  launch_hash_clear(ts.keys, slots, h->stream);
  GBA_CUDA(h, cudaGetLastError());
  return GBA_OK;
}

// Keeps every HASH table at most half full for the step about to run: the
// bound on its ids grows by the step's occurrences; when it passes half the
// slots the exact count is read, and if that is still too many the table
// doubles until it is not, every id moving to its slot in the larger table.
gba_status grow_hash_tables(gba_handle* h, const std::vector<int64_t>& nbase) {
  bool changed = false;
  for (int t = 0; t < h->T; ++t) {
    TableState& ts = h->tables[t];
    if (ts.desc.id_mode != GBA_ID_HASH) continue;
    const int64_t Nt = nbase[t + 1] - nbase[t];
    ts.id_bound += Nt;
    if (ts.id_bound <= ts.desc.rows / 2) continue;
    GBA_CUDA(h, sync_all(h));
    unsigned long long have = 0;
    GBA_CUDA(h, cudaMemcpy(&have, ts.count, 8, cudaMemcpyDeviceToHost));
    ts.id_bound = (int64_t)have + Nt;
    if (ts.id_bound <= ts.desc.rows / 2) continue;
    uint64_t slots = (uint64_t)ts.desc.rows;
    while ((int64_t)(slots / 2) < ts.id_bound) slots *= 2;
    const HashInfo from = hash_info(h, t);
    TableState old = ts;
    ts.w = ts.s0 = ts.s1 = nullptr;
    ts.ver = nullptr;
    ts.keys = nullptr;
    gba_status st = alloc_hash_arrays(h, ts, slots);
    if (st != GBA_OK) return st;
    ts.desc.rows = (int64_t)slots;
    launch_hash_rehash(from, hash_info(h, t), h->stream);
    GBA_CUDA(h, cudaGetLastError());
    GBA_CUDA(h, cudaStreamSynchronize(h->stream));
    cudaFree(old.w);
    cudaFree(old.s0);
    cudaFree(old.s1);
    cudaFree(old.ver);
    cudaFree(old.keys);
    changed = true;
  }
  return changed ? layout_keys(h) : GBA_OK;
}

gba_status ensure_step_capacity(gba_handle* h, int64_t N) {
  if (N > h->n_cap) {
    sync_all(h);
    int64_t cap = std::max<int64_t>(N + N / 4, 4096);
    const int64_t tiles = sort_tiles(cap);
    for (int b = 0; b < SLOTS; ++b) {
      for (int i = 0; i < 2; ++i) {
        cudaFree(h->d_keys[b][i]);
        cudaFree(h->d_vals[b][i]);
        h->d_keys[b][i] = h->d_vals[b][i] = nullptr;
        GBA_CUDA(h, cudaMalloc(&h->d_keys[b][i], cap * sizeof(uint32_t)));
        GBA_CUDA(h, cudaMalloc(&h->d_vals[b][i], cap * sizeof(uint32_t)));
      }
      cudaFree(h->d_status[b]);
      h->d_status[b] = nullptr;
      GBA_CUDA(h, cudaMalloc(&h->d_status[b], (size_t)tiles * 256 * sizeof(unsigned long long)));
      GBA_CUDA(h,
               cudaMemset(h->d_status[b], 0, (size_t)tiles * 256 * sizeof(unsigned long long)));
    }
    h->n_cap = cap;
    h->status_tiles = tiles;
    // row-kernel buffers: a record per possible row (and one per table for the
    // totals), a kept-list entry per occurrence, look-back words per scan tile,
    // long rows and their chunks
    for (void* p : {(void*)h->d_rr, (void*)h->d_kl, (void*)h->d_kw, (void*)h->d_scan_status,
                    (void*)h->d_long_rows, (void*)h->d_long_done, (void*)h->d_items,
                    (void*)h->d_part_hi, (void*)h->d_part_lo, (void*)h->d_small_rows})
      cudaFree(p);
    h->d_rr = nullptr;
    h->d_kl = nullptr;
    h->d_kw = h->d_part_hi = h->d_part_lo = nullptr;
    h->d_scan_status = nullptr;
    h->d_long_rows = nullptr;
    h->d_small_rows = nullptr;
    h->d_long_done = nullptr;
    h->d_items = nullptr;
    const int64_t stiles = scan_tiles(cap);
    const int64_t long_cap = cap / (LONG_ROW + 1) + h->T + 1;
    const int64_t items_cap = cap / LONG_CHUNK + long_cap;
    const int64_t parts_cap = 2 * (cap / LONG_CHUNK) + h->T + 1;
    GBA_CUDA(h, cudaMalloc(&h->d_rr, (size_t)(cap + h->T + 1) * sizeof(uint4)));
    GBA_CUDA(h, cudaMalloc(&h->d_kl, (size_t)cap * sizeof(float*)));
    GBA_CUDA(h, cudaMalloc(&h->d_kw, (size_t)cap * sizeof(float)));
    GBA_CUDA(h, cudaMalloc(&h->d_scan_status, (size_t)stiles * 4 * sizeof(unsigned long long)));
    GBA_CUDA(h, cudaMemset(h->d_scan_status, 0, (size_t)stiles * 4 * sizeof(unsigned long long)));
    GBA_CUDA(h, cudaMalloc(&h->d_long_rows, (size_t)long_cap * sizeof(uint4)));
    GBA_CUDA(h, cudaMalloc(&h->d_small_rows, (size_t)long_cap * sizeof(uint4)));
    GBA_CUDA(h, cudaMalloc(&h->d_long_done, (size_t)long_cap * sizeof(uint32_t)));
    GBA_CUDA(h, cudaMalloc(&h->d_items, (size_t)items_cap * sizeof(uint2)));
    GBA_CUDA(h, cudaMalloc(&h->d_part_hi, (size_t)parts_cap * h->d_max * sizeof(float)));
    GBA_CUDA(h, cudaMalloc(&h->d_part_lo, (size_t)parts_cap * h->d_max * sizeof(float)));
  }
  return GBA_OK;
}

gba_status ensure_arenas(gba_handle* h) {
  if (h->arenas_ready) return GBA_OK;
  for (auto& t : h->tables) {
    const int64_t cap = (int64_t)(h->max_buf + 1) * std::max<int64_t>(1, t.desc.max_ids_per_msg);
    t.arena.cap = cap;
    GBA_CUDA(h, cudaMalloc(&t.arena.ids, cap * sizeof(int64_t)));
    GBA_CUDA(h, cudaMalloc(&t.arena.rows, cap * (size_t)t.desc.dim * sizeof(float)));
  }
  if (h->D > 0) {
    const size_t bytes = (size_t)h->max_buf * h->D_pad * sizeof(float);
    GBA_CUDA(h, cudaMalloc(&h->dense_ring, bytes));
    GBA_CUDA(h, cudaMemset(h->dense_ring, 0, bytes));
  }
  h->arenas_ready = true;
  return GBA_OK;
}

// The dense weight of a message with this token applied at step k_apply
// (Eq. (1), or the decay strategy; the same numbers the kernels use).
float message_weight(const gba_handle* h, int64_t k_apply, int64_t token) {
  const int64_t diff = k_apply - token;
  const int64_t s = diff > 0 ? diff : 0;
  if (s > (int64_t)h->st.iota) return 0.f;
  if (h->st.decay == 0) return 1.f;
  return s < (int64_t)h->h_wtab.size() ? h->h_wtab[s] : 0.f;
}

gba_status push_common(gba_handle* h, int64_t token, const gba_sparse_grad* per_table,
                       const float* dense_grad, int32_t local_batch, bool copy) {
  if (!h) return GBA_E_ARG;
  if (h->failed) return set_err(h, GBA_E_STATE, "handle failed earlier");
  if (token < 0) return set_err(h, GBA_E_ARG, "token < 0");
  if (local_batch < 1) return set_err(h, GBA_E_ARG, "local_batch < 1");
  if (h->T > 0 && !per_table) return set_err(h, GBA_E_ARG, "per_table is NULL");
  if (h->D > 0 && !dense_grad) return set_err(h, GBA_E_ARG, "dense_grad is NULL");
  for (int t = 0; t < h->T; ++t) {
    const gba_sparse_grad& g = per_table[t];
    const gba_table_desc& d = h->tables[t].desc;
    if (g.n < 0 || g.n > d.max_ids_per_msg)
      return set_err(h, GBA_E_ARG, "ids per message outside [0, max_ids_per_msg]");
    if (g.n > 0 && (!g.ids || !g.rows)) return set_err(h, GBA_E_ARG, "NULL ids or rows");
    if (!copy && g.n > 0) {
      if (((uintptr_t)g.ids & 7u) != 0) return set_err(h, GBA_E_ARG, "ids not 8-byte aligned");
      if (d.dim % 4 == 0 && ((uintptr_t)g.rows & 15u) != 0)
        return set_err(h, GBA_E_ARG, "rows not 16-byte aligned");
      if (((uintptr_t)g.rows & 3u) != 0) return set_err(h, GBA_E_ARG, "rows not 4-byte aligned");
    }
  }
  if (!copy && h->D > 0 && ((uintptr_t)dense_grad & 15u) != 0)
    return set_err(h, GBA_E_ARG, "dense_grad not 16-byte aligned");
  if ((int64_t)h->fifo.size() >= h->max_buf) return set_err(h, GBA_E_FULL, "gradient buffer full");
  const bool eager = h->eager && h->D > 0;
  // eager: the step this message belongs to, and its accumulator
  const bool new_group = eager && (h->egroups.empty() || h->egroups.back().accB >= h->G);
  int new_slot = -1;
  if (new_group) {
    bool held[EAGER_SLOTS] = {};
    for (const auto& gr : h->egroups) held[gr.slot] = true;
    for (int i = 0; i < h->n_acc && new_slot < 0; ++i)
      if (!held[i]) new_slot = i;
    if (new_slot < 0)
      return set_err(h, GBA_E_FULL, "every eager accumulator holds a pending global step");
  }

  Msg m;
  m.token = token;
  m.B = local_batch;
  m.copied = copy;
  m.ids.resize(h->T);
  m.rows.resize(h->T);
  m.n.resize(h->T);
  m.arena_v.assign(h->T, -1);
  if (copy) {
    gba_status s = ensure_arenas(h);
    if (s != GBA_OK) return s;
    // The copy may overwrite buffer space of messages that earlier steps read.
    if (h->overlap) join_steps(h);
    if (h->D > 0 && !eager && h->slot_count >= h->max_buf)
      return set_err(h, GBA_E_FULL, "gradient buffer full");
    std::vector<int64_t> saved_tail(h->T);
    for (int t = 0; t < h->T; ++t) saved_tail[t] = h->tables[t].arena.vtail;
    for (int t = 0; t < h->T; ++t) {
      const int64_t n = per_table[t].n;
      const int64_t v = h->tables[t].arena.alloc(n);
      if (v < 0) {
        for (int u = 0; u < h->T; ++u) h->tables[u].arena.vtail = saved_tail[u];
        return set_err(h, GBA_E_FULL, "gradient buffer full (id storage)");
      }
      m.arena_v[t] = v;
    }
    for (int t = 0; t < h->T; ++t) {
      const int64_t n = per_table[t].n;
      Arena& ar = h->tables[t].arena;
      const int64_t p = m.arena_v[t] % ar.cap;
      const int32_t dim = h->tables[t].desc.dim;
      m.ids[t] = ar.ids + p;
      m.rows[t] = ar.rows + p * dim;
      m.n[t] = n;
      if (n > 0) {
        GBA_CUDA(h, cudaMemcpyAsync(ar.ids + p, per_table[t].ids, n * sizeof(int64_t),
                                    cudaMemcpyDefault, h->stream));
        GBA_CUDA(h, cudaMemcpyAsync(ar.rows + p * dim, per_table[t].rows,
                                    n * dim * sizeof(float), cudaMemcpyDefault, h->stream));
      }
    }
    if (h->D > 0 && !eager) {
      const int32_t slot = (h->slot_head + h->slot_count) % h->max_buf;
      float* dst = h->dense_ring + (size_t)slot * h->D_pad;
      GBA_CUDA(h, cudaMemcpyAsync(dst, dense_grad, h->D * sizeof(float), cudaMemcpyDefault,
                                  h->stream));
      h->slot_count++;
      m.dense = dst;
    } else {
      m.dense = nullptr;
    }
  } else {
    for (int t = 0; t < h->T; ++t) {
      m.ids[t] = per_table[t].ids;
      m.rows[t] = per_table[t].rows;
      m.n[t] = per_table[t].n;
    }
    m.dense = dense_grad;
  }
  if (eager) {  // the dense gradient joins its step's accumulator now
    if (new_group) {
      if (h->acc_ev_set[new_slot]) cudaStreamWaitEvent(h->stream, h->acc_ev[new_slot], 0);
      h->egroups.push_back(gba_handle::EagerGroup{0, new_slot, false});
    }
    gba_handle::EagerGroup& gr = h->egroups.back();
    const int64_t k_apply = h->k + (int64_t)h->egroups.size() - 1;
    const float f = message_weight(h, k_apply, token);
    if (f > 0.f) {
      const float* src = dense_grad;
      if (copy) {
        GBA_CUDA(h, cudaMemcpyAsync(h->d_stage_dense, dense_grad, h->D * sizeof(float),
                                    cudaMemcpyDefault, h->stream));
        src = h->d_stage_dense;
      }
      float* hi = h->d_acc + (size_t)gr.slot * 2 * h->D_pad;
      {
        Timed tm(h, GBA_K_DENSE, h->stream);
        launch_dense_accumulate(hi, hi + h->D_pad, src, h->D, f, !gr.has_sum, h->num_sms,
                                h->stream);
      }
      GBA_CUDA(h, cudaGetLastError());
      gr.has_sum = true;
    }
    gr.accB += local_batch;
    m.dense = nullptr;
  }
  h->fifo.push_back(std::move(m));
  return GBA_OK;
}

}  // namespace

extern "C" {

gba_status gba_create(const gba_table_desc* tables, int32_t n_tables, int64_t dense_size,
                      const gba_opt_desc* dense_opt, int64_t global_batch,
                      int32_t max_buffered_msgs, const gba_staleness_desc* st,
                      uint64_t init_seed, void* cuda_stream, gba_handle** out) {
  if (!out) return GBA_E_ARG;
  *out = nullptr;
  if (n_tables < 0 || (n_tables > 0 && !tables)) return GBA_E_ARG;
  if (dense_size < 0 || (dense_size > 0 && !dense_opt)) return GBA_E_ARG;
  if (global_batch < 1 || max_buffered_msgs < 1) return GBA_E_ARG;
  uint64_t total_rows = 0;
  for (int t = 0; t < n_tables; ++t) {
    const gba_table_desc& d = tables[t];
    if (d.rows < 1 || d.dim < 1 || d.dim > MAX_DIM) return GBA_E_ARG;
    if (d.id_mode != GBA_ID_DIRECT && d.id_mode != GBA_ID_MODULO && d.id_mode != GBA_ID_HASH)
      return GBA_E_ARG;
    if (d.id_mode == GBA_ID_HASH && d.rows > (1ll << 30)) return GBA_E_ARG;
    if (d.max_ids_per_msg < 0 || d.max_ids_per_msg > MAX_STEP_OCC) return GBA_E_ARG;
    if (validate_opt(d.opt) != GBA_OK) return GBA_E_ARG;
    uint64_t r = (uint64_t)d.rows;
    if (d.id_mode == GBA_ID_HASH) {  // a power of two of slots, at least 1024
      uint64_t slots = 1024;
      while (slots < r) slots *= 2;
      r = slots;
    }
    total_rows += r;
  }
  if (total_rows >= 0xFFFFFFFFull) return GBA_E_ARG;  // keys are 32-bit, one value reserved
  if (dense_size > 0 && validate_opt(*dense_opt) != GBA_OK) return GBA_E_ARG;
  gba_staleness_desc rule{0x7FFFFFFF, 0, 0, 0, 1.0f, 0};
  if (st) rule = *st;
  if (rule.iota < 0 || (rule.row_staleness != 0 && rule.row_staleness != 1) ||
      rule.sparse_denominator < 0 || rule.sparse_denominator > 2 ||
      (rule.decay != 0 && rule.decay != 1) || rule.drop_latest < 0)
    return GBA_E_ARG;
  if (rule.decay == 1 &&
      (!(rule.lambda > 0.f && rule.lambda <= 1.f) || rule.iota >= MAX_WTAB))
    return GBA_E_ARG;

  gba_handle* h = new (std::nothrow) gba_handle();
  if (!h) return GBA_E_OOM;
  h->T = n_tables;
  h->D = dense_size;
  h->D_pad = (dense_size + 3) & ~3ll;
  if (dense_opt) h->dense_opt = *dense_opt;
  h->G = global_batch;
  h->max_buf = max_buffered_msgs;
  h->st = rule;
  h->seed = init_seed;

  auto fail = [&](gba_status s) {
    free_all(h);
    delete h;
    return s;
  };
  cudaError_t e = cudaGetDevice(&h->device);
  if (e != cudaSuccess) {
    cudaGetLastError();
    return fail(GBA_E_CUDA);
  }
  int sms = 0;
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, h->device) == cudaSuccess &&
      sms > 0)
    h->num_sms = sms;
  if (cuda_stream) {
    h->stream = (cudaStream_t)cuda_stream;
  } else {
    if (cudaStreamCreateWithFlags(&h->stream, cudaStreamNonBlocking) != cudaSuccess)
      return fail(GBA_E_CUDA);
    h->own_stream = true;
  }
  // Stream priorities (GBA_STREAM_PRIO): 0 all equal; 1 the row path first and
  // the next step's sort last; 2 the row path first, the others equal.
  int prio_lo = 0, prio_hi = 0;
  if (GBA_STREAM_PRIO != 0 && cudaDeviceGetStreamPriorityRange(&prio_lo, &prio_hi) != cudaSuccess)
    prio_lo = prio_hi = 0;
  const int p_rows = GBA_STREAM_PRIO != 0 ? prio_hi : 0;
  const int p_sort = GBA_STREAM_PRIO == 1 ? prio_lo : (GBA_STREAM_PRIO == 2 ? (prio_lo + prio_hi) / 2 : 0);
  const int p_side = GBA_STREAM_PRIO != 0 ? (prio_lo + prio_hi) / 2 : 0;
  if (cudaStreamCreateWithPriority(&h->side, cudaStreamNonBlocking, p_side) != cudaSuccess ||
      cudaStreamCreateWithPriority(&h->sorts, cudaStreamNonBlocking, p_sort) != cudaSuccess ||
      cudaStreamCreateWithPriority(&h->applys, cudaStreamNonBlocking, p_rows) != cudaSuccess ||
      cudaEventCreateWithFlags(&h->ev_pushes, cudaEventDisableTiming) != cudaSuccess)
    return fail(GBA_E_CUDA);
  for (int b = 0; b < SLOTS; ++b)
    for (cudaEvent_t* e : {&h->ev_hist[b], &h->ev_sorted[b], &h->ev_applied[b], &h->ev_densed[b]})
      if (cudaEventCreateWithFlags(e, cudaEventDisableTiming) != cudaSuccess)
        return fail(GBA_E_CUDA);
  if (configure_dense() != cudaSuccess) return fail(GBA_E_CUDA);

  // tables (a HASH table starts with a power of two of slots)
  h->tables.resize(n_tables);
  h->h_tinfo.resize(n_tables);
  h->h_hinfo.resize(n_tables);
  for (int t = 0; t < n_tables; ++t) {
    TableState& ts = h->tables[t];
    ts.desc = tables[t];
    if (ts.desc.id_mode == GBA_ID_HASH) {
      int64_t slots = 1024;
      while (slots < ts.desc.rows) slots *= 2;
      ts.desc.rows = slots;
    }
    h->d_max = std::max(h->d_max, (int)tables[t].dim);
  }

  auto dev_alloc = [&](void** p, size_t bytes) -> bool {
    if (bytes == 0) return true;
    return cudaMalloc(p, bytes) == cudaSuccess;
  };
  for (int t = 0; t < n_tables; ++t) {
    TableState& ts = h->tables[t];
    if (ts.desc.id_mode == GBA_ID_HASH) {
      if (alloc_hash_arrays(h, ts, (uint64_t)ts.desc.rows) != GBA_OK ||
          !dev_alloc((void**)&ts.count, 8) || cudaMemset(ts.count, 0, 8) != cudaSuccess)
        return fail(GBA_E_OOM);
      continue;
    }
    const size_t n = (size_t)ts.desc.rows * ts.desc.dim;
    if (!dev_alloc((void**)&ts.w, n * 4) || !dev_alloc((void**)&ts.s0, n * 4) ||
        (ts.desc.opt.kind == GBA_ADAM && !dev_alloc((void**)&ts.s1, n * 4)) ||
        !dev_alloc((void**)&ts.ver, (size_t)ts.desc.rows * 4))
      return fail(GBA_E_OOM);
  }
  if (h->D > 0) {
    if (!dev_alloc((void**)&h->dw, h->D_pad * 4) || !dev_alloc((void**)&h->ds0, h->D_pad * 4) ||
        (h->dense_opt.kind == GBA_ADAM && !dev_alloc((void**)&h->ds1, h->D_pad * 4)))
      return fail(GBA_E_OOM);
  }
  h->seed = init_seed;
  if (n_tables > 0) {
    if (!dev_alloc((void**)&h->d_tinfo, n_tables * sizeof(TableInfo)) ||
        !dev_alloc((void**)&h->d_hinfo, n_tables * sizeof(HashInfo)))
      return fail(GBA_E_OOM);
  }
  if (layout_keys(h) != GBA_OK) return fail(GBA_E_CUDA);
  // step descriptor buffers
  {
    const size_t M = (size_t)max_buffered_msgs, T = (size_t)n_tables;
    h->meta_bytes = align16(M * 8) + align16(M * 8) + align16(T * (M + 1) * 4) +
                    align16(T * M * 8) + align16(T * M * 8) + align16((T + 1) * 8);
    for (int b = 0; b < SLOTS; ++b)
      if (!dev_alloc((void**)&h->d_meta[b], h->meta_bytes)) return fail(GBA_E_OOM);
    for (int i = 0; i < META_SLOTS; ++i) {
      if (cudaHostAlloc((void**)&h->h_meta[i], h->meta_bytes, cudaHostAllocDefault) !=
              cudaSuccess ||
          cudaEventCreateWithFlags(&h->meta_ev[i], cudaEventDisableTiming) != cudaSuccess)
        return fail(GBA_E_OOM);
    }
  }
  {
    const size_t M = (size_t)max_buffered_msgs;
    const size_t bytes = align16(MAX_PASSES * 256 * 4) + align16(MAX_PASSES * 4) +
                         align16(M * 4) + align16(M * 4) + align16(4) + align16(4) +
                         align16((size_t)std::max(h->T, 1) * 32) + align16(M * 4);
    for (int b = 0; b < SLOTS; ++b) {
      if (!dev_alloc((void**)&h->d_step_scratch[b], bytes)) return fail(GBA_E_OOM);
      if (cudaMemset(h->d_step_scratch[b], 0, bytes) != cudaSuccess) return fail(GBA_E_CUDA);
      char* p = h->d_step_scratch[b];
      StepScratch& sc = h->sc[b];
      sc.hist = (uint32_t*)p;
      p += align16(MAX_PASSES * 256 * 4);
      sc.tile_counter = (uint32_t*)p;
      p += align16(MAX_PASSES * 4);
      sc.keep = (int32_t*)p;
      p += align16(M * 4);
      sc.kept_list = (int32_t*)p;
      p += align16(M * 4);
      sc.n_kept = (int32_t*)p;
      p += align16(4);
      sc.step_err = (uint32_t*)p;
      p += align16(4);
      sc.seg_ticket = (uint32_t*)p;
      p += align16((size_t)std::max(h->T, 1) * 32);
      sc.fw = (float*)p;
    }
  }
  if (!dev_alloc((void**)&h->d_seg_total, (size_t)std::max(h->T, 1) * 4)) return fail(GBA_E_OOM);
  if (rule.decay == 1) {  // lambda^s as s products in double, rounded once, s = 0 .. iota
    h->n_wtab = rule.iota + 1;
    std::vector<float>& wt = h->h_wtab;
    wt.resize(h->n_wtab);
    double pw = 1.0;
    for (int32_t s2 = 0; s2 < h->n_wtab; ++s2) {
      wt[s2] = (float)pw;
      pw = pw * (double)rule.lambda;
    }
    if (!dev_alloc((void**)&h->d_wtab, wt.size() * sizeof(float))) return fail(GBA_E_OOM);
    if (cudaMemcpy(h->d_wtab, wt.data(), wt.size() * sizeof(float), cudaMemcpyHostToDevice) !=
        cudaSuccess)
      return fail(GBA_E_CUDA);
  }
  if (!dev_alloc((void**)&h->d_err, 4) || !dev_alloc((void**)&h->d_stats, sizeof(DevStats)))
    return fail(GBA_E_OOM);
  if (cudaHostAlloc((void**)&h->h_err, 4, cudaHostAllocMapped) != cudaSuccess)
    return fail(GBA_E_OOM);
  *h->h_err = 0u;
  uint32_t* h_err_dev = nullptr;
  if (cudaHostGetDevicePointer((void**)&h_err_dev, h->h_err, 0) != cudaSuccess)
    return fail(GBA_E_CUDA);
  h->sink = ErrSink{nullptr, h->d_err, h_err_dev};  // .step is set per slot
  if (cudaMemsetAsync(h->d_err, 0, 4, h->stream) != cudaSuccess ||
      cudaMemsetAsync(h->d_stats, 0, sizeof(DevStats), h->stream) != cudaSuccess)
    return fail(GBA_E_CUDA);

  // initial values (R11 of the design notes: counter-based hash of (seed, array, element))
  for (int t = 0; t < n_tables; ++t) {
    TableState& ts = h->tables[t];
    if (ts.desc.id_mode == GBA_ID_HASH) continue;  // rows start when their id arrives
    Timed tm(h, GBA_K_INIT, h->stream);
    launch_init_table(ts.w, ts.s0, ts.s1, ts.ver, ts.desc.rows, ts.desc.dim, ts.desc.opt.kind,
                      ts.desc.opt.adagrad_init_acc, init_seed, ((uint64_t)(uint32_t)t + 1u) << 48,
                      h->stream);
  }
  if (h->D > 0) {
    Timed tm(h, GBA_K_INIT, h->stream);
    launch_init_dense(h->dw, h->ds0, h->ds1, h->D, h->dense_opt.kind,
                      h->dense_opt.adagrad_init_acc, init_seed, (uint64_t)0xFFFFu << 48,
                      h->stream);
  }
  e = cudaGetLastError();
  if (e != cudaSuccess) return fail(GBA_E_CUDA);
  if (cudaStreamSynchronize(h->stream) != cudaSuccess) return fail(GBA_E_CUDA);
  collect_timing(h);
  *out = h;
  return GBA_OK;
}

gba_status gba_push(gba_handle* h, int64_t token, const gba_sparse_grad* per_table,
                    const float* dense_grad, int32_t local_batch) {
  return push_common(h, token, per_table, dense_grad, local_batch, true);
}

gba_status gba_push_ref(gba_handle* h, int64_t token, const gba_sparse_grad* per_table,
                        const float* dense_grad, int32_t local_batch) {
  return push_common(h, token, per_table, dense_grad, local_batch, false);
}

int32_t gba_try_apply(gba_handle* h) {
  if (!h) return GBA_E_ARG;
  if (h->failed) return GBA_E_STATE;
  {
    gba_status s = poll_device_error(h, false);
    if (s != GBA_OK) return s;
  }
  // Alg. 2: apply once the buffered local batches reach the global batch.
  int64_t acc = 0;
  int32_t M = 0;
  for (const Msg& m : h->fifo) {
    acc += m.B;
    ++M;
    if (acc >= h->G) break;
  }
  if (acc < h->G) return 0;
  const int T = h->T;
  std::vector<int64_t> nbase(T + 1, 0);
  for (int t = 0; t < T; ++t) {
    int64_t nt = 0;
    for (int i = 0; i < M; ++i) nt += h->fifo[i].n[t];
    nbase[t + 1] = nbase[t] + nt;
  }
  const int64_t N = nbase[T];
  if (N > MAX_STEP_OCC) return set_err(h, GBA_E_ARG, "more than 2^30-1 ids in one global step");
  cudaSetDevice(h->device);
  {
    gba_status s = grow_hash_tables(h, nbase);
    if (s == GBA_OK) s = ensure_step_capacity(h, N);
    if (s != GBA_OK) return s;
  }

  // ---- the step's buffers (slot b) and stream dependencies.  The sort stream
  // runs message weights, histogram and sort passes; the handle's stream the
  // segment-sum and row update; the side stream the dense update.
  const int b = (int)(h->k & 1);
  // everything the caller enqueued before this call (pushes included)
  cudaEventRecord(h->ev_pushes, h->stream);
  cudaStreamWaitEvent(h->sorts, h->ev_pushes, 0);
  if (h->slot_busy[b]) {  // step k - 2 used these buffers
    cudaStreamWaitEvent(h->sorts, h->ev_applied[b], 0);
    cudaStreamWaitEvent(h->sorts, h->ev_densed[b], 0);
  }
  StepScratch& sc = h->sc[b];
  ErrSink sink = h->sink;
  sink.step = sc.step_err;
  char* dmeta = h->d_meta[b];

  // ---- step descriptor
  const int slot = h->meta_slot;
  h->meta_slot = (h->meta_slot + 1) % META_SLOTS;
  cudaEventSynchronize(h->meta_ev[slot]);
  char* hp = h->h_meta[slot];
  const size_t Mx = (size_t)h->max_buf;
  size_t off = 0;
  auto section = [&](size_t bytes) {
    size_t o = off;
    off += align16(bytes);
    return o;
  };
  const size_t o_tok = section(Mx * 8), o_dense = section(Mx * 8),
               o_off = section((size_t)T * (Mx + 1) * 4), o_ids = section((size_t)T * Mx * 8),
               o_rows = section((size_t)T * Mx * 8), o_nbase = section((size_t)(T + 1) * 8);
  int64_t* tok = (int64_t*)(hp + o_tok);
  const float** dptr = (const float**)(hp + o_dense);
  uint32_t* moff = (uint32_t*)(hp + o_off);
  const int64_t** iptr = (const int64_t**)(hp + o_ids);
  const float** rptr = (const float**)(hp + o_rows);
  int64_t* nb = (int64_t*)(hp + o_nbase);
  for (int i = 0; i < M; ++i) {
    const Msg& m = h->fifo[i];
    tok[i] = m.token;
    dptr[i] = m.dense;
  }
  for (int t = 0; t < T; ++t) {
    uint32_t run = 0;
    for (int i = 0; i < M; ++i) {
      const Msg& m = h->fifo[i];
      moff[(size_t)t * (M + 1) + i] = run;
      run += (uint32_t)m.n[t];
      iptr[(size_t)t * M + i] = m.ids[t];
      rptr[(size_t)t * M + i] = m.rows[t];
    }
    moff[(size_t)t * (M + 1) + M] = run;
  }
  for (int t = 0; t <= T; ++t) nb[t] = nbase[t];
  GBA_CUDA(h, cudaMemcpyAsync(dmeta, hp, h->meta_bytes, cudaMemcpyHostToDevice, h->sorts));
  cudaEventRecord(h->meta_ev[slot], h->sorts);

  StepArgs a{};
  a.k = h->k;
  a.M = M;
  a.T = T;
  a.N = N;
  a.iota = h->st.iota;
  a.row_staleness = h->st.row_staleness;
  a.sparse_den = h->st.sparse_denominator;
  a.decay = h->st.decay;
  a.drop_latest = h->st.drop_latest;
  a.n_wtab = h->n_wtab;
  a.wtab = h->d_wtab;
  a.tokens = (const int64_t*)(dmeta + o_tok);
  a.dense_ptr = (const float* const*)(dmeta + o_dense);
  a.msg_off = (const uint32_t*)(dmeta + o_off);
  a.ids_ptr = (const int64_t* const*)(dmeta + o_ids);
  a.rows_ptr = (const float* const*)(dmeta + o_rows);
  a.nbase = (const int64_t*)(dmeta + o_nbase);
  a.tinfo = h->d_tinfo;
  a.hinfo = h->d_hinfo;

  // ---- K1: message weights (Eq. (1)); clears the per-step scratch
  {
    Timed tm(h, GBA_K_WEIGHTS, h->sorts);
    launch_weights(a, sc, h->d_stats, MAX_PASSES * 256, h->sorts);
  }
  // ---- K5 on the side stream, concurrently with the sort and segment-sum.
  // It is forked after the histogram kernel has validated every id, so a step
  // that fails its id check leaves the dense parameters untouched too.
  auto launch_dense_side = [&]() {
    if (h->D <= 0) return;
    const double p1 = h->dbpow1 * (double)h->dense_opt.beta1;
    const double p2 = h->dbpow2 * (double)h->dense_opt.beta2;
    DenseArgs da{h->dw, h->ds0, h->ds1, h->D, M, make_opt_step(h->dense_opt, p1, p2),
                 h->withhold_dense ? 1 : 0};
    cudaEventRecord(h->ev_hist[b], h->sorts);
    cudaStreamWaitEvent(h->side, h->ev_hist[b], 0);
    if (h->eager) {  // the step's sum was accumulated at push time
      const gba_handle::EagerGroup gr = h->egroups.front();
      h->egroups.pop_front();
      const float* hi = h->d_acc + (size_t)gr.slot * 2 * h->D_pad;
      {
        Timed tm(h, GBA_K_DENSE, h->side);
        launch_dense_eager(da, hi, hi + h->D_pad, gr.has_sum, sink, h->num_sms, h->side);
      }
      cudaEventRecord(h->acc_ev[gr.slot], h->side);
      h->acc_ev_set[gr.slot] = true;
    } else {
      Timed tm(h, GBA_K_DENSE, h->side);
      launch_dense(a, da, sc, sink, h->wait_ns, h->num_sms, h->side);
    }
    h->dbpow1 = p1;
    h->dbpow2 = p2;
  };
  // ---- K2 sort, K3+K4 segment-sum and row update
  int final_buf = 0;
  if (N > 0) {
    {
      Timed tm(h, GBA_K_SORT_HIST, h->sorts);
      int grid = (int)std::min<int64_t>((N + 255) / 256, (int64_t)h->num_sms * 8);
      // the first pass writes buffer 0, so its input keys go to buffer 1
      launch_sort_histogram(a, h->passes, sc, h->d_keys[b][1], sink, std::max(grid, 1), h->sorts);
    }
    launch_dense_side();
    const uint32_t* kin = h->d_keys[b][1];
    const uint32_t* vin = nullptr;
    for (int p = 0; p < h->passes; ++p) {
      const int ob = p & 1;
      if (++h->epoch == 0u) h->epoch = 1u;
      Timed tm(h, GBA_K_SORT_PASS, h->sorts);
      launch_onesweep(a, p == 0, p, kin, vin, h->d_keys[b][ob], h->d_vals[b][ob], sc,
                      h->d_status[b], h->epoch, sink, h->wait_ns, h->sorts);
      kin = h->d_keys[b][ob];
      vin = h->d_vals[b][ob];
      final_buf = ob;
    }
    cudaEventRecord(h->ev_sorted[b], h->sorts);
    cudaStreamWaitEvent(h->applys, h->ev_sorted[b], 0);
    for (int t = 0; t < T; ++t) {
      const int64_t Nt = nbase[t + 1] - nbase[t];
      if (Nt == 0) continue;
      TableState& ts = h->tables[t];
      const double p1 = ts.bpow1 * (double)ts.desc.opt.beta1;
      const double p2 = ts.bpow2 * (double)ts.desc.opt.beta2;
      SegTable tb{};
      tb.w = ts.w;
      tb.s0 = ts.s0;
      tb.s1 = ts.s1;
      tb.ver = ts.ver;
      tb.d = ts.desc.dim;
      tb.t = t;
      tb.key_base = ts.key_base;
      tb.rows = ts.desc.rows;
      tb.pos_begin = nbase[t];
      tb.pos_end = nbase[t + 1];
      tb.opt = make_opt_step(ts.desc.opt, p1, p2);
      if (++h->epoch == 0u) h->epoch = 1u;
      SegOut so{};
      so.rr = h->d_rr + nbase[t] + t;
      so.kl = h->d_kl + nbase[t];
      so.kw = h->d_kw + nbase[t];
      so.status = h->d_scan_status;
      so.epoch = h->epoch;
      so.ticket = sc.seg_ticket + 8 * t;
      so.n_long = sc.seg_ticket + 8 * t + 1;
      so.n_items = sc.seg_ticket + 8 * t + 2;
      so.n_parts = sc.seg_ticket + 8 * t + 3;
      so.item_ticket = sc.seg_ticket + 8 * t + 4;
      so.total = h->d_seg_total + t;
      so.long_rows = h->d_long_rows;
      so.long_done = h->d_long_done;
      so.items = h->d_items;
      so.part_hi = h->d_part_hi;
      so.part_lo = h->d_part_lo;
      so.pstride = h->d_max;
      so.small_rows = h->d_small_rows;
      so.n_small = sc.seg_ticket + 8 * t + 5;
      so.small_ticket = sc.seg_ticket + 8 * t + 6;
      {
        Timed tm(h, GBA_K_SEG_SCAN, h->applys);
        launch_seg_scan(a, tb, so, h->d_keys[b][final_buf], h->d_vals[b][final_buf], h->d_stats,
                        sink, h->wait_ns, h->applys);
      }
      {
        Timed tm(h, GBA_K_SEG_SCAN, h->applys);
        launch_row_classify(a, tb, so, sink, h->num_sms, h->applys);
      }
      {
        Timed tm(h, GBA_K_ROW_APPLY, h->applys);
        launch_row_apply(a, tb, so, h->d_stats, sink, h->num_sms, h->applys);
      }
      {
        Timed tm(h, GBA_K_ROW_LONG, h->applys);
        launch_row_long(a, tb, so, h->d_stats, sink, h->num_sms, h->applys);
      }
    }
  }
  if (N == 0) {
    launch_dense_side();
    cudaEventRecord(h->ev_sorted[b], h->sorts);
    cudaStreamWaitEvent(h->applys, h->ev_sorted[b], 0);
  }
  // Adam step counts advance every global step, whether or not a row moved.
  for (auto& ts : h->tables) {
    ts.bpow1 *= (double)ts.desc.opt.beta1;
    ts.bpow2 *= (double)ts.desc.opt.beta2;
  }
  cudaEventRecord(h->ev_applied[b], h->applys);
  cudaEventRecord(h->ev_densed[b], h->side);
  h->slot_busy[b] = true;
  // Unless steps may overlap, work the caller orders after this call on its
  // stream sees the whole step.
  if (!h->overlap) join_steps(h);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) {
    h->failed = true;
    h->fail_code = cuda_fail(h, e, "kernel launch");
    return h->fail_code;
  }

  // ---- pop the applied messages
  for (int i = 0; i < M; ++i) {
    Msg& m = h->fifo.front();
    if (m.copied) {
      for (int t = 0; t < T; ++t)
        if (m.n[t] > 0) h->tables[t].arena.release_through(m.arena_v[t] + m.n[t]);
      if (h->D > 0 && m.dense != nullptr) {  // a dense ring slot (not eager)
        h->slot_head = (h->slot_head + 1) % h->max_buf;
        h->slot_count--;
      }
    }
    h->fifo.pop_front();
  }
  h->k += 1;
  h->have_last = true;
  h->last_N = N;
  h->last_nbase = nbase;
  h->last_buf = final_buf;
  h->last_slot = b;
  h->last_M = M;
  return 1;
}

int64_t gba_pull_version(gba_handle* h) { return h ? h->k : -1; }

gba_status gba_sync(gba_handle* h) {
  if (!h) return GBA_E_ARG;
  if (h->failed) return h->fail_code == GBA_OK ? GBA_E_STATE : h->fail_code;
  cudaSetDevice(h->device);
  return poll_device_error(h, true);
}

gba_status gba_get_table(gba_handle* h, int32_t t, float** w, float** slot0, float** slot1,
                         int32_t** ver) {
  if (!h || t < 0 || t >= h->T) return GBA_E_ARG;
  const TableState& ts = h->tables[t];
  if (w) *w = ts.w;
  if (slot0) *slot0 = ts.s0;
  if (slot1) *slot1 = ts.s1;
  if (ver) *ver = ts.ver;
  return GBA_OK;
}

gba_status gba_get_dense(gba_handle* h, float** w, float** slot0, float** slot1) {
  if (!h) return GBA_E_ARG;
  if (w) *w = h->dw;
  if (slot0) *slot0 = h->ds0;
  if (slot1) *slot1 = h->ds1;
  return GBA_OK;
}

gba_status gba_stats(gba_handle* h, gba_stats_t* out) {
  if (!h || !out) return GBA_E_ARG;
  cudaSetDevice(h->device);
  sync_all(h);
  DevStats s{};
  GBA_CUDA(h, cudaMemcpyAsync(&s, h->d_stats, sizeof s, cudaMemcpyDeviceToHost, h->stream));
  GBA_CUDA(h, cudaStreamSynchronize(h->stream));
  out->steps = (int64_t)s.steps;
  out->msgs_kept = (int64_t)s.msgs_kept;
  out->msgs_dropped = (int64_t)s.msgs_dropped;
  out->dense_stale_sum = (int64_t)s.dense_stale_sum;
  out->dense_stale_max = (int64_t)s.dense_stale_max;
  out->pairs = (int64_t)s.pairs;
  out->pairs_dropped = (int64_t)s.pairs_dropped;
  out->row_stale_sum = (int64_t)s.row_stale_sum;
  out->row_stale_max = (int64_t)s.row_stale_max;
  out->occurrences = (int64_t)s.occurrences;
  out->rows_touched = (int64_t)s.rows_touched;
  out->rows_applied = (int64_t)s.rows_applied;
  out->occurrences_kept = (int64_t)s.occ_kept;
  return GBA_OK;
}

const char* gba_last_error(gba_handle* h) { return h ? h->last_error.c_str() : ""; }

void gba_destroy(gba_handle* h) {
  if (!h) return;
  free_all(h);
  delete h;
}

gba_status gba_set_timing(gba_handle* h, int32_t on) {
  if (!h) return GBA_E_ARG;
  sync_all(h);
  collect_timing(h);
  h->times = gba_kernel_times_t{};
  h->timing = on != 0;
  return GBA_OK;
}

gba_status gba_kernel_times(gba_handle* h, gba_kernel_times_t* out) {
  if (!h || !out) return GBA_E_ARG;
  cudaSetDevice(h->device);
  GBA_CUDA(h, sync_all(h));
  collect_timing(h);
  *out = h->times;
  return GBA_OK;
}

gba_status gba_pull(gba_handle* h, int32_t t, const int64_t* ids, int64_t n, float* out) {
  if (!h || t < 0 || t >= h->T || n < 0) return GBA_E_ARG;
  if (n > 0 && (!ids || !out)) return set_err(h, GBA_E_ARG, "NULL ids or out");
  if (h->failed) return set_err(h, GBA_E_STATE, "handle failed earlier");
  if (((uintptr_t)ids & 7u) != 0) return set_err(h, GBA_E_ARG, "ids not 8-byte aligned");
  if (n == 0) return GBA_OK;
  cudaSetDevice(h->device);
  join_steps(h);  // the rows as of every step enqueued so far
  const TableState& ts = h->tables[t];
  ErrSink sink = h->sink;
  sink.step = h->d_err;  // no step of its own: the handle's word takes both roles
  launch_pull_rows(ts.w, ts.desc.rows, ts.desc.dim, ts.desc.id_mode, h->h_tinfo[t].mod_magic,
                   h->d_hinfo + t, ids, n, out, sink, h->num_sms, h->stream);
  GBA_CUDA(h, cudaGetLastError());
  return GBA_OK;
}

gba_status gba_set_eager_dense(gba_handle* h, int32_t on) {
  if (!h) return GBA_E_ARG;
  if (h->failed) return set_err(h, GBA_E_STATE, "handle failed earlier");
  if (!h->fifo.empty()) return set_err(h, GBA_E_STATE, "messages are buffered");
  if (on && h->st.drop_latest > 0)
    return set_err(h, GBA_E_ARG, "eager aggregation cannot know the latest messages of a step");
  cudaSetDevice(h->device);
  if (on && h->D > 0 && !h->d_acc) {
    h->n_acc = std::min(EAGER_SLOTS, std::max(1, (int)h->max_buf));
    GBA_CUDA(h, cudaMalloc(&h->d_acc, (size_t)h->n_acc * 2 * h->D_pad * sizeof(float)));
    GBA_CUDA(h, cudaMalloc(&h->d_stage_dense, (size_t)h->D_pad * sizeof(float)));
    for (int i = 0; i < h->n_acc; ++i)
      GBA_CUDA(h, cudaEventCreateWithFlags(&h->acc_ev[i], cudaEventDisableTiming));
  }
  h->eager = on != 0;
  return GBA_OK;
}

gba_status gba_table_capacity(gba_handle* h, int32_t t, int64_t* rows) {
  if (!h || t < 0 || t >= h->T || !rows) return GBA_E_ARG;
  *rows = h->tables[t].desc.rows;
  return GBA_OK;
}

gba_status gba_lookup_rows(gba_handle* h, int32_t t, const int64_t* ids, int64_t n,
                           int64_t* rows_out) {
  if (!h || t < 0 || t >= h->T || n < 0) return GBA_E_ARG;
  if (h->tables[t].desc.id_mode != GBA_ID_HASH) return set_err(h, GBA_E_ARG, "not a HASH table");
  if (n > 0 && (!ids || !rows_out)) return set_err(h, GBA_E_ARG, "NULL ids or rows_out");
  cudaSetDevice(h->device);
  join_steps(h);
  launch_hash_lookup(h->d_hinfo + t, ids, n, rows_out, h->stream);
  GBA_CUDA(h, cudaGetLastError());
  return GBA_OK;
}

gba_status gba_join(gba_handle* h) {
  if (!h) return GBA_E_ARG;
  cudaSetDevice(h->device);
  join_steps(h);
  GBA_CUDA(h, cudaGetLastError());
  return GBA_OK;
}

gba_status gba_set_overlap(gba_handle* h, int32_t on) {
  if (!h) return GBA_E_ARG;
  cudaSetDevice(h->device);
  if (!on) join_steps(h);
  h->overlap = on != 0;
  return GBA_OK;
}

gba_status gba_set_debug(gba_handle* h, int32_t on) {
  if (!h) return GBA_E_ARG;
  h->debug = on != 0;
  return GBA_OK;
}

gba_status gba_debug_segments(gba_handle* h, int64_t cap, int32_t* table, int64_t* row,
                              int64_t* count, int64_t* kept, int64_t* n_unique) {
  if (!h || !n_unique) return GBA_E_ARG;
  if (!h->have_last || !h->debug)
    return set_err(h, GBA_E_STATE, "no debug record of a step (enable debug before the step)");
  cudaSetDevice(h->device);
  GBA_CUDA(h, sync_all(h));
  // the step's row records, table by table: (row, prefixes of kept occurrences
  // and of (message, row) pairs at the row's head), closed by the totals
  std::vector<uint32_t> U(h->T, 0u);
  if (h->T > 0 && h->last_N > 0)
    GBA_CUDA(h, cudaMemcpy(U.data(), h->d_seg_total, h->T * sizeof(uint32_t),
                           cudaMemcpyDeviceToHost));
  int64_t u_all = 0;
  for (int t = 0; t < h->T; ++t) {
    const int64_t Nt = h->last_nbase[t + 1] - h->last_nbase[t];
    if (Nt == 0) continue;
    std::vector<uint4> rr((size_t)U[t] + 1);
    GBA_CUDA(h, cudaMemcpy(rr.data(), h->d_rr + h->last_nbase[t] + t, rr.size() * sizeof(uint4),
                           cudaMemcpyDeviceToHost));
    std::vector<unsigned long long> keys;  // HASH tables report the id of each slot
    if (h->tables[t].desc.id_mode == GBA_ID_HASH) {
      keys.resize((size_t)h->tables[t].desc.rows);
      GBA_CUDA(h, cudaMemcpy(keys.data(), h->tables[t].keys, keys.size() * 8,
                             cudaMemcpyDeviceToHost));
    }
    for (uint32_t u = 0; u < U[t]; ++u, ++u_all) {
      if (u_all >= cap) continue;
      if (table) table[u_all] = t;
      if (row) row[u_all] = keys.empty() ? (int64_t)rr[u].x : (int64_t)keys[rr[u].x];
      if (count) count[u_all] = (int64_t)(rr[u + 1].z - rr[u].z);
      if (kept) kept[u_all] = (int64_t)(rr[u + 1].y - rr[u].y);
    }
  }
  *n_unique = u_all;
  return u_all > cap ? set_err(h, GBA_E_ARG, "capacity too small") : GBA_OK;
}

gba_status gba_debug_sorted(gba_handle* h, int64_t cap, uint32_t* keys, uint32_t* occ,
                            int64_t* n) {
  if (!h || !n) return GBA_E_ARG;
  if (!h->have_last) return set_err(h, GBA_E_STATE, "no step applied yet");
  cudaSetDevice(h->device);
  GBA_CUDA(h, sync_all(h));
  *n = h->last_N;
  if (h->last_N > cap) return set_err(h, GBA_E_ARG, "capacity too small");
  if (h->last_N > 0) {
    if (keys)
      GBA_CUDA(h, cudaMemcpy(keys, h->d_keys[h->last_slot][h->last_buf], h->last_N * 4, cudaMemcpyDeviceToHost));
    if (occ)
      GBA_CUDA(h, cudaMemcpy(occ, h->d_vals[h->last_slot][h->last_buf], h->last_N * 4, cudaMemcpyDeviceToHost));
  }
  return GBA_OK;
}

gba_status gba_debug_keep(gba_handle* h, int32_t cap, int32_t* keep, int32_t* M) {
  if (!h || !M) return GBA_E_ARG;
  if (!h->have_last) return set_err(h, GBA_E_STATE, "no step applied yet");
  cudaSetDevice(h->device);
  GBA_CUDA(h, sync_all(h));
  *M = h->last_M;
  if (h->last_M > cap) return set_err(h, GBA_E_ARG, "capacity too small");
  if (keep && h->last_M > 0)
    GBA_CUDA(h, cudaMemcpy(keep, h->sc[h->last_slot].keep, h->last_M * 4, cudaMemcpyDeviceToHost));
  return GBA_OK;
}

gba_status gba_debug_set_wait_limit(gba_handle* h, int64_t ns) {
  if (!h || ns < 0) return GBA_E_ARG;
  h->wait_ns = ns;
  return GBA_OK;
}

gba_status gba_debug_withhold_dense_copies(gba_handle* h, int32_t on) {
  if (!h || (on != 0 && on != 1)) return GBA_E_ARG;
  h->withhold_dense = on != 0;
  return GBA_OK;
}

gba_status gba_selftest_wait_timeout(int64_t limit_ns, void* cuda_stream) {
  if (limit_ns < 0 || limit_ns > 10000000000ll) return GBA_E_ARG;
  uint32_t* d = nullptr;
  if (cudaMalloc(&d, 2 * sizeof(uint32_t)) != cudaSuccess) return GBA_E_OOM;
  uint32_t result = 0;
  const int rc = launch_wait_selftest(limit_ns, (cudaStream_t)cuda_stream, d, &result);
  cudaFree(d);
  if (rc != 0) return GBA_E_CUDA;
  return result ? GBA_E_DEVICE_TIMEOUT : GBA_OK;
}

int32_t gba_device_binary_version(void) {
  const int v = kernel_binary_version();
  if (v < 0) {
    cudaGetLastError();
    return GBA_E_CUDA;
  }
  return v;
}

const char* gba_version_string(void) { return "libgba 0.2 (sm_103a)"; }

}  // extern "C"
