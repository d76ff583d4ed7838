// Internal declarations shared by the translation units of libgba.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace gba {

// ---- device error word bits -------------------------------------------------
constexpr uint32_t ERR_ID_RANGE = 1u;
constexpr uint32_t ERR_TIMEOUT = 2u;
constexpr uint32_t ERR_INTERNAL = 4u;

// Where kernels report a failure: the step's own word (later kernels of the
// same step skip their work when it is set), the handle's word (what the host
// reports), and a flag in mapped pinned host memory the host polls without
// synchronising.
struct ErrSink {
  uint32_t* step;
  uint32_t* dev;
  volatile uint32_t* host;
};

__device__ __forceinline__ void raise_error(const ErrSink& e, uint32_t code) {
  atomicOr(e.step, code);
  atomicOr(e.dev, code);
  *e.host = 1u;
}

__device__ __forceinline__ uint64_t globaltimer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// ---- mbarriers and 1-D bulk async copies (shared memory, this CTA) ----------
__device__ __forceinline__ uint32_t smem_addr(const void* p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count)
               : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)),
               "r"(bytes)
               : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_addr(bar)) : "memory");
}

// Waits for the phase with the given parity to complete; the thread may be
// suspended in the instruction for up to the hinted time instead of spinning.
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_addr(bar)), "r"(parity), "r"(100000u)
      : "memory");
  return ok != 0u;
}

// Bounded wait for the phase with the given parity; false if it gave up.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, int64_t limit_ns) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  while (!mbar_try_wait(bar, parity)) {
    if ((int64_t)(globaltimer_ns() - t0) > limit_ns) return false;
  }
  return true;
}

__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes,
                                         uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::
          "r"(smem_addr(dst)),
      "l"(src), "r"(bytes), "r"(smem_addr(bar))
      : "memory");
}

// ---- per-table static description (device copy) ----------------------------
struct TableInfo {
  int64_t V;
  uint32_t key_base;  // first global key of the table
  int32_t id_mode;    // 0 DIRECT, 1 MODULO
  uint64_t mod_magic; // floor((2^64 - 1) / V), for mod_u64
};

// x mod V for a 64-bit x and V < 2^32, without a 64-bit division: the
// quotient estimate floor(x * m / 2^64) with m = floor((2^64 - 1) / V) is at
// most 2 below floor(x / V) (division by an invariant integer through a
// precomputed reciprocal, after Granlund and Montgomery 1994), so at most two
// corrections give the exact remainder.
__device__ __forceinline__ uint64_t mod_u64(uint64_t x, uint64_t V, uint64_t m) {
  uint64_t r = x - __umul64hi(x, m) * V;
  if (r >= V) r -= V;
  if (r >= V) r -= V;
  return r;
}

// ---- counter-based initial values (shared by table init and hash inserts) ---
// SplitMix64 (Steele, Lea, Flood 2014): output for state x.
__device__ __forceinline__ uint64_t splitmix64(uint64_t x) {
  uint64_t z = x + 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

// Weight of element e of an array: top 24 bits of the hash, centred, times
// 2^-27 (an exact float in [-1/16, 1/16)).
__device__ __forceinline__ float init_weight(uint64_t seed, uint64_t tag, uint64_t e) {
  const uint64_t h = splitmix64(seed ^ tag ^ e);
  const int32_t top = (int32_t)(h >> 40) - 8388608;
  return (float)top * 0x1p-27f;
}

// ---- expandable hash tables of 64-bit ids (id_mode HASH) --------------------
// Open addressing with linear probing over a power-of-two number of slots; the
// row of an id is the slot it occupies, so the embedding arrays are indexed by
// slot.  A new id is inserted by compare-and-swap on its slot's key and its
// row is initialised from the id (element e = id * d + j of the table's
// counter-based stream), so every id starts from the same values whichever
// slot it lands in.
constexpr unsigned long long HASH_EMPTY = 0x8000000000000000ull;  // INT64_MIN: not a valid id
struct HashInfo {
  unsigned long long* keys;  // [slots] id per slot, HASH_EMPTY when free
  uint64_t mask;             // slots - 1
  float* w;
  float* s0;
  float* s1;
  int32_t* ver;
  unsigned long long* count;  // ids inserted so far
  uint64_t seed, tag;
  int32_t d, kind;
  float init_acc;
  int32_t pad;
};

__device__ __forceinline__ void hash_init_row(const HashInfo& hi, uint64_t slot, int64_t id) {
  const float a0 = hi.kind == 0 ? hi.init_acc : 0.f;
  for (int j = 0; j < hi.d; ++j) {
    const size_t e = (size_t)slot * hi.d + j;
    hi.w[e] = init_weight(hi.seed, hi.tag, (uint64_t)id * (uint64_t)hi.d + (uint64_t)j);
    hi.s0[e] = a0;
    if (hi.kind == 1) hi.s1[e] = 0.f;
  }
  hi.ver[slot] = 0;
}

// The slot of id, inserting it when absent; returns mask + 1 when the table
// is full (cannot happen while the host keeps it at most half full).
__device__ __forceinline__ uint64_t hash_find_or_insert(const HashInfo& hi, int64_t id) {
  const unsigned long long key = (unsigned long long)id;
  uint64_t slot = splitmix64(key) & hi.mask;
  for (uint64_t probe = 0; probe <= hi.mask; ++probe, slot = (slot + 1) & hi.mask) {
    const unsigned long long k = *(volatile unsigned long long*)(hi.keys + slot);
    if (k == key) return slot;
    if (k == HASH_EMPTY) {
      const unsigned long long old = atomicCAS(hi.keys + slot, HASH_EMPTY, key);
      if (old == HASH_EMPTY) {
        hash_init_row(hi, slot, id);
        atomicAdd(hi.count, 1ull);
        return slot;
      }
      if (old == key) return slot;
    }
  }
  return hi.mask + 1;
}

// The slot of id, or mask + 1 when it is absent.
__device__ __forceinline__ uint64_t hash_find(const HashInfo& hi, int64_t id) {
  const unsigned long long key = (unsigned long long)id;
  uint64_t slot = splitmix64(key) & hi.mask;
  for (uint64_t probe = 0; probe <= hi.mask; ++probe, slot = (slot + 1) & hi.mask) {
    const unsigned long long k = hi.keys[slot];
    if (k == key) return slot;
    if (k == HASH_EMPTY) break;
  }
  return hi.mask + 1;
}

// ---- optimizer parameters of one parameter group for one step ---------------
struct OptStep {
  int32_t kind;  // 0 Adagrad, 1 Adam
  float lr, b1, b2, eps;
  float c1, c2;    // 1 - b1, 1 - b2 (float arithmetic)
  float bc1, bc2;  // Adam bias corrections of this step
};

// Adagrad and Adam, one IEEE float operation at a time in a fixed order.
__device__ __forceinline__ void opt_update(const OptStep& o, float& w, float& s0, float& s1,
                                           float g) {
  if (o.kind == 0) {
    float gg = __fmul_rn(g, g);
    float an = __fadd_rn(s0, gg);
    float step = __fmul_rn(o.lr, g);
    float den = __fsqrt_rn(an);
    s0 = an;
    w = __fsub_rn(w, __fdiv_rn(step, den));
  } else {
    float mn = __fadd_rn(__fmul_rn(o.b1, s0), __fmul_rn(o.c1, g));
    float gg = __fmul_rn(g, g);
    float vn = __fadd_rn(__fmul_rn(o.b2, s1), __fmul_rn(o.c2, gg));
    float mhat = __fdiv_rn(mn, o.bc1);
    float vhat = __fdiv_rn(vn, o.bc2);
    float num = __fmul_rn(o.lr, mhat);
    float den = __fadd_rn(__fsqrt_rn(vhat), o.eps);
    s0 = mn;
    s1 = vn;
    w = __fsub_rn(w, __fdiv_rn(num, den));
  }
}

// Error-free transformation of a + b (Knuth's TwoSum): s + e == a + b exactly.
__device__ __forceinline__ void two_sum(float a, float b, float& s, float& e) {
  s = __fadd_rn(a, b);
  float bp = __fsub_rn(s, a);
  float ap = __fsub_rn(s, bp);
  e = __fadd_rn(__fsub_rn(a, ap), __fsub_rn(b, bp));
}

// Compensated accumulator: value = hi + lo.
struct CSum {
  float hi, lo;
};
__device__ __forceinline__ void csum_add(CSum& c, float x) {
  float s, e;
  two_sum(c.hi, x, s, e);
  c.hi = s;
  c.lo = __fadd_rn(c.lo, e);
}
__device__ __forceinline__ void csum_merge(CSum& c, float hi, float lo) {
  float s, e;
  two_sum(c.hi, hi, s, e);
  c.hi = s;
  c.lo = __fadd_rn(__fadd_rn(c.lo, lo), e);
}
__device__ __forceinline__ float csum_value(const CSum& c) { return __fadd_rn(c.hi, c.lo); }

// ---- one global step, as seen by the kernels ---------------------------------
// Passed by value to every kernel of a step; the arrays live in a device
// buffer the host fills before the step.
struct StepArgs {
  int64_t k;
  int32_t M;           // messages popped
  int32_t T;           // tables
  int64_t N;           // id occurrences over all tables
  int32_t iota;
  int32_t row_staleness;
  int32_t sparse_den;
  int32_t decay;        // 0: f in {0, 1} (Eq. (1)); 1: f = lambda^s for s <= iota
  int32_t drop_latest;  // the last drop_latest popped messages are excluded (0: none)
  int32_t n_wtab;       // entries of wtab (decay 1): wtab[s] = lambda^s, s < n_wtab
  const float* wtab;    // [n_wtab] device
  const int64_t* tokens;          // [M]
  const float* const* dense_ptr;  // [M]
  const uint32_t* msg_off;        // [T][M+1] occurrence offsets within the table
  const int64_t* const* ids_ptr;  // [T][M]
  const float* const* rows_ptr;   // [T][M]
  const int64_t* nbase;           // [T+1] first global occurrence of each table
  const TableInfo* tinfo;         // [T]
  const HashInfo* hinfo;          // [T] (tables with id_mode HASH)
};

// Per-step device scratch that K1 clears at the start of a step.
struct StepScratch {
  uint32_t* hist;          // [4][256] digit histograms of the key passes
  uint32_t* tile_counter;  // [4] onesweep tile tickets
  int32_t* keep;           // [M] message weights f
  int32_t* kept_list;      // [M] indices of kept messages, in pop order
  int32_t* n_kept;         // [1]
  uint32_t* step_err;      // [1] failures of this step
  uint32_t* seg_ticket;    // [T][8] per table: scan tile tickets, long rows, their items,
                           // chunk-sum slots, item tickets, unused
  float* fw;               // [M] message weights of the dense sum (decay 1; 1 or 0 otherwise)
};

// Weight of a gradient with staleness s (s >= 0), or 0 when it is excluded:
// Eq. (1) keeps s <= iota; decay 1 scales a kept gradient by lambda^s.
__device__ __forceinline__ float decay_weight(const StepArgs& a, uint64_t s) {
  if (s > (uint64_t)(int64_t)a.iota) return 0.f;
  if (a.decay == 0) return 1.f;
  return s < (uint64_t)a.n_wtab ? __ldg(a.wtab + s) : 0.f;
}

// Compensated accumulation of a product f * g: the product's rounding error
// (from a fused multiply-add) joins the compensation term, so with f = 1 this
// is exactly csum_add.
__device__ __forceinline__ void csum_add_prod(CSum& c, float f, float g) {
  const float p = __fmul_rn(f, g);
  const float e = __fmaf_rn(f, g, -p);
  float s, t;
  two_sum(c.hi, p, s, t);
  c.hi = s;
  c.lo = __fadd_rn(c.lo, __fadd_rn(t, e));
}

// A kept term of a weighted sum.  With decay strategy 0 every kept weight is
// exactly 1 and the term is added by csum_add, which gives what csum_add_prod
// gives for f = 1 (the product and its error are g and 0) with fewer operations.
__device__ __forceinline__ void csum_add_w(CSum& c, bool unit, float f, float g) {
  if (unit)
    csum_add(c, g);
  else
    csum_add_prod(c, f, g);
}

// Accumulated statistics (device).
struct DevStats {
  unsigned long long steps, msgs_kept, msgs_dropped, dense_stale_sum, dense_stale_max, pairs,
      pairs_dropped, row_stale_sum, row_stale_max, occurrences, rows_touched, rows_applied,
      occ_kept;
};

// The message that holds table-local occurrence x: the largest m in [0, M)
// with off[m] <= x, given off[0] = 0 <= x < off[M] (empty messages repeat an
// offset and are skipped by taking the largest such m).
__device__ __forceinline__ int message_of(const uint32_t* off, int M, uint32_t x) {
  int lo = 0, hi = M;  // off[lo] <= x < off[hi]
  while (hi - lo > 1) {
    int mid = (lo + hi) >> 1;
    if (__ldg(off + mid) <= x)
      lo = mid;
    else
      hi = mid;
  }
  return lo;
}

// ---- launch wrappers (defined in the kernel translation units) ---------------
void launch_weights(const StepArgs& a, StepScratch sc, DevStats* stats, int n_hist_words,
                    cudaStream_t s);

// Keys per onesweep tile (also sizes the look-back words of the static sort).
#ifndef GBA_SORT_TILE
#define GBA_SORT_TILE 2048
#endif
constexpr int SORT_TILE_KEYS = GBA_SORT_TILE;  // keys per onesweep tile

// Digit histograms of every pass; writes each occurrence's key to keys0 (the
// first onesweep pass's input).
void launch_sort_histogram(const StepArgs& a, int passes, StepScratch sc, uint32_t* keys0,
                           ErrSink err, int grid, cudaStream_t s);

void launch_onesweep(const StepArgs& a, bool first, int pass, const uint32_t* keys_in,
                     const uint32_t* vals_in, uint32_t* keys_out, uint32_t* vals_out,
                     StepScratch sc, unsigned long long* status, uint32_t epoch, ErrSink err,
                     int64_t wait_ns, cudaStream_t s);

int sort_tiles(int64_t N);

struct SegTable {
  float* w;
  float* s0;
  float* s1;
  int32_t* ver;
  int32_t d;
  int32_t t;
  uint32_t key_base;
  int32_t pad;
  int64_t rows;                // V of the table
  int64_t pos_begin, pos_end;  // range of the sorted array holding this table's keys
  OptStep opt;
};

// Buffers of the row kernels (one set, used in stream order by the apply
// stream; every table of a step uses its own ranges of rr / kl / kw).
//  rr[u]   row u of the table in sorted order: (row x, and the exclusive
//          prefixes at its head of kept occurrences K, (message, row) pairs C
//          and kept pairs CK); rr[U] holds the totals, so row u's kept
//          occurrences are kl[rr[u].K .. rr[u+1].K), c_x = rr[u+1].C - rr[u].C
//  kl[j]   address of the j-th kept occurrence's gradient row, sorted by row
//  kw[j]   its weight f (1 under Eq. (1))
struct SegOut {
  uint4* rr;                   // this table's range
  const float** kl;            // this table's range
  float* kw;                   // this table's range
  unsigned long long* status;  // [tiles][4] look-back words of the scan
  uint32_t epoch;              // tag of this launch's look-back words
  uint32_t* ticket;            // scan tile tickets (cleared by K1)
  uint32_t* n_long;            // rows with more than LONG_ROW kept occurrences (cleared by K1)
  uint32_t* n_items;           // chunks of those rows (cleared by K1)
  uint32_t* n_parts;           // chunk-sum slots of rows split into chunks (cleared by K1)
  uint32_t* item_ticket;       // items claimed by warps of the long-row kernel (cleared by K1)
  uint32_t* total;             // this table's U (written by the last scan tile)
  uint4* long_rows;            // [n_long] (u, first kept, kept count, first chunk-sum slot)
  uint32_t* long_done;         // [n_long] chunks of the row finished
  uint2* items;                // [n_items] (long row, chunk)
  float* part_hi;              // [n_parts][pstride] compensated chunk sums
  float* part_lo;
  int32_t pstride;
  uint4* small_rows;           // [n_small] (row, first kept, kept count, denominator bits)
  uint32_t* n_small;           // long rows of at most SMALL_MAX kept occurrences (cleared by K1)
  uint32_t* small_ticket;      // small rows claimed by the long-row kernel (cleared by K1)
};

// Rows with at most LONG_ROW kept occurrences are applied by one lane group
// each with all their gradient rows staged in shared memory; longer rows by a
// whole warp each, in chunks of LONG_CHUNK kept occurrences.
constexpr int LONG_ROW = 4;
#ifndef GBA_LONG_CHUNK
#define GBA_LONG_CHUNK 128
#endif
constexpr int LONG_CHUNK = GBA_LONG_CHUNK;
// Long rows of at most SMALL_MAX kept occurrences are applied by one lane
// group each, with all their gradient rows staged in shared memory.
#ifndef GBA_SMALL_MAX
#define GBA_SMALL_MAX 32
#endif
constexpr int SMALL_MAX = GBA_SMALL_MAX;
#ifndef GBA_SCAN_TILE
#define GBA_SCAN_TILE 2048
#endif
constexpr int SCAN_TILE = GBA_SCAN_TILE;  // sorted positions per segment-scan tile

int64_t scan_tiles(int64_t N);

void launch_seg_scan(const StepArgs& a, const SegTable& tb, const SegOut& so, const uint32_t* keys,
                     const uint32_t* vals, DevStats* stats, ErrSink err, int64_t wait_ns,
                     cudaStream_t s);

void launch_row_apply(const StepArgs& a, const SegTable& tb, const SegOut& so, DevStats* stats,
                      ErrSink err, int num_sms, cudaStream_t s);

void launch_row_long(const StepArgs& a, const SegTable& tb, const SegOut& so, DevStats* stats,
                     ErrSink err, int num_sms, cudaStream_t s);

// Lists the long rows and their chunks (after the scan, before both row kernels).
void launch_row_classify(const StepArgs& a, const SegTable& tb, const SegOut& so, ErrSink err,
                         int num_sms, cudaStream_t s);

struct DenseArgs {
  float* w;
  float* s0;
  float* s1;
  int64_t D;
  int32_t M;
  OptStep opt;
  int32_t withhold = 0;  // test hook: the producer issues no copies, so every
                         // consumer wait runs out and reports ERR_TIMEOUT
};

size_t dense_smem_bytes();
cudaError_t configure_dense();
void launch_dense(const StepArgs& a, const DenseArgs& da, StepScratch sc, ErrSink err,
                  int64_t wait_ns, int num_sms, cudaStream_t s);

// Eager dense aggregation: add f * g to a step's accumulator (first: start it),
// and the step's update from the accumulator.
void launch_dense_accumulate(float* hi, float* lo, const float* g, int64_t D, float f, bool first,
                             int num_sms, cudaStream_t s);
void launch_dense_eager(const DenseArgs& da, const float* hi, const float* lo, bool has_sum,
                        ErrSink err, int num_sms, cudaStream_t s);

void launch_init_table(float* w, float* s0, float* s1, int32_t* ver, int64_t rows, int32_t d,
                       int32_t kind, float init_acc, uint64_t seed, uint64_t tag,
                       cudaStream_t s);

void launch_init_dense(float* w, float* s0, float* s1, int64_t D, int32_t kind, float init_acc,
                       uint64_t seed, uint64_t tag, cudaStream_t s);

int launch_wait_selftest(int64_t limit_ns, cudaStream_t s, uint32_t* d_word, uint32_t* result);

// Rows of one table for n ids (pull responding), into out[n][d].
void launch_pull_rows(const float* w, int64_t V, int d, int id_mode, uint64_t mod_magic,
                      const HashInfo* hinfo, const int64_t* ids, int64_t n, float* out,
                      ErrSink err, int num_sms, cudaStream_t s);

// Hash tables: fill keys with HASH_EMPTY; move every id of one table into a
// larger one (keys, rows and tags); slots of ids (mask + 1 when absent).
void launch_hash_clear(unsigned long long* keys, uint64_t slots, cudaStream_t s);
void launch_hash_rehash(HashInfo from, HashInfo to, cudaStream_t s);
void launch_hash_lookup(const HashInfo* hinfo, const int64_t* ids, int64_t n, int64_t* slots,
                        cudaStream_t s);

// Compute capability (major * 10 + minor) of the device code the library's
// kernels were loaded from on the current device, or -1.
int kernel_binary_version();

}  // namespace gba
