// K1 (message weights, Eq. (1)) and K2 (stable LSD radix sort of the step's
// row keys) of the GBA aggregate-and-apply step.
//
// The sort follows the onesweep method (Adinets & Merrill 2022): one kernel
// counts the digits of every pass, then each pass is a single kernel in which
// tiles rank their keys locally and find their global output offsets by
// decoupled look-back over the per-tile digit counts of earlier tiles
// (Merrill & Garland 2016).  Tiles take tickets from an atomic counter, so a
// tile only ever waits on tiles that are already running; every wait is
// bounded in time and latches ERR_TIMEOUT instead of hanging.
//
// The first pass reads the int64 ids straight from the messages and computes
// the 32-bit key (global row = table key base + row) on the fly, with the
// global occurrence index as payload; later passes move (key, payload) pairs.
#include "gba_internal.cuh"

namespace gba {

namespace {

constexpr int RADIX = 256;
constexpr int SORT_THREADS = 256;  // one thread per digit in the look-back
constexpr int SORT_WARPS = SORT_THREADS / 32;
constexpr int SORT_ITEMS = SORT_TILE_KEYS / SORT_THREADS;
constexpr int SORT_TILE = SORT_TILE_KEYS;
static_assert(SORT_TILE_KEYS % SORT_THREADS == 0, "tile must fill the block");
constexpr int MAX_PASSES = 4;
constexpr int LB_WIN = 8;  // look-back window
constexpr int OFF_CACHE = 1024;  // message offsets kept in shared memory

// Copies the step's message offsets into shared memory when they fit;
// returns the array the key computation should read.
__device__ __forceinline__ const uint32_t* cache_offsets(const StepArgs& a, uint32_t* s_off) {
  const int n = a.T * (a.M + 1);
  if (n > OFF_CACHE) return a.msg_off;
  for (int i = threadIdx.x; i < n; i += blockDim.x) s_off[i] = a.msg_off[i];
  __syncthreads();
  return s_off;
}

// Look-back status word: [63:32] epoch of the launch, [31:30] flag, [29:0] count.
constexpr unsigned long long FLAG_AGG = 1ull << 30;
constexpr unsigned long long FLAG_INCL = 2ull << 30;
constexpr unsigned long long FLAG_MASK = 3ull << 30;
constexpr unsigned long long COUNT_MASK = (1ull << 30) - 1;

__device__ __forceinline__ unsigned long long ld_relaxed_u64(const unsigned long long* p) {
  unsigned long long v;
  asm volatile("ld.relaxed.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ void st_relaxed_u64(unsigned long long* p, unsigned long long v) {
  asm volatile("st.relaxed.gpu.global.u64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}
__device__ __forceinline__ uint32_t ld_volatile_u32(const uint32_t* p) {
  return *(const volatile uint32_t*)p;
}
__device__ __forceinline__ uint32_t lanemask_lt() {
  uint32_t m;
  asm("mov.u32 %0, %%lanemask_lt;" : "=r"(m));
  return m;
}

// Key of global occurrence o: the table holding o, the message holding it, the
// id, and the row it maps to (DIRECT ids outside [0, V) latch ERR_ID_RANGE and
// are clamped to row 0; the whole step is then skipped by later kernels).
__device__ __forceinline__ uint32_t occurrence_key(const StepArgs& a, const uint32_t* offs,
                                                   int64_t o, const ErrSink& err) {
  int t = 0;
  while (t + 1 < a.T && __ldg(a.nbase + t + 1) <= o) ++t;
  const uint32_t ot = (uint32_t)(o - __ldg(a.nbase + t));
  const uint32_t* off = offs + (size_t)t * (a.M + 1);
  int lo = 0, hi = a.M;  // the message holding ot: off[lo] <= ot < off[lo + 1]
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (off[mid] <= ot)
      lo = mid;
    else
      hi = mid;
  }
  const int m = lo;
  const uint32_t p = ot - off[m];
  const int64_t* ids = a.ids_ptr[(size_t)t * a.M + m];
  const int64_t id = __ldg(ids + p);
  const TableInfo ti = a.tinfo[t];
  uint64_t row;
  if (ti.id_mode == 0) {
    if (id < 0 || id >= ti.V) {
      raise_error(err, ERR_ID_RANGE);
      row = 0;
    } else {
      row = (uint64_t)id;
    }
  } else if (ti.id_mode == 1) {
    row = mod_u64((uint64_t)id, (uint64_t)ti.V, ti.mod_magic);
  } else {  // HASH: the id's slot, inserted on first sight
    if ((unsigned long long)id == HASH_EMPTY) {
      raise_error(err, ERR_ID_RANGE);
      row = 0;
    } else {
      row = hash_find_or_insert(a.hinfo[t], id);
      if (row > a.hinfo[t].mask) {
        raise_error(err, ERR_INTERNAL);
        row = 0;
      }
    }
  }
  return ti.key_base + (uint32_t)row;
}

// Exclusive scan of one value per thread over a 256-thread block.
__device__ __forceinline__ uint32_t block_excl_scan_256(uint32_t v, uint32_t* s_tmp) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  uint32_t x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    uint32_t y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) s_tmp[warp] = x;
  __syncthreads();
  uint32_t wsum = 0;
#pragma unroll
  for (int w = 0; w < SORT_WARPS; ++w)
    if (w < warp) wsum += s_tmp[w];
  __syncthreads();
  return wsum + x - v;
}

// ---------------------------------------------------------------------------
// K1: message weights of Eq. (1), kept-message list, dense staleness counters;
// also clears the per-step sort scratch.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256) k_message_weights(StepArgs a, StepScratch sc,
                                                         DevStats* st, int n_hist_words) {
  const int tid = threadIdx.x;
  for (int i = tid; i < n_hist_words; i += blockDim.x) sc.hist[i] = 0u;
  if (tid < MAX_PASSES) sc.tile_counter[tid] = 0u;
  if (tid == 0) *sc.step_err = 0u;
  if (sc.seg_ticket)
    for (int i = tid; i < 8 * a.T; i += blockDim.x) sc.seg_ticket[i] = 0u;
  if (tid >= 32) return;
  const int lane = tid;
  int kept = 0;
  unsigned long long s_sum = 0, s_max = 0;
  for (int base = 0; base < a.M; base += 32) {
    const int m = base + lane;
    int keep = 0;
    unsigned long long s = 0;
    float f = 0.f;
    if (m < a.M) {
      const int64_t diff = a.k - a.tokens[m];
      s = diff > 0 ? (unsigned long long)diff : 0ull;
      // Eq. (1) (or the decay strategy), and Hop-BW's ignored latest messages
      f = m < a.M - a.drop_latest ? decay_weight(a, s) : 0.f;
      keep = f > 0.f ? 1 : 0;
      sc.keep[m] = keep;
    }
    const uint32_t b = __ballot_sync(0xffffffffu, keep != 0);
    if (keep) {
      const int j = kept + __popc(b & lanemask_lt());
      sc.kept_list[j] = m;
      if (sc.fw) sc.fw[j] = f;
    }
    kept += __popc(b);
    s_sum += s;
    s_max = s > s_max ? s : s_max;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    s_sum += __shfl_xor_sync(0xffffffffu, s_sum, o);
    unsigned long long y = __shfl_xor_sync(0xffffffffu, s_max, o);
    s_max = y > s_max ? y : s_max;
  }
  if (lane == 0) {
    *sc.n_kept = kept;
    atomicAdd(&st->steps, 1ull);
    atomicAdd(&st->msgs_kept, (unsigned long long)kept);
    atomicAdd(&st->msgs_dropped, (unsigned long long)(a.M - kept));
    atomicAdd(&st->dense_stale_sum, s_sum);
    atomicMax(&st->dense_stale_max, s_max);
    atomicAdd(&st->occurrences, (unsigned long long)a.N);
  }
}

// ---------------------------------------------------------------------------
// Digit counts of every pass in one read of the ids; also writes every
// occurrence's key (keys0) for the first onesweep pass.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(SORT_THREADS) k_sort_histogram(StepArgs a, int passes,
                                                                 StepScratch sc, uint32_t* keys0,
                                                                 ErrSink err) {
  __shared__ uint32_t h[MAX_PASSES][RADIX];
  __shared__ uint32_t s_off[OFF_CACHE];
  for (int i = threadIdx.x; i < MAX_PASSES * RADIX; i += SORT_THREADS) (&h[0][0])[i] = 0u;
  const uint32_t* offs = cache_offsets(a, s_off);
  __syncthreads();
  const int64_t stride = (int64_t)gridDim.x * SORT_THREADS;
  for (int64_t o = (int64_t)blockIdx.x * SORT_THREADS + threadIdx.x; o < a.N; o += stride) {
    const uint32_t key = occurrence_key(a, offs, o, err);
    keys0[o] = key;
    for (int p = 0; p < passes; ++p) atomicAdd(&h[p][(key >> (8 * p)) & (RADIX - 1)], 1u);
  }
  __syncthreads();
  for (int i = threadIdx.x; i < passes * RADIX; i += SORT_THREADS) {
    const uint32_t v = (&h[0][0])[i];
    if (v) atomicAdd(sc.hist + i, v);
  }
}

// ---------------------------------------------------------------------------
// One onesweep pass over 8 bits of the key.
// ---------------------------------------------------------------------------
#ifndef GBA_LOOKBACK_SLEEP_NS
#define GBA_LOOKBACK_SLEEP_NS 64
#endif
template <bool FIRST>
__global__ void __launch_bounds__(SORT_THREADS)
    k_onesweep(StepArgs a, int pass, const uint32_t* __restrict__ keys_in,
               const uint32_t* __restrict__ vals_in, uint32_t* __restrict__ keys_out,
               uint32_t* __restrict__ vals_out, StepScratch sc, unsigned long long* status,
               uint32_t epoch, ErrSink err, int64_t wait_ns) {
  __shared__ uint32_t s_warp[SORT_WARPS][RADIX];  // per-warp digit counts, then offsets
  __shared__ uint32_t s_tile_excl[RADIX];         // first tile slot of each digit
  __shared__ uint32_t s_out_base[RADIX];          // global position of that slot
  __shared__ uint32_t s_tmp[SORT_WARPS];
  __shared__ uint32_t s_keys[SORT_TILE];
  __shared__ uint32_t s_vals[SORT_TILE];
  __shared__ uint32_t s_tile;

  // An id range error was latched before this launch (by the histogram):
  // every tile of every pass skips, consistently.
  if (__syncthreads_or((ld_volatile_u32(err.step) & ERR_ID_RANGE) != 0u)) return;

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  if (tid == 0) s_tile = atomicAdd(sc.tile_counter + pass, 1u);
  for (int i = tid; i < SORT_WARPS * RADIX; i += SORT_THREADS) (&s_warp[0][0])[i] = 0u;
  __syncthreads();

  const uint32_t tile = s_tile;
  const int64_t N = a.N;
  const int64_t base = (int64_t)tile * SORT_TILE;
  const int shift = 8 * pass;

  uint32_t key[SORT_ITEMS], val[SORT_ITEMS], rank[SORT_ITEMS];
#pragma unroll
  for (int j = 0; j < SORT_ITEMS; ++j) {
    const int64_t idx = base + (int64_t)warp * (SORT_ITEMS * 32) + j * 32 + lane;
    if (idx < N) {
      if (FIRST) {  // keys written by the histogram kernel; payload = occurrence
        key[j] = keys_in[idx];
        val[j] = (uint32_t)idx;
      } else {
        key[j] = keys_in[idx];
        val[j] = vals_in[idx];
      }
    } else {
      key[j] = 0u;
      val[j] = 0u;
    }
  }

  // Warp-level multi-split: stable rank of each key among equal digits.
  const uint32_t lt = lanemask_lt();
#pragma unroll
  for (int j = 0; j < SORT_ITEMS; ++j) {
    const int64_t idx = base + (int64_t)warp * (SORT_ITEMS * 32) + j * 32 + lane;
    const bool valid = idx < N;
    const uint32_t d = valid ? ((key[j] >> shift) & (RADIX - 1)) : (uint32_t)RADIX;
    const uint32_t peers = __match_any_sync(0xffffffffu, d);
    uint32_t before = 0;
    if (valid) before = s_warp[warp][d];
    rank[j] = before + __popc(peers & lt);
    __syncwarp();
    if (valid && (peers & lt) == 0u) s_warp[warp][d] = before + __popc(peers);
    __syncwarp();
  }
  __syncthreads();

  // Thread d: this tile's count of digit d, then its global offset.
  const int d = tid;
  uint32_t run = 0;
#pragma unroll
  for (int w = 0; w < SORT_WARPS; ++w) {
    const uint32_t c = s_warp[w][d];
    s_warp[w][d] = run;
    run += c;
  }
  const uint32_t tile_count = run;
  unsigned long long* my = status + (size_t)tile * RADIX + d;
  const unsigned long long ep = (unsigned long long)epoch << 32;
  st_relaxed_u64(my, ep | (tile == 0 ? FLAG_INCL : FLAG_AGG) | tile_count);

  const uint32_t g_excl = block_excl_scan_256(sc.hist[pass * RADIX + d], s_tmp);
  const uint32_t t_excl = block_excl_scan_256(tile_count, s_tmp);
  s_tile_excl[d] = t_excl;

  // Decoupled look-back over a window of LB_WIN predecessors at a time: the
  // window's status words are read with independent loads, then consumed from
  // the nearest tile backwards until an inclusive prefix is found.  The words
  // are self-contained (no other data is published with them), so relaxed
  // loads and stores suffice.
  uint32_t prefix = 0;
  if (tile > 0) {
    int64_t j = (int64_t)tile - 1;
    const uint64_t t0 = globaltimer_ns();
    bool done = false;
    while (!done) {
      unsigned long long v[LB_WIN];
#pragma unroll
      for (int i = 0; i < LB_WIN; ++i)
        v[i] = (j - i >= 0) ? ld_relaxed_u64(status + (size_t)(j - i) * RADIX + d) : 0ull;
      int used = 0;
#pragma unroll
      for (int i = 0; i < LB_WIN; ++i) {
        if (done || used != i || j - i < 0) continue;
        const unsigned long long x = v[i];
        if ((x & ~0xFFFFFFFFull) != ep || (x & FLAG_MASK) == 0ull) continue;  // not ready
        prefix += (uint32_t)(x & COUNT_MASK);
        used = i + 1;
        if (x & FLAG_INCL) done = true;
      }
      if (done) break;
      j -= used;
      if (j < 0) break;  // cannot happen: tile 0 publishes an inclusive prefix
      if (used == 0) {
        if ((ld_volatile_u32(err.step) & ERR_TIMEOUT) ||
            (int64_t)(globaltimer_ns() - t0) > wait_ns) {
          raise_error(err, ERR_TIMEOUT);
          break;
        }
        if (GBA_LOOKBACK_SLEEP_NS > 0) __nanosleep(GBA_LOOKBACK_SLEEP_NS);  // back off: spinning takes issue slots from the tiles it waits for
      }
    }
    st_relaxed_u64(my, ep | FLAG_INCL | ((prefix + tile_count) & COUNT_MASK));
  }
  s_out_base[d] = g_excl + prefix;
  __syncthreads();

  // Place keys in digit order in shared memory, then write runs of equal digits.
#pragma unroll
  for (int j = 0; j < SORT_ITEMS; ++j) {
    const int64_t idx = base + (int64_t)warp * (SORT_ITEMS * 32) + j * 32 + lane;
    if (idx < N) {
      const uint32_t dg = (key[j] >> shift) & (RADIX - 1);
      const uint32_t pos = s_tile_excl[dg] + s_warp[warp][dg] + rank[j];
      s_keys[pos] = key[j];
      s_vals[pos] = val[j];
    }
  }
  __syncthreads();
  const int n_valid = (int)((N - base) < SORT_TILE ? (N - base) : SORT_TILE);
  for (int i = tid; i < n_valid; i += SORT_THREADS) {
    const uint32_t k = s_keys[i];
    const uint32_t dg = (k >> shift) & (RADIX - 1);
    const uint32_t out = s_out_base[dg] + ((uint32_t)i - s_tile_excl[dg]);
    if (out < (uint32_t)N) {
      keys_out[out] = k;
      vals_out[out] = s_vals[i];
    } else {
      raise_error(err, ERR_INTERNAL);
    }
  }
}

}  // namespace

int sort_tiles(int64_t N) { return (int)((N + SORT_TILE - 1) / SORT_TILE); }

void launch_weights(const StepArgs& a, StepScratch sc, DevStats* stats, int n_hist_words,
                    cudaStream_t s) {
  k_message_weights<<<1, 256, 0, s>>>(a, sc, stats, n_hist_words);
}

void launch_sort_histogram(const StepArgs& a, int passes, StepScratch sc, uint32_t* keys0,
                           ErrSink err, int grid, cudaStream_t s) {
  k_sort_histogram<<<grid, SORT_THREADS, 0, s>>>(a, passes, sc, keys0, err);
}

void launch_onesweep(const StepArgs& a, bool first, int pass, const uint32_t* keys_in,
                     const uint32_t* vals_in, uint32_t* keys_out, uint32_t* vals_out,
                     StepScratch sc, unsigned long long* status, uint32_t epoch, ErrSink err,
                     int64_t wait_ns, cudaStream_t s) {
  const int tiles = sort_tiles(a.N);
  if (first)
    k_onesweep<true><<<tiles, SORT_THREADS, 0, s>>>(a, pass, keys_in, vals_in, keys_out,
                                                    vals_out, sc, status, epoch, err, wait_ns);
  else
    k_onesweep<false><<<tiles, SORT_THREADS, 0, s>>>(a, pass, keys_in, vals_in, keys_out,
                                                     vals_out, sc, status, epoch, err, wait_ns);
}

}  // namespace gba
