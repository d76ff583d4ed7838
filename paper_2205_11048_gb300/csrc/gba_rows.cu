// K3 + K4 of the GBA aggregate-and-apply step: per unique row of the sorted
// occurrence array, decay each occurrence by the row's step tag against its
// message's token (Eq. (1); Alg. 2, push responding), sum the kept gradient
// rows, divide by the number of messages whose ids include the row, apply the
// optimizer to the row and its state in place, and set the row's tag to k + 1.
//
// Three kernels per table:
//
//  k_seg_scan   Tiles of 2048 sorted positions.  Every position's message,
//               tag, staleness and weight are decided here (the tag is read
//               before any row of the step is updated), then one block-wide
//               scan of four counters -- row heads, kept occurrences,
//               (message, row) pairs and kept pairs -- continued across tiles
//               by a decoupled look-back over epoch-tagged words.  Each row
//               head writes its record (row, prefixes); each kept occurrence
//               writes the address of its gradient row (and its weight) into
//               a list sorted by row.  Rows that cross tiles need no special
//               care: a row's counts are differences of prefixes.
//  k_row_apply_staged  Rows with at most LONG_ROW kept occurrences (widths a
//               multiple of 4): one lane group per row, grid-stride over the
//               rows; the row's records, kept-list entries, weights, state and
//               gradient rows are copied into shared memory by a three-level
//               cp.async pipeline several rows ahead, then the kept gradients
//               are summed in sorted order with compensated (TwoSum)
//               arithmetic, divided by the denominator and applied.
//  k_row_apply  The same with register-held rows, for other widths.
//  k_row_long   Rows with more kept occurrences, in chunks of LONG_CHUNK of
//               them, one warp per chunk claimed in list order: the warp's
//               lane groups sum contiguous parts that are merged in order,
//               and a row split into several chunks is finished by the warp
//               that completes its last chunk, merging the chunk sums in
//               chunk order.
//
// Every summation order is fixed (sorted order, then fixed parts and chunks),
// so results are bit-identical run to run; no float atomics anywhere.
#include <algorithm>

#include "gba_internal.cuh"

namespace gba {

namespace {

constexpr uint32_t FULL = 0xffffffffu;
constexpr uint32_t NO_KEY = 0xFFFFFFFFu;
constexpr int MSG_CACHE = 256;  // messages whose lookups are cached in shared memory
constexpr int SCAN_THREADS = 256;
constexpr int SCAN_ITEMS = SCAN_TILE / SCAN_THREADS;
constexpr int SCAN_WARPS = SCAN_THREADS / 32;
static_assert(SCAN_TILE % SCAN_THREADS == 0, "scan tile must fill the block");
constexpr int ROW_THREADS = 256;
#define SCAN_PAD(i) ((i) + ((i) >> 3))
// shared staging of one scan tile's outputs: row records and kept-list entries
constexpr size_t SCAN_OUT_BYTES = (size_t)SCAN_TILE * (sizeof(uint4) + sizeof(void*) + sizeof(float));

// look-back word: [63:32] epoch of the launch, [31:30] flag, [29:0] count
constexpr unsigned long long ST_AGG = 1ull << 30;
constexpr unsigned long long ST_INCL = 2ull << 30;
constexpr unsigned long long ST_FLAGS = 3ull << 30;
constexpr unsigned long long ST_COUNT = (1ull << 30) - 1;

__device__ __forceinline__ uint32_t ld_volatile_u32(const uint32_t* p) {
  return *(const volatile uint32_t*)p;
}
__device__ __forceinline__ unsigned long long ld_relaxed_u64(const unsigned long long* p) {
  unsigned long long v;
  asm volatile("ld.relaxed.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ void st_relaxed_u64(unsigned long long* p, unsigned long long v) {
  asm volatile("st.relaxed.gpu.global.u64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}

// The message of table-local occurrence x in the offsets off[0..M]: the
// largest m with off[m] <= x (empty messages repeat an offset).
__device__ __forceinline__ int message_of_any(const uint32_t* off, int M, uint32_t x) {
  int lo = 0, hi = M;
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (off[mid] <= x)
      lo = mid;
    else
      hi = mid;
  }
  return lo;
}

// The same, starting from the message an even split would give (exact when
// every message holds the same number of ids, as with one-hot fields; scale
// is M over the table's occurrences) and falling back to the binary search
// when that guess is more than two messages off.
__device__ __forceinline__ int message_of(const uint32_t* off, int M, uint32_t x, float scale) {
  int m = (int)((float)x * scale);
  m = m < 0 ? 0 : (m < M - 1 ? m : M - 1);
#pragma unroll
  for (int s = 0; s < 2; ++s) {
    if (m > 0 && off[m] > x)
      --m;
    else if (m + 1 < M && off[m + 1] <= x)
      ++m;
  }
  if (off[m] <= x && (m + 1 >= M || off[m + 1] > x)) return m;
  return message_of_any(off, M, x);
}

// Denominator of a row's weighted sum (Alg. 2: messages whose ids include the
// row; or the messages whose occurrence was kept; or all M messages).
__device__ __forceinline__ float row_denominator(int mode, uint32_t c_all, uint32_t c_kept, int M) {
  const uint32_t den = mode == 0 ? c_all : (mode == 1 ? c_kept : (uint32_t)M);
  return (float)den;
}

// ---------------------------------------------------------------------------
// k_seg_scan
// ---------------------------------------------------------------------------
#ifndef GBA_LOOKBACK_SLEEP_NS
#define GBA_LOOKBACK_SLEEP_NS 64
#endif
#ifndef GBA_SCAN_MINB
#define GBA_SCAN_MINB 2
#endif
__global__ void __launch_bounds__(SCAN_THREADS, GBA_SCAN_MINB)
    k_seg_scan(StepArgs a, SegTable tb, SegOut so, const uint32_t* __restrict__ keys,
               const uint32_t* __restrict__ vals, DevStats* st, ErrSink err, int64_t wait_ns) {
  __shared__ uint32_t s_off[MSG_CACHE + 1];
  __shared__ int64_t s_tok[MSG_CACHE];
  __shared__ const float* s_rowp[MSG_CACHE];
  // keys and occurrences of the tile at padded slots (one spare word after
  // every 8, so the threads' runs of 8 fall in distinct banks); slot 0 holds
  // the position before the tile
  __shared__ uint32_t s_k[SCAN_PAD(SCAN_TILE) + 1];
  __shared__ uint32_t s_v[SCAN_PAD(SCAN_TILE) + 1];
  extern __shared__ __align__(16) unsigned char s_out[];  // the tile's records and list entries
  __shared__ uint32_t s_wsum[4][SCAN_WARPS];
  __shared__ uint32_t s_base[4];
  __shared__ uint32_t s_tile;

  // block-uniform: another kernel may set the word while this block reads it
  if (__syncthreads_or((ld_volatile_u32(err.step) & (ERR_ID_RANGE | ERR_TIMEOUT)) != 0u)) return;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int M = a.M;
  const uint32_t* off_g = a.msg_off + (size_t)tb.t * (M + 1);
  const float* const* rows_g = a.rows_ptr + (size_t)tb.t * M;
  const bool cached = M <= MSG_CACHE;
  if (cached) {
    for (int i = tid; i <= M; i += SCAN_THREADS) s_off[i] = off_g[i];
    for (int i = tid; i < M; i += SCAN_THREADS) {
      s_tok[i] = a.tokens[i];
      s_rowp[i] = rows_g[i];
    }
  }
  if (tid == 0) s_tile = atomicAdd(so.ticket, 1u);
  __syncthreads();
  const uint32_t* off = cached ? s_off : off_g;
  const uint32_t tile = s_tile;
  const int64_t Nt = tb.pos_end - tb.pos_begin;
  const int64_t n_tiles = (Nt + SCAN_TILE - 1) / SCAN_TILE;
  const int64_t p0 = tb.pos_begin + (int64_t)tile * SCAN_TILE;
  const int n_valid = (int)(tb.pos_end - p0 < SCAN_TILE ? tb.pos_end - p0 : SCAN_TILE);
  for (int i = tid; i < n_valid; i += SCAN_THREADS) {  // coalesced
    s_k[SCAN_PAD(i + 1)] = keys[p0 + i];
    s_v[SCAN_PAD(i + 1)] = vals[p0 + i];
  }
  if (tid == 0) {
    s_k[0] = p0 > tb.pos_begin ? keys[p0 - 1] : NO_KEY;
    s_v[0] = p0 > tb.pos_begin ? vals[p0 - 1] : 0u;
  }
  __syncthreads();

  const int64_t nbase = a.nbase[tb.t];
  const uint32_t n_t = (uint32_t)Nt;
  const uint32_t v_t = (uint32_t)tb.rows;
  const int hop_limit = M - a.drop_latest;  // messages at or past this index are dropped
  const float mscale = (float)M / (float)(n_t > 0u ? n_t : 1u);

  // ---- pass 1: decide every position of this thread's 8 (blocked layout)
  const int i0 = tid * SCAN_ITEMS;
  uint32_t x_[SCAN_ITEMS];
  const float* p_[SCAN_ITEMS];
  float f_[SCAN_ITEMS];
  uint32_t flags = 0u;  // bit 4j: head, 4j+1: keep, 4j+2: new (message, row) pair
  uint32_t cnt[4] = {0u, 0u, 0u, 0u};
  uint32_t n_drop_pairs = 0u;
  unsigned long long stale_sum = 0ull, stale_max = 0ull;
  int m_prev = -1;
  if (i0 < n_valid && s_k[SCAN_PAD(i0)] != NO_KEY) {  // message of the position before
    const uint32_t o_t = (uint32_t)((int64_t)s_v[SCAN_PAD(i0)] - nbase);
    if (o_t < n_t) m_prev = message_of(off, M, o_t, mscale);
  }
  // the rows' step tags first, all eight loads in flight together (positions
  // of one row read the same tag, so only a row's first read reaches DRAM)
  int32_t tg_[SCAN_ITEMS];
#pragma unroll
  for (int j = 0; j < SCAN_ITEMS; ++j) {
    const int i = i0 + j;
    x_[j] = i < n_valid ? s_k[SCAN_PAD(i + 1)] - tb.key_base : 0u;
    tg_[j] = 0;
    if (a.row_staleness == 0 && i < n_valid && x_[j] < v_t) tg_[j] = __ldg(tb.ver + x_[j]);
  }
#pragma unroll
  for (int j = 0; j < SCAN_ITEMS; ++j) {
    const int i = i0 + j;
    p_[j] = nullptr;
    f_[j] = 0.f;
    if (i < n_valid) {
      const uint32_t key = s_k[SCAN_PAD(i + 1)];
      const bool head = key != s_k[SCAN_PAD(i)];
      const uint32_t o_t = (uint32_t)((int64_t)s_v[SCAN_PAD(i + 1)] - nbase);
      const uint32_t x = x_[j];
      if (o_t >= n_t || x >= v_t) {
        raise_error(err, ERR_INTERNAL);  // cannot happen for a correctly sorted array
        continue;
      }
      const int m = message_of(off, M, o_t, mscale);
      const int64_t tok = cached ? s_tok[m] : a.tokens[m];
      const int64_t ref = a.row_staleness == 0 ? (int64_t)tg_[j] : a.k;
      const int64_t diff = ref - tok;
      const uint64_t sl = diff > 0 ? (uint64_t)diff : 0ull;
      const float f = m < hop_limit ? decay_weight(a, sl) : 0.f;
      const bool keep = f > 0.f;
      const bool newp = head || m != m_prev;
      m_prev = m;
      f_[j] = f;
      if (keep)
        p_[j] = (cached ? s_rowp[m] : rows_g[m]) + (size_t)(o_t - off[m]) * (size_t)tb.d;
      flags |= ((head ? 1u : 0u) | (keep ? 2u : 0u) | (newp ? 4u : 0u)) << (4 * j);
      cnt[0] += head;
      cnt[1] += keep;
      cnt[2] += newp;
      cnt[3] += newp && keep;
      if (newp) {
        if (!keep) ++n_drop_pairs;
        const uint32_t s32 = (uint32_t)(sl > 0xFFFFFFFFull ? 0xFFFFFFFFull : sl);
        stale_sum += s32;
        stale_max = s32 > stale_max ? s32 : stale_max;
      }
    }
  }

  // ---- block-wide exclusive scan of the four counters
  uint32_t excl[4];
#pragma unroll
  for (int c = 0; c < 4; ++c) {
    uint32_t v = cnt[c];
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t y = __shfl_up_sync(FULL, v, o);
      if (lane >= o) v += y;
    }
    excl[c] = v - cnt[c];
    if (lane == 31) s_wsum[c][warp] = v;
  }
  __syncthreads();
  uint32_t tile_tot[4];
#pragma unroll
  for (int c = 0; c < 4; ++c) {
    uint32_t before = 0u, tot = 0u;
#pragma unroll
    for (int w = 0; w < SCAN_WARPS; ++w) {
      const uint32_t y = s_wsum[c][w];
      if (w < warp) before += y;
      tot += y;
    }
    excl[c] += before;
    tile_tot[c] = tot;
  }

  // ---- the tile's prefixes: the whole block looks back over earlier tiles,
  // SCAN_THREADS of them at a time (thread i reads tile j - i)
  {
    unsigned long long* my = so.status + (size_t)tile * 4;
    const unsigned long long ep = (unsigned long long)so.epoch << 32;
    if (tid == 0)
      for (int c = 0; c < 4; ++c)
        st_relaxed_u64(my + c, ep | (tile == 0 ? ST_INCL : ST_AGG) | (unsigned long long)tile_tot[c]);
    __shared__ uint32_t s_first_nr[SCAN_WARPS], s_first_in[SCAN_WARPS];
    __shared__ uint32_t s_part[4][SCAN_WARPS];
    __shared__ int s_done;
    uint32_t pre[4] = {0u, 0u, 0u, 0u};
    if (tile > 0) {
      int64_t j = (int64_t)tile - 1;
      const uint64_t t0 = globaltimer_ns();
      for (;;) {
        const int64_t q = j - tid;
        unsigned long long v[4];
#pragma unroll
        for (int c = 0; c < 4; ++c)
          v[c] = q >= 0 ? ld_relaxed_u64(so.status + (size_t)q * 4 + c) : (ep | ST_INCL);
        // a tile is usable once its four words carry this launch's epoch and
        // the same flag (the writer replaces all four, so a mix is transient)
        bool ready = true, incl = true;
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          ready = ready && (v[c] & ~0xFFFFFFFFull) == ep && (v[c] & ST_FLAGS) != 0ull &&
                  (v[c] & ST_FLAGS) == (v[0] & ST_FLAGS);
          incl = incl && (v[c] & ST_INCL) != 0ull;
        }
        incl = incl && ready;
        const uint32_t rm = __ballot_sync(FULL, ready), im = __ballot_sync(FULL, incl);
        if (lane == 0) {
          s_first_nr[warp] = ~rm ? (uint32_t)(warp * 32 + __ffs(~rm) - 1) : 0xFFFFFFFFu;
          s_first_in[warp] = im ? (uint32_t)(warp * 32 + __ffs(im) - 1) : 0xFFFFFFFFu;
        }
        __syncthreads();
        uint32_t first_nr = 0xFFFFFFFFu, first_in = 0xFFFFFFFFu;
#pragma unroll
        for (int w = 0; w < SCAN_WARPS; ++w) {
          first_nr = min(first_nr, s_first_nr[w]);
          first_in = min(first_in, s_first_in[w]);
        }
        first_nr = min(first_nr, (uint32_t)SCAN_THREADS);
        const uint32_t take = first_in < first_nr ? first_in + 1 : first_nr;
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          uint32_t cc = (uint32_t)tid < take ? (uint32_t)(v[c] & ST_COUNT) : 0u;
#pragma unroll
          for (int o = 16; o > 0; o >>= 1) cc += __shfl_xor_sync(FULL, cc, o);
          if (lane == 0) s_part[c][warp] = cc;
        }
        if (tid == 0) {
          s_done = first_in < first_nr ? 1 : 0;
          if (take == 0u && ((ld_volatile_u32(err.step) & ERR_TIMEOUT) ||
                             (int64_t)(globaltimer_ns() - t0) > wait_ns)) {
            raise_error(err, ERR_TIMEOUT);
            s_done = 1;
          }
        }
        __syncthreads();
#pragma unroll
        for (int c = 0; c < 4; ++c)
#pragma unroll
          for (int w = 0; w < SCAN_WARPS; ++w) pre[c] += s_part[c][w];
        const bool done = s_done != 0;
        __syncthreads();  // the shared words are rewritten by the next round
        if (done) break;
        if (take == 0u && GBA_LOOKBACK_SLEEP_NS > 0) __nanosleep(GBA_LOOKBACK_SLEEP_NS);  // back off while predecessors work
        j -= take;
      }
      if (tid == 0)
        for (int c = 0; c < 4; ++c)
          st_relaxed_u64(my + c, ep | ST_INCL | (unsigned long long)((pre[c] + tile_tot[c]) & ST_COUNT));
    }
    if (tid == 0) {
      for (int c = 0; c < 4; ++c) s_base[c] = pre[c];
      if ((int64_t)tile == n_tiles - 1) {  // the totals close the record array
        so.rr[pre[0] + tile_tot[0]] =
            make_uint4(0u, pre[1] + tile_tot[1], pre[2] + tile_tot[2], pre[3] + tile_tot[3]);
        *so.total = pre[0] + tile_tot[0];
      }
    }
  }
  __syncthreads();

  // ---- pass 2: row records and the kept list, staged in shared memory in
  // order, then written out in contiguous runs
  uint4* o_rr = reinterpret_cast<uint4*>(s_out);
  const float** o_kl = reinterpret_cast<const float**>(s_out + (size_t)SCAN_TILE * sizeof(uint4));
  float* o_kw = reinterpret_cast<float*>(s_out + (size_t)SCAN_TILE * (sizeof(uint4) + sizeof(void*)));
  uint32_t run[4];
#pragma unroll
  for (int c = 0; c < 4; ++c) run[c] = s_base[c] + excl[c];
  uint32_t lh = excl[0], lk = excl[1];  // indices within the tile
#pragma unroll
  for (int j = 0; j < SCAN_ITEMS; ++j) {
    const uint32_t fl = (flags >> (4 * j)) & 7u;
    if (fl & 1u) o_rr[lh] = make_uint4(x_[j], run[1], run[2], run[3]);
    if (fl & 2u) {
      o_kl[lk] = p_[j];
      o_kw[lk] = f_[j];
    }
    lh += fl & 1u;
    lk += (fl >> 1) & 1u;
    run[0] += fl & 1u;
    run[1] += (fl >> 1) & 1u;
    run[2] += (fl >> 2) & 1u;
    run[3] += ((fl >> 2) & (fl >> 1)) & 1u;
  }
  __syncthreads();
  {
    const uint32_t h0 = s_base[0], k0 = s_base[1];
    for (uint32_t i = tid; i < tile_tot[0]; i += SCAN_THREADS) so.rr[h0 + i] = o_rr[i];
    for (uint32_t i = tid; i < tile_tot[1]; i += SCAN_THREADS) {
      so.kl[k0 + i] = o_kl[i];
      so.kw[k0 + i] = o_kw[i];
    }
  }

  // ---- counters of Table 3's kind (pairs, dropped pairs, row staleness)
  uint32_t n_pairs = cnt[2], n_kept_occ = cnt[1], n_heads = cnt[0];
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    n_pairs += __shfl_xor_sync(FULL, n_pairs, o);
    n_drop_pairs += __shfl_xor_sync(FULL, n_drop_pairs, o);
    n_kept_occ += __shfl_xor_sync(FULL, n_kept_occ, o);
    n_heads += __shfl_xor_sync(FULL, n_heads, o);
    stale_sum += __shfl_xor_sync(FULL, stale_sum, o);
    const unsigned long long y = __shfl_xor_sync(FULL, stale_max, o);
    stale_max = y > stale_max ? y : stale_max;
  }
  if (lane == 0) {
    if (n_pairs) atomicAdd(&st->pairs, (unsigned long long)n_pairs);
    if (n_drop_pairs) atomicAdd(&st->pairs_dropped, (unsigned long long)n_drop_pairs);
    if (stale_sum) atomicAdd(&st->row_stale_sum, stale_sum);
    if (stale_max) atomicMax(&st->row_stale_max, stale_max);
    if (n_kept_occ) atomicAdd(&st->occ_kept, (unsigned long long)n_kept_occ);
    if (n_heads) atomicAdd(&st->rows_touched, (unsigned long long)n_heads);
  }
}

// ---------------------------------------------------------------------------
// shared pieces of the two row kernels
// ---------------------------------------------------------------------------
// A lane's part of one row: CPL pieces of CH floats; piece q of the row is
// held by lane q mod L as its piece number q / L.
template <int CH, int CPL>
struct Part {
  float v[CH * CPL];
};

template <int CH, int CPL>
__device__ __forceinline__ void load_part(const float* row, int l, int L, int C, Part<CH, CPL>& p) {
#pragma unroll
  for (int c = 0; c < CPL; ++c) {
    const int q = l + c * L;
    if (q < C) {
      if constexpr (CH == 4) {
        const float4 t = *reinterpret_cast<const float4*>(row + 4 * q);
        p.v[4 * c] = t.x;
        p.v[4 * c + 1] = t.y;
        p.v[4 * c + 2] = t.z;
        p.v[4 * c + 3] = t.w;
      } else {
        p.v[c] = row[q];
      }
    }
  }
}

template <int CH, int CPL>
__device__ __forceinline__ void store_part(float* row, int l, int L, int C, const Part<CH, CPL>& p) {
#pragma unroll
  for (int c = 0; c < CPL; ++c) {
    const int q = l + c * L;
    if (q < C) {
      if constexpr (CH == 4) {
        *reinterpret_cast<float4*>(row + 4 * q) =
            make_float4(p.v[4 * c], p.v[4 * c + 1], p.v[4 * c + 2], p.v[4 * c + 3]);
      } else {
        row[q] = p.v[c];
      }
    }
  }
}

// The optimizer step of row x with its summed gradient (acc) and denominator.
template <int CH, int CPL>
__device__ __forceinline__ void finish_row(const SegTable& tb, uint32_t x, float den,
                                           const CSum (&acc)[CH * CPL], Part<CH, CPL>& w,
                                           Part<CH, CPL>& s0, Part<CH, CPL>& s1, int l, int L,
                                           int C, bool adam) {
  const size_t base = (size_t)x * (size_t)tb.d;
#pragma unroll
  for (int c = 0; c < CPL; ++c) {
    if (l + c * L >= C) continue;
#pragma unroll
    for (int k = 0; k < CH; ++k) {
      const int i = c * CH + k;
      const float v = csum_value(acc[i]);
      const float g = den == 1.f ? v : __fdiv_rn(v, den);  // x / 1 is exact
      float b = adam ? s1.v[i] : 0.f;
      opt_update(tb.opt, w.v[i], s0.v[i], b, g);
      s1.v[i] = b;
    }
  }
  store_part<CH, CPL>(tb.w + base, l, L, C, w);
  store_part<CH, CPL>(tb.s0 + base, l, L, C, s0);
  if (adam) store_part<CH, CPL>(tb.s1 + base, l, L, C, s1);
}

struct RowMeta {
  uint32_t x, ks, n;
  float den;
};

__device__ __forceinline__ RowMeta row_meta(const SegOut& so, uint32_t u, uint32_t U, int mode,
                                            int M) {
  RowMeta r{0u, 0u, 0u, 0.f};
  if (u < U) {
    const uint4 a = so.rr[u];
    const uint4 b = so.rr[u + 1];
    r.x = a.x;
    r.ks = a.y;
    r.n = b.y - a.y;
    r.den = row_denominator(mode, b.z - a.z, b.w - a.w, M);
  }
  return r;
}

// ---------------------------------------------------------------------------
// k_row_classify: lists the rows with more than LONG_ROW kept occurrences for
// the long-row kernel.  With small_ok, rows of at most SMALL_MAX kept
// occurrences go to a list of their own (row, first kept entry, count,
// denominator), each applied there by one lane group; longer rows are listed
// with their chunks of LONG_CHUNK, each chunk summed by one warp.  Tiles of
// 2048 row records (8 per thread); a block reserves a tile's entries with one
// atomic per counter.  The order of the lists depends on the atomics, the
// results do not: every row's chunks are summed and merged in chunk order.
// ---------------------------------------------------------------------------
constexpr int CLS_THREADS = 256, CLS_ITEMS = 8;  // rows per tile: 2048

__global__ void __launch_bounds__(CLS_THREADS)
    k_row_classify(StepArgs a, SegOut so, ErrSink err, int small_ok) {
  __shared__ uint32_t s_w[4][CLS_THREADS / 32];
  __shared__ uint32_t s_b[4];
  if (__syncthreads_or(ld_volatile_u32(err.step) != 0u)) return;
  const uint32_t U = ld_volatile_u32(so.total);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const uint32_t small_max = small_ok ? (uint32_t)SMALL_MAX : (uint32_t)LONG_ROW;
  const uint32_t tile_rows = CLS_THREADS * CLS_ITEMS;
  for (uint32_t t0 = blockIdx.x * tile_rows; t0 < U; t0 += gridDim.x * tile_rows) {
    // this thread's rows t0 + tid*8 .. +7: kind and sizes
    const uint32_t u0 = t0 + (uint32_t)tid * CLS_ITEMS;
    uint32_t n_[CLS_ITEMS];
    uint32_t cnt[4] = {0u, 0u, 0u, 0u};  // small rows, long rows, chunks, chunk-sum slots
    uint4 prev = u0 < U ? so.rr[u0] : make_uint4(0u, 0u, 0u, 0u);
#pragma unroll
    for (int k = 0; k < CLS_ITEMS; ++k) {
      const uint32_t u = u0 + k;
      n_[k] = 0u;
      if (u < U) {
        const uint4 nx = so.rr[u + 1];
        n_[k] = nx.y - prev.y;
        prev = nx;
      }
      const uint32_t n = n_[k];
      if (n > (uint32_t)LONG_ROW && n <= small_max) {
        ++cnt[0];
      } else if (n > small_max) {
        const uint32_t nch = (n + LONG_CHUNK - 1) / LONG_CHUNK;
        ++cnt[1];
        cnt[2] += nch;
        cnt[3] += nch > 1u ? nch : 0u;
      }
    }
    // block-wide exclusive scans of the four counters; one atomic per counter
    uint32_t excl[4];
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      uint32_t v = cnt[c];
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const uint32_t y = __shfl_up_sync(FULL, v, o);
        if (lane >= o) v += y;
      }
      excl[c] = v - cnt[c];
      if (lane == 31) s_w[c][warp] = v;
    }
    __syncthreads();
    if (tid < 4) {
      uint32_t tot = 0u;
      for (int w = 0; w < CLS_THREADS / 32; ++w) tot += s_w[tid][w];
      uint32_t* ctr = tid == 0 ? so.n_small : (tid == 1 ? so.n_long : (tid == 2 ? so.n_items : so.n_parts));
      s_b[tid] = tot ? atomicAdd(ctr, tot) : 0u;
    }
    __syncthreads();
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      uint32_t before = 0u;
      for (int w = 0; w < warp; ++w) before += s_w[c][w];
      excl[c] += before + s_b[c];
    }
    if (cnt[0] | cnt[1]) {
      prev = so.rr[u0];
#pragma unroll
      for (int k = 0; k < CLS_ITEMS; ++k) {
        const uint32_t u = u0 + k;
        const uint32_t n = n_[k];
        if (u >= U) break;
        const uint4 nx = so.rr[u + 1];
        if (n > (uint32_t)LONG_ROW && n <= small_max) {
          so.small_rows[excl[0]++] = make_uint4(
              prev.x, prev.y, n,
              __float_as_uint(row_denominator(a.sparse_den, nx.z - prev.z, nx.w - prev.w, a.M)));
        } else if (n > small_max) {
          const uint32_t nch = (n + LONG_CHUNK - 1) / LONG_CHUNK;
          const uint32_t li = excl[1]++;
          so.long_rows[li] = make_uint4(u, prev.y, n, nch > 1u ? excl[3] : 0u);
          so.long_done[li] = 0u;
          for (uint32_t c = 0; c < nch; ++c) so.items[excl[2] + c] = make_uint2(li, c);
          excl[2] += nch;
          excl[3] += nch > 1u ? nch : 0u;
        }
        prev = nx;
      }
    }
    __syncthreads();  // s_w and s_b are rewritten by the next tile
  }
}

// ---------------------------------------------------------------------------
// k_row_apply: one lane group per row
// ---------------------------------------------------------------------------
template <int CH, int CPL>
__global__ void __launch_bounds__(ROW_THREADS, (CH * CPL <= 4) ? 3 : 2)
    k_row_apply(StepArgs a, SegTable tb, SegOut so, DevStats* st, ErrSink err) {
  // a failed step changes no row (warp-uniform: the warp reduces at the end)
  if (__any_sync(FULL, ld_volatile_u32(err.step) != 0u)) return;
  constexpr int P = CH * CPL;
  const uint32_t U = ld_volatile_u32(so.total);
  const int d = tb.d;
  const int C = CH == 4 ? d / 4 : d;  // pieces per row
  int L = 1;
  while (L < C && L < 32) L <<= 1;
  const int lg = __ffs(L) - 1;
  const int G = 32 >> lg;  // rows per warp
  const int lane = threadIdx.x & 31;
  const int g = lane >> lg, l = lane & (L - 1);
  const int64_t gw = (int64_t)blockIdx.x * (ROW_THREADS / 32) + (threadIdx.x >> 5);
  const int64_t TG = (int64_t)gridDim.x * (ROW_THREADS / 32) * G;
  const bool adam = tb.opt.kind == 1;
  const bool unit = a.decay == 0;  // every kept weight is 1
  const int mode = a.sparse_den;
  const int32_t tag = (int32_t)(a.k + 1);
  uint32_t applied = 0u;

  int64_t u = gw * G + g;
  auto clamp_u = [&](int64_t v) { return (uint32_t)(v < (int64_t)U ? v : (int64_t)U); };
  RowMeta cur = row_meta(so, clamp_u(u), U, mode, a.M);
  RowMeta nxt = row_meta(so, clamp_u(u + TG), U, mode, a.M);
  // lane l of the group holds the l-th kept entry of the current row
  const float* kp_cur = nullptr;
  float kw_cur = 0.f;
  if (cur.n <= LONG_ROW && (uint32_t)l < cur.n) {
    kp_cur = so.kl[cur.ks + l];
    kw_cur = so.kw[cur.ks + l];
  }
  // warp-uniform loop: the warp's first row bounds the rows of all its groups
  for (int64_t uw = gw * G; uw < (int64_t)U; uw += TG, u += TG) {
    // ---- one row ahead: the next row's list entries; two ahead: its record
    const RowMeta n2 = row_meta(so, clamp_u(u + 2 * TG), U, mode, a.M);
    const float* kp_nxt = nullptr;
    float kw_nxt = 0.f;
    if (nxt.n <= LONG_ROW && (uint32_t)l < nxt.n) {
      kp_nxt = so.kl[nxt.ks + l];
      kw_nxt = so.kw[nxt.ks + l];
    }
    // ---- this row: state and gradients, then the sums in sorted order
    const bool active = u < (int64_t)U && cur.n > 0u && cur.n <= (uint32_t)LONG_ROW;
    Part<CH, CPL> w, s0, s1;
    if (active) {
      const size_t base = (size_t)cur.x * (size_t)d;
      load_part<CH, CPL>(tb.w + base, l, L, C, w);
      load_part<CH, CPL>(tb.s0 + base, l, L, C, s0);
      if (adam) load_part<CH, CPL>(tb.s1 + base, l, L, C, s1);
    }
    CSum acc[P];
#pragma unroll
    for (int i = 0; i < P; ++i) acc[i] = CSum{0.f, 0.f};
    const uint32_t n_here = active ? cur.n : 0u;
    uint32_t n_max = n_here;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) n_max = max(n_max, __shfl_xor_sync(FULL, n_max, o));
    for (uint32_t j0 = 0; j0 < n_max; j0 += 4) {
      Part<CH, CPL> gr[4];
      float fw[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const uint32_t j = j0 + e;
        const int src = (int)(j & (uint32_t)(L - 1));
        const float* p = (const float*)__shfl_sync(FULL, (unsigned long long)kp_cur, src, L);
        float f = __shfl_sync(FULL, kw_cur, src, L);
        if (j >= (uint32_t)L && j < n_here) {  // beyond the entries held by the lanes
          p = so.kl[cur.ks + j];
          f = so.kw[cur.ks + j];
        }
        fw[e] = f;
        if (j < n_here) load_part<CH, CPL>(p, l, L, C, gr[e]);
      }
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        if (j0 + e < n_here) {
#pragma unroll
          for (int c = 0; c < CPL; ++c) {
            if (l + c * L >= C) continue;
#pragma unroll
            for (int k = 0; k < CH; ++k) csum_add_w(acc[c * CH + k], unit, fw[e], gr[e].v[c * CH + k]);
          }
        }
      }
    }
    if (active) {
      finish_row<CH, CPL>(tb, cur.x, cur.den, acc, w, s0, s1, l, L, C, adam);
      if (l == 0) {
        tb.ver[cur.x] = tag;
        ++applied;
      }
    }
    cur = nxt;
    nxt = n2;
    kp_cur = kp_nxt;
    kw_cur = kw_nxt;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) applied += __shfl_xor_sync(FULL, applied, o);
  if (lane == 0 && applied) atomicAdd(&st->rows_applied, (unsigned long long)applied);
}

// ---------------------------------------------------------------------------
// k_row_apply_staged: the same per-row work for widths that are a multiple of
// 4, with every row's weights, state and (at most LONG_ROW) kept gradient rows
// copied into a per-lane-group ring of STAGE_P shared-memory slots by
// cp.async 16-byte copies, STAGE_P rows ahead of the row being applied; the
// list entries and records feeding those copies are loaded one and two rows
// further ahead.  Registers hold one row at a time, so many rows are in
// flight per SM.
// ---------------------------------------------------------------------------
#ifndef GBA_STAGE_P
#define GBA_STAGE_P 2
#endif
#ifndef GBA_STAGE_CPL
#define GBA_STAGE_CPL 1  // 16-byte pieces per lane for rows of up to 128 floats
#endif
constexpr int STAGE_P = GBA_STAGE_P;  // rows in flight per lane group
constexpr int STAGE_NG = LONG_ROW;  // every kept gradient row of a row applied here is staged
constexpr int STAGE_META = 8;       // floats of row metadata at the head of a data slot
constexpr int STAGE_THREADS = 128;
// per lane group: records of 3P rows ahead (2 x 16 B each), list entries of
// 2P rows ahead (4 addresses + 4 weights + the decoded record = 64 B each), P
// data slots
constexpr int STAGE_REC_FLOATS = 3 * STAGE_P * 8;
constexpr int STAGE_KL_FLOATS = 2 * STAGE_P * 16;

__device__ __forceinline__ void cp_async16(void* dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_addr(dst)), "l"(src)
               : "memory");
}
__device__ __forceinline__ void cp_async8(void* dst, const void* src) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 8;" ::"r"(smem_addr(dst)), "l"(src)
               : "memory");
}
__device__ __forceinline__ void cp_async4(void* dst, const void* src) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(smem_addr(dst)), "l"(src)
               : "memory");
}

__host__ __device__ constexpr int stage_floats_per_warp(int CPL, int regions, int G) {
  return G * (STAGE_REC_FLOATS + STAGE_KL_FLOATS) + STAGE_P * (G * STAGE_META + regions * 128 * CPL);
}

// k_row_apply_staged: rows with at most LONG_ROW kept occurrences and a width
// that is a multiple of 4.  Each lane group walks its rows (u, u + TG, ...)
// through a three-level pipeline of cp.async copies into shared memory, one
// commit group per row: the row's two records 3P rows ahead, its kept-list
// entries 2P rows ahead (they need the records), its weights, state and
// gradient rows P rows ahead (they need the entries); the row itself is then
// summed in sorted order and applied from shared memory.
#ifndef GBA_STAGE_MINB
#define GBA_STAGE_MINB 6
#endif
template <int CPL>
__global__ void __launch_bounds__(STAGE_THREADS, CPL == 1 ? GBA_STAGE_MINB : (CPL == 2 ? 4 : 2))
    k_row_apply_staged(StepArgs a, SegTable tb, SegOut so, DevStats* st, ErrSink err) {
  extern __shared__ __align__(16) float s_stage[];
  if (__any_sync(FULL, ld_volatile_u32(err.step) != 0u)) return;
  const uint32_t U = ld_volatile_u32(so.total);
  const int d = tb.d;
  const int C = d >> 2;  // 16-byte pieces per row
  int L = 1;
  while (L * CPL < C && L < 32) L <<= 1;  // lanes per row: CPL pieces each
  const int lg = __ffs(L) - 1;
  const int G = 32 >> lg;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int g = lane >> lg, l = lane & (L - 1);
  // row indices fit 32 bits (at most 2^30 occurrences per step)
  const uint32_t gw = blockIdx.x * (uint32_t)(STAGE_THREADS / 32) + (uint32_t)warp;
  const uint32_t TG = gridDim.x * (uint32_t)(STAGE_THREADS / 32) * (uint32_t)G;
  const bool adam = tb.opt.kind == 1;
  const bool unit = a.decay == 0;  // every kept weight is 1
  const int NS = adam ? 3 : 2;
  const int RS = L * CPL * 4;  // floats per region of a data slot
  const int SL = STAGE_META + (NS + STAGE_NG) * RS;
  float* wbase = s_stage + (size_t)warp * stage_floats_per_warp(CPL, NS + STAGE_NG, G);
  float* recs = wbase + (size_t)g * STAGE_REC_FLOATS;                       // [3P][8]
  float* kls = wbase + (size_t)G * STAGE_REC_FLOATS + (size_t)g * STAGE_KL_FLOATS;  // [2P][16]
  float* data = wbase + (size_t)G * (STAGE_REC_FLOATS + STAGE_KL_FLOATS) + (size_t)g * STAGE_P * SL;
  const int mode = a.sparse_den;
  const int32_t tag = (int32_t)(a.k + 1);
  float* const state[3] = {tb.w, tb.s0, tb.s1};
  uint32_t applied = 0u;
  const uint32_t u0 = gw * (uint32_t)G + (uint32_t)g;

  // level A: the records of row i (two 16-byte words), or an empty record
  auto level_a = [&](uint32_t i) {
    const uint32_t u = u0 + i * TG;
    uint4* r = reinterpret_cast<uint4*>(recs + (size_t)(i % (3 * STAGE_P)) * 8);
    if (u < U) {
      for (int e = l; e < 2; e += L) cp_async16(r + e, so.rr + u + e);  // L may be 1
    } else if (l == 0) {
      r[0] = make_uint4(0u, 0u, 0u, 0u);
      r[1] = make_uint4(0u, 0u, 0u, 0u);
    }
  };
  auto decode = [&](uint32_t i) {
    const uint4* r = reinterpret_cast<const uint4*>(recs + (size_t)(i % (3 * STAGE_P)) * 8);
    const uint4 ra = r[0], rb = r[1];
    RowMeta m;
    m.x = ra.x;
    m.ks = ra.y;
    m.n = rb.y - ra.y;
    m.den = row_denominator(mode, rb.z - ra.z, rb.w - ra.w, a.M);
    return m;
  };
  // level B: the kept entries of row i (addresses and weights); the decoded
  // record is kept beside them for level C
  auto level_b = [&](uint32_t i) {
    const RowMeta m = decode(i);
    float* k = kls + (size_t)(i % (2 * STAGE_P)) * 16;
    if (l == 0)
      *reinterpret_cast<float4*>(k + 12) =
          make_float4(__uint_as_float(m.x), __uint_as_float(m.n), m.den, 0.f);
    if (m.n > 0u && m.n <= (uint32_t)LONG_ROW) {
      for (uint32_t e = (uint32_t)l; e < m.n; e += (uint32_t)L) {  // L may be below LONG_ROW
        cp_async8(k + 2 * e, so.kl + m.ks + e);
        cp_async4(k + 8 + e, so.kw + m.ks + e);
      }
    }
  };
  // level C: weights, state and gradient rows of row i into data slot i % P
  auto level_c = [&](uint32_t i) {
    const float* k = kls + (size_t)(i % (2 * STAGE_P)) * 16;
    const float4 km = *reinterpret_cast<const float4*>(k + 12);
    RowMeta m;
    m.x = __float_as_uint(km.x);
    m.n = __float_as_uint(km.y);
    m.den = km.z;
    float* sl = data + (size_t)(i % STAGE_P) * SL;
    const bool live = u0 + i * TG < U;
    const bool short_row = live && m.n > 0u && m.n <= (uint32_t)LONG_ROW;
    if (l == 0) {
      *reinterpret_cast<float4*>(sl) =
          make_float4(__uint_as_float(m.x), __uint_as_float(short_row ? m.n : 0u), m.den, 0.f);
      *reinterpret_cast<float4*>(sl + 4) = short_row ? *reinterpret_cast<const float4*>(k + 8)
                                                     : make_float4(0.f, 0.f, 0.f, 0.f);
    }
    if (short_row) {
      const size_t base = (size_t)m.x * (size_t)d;
      const float* const* gp = reinterpret_cast<const float* const*>(k);
#pragma unroll
      for (int c = 0; c < CPL; ++c) {
        const int q = l + c * L;
        if (q < C) {
          float* dq = sl + STAGE_META + 4 * q;
          cp_async16(dq, state[0] + base + 4 * q);
          cp_async16(dq + RS, state[1] + base + 4 * q);
          if (adam) cp_async16(dq + 2 * RS, state[2] + base + 4 * q);
#pragma unroll
          for (int e = 0; e < STAGE_NG; ++e)
            if ((uint32_t)e < m.n) cp_async16(dq + (NS + e) * RS, gp[e] + 4 * q);
        }
      }
    }
  };
  auto commit = []() { asm volatile("cp.async.commit_group;" ::: "memory"); };
  auto wait_all = []() { asm volatile("cp.async.wait_group 0;" ::: "memory"); };

  // ---- prologue: records of rows 0 .. 3P-1, entries of 0 .. 2P-1, data of 0 .. P-1
  for (int i = 0; i < 3 * STAGE_P; ++i) level_a(i);
  commit();
  wait_all();
  __syncwarp();
  for (int i = 0; i < 2 * STAGE_P; ++i) level_b(i);
  commit();
  wait_all();
  __syncwarp();
  for (int i = 0; i < STAGE_P; ++i) {
    level_c(i);
    commit();
  }

  // every group of the warp runs the same iterations (the loop holds __syncwarp)
  const uint32_t uw = gw * (uint32_t)G;
  for (uint32_t i = 0; uw + i * TG < U; ++i) {
    asm volatile("cp.async.wait_group %0;" ::"n"(STAGE_P - 1) : "memory");
    __syncwarp();
    // ---- apply row i from its data slot: its kept gradients summed in sorted order
    {
      const float* sl = data + (size_t)(i % STAGE_P) * SL;
      const float4 m0 = *reinterpret_cast<const float4*>(sl);
      const float4 fw = *reinterpret_cast<const float4*>(sl + 4);
      const uint32_t x = __float_as_uint(m0.x);
      const uint32_t n = __float_as_uint(m0.y);
      const float f[4] = {fw.x, fw.y, fw.z, fw.w};
      if (n > 0u) {
        Part<4, CPL> w, s0, s1;
        CSum acc[4 * CPL];
#pragma unroll
        for (int c = 0; c < CPL; ++c) {
          const int q = l + c * L;
          if (q >= C) continue;
          const float* dq = sl + STAGE_META + 4 * q;
          const float4 wv = *reinterpret_cast<const float4*>(dq);
          const float4 av = *reinterpret_cast<const float4*>(dq + RS);
          const float4 bv = adam ? *reinterpret_cast<const float4*>(dq + 2 * RS)
                                 : make_float4(0.f, 0.f, 0.f, 0.f);
          const float4 g0 = *reinterpret_cast<const float4*>(dq + NS * RS);
          const float wa[4] = {wv.x, wv.y, wv.z, wv.w}, aa[4] = {av.x, av.y, av.z, av.w},
                      ba[4] = {bv.x, bv.y, bv.z, bv.w}, ga[4] = {g0.x, g0.y, g0.z, g0.w};
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            w.v[4 * c + k] = wa[k];
            s0.v[4 * c + k] = aa[k];
            s1.v[4 * c + k] = ba[k];
            if (f[0] == 1.f) {
              acc[4 * c + k] = CSum{ga[k], 0.f};  // 0 + g is exact: the first term as it is
            } else {
              acc[4 * c + k] = CSum{0.f, 0.f};
              csum_add_prod(acc[4 * c + k], f[0], ga[k]);
            }
          }
#pragma unroll
          for (int e = 1; e < STAGE_NG; ++e) {
            if ((uint32_t)e < n) {
              const float4 gv = *reinterpret_cast<const float4*>(dq + (NS + e) * RS);
              const float gb[4] = {gv.x, gv.y, gv.z, gv.w};
#pragma unroll
              for (int k = 0; k < 4; ++k) csum_add_w(acc[4 * c + k], unit, f[e], gb[k]);
            }
          }
        }
        finish_row<4, CPL>(tb, x, m0.z, acc, w, s0, s1, l, L, C, adam);
        if (l == 0) {
          tb.ver[x] = tag;
          ++applied;
        }
      }
    }
    __syncwarp();  // every lane is done with the slots being refilled
    level_c(i + STAGE_P);
    level_b(i + 2 * STAGE_P);
    level_a(i + 3 * STAGE_P);
    commit();
  }
  wait_all();
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) applied += __shfl_xor_sync(FULL, applied, o);
  if (lane == 0 && applied) atomicAdd(&st->rows_applied, (unsigned long long)applied);
}

// ---------------------------------------------------------------------------
// k_row_long: rows with more than LONG_ROW kept occurrences, one warp per
// chunk of at most LONG_CHUNK of them; warps claim chunks in list order.
// ---------------------------------------------------------------------------
#ifndef GBA_LONG_UNROLL
#define GBA_LONG_UNROLL 4
#endif
constexpr int LONG_UNROLL = GBA_LONG_UNROLL;
#ifndef GBA_LONG_BPS
#define GBA_LONG_BPS 0  // blocks per SM of the long-row kernel (0: as many as fit)
#endif
#ifndef GBA_STAGE_BPS_CUT
#define GBA_STAGE_BPS_CUT 0  // staged blocks per SM left free for other kernels
#endif
constexpr int LONG_SLOTS = 4;  // list entries per lane: a group's part is at most 4 L entries
static_assert(LONG_CHUNK <= 32 * LONG_SLOTS, "a chunk's part must fit the lanes' slots");

template <int CH, int CPL>
__global__ void __launch_bounds__(ROW_THREADS)
    k_row_long(StepArgs a, SegTable tb, SegOut so, DevStats* st, ErrSink err) {
  constexpr int P = CH * CPL;
  if (__any_sync(FULL, ld_volatile_u32(err.step) != 0u)) return;
  const uint32_t n_items = ld_volatile_u32(so.n_items);
  const uint32_t U = ld_volatile_u32(so.total);
  const int d = tb.d;
  const int C = CH == 4 ? d / 4 : d;
  int L = 1;
  while (L < C && L < 32) L <<= 1;
  const int lg = __ffs(L) - 1;
  const int G = 32 >> lg;  // lane groups per warp
  const int lane = threadIdx.x & 31;
  const int g = lane >> lg, l = lane & (L - 1);
  const bool adam = tb.opt.kind == 1;
  const bool unit = a.decay == 0;  // every kept weight is 1
  uint32_t applied = 0u;

  // the warp's next item is claimed and its description loaded while the
  // current one is summed
  auto claim = [&]() {
    uint32_t t = 0u;
    if (lane == 0) t = atomicAdd(so.item_ticket, 1u);
    return __shfl_sync(FULL, t, 0);
  };
  uint32_t it = claim();
  uint2 item = it < n_items ? so.items[it] : make_uint2(0u, 0u);
  uint4 lr = it < n_items ? so.long_rows[item.x] : make_uint4(0u, 0u, 0u, 0u);
  while (it < n_items) {
    const uint32_t it_next = claim();
    const uint2 item_next = it_next < n_items ? so.items[it_next] : make_uint2(0u, 0u);
    const uint32_t nch = (lr.z + LONG_CHUNK - 1) / LONG_CHUNK;
    const uint32_t e0 = lr.y + item.y * LONG_CHUNK;
    const uint32_t e1 = min(e0 + (uint32_t)LONG_CHUNK, lr.y + lr.z);
    // group g sums a contiguous part of the chunk
    const uint32_t per = (e1 - e0 + G - 1) / G;
    const uint32_t b0 = min(e0 + g * per, e1), b1 = min(b0 + per, e1);
    CSum acc[P];
#pragma unroll
    for (int i = 0; i < P; ++i) acc[i] = CSum{0.f, 0.f};
    const uint32_t mine = b1 - b0;
    // the part's list entries first: lane l holds entries l, l + L, l + 2L, l + 3L
    const float* ptr[LONG_SLOTS];
    float wgt[LONG_SLOTS];
#pragma unroll
    for (int s2 = 0; s2 < LONG_SLOTS; ++s2) {
      const uint32_t j = (uint32_t)(l + s2 * L);
      ptr[s2] = j < mine ? so.kl[b0 + j] : nullptr;
      wgt[s2] = j < mine ? so.kw[b0 + j] : 0.f;
    }
    uint32_t most = mine;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) most = max(most, __shfl_xor_sync(FULL, most, o));
    for (uint32_t j0 = 0; j0 < most; j0 += LONG_UNROLL) {
      Part<CH, CPL> gr[LONG_UNROLL];
      float fw[LONG_UNROLL];
#pragma unroll
      for (int e = 0; e < LONG_UNROLL; ++e) {
        const uint32_t j = j0 + e;
        const uint32_t s2 = j >> lg;  // slot and lane of entry j
        const int src = (int)(j & (uint32_t)(L - 1));
        const float* pj = s2 == 0 ? ptr[0] : (s2 == 1 ? ptr[1] : (s2 == 2 ? ptr[2] : ptr[3]));
        const float wj = s2 == 0 ? wgt[0] : (s2 == 1 ? wgt[1] : (s2 == 2 ? wgt[2] : wgt[3]));
        pj = (const float*)__shfl_sync(FULL, (unsigned long long)pj, src, L);
        fw[e] = __shfl_sync(FULL, wj, src, L);
        if (j < mine) load_part<CH, CPL>(pj, l, L, C, gr[e]);
      }
#pragma unroll
      for (int e = 0; e < LONG_UNROLL; ++e) {
        if (j0 + e < mine) {
#pragma unroll
          for (int c = 0; c < CPL; ++c) {
            if (l + c * L >= C) continue;
#pragma unroll
            for (int k = 0; k < CH; ++k) csum_add_w(acc[c * CH + k], unit, fw[e], gr[e].v[c * CH + k]);
          }
        }
      }
    }
    // the groups' parts in group order, into group 0
    for (int gg = 1; gg < G; ++gg) {
#pragma unroll
      for (int i = 0; i < P; ++i) {
        const float hi = __shfl_sync(FULL, acc[i].hi, gg * L + l);
        const float lo = __shfl_sync(FULL, acc[i].lo, gg * L + l);
        if (g == 0) csum_merge(acc[i], hi, lo);
      }
    }
    bool finish = nch == 1u;
    if (!finish) {  // one chunk of several: leave its sum; the last chunk finishes the row
      if (g == 0) {
        const size_t pb = (size_t)(lr.w + item.y) * (size_t)so.pstride;
#pragma unroll
        for (int c = 0; c < CPL; ++c)
#pragma unroll
          for (int k = 0; k < CH; ++k) {
            const int q = l + c * L;
            if (q < C) {
              so.part_hi[pb + (size_t)q * CH + k] = acc[c * CH + k].hi;
              so.part_lo[pb + (size_t)q * CH + k] = acc[c * CH + k].lo;
            }
          }
      }
      __threadfence();
      __syncwarp();
      uint32_t last = 0u;
      if (lane == 0) last = atomicAdd(so.long_done + item.x, 1u) == nch - 1u;
      finish = __shfl_sync(FULL, last, 0) != 0u;
      if (finish) {  // every chunk's sum is visible: merge them in chunk order
        __threadfence();
#pragma unroll
        for (int i = 0; i < P; ++i) acc[i] = CSum{0.f, 0.f};
        for (uint32_t cc = 0; cc < nch; ++cc) {
          const size_t qb = (size_t)(lr.w + cc) * (size_t)so.pstride;
#pragma unroll
          for (int c = 0; c < CPL; ++c)
#pragma unroll
            for (int k = 0; k < CH; ++k) {
              const int q = l + c * L;
              if (q < C && g == 0)
                csum_merge(acc[c * CH + k], __ldcg(so.part_hi + qb + (size_t)q * CH + k),
                           __ldcg(so.part_lo + qb + (size_t)q * CH + k));
            }
        }
      }
    }
    if (finish && g == 0) {
      const RowMeta r = row_meta(so, lr.x, U, a.sparse_den, a.M);
      Part<CH, CPL> w, s0, s1;
      const size_t base = (size_t)r.x * (size_t)d;
      load_part<CH, CPL>(tb.w + base, l, L, C, w);
      load_part<CH, CPL>(tb.s0 + base, l, L, C, s0);
      if (adam) load_part<CH, CPL>(tb.s1 + base, l, L, C, s1);
      finish_row<CH, CPL>(tb, r.x, r.den, acc, w, s0, s1, l, L, C, adam);
      if (l == 0) {
        tb.ver[r.x] = (int32_t)(a.k + 1);
        ++applied;
      }
    }
    __syncwarp();
    it = it_next;
    item = item_next;
    lr = it < n_items ? so.long_rows[item.x] : make_uint4(0u, 0u, 0u, 0u);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) applied += __shfl_xor_sync(FULL, applied, o);
  if (lane == 0 && applied) atomicAdd(&st->rows_applied, (unsigned long long)applied);
}

// ---------------------------------------------------------------------------
// k_row_long_staged: the long rows for widths that are a multiple of 4, with
// their gradient rows staged in shared memory by cp.async so that many rows
// are in flight per warp.
//  1. Chunks of rows with more than SMALL_MAX kept occurrences, one warp per
//     chunk as in k_row_long; each lane group's part of the chunk streams
//     through a double buffer of LUNR rows per group.
//  2. Rows of LONG_ROW + 1 .. SMALL_MAX kept occurrences, one lane group per
//     row: its list entries, then its state and every kept gradient row are
//     copied at once; warps claim G rows at a time.
// Sums run over the kept entries in list order (per lane group part, parts
// merged in group order, chunks in chunk order), as in k_row_long.
// ---------------------------------------------------------------------------
#ifndef GBA_LUNR
#define GBA_LUNR 16
#endif
constexpr int LUNR = GBA_LUNR;  // rows per lane group per buffer in part 1
constexpr int LONG_STAGE_THREADS = 128;

__host__ __device__ constexpr int long_group_floats(int L, int CPL) {
  // list entries (SMALL_MAX addresses + weights), state (3 rows), gradient rows
  return 3 * SMALL_MAX + (3 + SMALL_MAX) * L * 4 * CPL;
}
__host__ __device__ constexpr int long_warp_floats(int L, int CPL) {
  return (2 * LUNR * 32 * 4 * CPL) > ((32 / L) * long_group_floats(L, CPL))
             ? (2 * LUNR * 32 * 4 * CPL)
             : ((32 / L) * long_group_floats(L, CPL));
}

template <int CPL>
__global__ void __launch_bounds__(LONG_STAGE_THREADS)
    k_row_long_staged(StepArgs a, SegTable tb, SegOut so, DevStats* st, ErrSink err) {
  extern __shared__ __align__(16) float s_long[];
  if (__any_sync(FULL, ld_volatile_u32(err.step) != 0u)) return;
  const int d = tb.d;
  const int C = d >> 2;
  int L = 1;
  while (L * CPL < C && L < 32) L <<= 1;
  const int lg = __ffs(L) - 1;
  const int G = 32 >> lg;  // lane groups per warp
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int g = lane >> lg, l = lane & (L - 1);
  const bool adam = tb.opt.kind == 1;
  const bool unit = a.decay == 0;  // every kept weight is 1
  const int RS = L * 4 * CPL;      // floats of one row in shared memory
  const int32_t tag = (int32_t)(a.k + 1);
  float* wsm = s_long + (size_t)warp * long_warp_floats(L, CPL);
  uint32_t applied = 0u;

  // ---- 1. chunks of the longest rows, one warp per chunk
  {
    const uint32_t n_items = ld_volatile_u32(so.n_items);
    const uint32_t U = ld_volatile_u32(so.total);
    auto claim = [&]() {
      uint32_t t = 0u;
      if (lane == 0) t = atomicAdd(so.item_ticket, 1u);
      return __shfl_sync(FULL, t, 0);
    };
    uint32_t it = claim();
    uint2 item = it < n_items ? so.items[it] : make_uint2(0u, 0u);
    uint4 lr = it < n_items ? so.long_rows[item.x] : make_uint4(0u, 0u, 0u, 0u);
    while (it < n_items) {
      const uint32_t it_next = claim();
      const uint2 item_next = it_next < n_items ? so.items[it_next] : make_uint2(0u, 0u);
      const uint32_t nch = (lr.z + LONG_CHUNK - 1) / LONG_CHUNK;
      const uint32_t e0 = lr.y + item.y * LONG_CHUNK;
      const uint32_t e1 = min(e0 + (uint32_t)LONG_CHUNK, lr.y + lr.z);
      const uint32_t per = (e1 - e0 + G - 1) / G;
      const uint32_t b0 = min(e0 + g * per, e1), b1 = min(b0 + per, e1);
      const uint32_t mine = b1 - b0;
      const float* ptr[LONG_SLOTS];
      float wgt[LONG_SLOTS];
#pragma unroll
      for (int s2 = 0; s2 < LONG_SLOTS; ++s2) {
        const uint32_t j = (uint32_t)(l + s2 * L);
        ptr[s2] = j < mine ? so.kl[b0 + j] : nullptr;
        wgt[s2] = j < mine ? so.kw[b0 + j] : 0.f;
      }
      uint32_t most = mine;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) most = max(most, __shfl_xor_sync(FULL, most, o));
      CSum acc[4 * CPL];
#pragma unroll
      for (int i = 0; i < 4 * CPL; ++i) acc[i] = CSum{0.f, 0.f};
      // entries j0 .. j0 + LUNR - 1 of every group's part into buffer bsel
      auto stage = [&](uint32_t j0, int bsel) {
#pragma unroll 4
        for (int e = 0; e < LUNR; ++e) {
          const uint32_t j = j0 + (uint32_t)e;
          const uint32_t s2 = j >> lg;
          const int src = (int)(j & (uint32_t)(L - 1));
          const float* pj = s2 == 0 ? ptr[0] : (s2 == 1 ? ptr[1] : (s2 == 2 ? ptr[2] : ptr[3]));
          pj = (const float*)__shfl_sync(FULL, (unsigned long long)pj, src, L);
          if (j < mine) {
            float* dst = wsm + ((size_t)(bsel * G + g) * LUNR + e) * RS;
#pragma unroll
            for (int c = 0; c < CPL; ++c) {
              const int q = l + c * L;
              if (q < C) cp_async16(dst + 4 * q, pj + 4 * q);
            }
          }
        }
        asm volatile("cp.async.commit_group;" ::: "memory");
      };
      stage(0u, 0);
      int bsel = 0;
      for (uint32_t j0 = 0; j0 < most; j0 += LUNR, bsel ^= 1) {
        if (j0 + LUNR < most) {
          stage(j0 + LUNR, bsel ^ 1);
          asm volatile("cp.async.wait_group 1;" ::: "memory");
        } else {
          asm volatile("cp.async.wait_group 0;" ::: "memory");
        }
        __syncwarp();
        for (int e = 0; e < LUNR; ++e) {
          const uint32_t j = j0 + (uint32_t)e;
          const uint32_t s2 = j >> lg;
          const int src = (int)(j & (uint32_t)(L - 1));
          float wj = s2 == 0 ? wgt[0] : (s2 == 1 ? wgt[1] : (s2 == 2 ? wgt[2] : wgt[3]));
          wj = __shfl_sync(FULL, wj, src, L);
          if (j < mine) {
            const float* rowp = wsm + ((size_t)(bsel * G + g) * LUNR + e) * RS;
#pragma unroll
            for (int c = 0; c < CPL; ++c) {
              const int q = l + c * L;
              if (q >= C) continue;
              const float4 v = *reinterpret_cast<const float4*>(rowp + 4 * q);
              csum_add_w(acc[4 * c + 0], unit, wj, v.x);
              csum_add_w(acc[4 * c + 1], unit, wj, v.y);
              csum_add_w(acc[4 * c + 2], unit, wj, v.z);
              csum_add_w(acc[4 * c + 3], unit, wj, v.w);
            }
          }
        }
        __syncwarp();  // the buffer is refilled next
      }
      // the groups' parts in group order, into group 0
      for (int gg = 1; gg < G; ++gg) {
#pragma unroll
        for (int i = 0; i < 4 * CPL; ++i) {
          const float hi = __shfl_sync(FULL, acc[i].hi, gg * L + l);
          const float lo = __shfl_sync(FULL, acc[i].lo, gg * L + l);
          if (g == 0) csum_merge(acc[i], hi, lo);
        }
      }
      bool finish = nch == 1u;
      if (!finish) {  // one chunk of several: leave its sum; the last chunk finishes the row
        if (g == 0) {
          const size_t pb = (size_t)(lr.w + item.y) * (size_t)so.pstride;
#pragma unroll
          for (int c = 0; c < CPL; ++c)
#pragma unroll
            for (int k = 0; k < 4; ++k) {
              const int q = l + c * L;
              if (q < C) {
                so.part_hi[pb + (size_t)q * 4 + k] = acc[c * 4 + k].hi;
                so.part_lo[pb + (size_t)q * 4 + k] = acc[c * 4 + k].lo;
              }
            }
        }
        __threadfence();
        __syncwarp();
        uint32_t last = 0u;
        if (lane == 0) last = atomicAdd(so.long_done + item.x, 1u) == nch - 1u;
        finish = __shfl_sync(FULL, last, 0) != 0u;
        if (finish) {  // every chunk's sum is visible: merge them in chunk order
          __threadfence();
#pragma unroll
          for (int i = 0; i < 4 * CPL; ++i) acc[i] = CSum{0.f, 0.f};
          for (uint32_t cc = 0; cc < nch; ++cc) {
            const size_t qb = (size_t)(lr.w + cc) * (size_t)so.pstride;
#pragma unroll
            for (int c = 0; c < CPL; ++c)
#pragma unroll
              for (int k = 0; k < 4; ++k) {
                const int q = l + c * L;
                if (q < C && g == 0)
                  csum_merge(acc[c * 4 + k], __ldcg(so.part_hi + qb + (size_t)q * 4 + k),
                             __ldcg(so.part_lo + qb + (size_t)q * 4 + k));
              }
          }
        }
      }
      if (finish && g == 0) {
        const RowMeta r = row_meta(so, lr.x, U, a.sparse_den, a.M);
        Part<4, CPL> w, s0, s1;
        const size_t base = (size_t)r.x * (size_t)d;
        load_part<4, CPL>(tb.w + base, l, L, C, w);
        load_part<4, CPL>(tb.s0 + base, l, L, C, s0);
        if (adam) load_part<4, CPL>(tb.s1 + base, l, L, C, s1);
        finish_row<4, CPL>(tb, r.x, r.den, acc, w, s0, s1, l, L, C, adam);
        if (l == 0) {
          tb.ver[r.x] = tag;
          ++applied;
        }
      }
      __syncwarp();
      it = it_next;
      item = item_next;
      lr = it < n_items ? so.long_rows[item.x] : make_uint4(0u, 0u, 0u, 0u);
    }
  }

  // ---- 2. rows of LONG_ROW + 1 .. SMALL_MAX kept occurrences, one lane group each
  {
    const uint32_t n_small = ld_volatile_u32(so.n_small);
    const int GF = long_group_floats(L, CPL);
    float* gs = wsm + (size_t)g * GF;
    const float** pp = reinterpret_cast<const float**>(gs);  // [SMALL_MAX] addresses
    float* wt = gs + 2 * SMALL_MAX;                           // [SMALL_MAX] weights
    float* sst = gs + 3 * SMALL_MAX;                          // w, s0, s1
    float* rows = sst + 3 * RS;                               // [SMALL_MAX] gradient rows
    auto claim = [&]() {
      uint32_t t = 0u;
      if (lane == 0) t = atomicAdd(so.small_ticket, (uint32_t)G);
      return __shfl_sync(FULL, t, 0);
    };
    uint32_t base = claim();
    uint4 sr = base + g < n_small ? so.small_rows[base + g] : make_uint4(0u, 0u, 0u, 0u);
    while (base < n_small) {
      const uint32_t x = sr.x, ks = sr.y, n = sr.z;  // n = 0: no row for this group
      for (uint32_t e = (uint32_t)l; e < n; e += (uint32_t)L) {
        cp_async8(pp + e, so.kl + ks + e);
        cp_async4(wt + e, so.kw + ks + e);
      }
      asm volatile("cp.async.commit_group;" ::: "memory");
      asm volatile("cp.async.wait_group 0;" ::: "memory");
      __syncwarp();
      if (n > 0u) {
        const size_t rb = (size_t)x * (size_t)d;
#pragma unroll
        for (int c = 0; c < CPL; ++c) {
          const int q = l + c * L;
          if (q >= C) continue;
          cp_async16(sst + 4 * q, tb.w + rb + 4 * q);
          cp_async16(sst + RS + 4 * q, tb.s0 + rb + 4 * q);
          if (adam) cp_async16(sst + 2 * RS + 4 * q, tb.s1 + rb + 4 * q);
          for (uint32_t e = 0; e < n; ++e) cp_async16(rows + (size_t)e * RS + 4 * q, pp[e] + 4 * q);
        }
      }
      asm volatile("cp.async.commit_group;" ::: "memory");
      // the next rows are claimed while these land
      const uint32_t base_next = claim();
      const uint4 sr_next =
          base_next + g < n_small ? so.small_rows[base_next + g] : make_uint4(0u, 0u, 0u, 0u);
      asm volatile("cp.async.wait_group 0;" ::: "memory");
      __syncwarp();
      if (n > 0u) {
        CSum acc[4 * CPL];
#pragma unroll
        for (int i = 0; i < 4 * CPL; ++i) acc[i] = CSum{0.f, 0.f};
        for (uint32_t e = 0; e < n; ++e) {
          const float we = wt[e];
#pragma unroll
          for (int c = 0; c < CPL; ++c) {
            const int q = l + c * L;
            if (q >= C) continue;
            const float4 v = *reinterpret_cast<const float4*>(rows + (size_t)e * RS + 4 * q);
            csum_add_w(acc[4 * c + 0], unit, we, v.x);
            csum_add_w(acc[4 * c + 1], unit, we, v.y);
            csum_add_w(acc[4 * c + 2], unit, we, v.z);
            csum_add_w(acc[4 * c + 3], unit, we, v.w);
          }
        }
        Part<4, CPL> w, s0, s1;
        load_part<4, CPL>(sst, l, L, C, w);
        load_part<4, CPL>(sst + RS, l, L, C, s0);
        if (adam) load_part<4, CPL>(sst + 2 * RS, l, L, C, s1);
        finish_row<4, CPL>(tb, x, __uint_as_float(sr.w), acc, w, s0, s1, l, L, C, adam);
        if (l == 0) {
          tb.ver[x] = tag;
          ++applied;
        }
      }
      __syncwarp();  // every lane is done with the group's buffers
      base = base_next;
      sr = sr_next;
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) applied += __shfl_xor_sync(FULL, applied, o);
  if (lane == 0 && applied) atomicAdd(&st->rows_applied, (unsigned long long)applied);
}

// ---------------------------------------------------------------------------
// launchers
// ---------------------------------------------------------------------------
template <typename K>
int blocks_per_sm(K kernel, int threads, size_t smem) {
  int b = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&b, kernel, threads, smem) != cudaSuccess ||
      b < 1)
    b = 1;
  return b;
}

template <int CPL>
void launch_staged(const StepArgs& a, const SegTable& tb, const SegOut& so, DevStats* stats,
                   ErrSink err, int num_sms, cudaStream_t s) {
  const int C = tb.d / 4;
  int L = 1;
  while (L * CPL < C && L < 32) L <<= 1;
  const int G = 32 / L;
  const int regions = (tb.opt.kind == 1 ? 3 : 2) + STAGE_NG;
  const size_t smem = (size_t)(STAGE_THREADS / 32) * stage_floats_per_warp(CPL, regions, G) * 4;
  static const size_t smem_max =
      (size_t)(STAGE_THREADS / 32) * stage_floats_per_warp(CPL, 3 + STAGE_NG, 32) * 4;
  static const bool configured =
      cudaFuncSetAttribute(k_row_apply_staged<CPL>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)smem_max) == cudaSuccess;
  (void)configured;
  const int bps = std::max(1, blocks_per_sm(k_row_apply_staged<CPL>, STAGE_THREADS, smem) -
                                 GBA_STAGE_BPS_CUT);
  const int64_t Nt = tb.pos_end - tb.pos_begin;  // bounds the rows
  const int64_t rows_per_block = (int64_t)(STAGE_THREADS / 32) * G * STAGE_P;
  const int64_t grid = std::max<int64_t>(
      1, std::min<int64_t>((int64_t)num_sms * bps, (Nt + rows_per_block - 1) / rows_per_block));
  k_row_apply_staged<CPL><<<(unsigned)grid, STAGE_THREADS, smem, s>>>(a, tb, so, stats, err);
}

template <int CH, int CPL>
void launch_apply_cfg(const StepArgs& a, const SegTable& tb, const SegOut& so, DevStats* stats,
                      ErrSink err, int num_sms, cudaStream_t s) {
  if constexpr (CH == 4) {
    if (CPL == 1 && GBA_STAGE_CPL != 1 && tb.d >= 32)  // wider pieces per lane for wide rows
      launch_staged<GBA_STAGE_CPL>(a, tb, so, stats, err, num_sms, s);
    else
      launch_staged<CPL>(a, tb, so, stats, err, num_sms, s);
    return;
  }
  static const int bps = blocks_per_sm(k_row_apply<CH, CPL>, ROW_THREADS, 0);
  const int64_t Nt = tb.pos_end - tb.pos_begin;  // bounds the rows
  const int C = CH == 4 ? tb.d / 4 : tb.d;
  int L = 1;
  while (L < C && L < 32) L <<= 1;
  const int64_t rows_per_block = (int64_t)(ROW_THREADS / 32) * (32 / L);
  const int64_t grid = std::max<int64_t>(
      1, std::min<int64_t>((int64_t)num_sms * bps, (Nt + rows_per_block - 1) / rows_per_block));
  k_row_apply<CH, CPL><<<(unsigned)grid, ROW_THREADS, 0, s>>>(a, tb, so, stats, err);
}

template <int CPL>
void launch_long_staged(const StepArgs& a, const SegTable& tb, const SegOut& so, DevStats* stats,
                        ErrSink err, int num_sms, cudaStream_t s) {
  const int C = tb.d / 4;
  int L = 1;
  while (L * CPL < C && L < 32) L <<= 1;
  const size_t smem = (size_t)(LONG_STAGE_THREADS / 32) * long_warp_floats(L, CPL) * 4;
  static size_t attr = 0;  // the largest dynamic shared memory size set so far
  if (smem > attr &&
      cudaFuncSetAttribute(k_row_long_staged<CPL>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)smem) == cudaSuccess)
    attr = smem;
  const int bps = GBA_LONG_BPS > 0
                      ? GBA_LONG_BPS
                      : blocks_per_sm(k_row_long_staged<CPL>, LONG_STAGE_THREADS, smem);
  const int64_t Nt = tb.pos_end - tb.pos_begin;
  const int64_t max_items = Nt / (LONG_ROW + 1) + Nt / LONG_CHUNK + 1;
  const int64_t grid = std::max<int64_t>(
      1, std::min<int64_t>((int64_t)num_sms * bps,
                           (max_items + LONG_STAGE_THREADS / 32 - 1) / (LONG_STAGE_THREADS / 32)));
  k_row_long_staged<CPL><<<(unsigned)grid, LONG_STAGE_THREADS, smem, s>>>(a, tb, so, stats, err);
}

template <int CH, int CPL>
void launch_long_cfg(const StepArgs& a, const SegTable& tb, const SegOut& so, DevStats* stats,
                     ErrSink err, int num_sms, cudaStream_t s) {
  if constexpr (CH == 4) {
    launch_long_staged<CPL>(a, tb, so, stats, err, num_sms, s);
    return;
  }
  static const int bps = GBA_LONG_BPS > 0 ? GBA_LONG_BPS
                                         : blocks_per_sm(k_row_long<CH, CPL>, ROW_THREADS, 0);
  const int64_t Nt = tb.pos_end - tb.pos_begin;
  const int64_t max_items = Nt / (LONG_ROW + 1) + Nt / LONG_CHUNK + 1;
  const int64_t grid = std::max<int64_t>(
      1, std::min<int64_t>((int64_t)num_sms * bps, (max_items + ROW_THREADS / 32 - 1) / (ROW_THREADS / 32)));
  k_row_long<CH, CPL><<<(unsigned)grid, ROW_THREADS, 0, s>>>(a, tb, so, stats, err);
}

}  // namespace

int64_t scan_tiles(int64_t N) { return (N + SCAN_TILE - 1) / SCAN_TILE; }

void launch_row_classify(const StepArgs& a, const SegTable& tb, const SegOut& so, ErrSink err,
                         int num_sms, cudaStream_t s) {
  const int64_t Nt = tb.pos_end - tb.pos_begin;  // bounds the rows
  const int64_t tile_rows = CLS_THREADS * CLS_ITEMS;
  const int64_t grid =
      std::max<int64_t>(1, std::min<int64_t>((int64_t)num_sms * 4, (Nt + tile_rows - 1) / tile_rows));
  // widths that are a multiple of 4 use the staged long-row kernel and its list of small rows
  k_row_classify<<<(unsigned)grid, CLS_THREADS, 0, s>>>(a, so, err, (tb.d & 3) == 0 ? 1 : 0);
}

void launch_seg_scan(const StepArgs& a, const SegTable& tb, const SegOut& so, const uint32_t* keys,
                     const uint32_t* vals, DevStats* stats, ErrSink err, int64_t wait_ns,
                     cudaStream_t s) {
  const int64_t tiles = scan_tiles(tb.pos_end - tb.pos_begin);
  if (tiles <= 0) return;
  static const bool configured =
      cudaFuncSetAttribute(k_seg_scan, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)SCAN_OUT_BYTES) == cudaSuccess;
  (void)configured;
  k_seg_scan<<<(unsigned)tiles, SCAN_THREADS, SCAN_OUT_BYTES, s>>>(a, tb, so, keys, vals, stats,
                                                                    err, wait_ns);
}

#define GBA_ROW_DISPATCH(FN)                                                       \
  const int d = tb.d;                                                              \
  if ((d & 3) == 0) {                                                              \
    if (d <= 128) return FN<4, 1>(a, tb, so, stats, err, num_sms, s);              \
    return FN<4, 2>(a, tb, so, stats, err, num_sms, s);                            \
  }                                                                                \
  if (d <= 32) return FN<1, 1>(a, tb, so, stats, err, num_sms, s);                 \
  if (d <= 64) return FN<1, 2>(a, tb, so, stats, err, num_sms, s);                 \
  if (d <= 128) return FN<1, 4>(a, tb, so, stats, err, num_sms, s);                \
  return FN<1, 8>(a, tb, so, stats, err, num_sms, s);

void launch_row_apply(const StepArgs& a, const SegTable& tb, const SegOut& so, DevStats* stats,
                      ErrSink err, int num_sms, cudaStream_t s) {
  GBA_ROW_DISPATCH(launch_apply_cfg)
}

void launch_row_long(const StepArgs& a, const SegTable& tb, const SegOut& so, DevStats* stats,
                     ErrSink err, int num_sms, cudaStream_t s) {
  GBA_ROW_DISPATCH(launch_long_cfg)
}

#undef GBA_ROW_DISPATCH

}  // namespace gba
