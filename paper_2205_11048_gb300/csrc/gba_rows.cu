// K3 + K4 of the GBA aggregate-and-apply step: per unique row of the sorted
// occurrence array, decay each occurrence by the row's step tag against its
// message's token (Eq. (1), Alg. 2), sum the kept gradient rows, divide by the
// number of messages that encountered the row, apply the optimizer to the row
// and its state in place, and set the row's tag to k + 1.
//
// Three kernels, each with work that is balanced by construction:
//
//  k_seg_reduce   Windows of at most 256 sorted positions, claimed in order by
//                 persistent warps.  A metadata pass decides every
//                 occurrence's weight (the tag is read here, before any row is
//                 updated) and counts the window's row heads; a decoupled
//                 look-back over the windows turns the counts into each row's
//                 index u in a compact list of the step's rows.  A second pass
//                 gathers the kept gradient rows of rows with two or more kept
//                 occurrences (staged in shared memory with cp.async, each lane
//                 copying its own row, all of a round's rows in flight) and
//                 sums them with compensated
//                 (TwoSum) arithmetic, lane = element, in sorted order.  A row
//                 with one kept occurrence needs no sum: its list entry points
//                 at the message's gradient row.  Rows that cross a window
//                 boundary leave compensated partial sums in per-window records.
//  k_seg_cross    One block per row that crosses windows: finds the window
//                 where the row ends, merges the partial sums (warps take
//                 interleaved records, then the warps' results are merged in
//                 order) and completes the row's list entry.
//  k_row_update   The optimizer step over the compact list: L = d/4 lanes per
//                 row, each lane one 16-byte piece of the gradient, weights and
//                 state, two rows per lane group in flight, grid-stride over
//                 the list.
//
// The row tags are read only in k_seg_reduce and written only in k_row_update,
// so no read of a tag can see this step's update.  Every summation order is
// fixed, so results are bit-identical run to run.
#include <algorithm>

#include "gba_internal.cuh"

namespace gba {

namespace {

constexpr int MSG_CACHE = 256;  // messages whose lookups are cached in shared memory
constexpr int WIN_ROUNDS = 8;   // a window is at most 8 rounds of 32 positions
constexpr uint32_t FULL = 0xffffffffu;
constexpr uint32_t NO_KEY = 0xFFFFFFFFu;

// record types (slot 0: the part of a row that began in an earlier window;
// slot 1: a row that begins in this window and continues past its end)
constexpr uint32_t REC_NONE = 0u, REC_PASS = 1u, REC_CLOSED = 2u, REC_OWNER = 3u;

// look-back status word: [63:32] epoch of the launch, [31:30] flag, [29:0] count
constexpr unsigned long long ST_AGG = 1ull << 30;
constexpr unsigned long long ST_INCL = 2ull << 30;
constexpr unsigned long long ST_FLAGS = 3ull << 30;
constexpr unsigned long long ST_COUNT = (1ull << 30) - 1;

// Per warp: one buffer of 32 staged gradient rows, then the window's keys and
// occurrence indices (written by the first pass, read by the second).
template <int EPL>
struct ReduceCfg {
  static constexpr int WARPS = EPL <= 2 ? 8 : (EPL == 4 ? 4 : 2);
  static constexpr int THREADS = WARPS * 32;
  static constexpr int MIN_BLOCKS = EPL == 1 ? 4 : (EPL == 2 ? 3 : 2);
  static constexpr size_t WARP_BYTES =
      (size_t)32 * 32 * EPL * sizeof(float) + (size_t)32 * WIN_ROUNDS * 2 * sizeof(uint32_t);
  static constexpr size_t SMEM = (size_t)WARPS * WARP_BYTES;
};
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
__device__ __forceinline__ uint32_t lanemask_lt() {
  uint32_t m;
  asm("mov.u32 %0, %%lanemask_lt;" : "=r"(m));
  return m;
}
__device__ __forceinline__ uint32_t bits_from(int j) { return j >= 32 ? 0u : (FULL << j); }
__device__ __forceinline__ uint32_t bits_below(int j) { return j >= 32 ? FULL : ((1u << j) - 1u); }

// Denominator of the row's weighted sum (R6: messages that encountered the
// row; or the kept ones; or all M messages).
__device__ __forceinline__ float row_denominator(int mode, uint32_t c_all, uint32_t c_kept,
                                                 int M) {
  const uint32_t den = mode == 0 ? c_all : (mode == 1 ? c_kept : (uint32_t)M);
  return (float)den;
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

struct RunCounts {
  uint32_t c_all, c_kept, k_occ;
};

__device__ __forceinline__ void store_desc(RowDesc* d, const float* src, uint32_t x, float den) {
  ulonglong2 v;
  v.x = (unsigned long long)src;
  v.y = (unsigned long long)x | ((unsigned long long)__float_as_uint(den) << 32);
  *reinterpret_cast<ulonglong2*>(d) = v;
}

template <int EPL>
__device__ __forceinline__ void write_record(const SegOut& so, int64_t w, int slot, int d,
                                             uint32_t type, uint32_t x, const RunCounts& c,
                                             uint32_t head_pos, uint32_t u, int lane,
                                             const CSum* acc) {
  const size_t base = ((size_t)w * 2 + slot) * (size_t)so.rec_stride;
#pragma unroll
  for (int e = 0; e < EPL; ++e) {
    const int el = lane * EPL + e;
    if (el < d) {
      so.rec_hi[base + el] = acc[e].hi;
      so.rec_lo[base + el] = acc[e].lo;
    }
  }
  if (lane == 0) {
    uint32_t* m = so.rec_meta + ((size_t)w * 2 + slot) * REC_META;
    m[1] = x;
    m[2] = c.c_all;
    m[3] = c.c_kept;
    m[4] = c.k_occ;
    m[5] = head_pos;
    m[6] = u;
    m[0] = type;
  }
}

// A row that began and ended in this window: its list entry (and, when two
// or more occurrences were kept, its sum in the compact buffer).
template <int EPL>
__device__ __forceinline__ void finish_local_row(const SegOut& so, int d, int mode, int M,
                                                 uint32_t x, uint32_t u, uint32_t head_pos,
                                                 const RunCounts& rc, const CSum* acc, int lane,
                                                 uint32_t* dbg_count, uint32_t* dbg_kept) {
  float* dst = so.compact + (size_t)u * so.cs;
  if (rc.k_occ > 0u) {
#pragma unroll
    for (int e = 0; e < EPL; ++e) {
      const int el = lane * EPL + e;
      if (el < d) dst[el] = csum_value(acc[e]);
    }
  }
  if (lane == 0) {
    const float den = rc.k_occ > 0u ? row_denominator(mode, rc.c_all, rc.c_kept, M) : 0.f;
    store_desc(so.desc + u, dst, x, den);
    if (dbg_count) {
      dbg_count[head_pos] = rc.c_all;
      dbg_kept[head_pos] = rc.k_occ;
    }
  }
}

// ---------------------------------------------------------------------------
// k_seg_reduce
// ---------------------------------------------------------------------------
template <int EPL>
__global__ void __launch_bounds__(ReduceCfg<EPL>::THREADS, ReduceCfg<EPL>::MIN_BLOCKS)
    k_seg_reduce(StepArgs a, SegTable tb, SegOut so, const uint32_t* __restrict__ keys,
                 const uint32_t* __restrict__ vals, int64_t wp, int64_t n_win, DevStats* st,
                 uint32_t* dbg_count, uint32_t* dbg_kept, ErrSink err, int64_t wait_ns) {
  using Cfg = ReduceCfg<EPL>;
  __shared__ uint32_t s_off[MSG_CACHE + 1];
  __shared__ int64_t s_tok[MSG_CACHE];
  __shared__ const float* s_rowp[MSG_CACHE];
  extern __shared__ __align__(128) unsigned char s_dyn[];

  // block-uniform: another kernel may set the word while this block reads it
  if (__syncthreads_or((ld_volatile_u32(err.step) & (ERR_ID_RANGE | ERR_TIMEOUT)) != 0u)) return;
  const int M = a.M;
  const uint32_t* off_g = a.msg_off + (size_t)tb.t * (M + 1);
  const float* const* rows_g = a.rows_ptr + (size_t)tb.t * M;
  const bool cached = M <= MSG_CACHE;
  if (cached) {
    for (int i = threadIdx.x; i <= M; i += Cfg::THREADS) s_off[i] = off_g[i];
    for (int i = threadIdx.x; i < M; i += Cfg::THREADS) {
      s_tok[i] = a.tokens[i];
      s_rowp[i] = rows_g[i];
    }
  }
  __syncthreads();
  const uint32_t* off = cached ? s_off : off_g;

  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  constexpr int SS = 32 * EPL;  // staged row stride (floats)
  float* stage = reinterpret_cast<float*>(s_dyn + (size_t)warp * Cfg::WARP_BYTES);
  uint2* pkv = reinterpret_cast<uint2*>(stage + 32 * SS);  // [position in window]: key, occurrence
  const int d = tb.d;
  const bool vec16 = (d & 3) == 0;  // gradient rows are 16-byte aligned
  const int64_t nbase = a.nbase[tb.t];
  const uint32_t n_t = (uint32_t)(tb.pos_end - tb.pos_begin);
  const uint32_t v_t = (uint32_t)tb.rows;
  const int mode = a.sparse_den;
  const unsigned long long ep = (unsigned long long)so.epoch << 32;

  uint32_t n_pairs = 0, n_pairs_dropped = 0, n_kept_occ = 0, n_heads = 0;
  unsigned long long stale_sum = 0, stale_max = 0;
  __shared__ uint32_t s_tile, s_base, s_cnt[Cfg::WARPS];
  const int64_t n_tiles = (n_win + Cfg::WARPS - 1) / Cfg::WARPS;

  // A block claims a tile of WARPS consecutive windows (in order, by ticket);
  // warp j takes window WARPS * tile + j.
  for (;;) {
    if (threadIdx.x == 0) s_tile = atomicAdd(so.ticket, 1u);
    __syncthreads();
    const int64_t bt = (int64_t)s_tile;
    if (bt >= n_tiles) break;
    const int64_t w = bt * Cfg::WARPS + warp;
    if (w >= n_win) {  // past the last window: only the barriers
      s_cnt[warp] = 0u;
      __syncthreads();
      __syncthreads();
      continue;
    }
    const int64_t p0 = tb.pos_begin + w * wp;
    const int64_t p1 = (p0 + wp < tb.pos_end) ? p0 + wp : tb.pos_end;
    const int R = (int)((p1 - p0 + 31) >> 5);

    // ---- pass 1a: the window's keys; its row heads and their count -------------
    uint32_t kk[WIN_ROUNDS], vv[WIN_ROUNDS];
#pragma unroll
    for (int r = 0; r < WIN_ROUNDS; ++r) {
      const int64_t pos = p0 + 32 * r + lane;
      kk[r] = NO_KEY;
      vv[r] = 0u;
      if (r < R && pos < p1) {
        kk[r] = keys[pos];
        vv[r] = vals[pos];
      }
    }
#pragma unroll
    for (int r = 0; r < WIN_ROUNDS; ++r)
      if (r < R) pkv[32 * r + lane] = make_uint2(kk[r], vv[r]);
    // the neighbours outside the window: lane 0 the position before, lane 1 after
    uint32_t edge_k = NO_KEY, edge_v = 0u;
    if (lane == 0 && p0 > tb.pos_begin) {
      edge_k = keys[p0 - 1];
      edge_v = vals[p0 - 1];
    }
    if (lane == 1 && p1 < tb.pos_end) edge_k = keys[p1];
    const uint32_t first_prev = __shfl_sync(FULL, edge_k, 0);
    const uint32_t next_key = __shfl_sync(FULL, edge_k, 1);
    uint32_t myH = 0u, nh = 0u, last_key = NO_KEY;
    {
      uint32_t prev_key = first_prev;
#pragma unroll
      for (int r = 0; r < WIN_ROUNDS; ++r) {
        if (r < R) {
          uint32_t pk = __shfl_up_sync(FULL, kk[r], 1);
          if (lane == 0) pk = prev_key;
          const uint32_t Hm = __ballot_sync(FULL, kk[r] != NO_KEY && kk[r] != pk);
          if (lane == r) myH = Hm;
          nh += __popc(Hm);
          const uint32_t Vm = __ballot_sync(FULL, kk[r] != NO_KEY);
          if (Vm) last_key = __shfl_sync(FULL, kk[r], 31 - __clz(Vm));
          prev_key = __shfl_sync(FULL, kk[r], 31);
        }
      }
    }
    const bool cont_end = p1 < tb.pos_end && next_key == last_key;  // last row goes on
    const uint32_t key0 = __shfl_sync(FULL, kk[0], 0);
    if (lane == 0) s_cnt[warp] = nh;

    // ---- pass 1b: messages, tags, weights (Eq. (1)), new-message flags ----------
    uint32_t mm[WIN_ROUNDS];
    int32_t tg[WIN_ROUNDS];
#pragma unroll
    for (int r = 0; r < WIN_ROUNDS; ++r) {
      mm[r] = 0xFFFFFFFEu;
      tg[r] = 0;
      if (kk[r] != NO_KEY) {
        const uint32_t o_t = (uint32_t)((int64_t)vv[r] - nbase);
        const uint32_t x = kk[r] - tb.key_base;
        if (o_t >= n_t || x >= v_t) {
          raise_error(err, ERR_INTERNAL);  // cannot happen for a correctly sorted array
        } else {
          mm[r] = (uint32_t)message_of_any(off, M, o_t);
          if (a.row_staleness == 0) tg[r] = tb.ver[x];  // the row's step tag (Alg. 2)
        }
      }
    }
    uint32_t prev_m = 0xFFFFFFFFu;
    {
      const uint32_t o_t = (uint32_t)((int64_t)edge_v - nbase);
      uint32_t pm = 0xFFFFFFFFu;
      if (lane == 0 && first_prev != NO_KEY && o_t < n_t)
        pm = (uint32_t)message_of_any(off, M, o_t);
      prev_m = __shfl_sync(FULL, pm, 0);
    }
    uint32_t myK = 0u, myN = 0u;  // lane r keeps round r's kept / new-message masks
#pragma unroll
    for (int r = 0; r < WIN_ROUNDS; ++r) {
      if (r < R) {
        const bool valid = mm[r] != 0xFFFFFFFEu;
        bool keep = false;
        uint32_t stale = 0u;
        if (valid) {
          const uint32_t m = mm[r];
          const int64_t tok = cached ? s_tok[m] : a.tokens[m];
          const int64_t ref = a.row_staleness == 0 ? (int64_t)tg[r] : a.k;
          const int64_t diff = ref - tok;
          const uint64_t sl = diff > 0 ? (uint64_t)diff : 0ull;
          keep = sl <= (uint64_t)(int64_t)a.iota;
          stale = (uint32_t)(sl > 0xFFFFFFFFull ? 0xFFFFFFFFull : sl);
        }
        uint32_t pm = __shfl_up_sync(FULL, mm[r], 1);
        if (lane == 0) pm = prev_m;
        const bool head = (__shfl_sync(FULL, myH, r) >> lane) & 1u;
        const bool newmsg = valid && (head || mm[r] != pm);
        if (keep) ++n_kept_occ;
        if (newmsg) {
          ++n_pairs;
          if (!keep) ++n_pairs_dropped;
          stale_sum += stale;
          stale_max = stale > stale_max ? stale : stale_max;
        }
        const uint32_t Km = __ballot_sync(FULL, keep);
        const uint32_t Nm = __ballot_sync(FULL, newmsg);
        if (lane == r) {
          myK = Km;
          myN = Nm;
        }
        prev_m = __shfl_sync(FULL, mm[r], 31);
      }
    }

    // ---- the window's first list index: warp 0 looks back over block tiles
    __syncthreads();
    if (warp == 0) {
      uint32_t c = lane < Cfg::WARPS ? s_cnt[lane] : 0u;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) c += __shfl_xor_sync(FULL, c, o);
      const uint32_t tile_cnt = c;
      if (lane == 0)
        st_relaxed_u64(so.status + bt,
                       ep | (bt == 0 ? ST_INCL : ST_AGG) | (unsigned long long)tile_cnt);
      uint32_t tp = 0u;
      if (bt > 0) {
        int64_t j = bt - 1;
        const uint64_t t0 = globaltimer_ns();
        for (;;) {
          const int64_t q = j - lane;
          unsigned long long v = ep | ST_INCL;  // before tile 0: nothing
          if (q >= 0) v = ld_relaxed_u64(so.status + q);
          const bool ready = (v & ~0xFFFFFFFFull) == ep && (v & ST_FLAGS) != 0ull;
          const bool incl = ready && (v & ST_INCL) != 0ull;
          const uint32_t rm = __ballot_sync(FULL, ready), im = __ballot_sync(FULL, incl);
          const int first_nr = ~rm ? __ffs(~rm) - 1 : 32;
          const int first_in = im ? __ffs(im) - 1 : 32;
          const int take = first_in < first_nr ? first_in + 1 : first_nr;
          uint32_t cc = lane < take ? (uint32_t)(v & ST_COUNT) : 0u;
#pragma unroll
          for (int o = 16; o > 0; o >>= 1) cc += __shfl_xor_sync(FULL, cc, o);
          tp += cc;
          if (first_in < first_nr) break;
          j -= take;
          if (take == 0 && ((ld_volatile_u32(err.step) & ERR_TIMEOUT) ||
                            (int64_t)(globaltimer_ns() - t0) > wait_ns)) {
            if (lane == 0) raise_error(err, ERR_TIMEOUT);
            break;
          }
        }
        if (lane == 0)
          st_relaxed_u64(so.status + bt,
                         ep | ST_INCL | (unsigned long long)((tp + tile_cnt) & ST_COUNT));
      }
      if (lane == 0) {
        s_base = tp;
        if (bt == n_tiles - 1) *so.total = tp + tile_cnt;
      }
    }
    __syncthreads();
    uint32_t prefix = s_base;
    for (int j = 0; j < warp; ++j) prefix += s_cnt[j];
    n_heads += nh;

    // ---- pass 2: gather and sum, round by round ----------------------------------
    // prepare() analyses a round, writes the list entries of rows that begin
    // and end inside it and issues its gathers; the sums follow in order and
    // carry the open row from round to round.
    CSum acc[EPL];
#pragma unroll
    for (int e = 0; e < EPL; ++e) acc[e] = CSum{0.f, 0.f};
    RunCounts rc{0u, 0u, 0u};
    uint32_t ox = 0u, ou = 0u, ohead = 0u;
    bool open_head = false;  // the open row's head lies in this window
    bool wrote_slot0 = false;
    uint32_t hb = 0u;  // heads of the window before the next round to prepare
    if (p0 > tb.pos_begin && !(__shfl_sync(FULL, myH, 0) & 1u))
      ox = key0 - tb.key_base;  // a row that began in an earlier window is open

    struct Round {
      uint32_t Hm, Km, Nm, Gm, Fm, u_fl, key, hb;
      int n_round;
      bool cont;
    };
    auto prepare = [&](int r, float* buf) -> Round {
      Round st;
      const int64_t rb = p0 + 32 * r;
      const int n_round = (int)((p1 - rb) < 32 ? (p1 - rb) : 32);
      const uint32_t Hm = __shfl_sync(FULL, myH, r);
      const uint32_t Km = __shfl_sync(FULL, myK, r);
      const uint32_t Nm = __shfl_sync(FULL, myN, r);
      const uint32_t Vm = bits_below(n_round);
      const uint32_t Hn = __shfl_sync(FULL, myH, r + 1 < 32 ? r + 1 : 31);
      const bool cont = (r + 1 < R) ? !(Hn & 1u) : cont_end;  // the round's last row goes on
      const bool valid = lane < n_round;
      // lane metadata again, from the keys and occurrences pass 1 kept
      uint32_t key = NO_KEY;
      const float* rowp = nullptr;
      if (valid) {
        const uint2 kv = pkv[32 * r + lane];
        key = kv.x;
        const uint32_t o_t = (uint32_t)((int64_t)kv.y - nbase);
        if (o_t < n_t) {
          const uint32_t m = (uint32_t)message_of_any(off, M, o_t);
          rowp = (cached ? s_rowp[m] : rows_g[m]) + (size_t)(o_t - off[m]) * (size_t)d;
        }
      }
      const bool keep = (Km >> lane) & 1u;
      // pieces: maximal runs of one row inside the round
      const uint32_t Bm = (Hm | 1u) & Vm;
      const int s_of = 31 - __clz(Bm & bits_below(lane + 1));  // my piece's first lane
      const uint32_t after = Bm & ~bits_below(s_of + 1);
      const int e_of = after ? __ffs(after) - 1 : n_round;  // and its end
      const uint32_t rng = bits_below(e_of) & bits_from(s_of);
      const bool starts = valid && s_of == lane;
      const bool is_head = (Hm >> lane) & 1u;
      const bool closes = e_of < n_round || !cont;
      const uint32_t kmask = Km & rng;
      const uint32_t kc = __popc(kmask);
      const uint32_t ca = __popc(Nm & rng), ck = __popc(Nm & Km & rng);
      // rows that begin and end inside the round: the lane of the head writes
      // the list entry -- pointing at the single kept gradient row, or at the
      // compact slot that the sum fills
      const bool single = starts && is_head && closes && kc <= 1u;
      const bool local_sum = starts && is_head && closes && kc >= 2u;
      const uint32_t u_me = prefix + hb + __popc(Hm & lanemask_lt());
      const int jk = single && kc ? __ffs(kmask) - 1 : lane;
      const float* src1 = (const float*)__shfl_sync(FULL, (unsigned long long)rowp, jk);
      if (single || local_sum) {
        const float den = kc ? row_denominator(mode, ca, ck, M) : 0.f;
        store_desc(so.desc + u_me, single ? src1 : so.compact + (size_t)u_me * so.cs,
                   key - tb.key_base, den);
        if (dbg_count) {
          dbg_count[rb + lane] = ca;
          dbg_kept[rb + lane] = kc;
        }
      }
      const uint32_t Sm = __ballot_sync(FULL, single);
      const uint32_t Lm = __ballot_sync(FULL, local_sum);
      // gathered positions: kept, outside single rows; flush positions: the last
      // kept position of a local sum, which also learns the row's list index
      const bool gather = valid && keep && !((Sm >> s_of) & 1u);
      const bool flush = gather && ((Lm >> s_of) & 1u) && (31 - __clz(kmask)) == lane;
      st.Gm = __ballot_sync(FULL, gather);
      st.Fm = __ballot_sync(FULL, flush);
      st.u_fl = __shfl_sync(FULL, u_me, s_of);
      if (gather) {  // each gathering lane copies its own row
        float* dst = buf + lane * SS;
        if (vec16) {
          for (int q = 0; q < d; q += 4)
            asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_addr(dst + q)),
                         "l"(rowp + q)
                         : "memory");
        } else {
          for (int q = 0; q < d; ++q)
            asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(smem_addr(dst + q)),
                         "l"(rowp + q)
                         : "memory");
        }
      }
      asm volatile("cp.async.commit_group;" ::: "memory");
      st.Hm = Hm;
      st.Km = Km;
      st.Nm = Nm;
      st.key = __shfl_sync(FULL, key, 31 - __clz(Bm));  // key where the round's last piece starts
      st.hb = hb;
      st.n_round = n_round;
      st.cont = cont;
      hb += __popc(Hm);
      return st;
    };

    for (int r = 0; r < R; ++r) {
      float* buf = stage;
      const Round cur = prepare(r, buf);
      asm volatile("cp.async.wait_group 0;" ::: "memory");
      __syncwarp();
      const uint32_t Hm = cur.Hm, Km = cur.Km, Nm = cur.Nm, Gm = cur.Gm, Fm = cur.Fm;
      const int n_round = cur.n_round;
      const bool cont = cur.cont;
      const uint32_t Vm = bits_below(n_round);
      const uint32_t Bm = (Hm | 1u) & Vm;
      const int64_t rb = p0 + 32 * r;
      // ---- the sums, lane = element, in sorted order
      uint32_t gm = Gm;
      if (Hm == 0u) {
        // The whole round continues the open row (a Zipf-hot row): the same
        // compensated sum in the same order, unrolled, positions that were not
        // gathered adding an exact zero.
#pragma unroll
        for (int j = 0; j < 32; ++j) {
          const bool on = (Gm >> j) & 1u;
#pragma unroll
          for (int q = 0; q < EPL; ++q) {
            const float x = buf[j * SS + lane * EPL + q];
            csum_add(acc[q], on ? x : 0.f);
          }
        }
        gm = 0u;
      }
      if (!(Hm & 1u)) {  // position 0 continues the open row
        const uint32_t a0 = Bm & ~1u;
        const int e0 = a0 ? __ffs(a0) - 1 : n_round;
        const uint32_t r0 = bits_below(e0);
        uint32_t g0 = gm & r0;
        gm &= ~r0;
        while (g0) {
          const int j = __ffs(g0) - 1;
          g0 &= g0 - 1u;
          const float* sp = buf + j * SS + lane * EPL;
#pragma unroll
          for (int q = 0; q < EPL; ++q) csum_add(acc[q], sp[q]);
        }
        rc.c_all += __popc(Nm & r0);
        rc.c_kept += __popc(Nm & Km & r0);
        rc.k_occ += __popc(Km & r0);
        if (e0 < n_round || !cont) {  // the open row ends in this round
          if (open_head) {
            finish_local_row<EPL>(so, d, mode, M, ox, ou, ohead, rc, acc, lane, dbg_count,
                                  dbg_kept);
          } else {
            write_record<EPL>(so, w, 0, d, REC_CLOSED, ox, rc, 0u, 0u, lane, acc);
            wrote_slot0 = true;
            // the row's head is the last one before this window: list index prefix - 1
            if (lane == 0 && prefix > 0u) so.cross_end[prefix - 1u] = (uint32_t)w;
          }
          open_head = false;
#pragma unroll
          for (int q = 0; q < EPL; ++q) acc[q] = CSum{0.f, 0.f};
        }
      }
      while (gm) {
        const int j = __ffs(gm) - 1;
        gm &= gm - 1u;
        const float* sp = buf + j * SS + lane * EPL;
#pragma unroll
        for (int q = 0; q < EPL; ++q) csum_add(acc[q], sp[q]);
        if ((Fm >> j) & 1u) {
          const uint32_t uj = __shfl_sync(FULL, cur.u_fl, j);
          float* dst = so.compact + (size_t)uj * so.cs;
#pragma unroll
          for (int q = 0; q < EPL; ++q) {
            const int el = lane * EPL + q;
            if (el < d) dst[el] = csum_value(acc[q]);
            acc[q] = CSum{0.f, 0.f};
          }
        }
      }
      // a row that begins in this round and goes on past it becomes the open row
      const int ls = 31 - __clz(Bm);
      if (cont && ((Hm >> ls) & 1u)) {
        const uint32_t rl = Vm & bits_from(ls);
        ox = cur.key - tb.key_base;
        ou = prefix + cur.hb + __popc(Hm & bits_below(ls));
        ohead = (uint32_t)(rb + ls);
        rc = RunCounts{(uint32_t)__popc(Nm & rl), (uint32_t)__popc(Nm & Km & rl),
                       (uint32_t)__popc(Km & rl)};
        open_head = true;
      }
      __syncwarp();  // the buffer is refilled by the next round
    }
    bool wrote_slot1 = false;
    if (cont_end) {  // the open row goes on in the next window
      if (open_head) {
        write_record<EPL>(so, w, 1, d, REC_OWNER, ox, rc, ohead, ou, lane, acc);
        wrote_slot1 = true;
        if (lane == 0) so.cross_list[atomicAdd(so.cross_count, 1u)] = (uint32_t)w;
      } else {
        write_record<EPL>(so, w, 0, d, REC_PASS, ox, rc, 0u, 0u, lane, acc);
        wrote_slot0 = true;
      }
    }
    if (lane == 0) {
      if (!wrote_slot0) so.rec_meta[((size_t)w * 2 + 0) * REC_META] = REC_NONE;
      if (!wrote_slot1) so.rec_meta[((size_t)w * 2 + 1) * REC_META] = REC_NONE;
    }
    __syncwarp();
  }

#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    n_pairs += __shfl_xor_sync(FULL, n_pairs, o);
    n_pairs_dropped += __shfl_xor_sync(FULL, n_pairs_dropped, o);
    stale_sum += __shfl_xor_sync(FULL, stale_sum, o);
    const unsigned long long y = __shfl_xor_sync(FULL, stale_max, o);
    stale_max = y > stale_max ? y : stale_max;
    n_kept_occ += __shfl_xor_sync(FULL, n_kept_occ, o);
  }
  if (lane == 0) {
    if (n_pairs) atomicAdd(&st->pairs, (unsigned long long)n_pairs);
    if (n_pairs_dropped) atomicAdd(&st->pairs_dropped, (unsigned long long)n_pairs_dropped);
    if (stale_sum) atomicAdd(&st->row_stale_sum, stale_sum);
    if (stale_max) atomicMax(&st->row_stale_max, stale_max);
    if (n_kept_occ) atomicAdd(&st->occ_kept, (unsigned long long)n_kept_occ);
    if (n_heads) atomicAdd(&st->rows_touched, (unsigned long long)n_heads);
  }
}

// ---------------------------------------------------------------------------
// k_seg_cross: rows whose occurrences span two or more windows
// ---------------------------------------------------------------------------
constexpr int CROSS_THREADS = 256;
constexpr int CROSS_WARPS = CROSS_THREADS / 32;

template <int EPL>
__device__ __forceinline__ void cross_row(const StepArgs& a, const SegTable& tb, const SegOut& so,
                                          int64_t n_win, int64_t w, uint32_t* dbg_count,
                                          uint32_t* dbg_kept, const ErrSink& err) {
  __shared__ float s_hi[CROSS_WARPS][32 * EPL];
  __shared__ float s_lo[CROSS_WARPS][32 * EPL];
  __shared__ uint32_t s_bad, s_call, s_ckept, s_kocc;
  const uint32_t* m1 = so.rec_meta + ((size_t)w * 2 + 1) * REC_META;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const uint32_t type = m1[0], x = m1[1], head_pos = m1[5], u = m1[6];
  const int64_t end = type == REC_OWNER ? (int64_t)so.cross_end[u] : -1;
  if (tid == 0) {
    s_bad = 0u;
    s_call = m1[2];
    s_ckept = m1[3];
    s_kocc = m1[4];
  }
  __syncthreads();
  // the list holds owners only; the row ends in a later window
  if (end <= w || end >= n_win || x >= (uint32_t)tb.rows) {
    if (tid == 0) raise_error(err, ERR_INTERNAL);
    __syncthreads();
    return;
  }
  // Merge the partial sums: warp j takes the records of windows w+1+j,
  // w+1+j+W, ... in order (warp 0 starts from the owner's), then warp 0 merges
  // the warps' results in warp order.  Each record must carry the row on
  // (PASS) but the last, which closes it (CLOSED).
  const int d = tb.d;
  const int64_t R = end - w;
  CSum acc[EPL];
#pragma unroll
  for (int e = 0; e < EPL; ++e) acc[e] = CSum{0.f, 0.f};
  if (warp == 0) {
    const size_t b = ((size_t)w * 2 + 1) * (size_t)so.rec_stride;
#pragma unroll
    for (int e = 0; e < EPL; ++e) {
      const int el = lane * EPL + e;
      if (el < d) acc[e] = CSum{so.rec_hi[b + el], so.rec_lo[b + el]};
    }
  }
  constexpr int U4 = EPL == 1 ? 8 : (EPL == 2 ? 4 : 2);  // records in flight per warp
  uint32_t c_all = 0u, c_kept = 0u, k_occ = 0u;
  bool bad = false;
  for (int64_t i0 = warp; i0 < R; i0 += CROSS_WARPS * U4) {
    float hi[U4][EPL], lo[U4][EPL];
#pragma unroll
    for (int k = 0; k < U4; ++k) {
      const int64_t i = i0 + (int64_t)k * CROSS_WARPS;
      const size_t rw = (size_t)(w + 1 + i) * 2 + 0;
      const size_t b = rw * (size_t)so.rec_stride;
#pragma unroll
      for (int e = 0; e < EPL; ++e) {
        const int el = lane * EPL + e;
        hi[k][e] = 0.f;
        lo[k][e] = 0.f;
        if (i < R && el < d) {
          hi[k][e] = so.rec_hi[b + el];
          lo[k][e] = so.rec_lo[b + el];
        }
      }
      if (i < R && lane == 0) {
        const uint32_t* m0 = so.rec_meta + rw * REC_META;
        const uint32_t want = i + 1 == R ? REC_CLOSED : REC_PASS;
        if (m0[0] != want || m0[1] != x) bad = true;
        c_all += m0[2];
        c_kept += m0[3];
        k_occ += m0[4];
      }
    }
#pragma unroll
    for (int k = 0; k < U4; ++k)
      if (i0 + (int64_t)k * CROSS_WARPS < R) {
#pragma unroll
        for (int e = 0; e < EPL; ++e) csum_merge(acc[e], hi[k][e], lo[k][e]);
      }
  }
  if (lane == 0) {
    if (bad) s_bad = 1u;
    atomicAdd(&s_call, c_all);
    atomicAdd(&s_ckept, c_kept);
    atomicAdd(&s_kocc, k_occ);
  }
#pragma unroll
  for (int e = 0; e < EPL; ++e) {
    s_hi[warp][lane * EPL + e] = acc[e].hi;
    s_lo[warp][lane * EPL + e] = acc[e].lo;
  }
  __syncthreads();
  if (warp == 0) {
    if (s_bad) {
      if (lane == 0) raise_error(err, ERR_INTERNAL);
    } else {
#pragma unroll
      for (int j = 1; j < CROSS_WARPS; ++j)
#pragma unroll
        for (int e = 0; e < EPL; ++e)
          csum_merge(acc[e], s_hi[j][lane * EPL + e], s_lo[j][lane * EPL + e]);
      const RunCounts rc{s_call, s_ckept, s_kocc};
      finish_local_row<EPL>(so, d, a.sparse_den, a.M, x, u, head_pos, rc, acc, lane, dbg_count,
                            dbg_kept);
    }
  }
  __syncthreads();  // the shared scratch is reused by the block's next row
}

// One block per listed row (the list order does not matter: rows are
// independent and each row's merge order is fixed).
template <int EPL>
__global__ void __launch_bounds__(CROSS_THREADS, EPL <= 2 ? 4 : 2)
    k_seg_cross(StepArgs a, SegTable tb, SegOut so, int64_t n_win, uint32_t* dbg_count,
                uint32_t* dbg_kept, ErrSink err) {
  if (__syncthreads_or(ld_volatile_u32(err.step) != 0u)) return;
  const uint32_t n = ld_volatile_u32(so.cross_count);
  for (uint32_t i = blockIdx.x; i < n; i += gridDim.x)
    cross_row<EPL>(a, tb, so, n_win, (int64_t)so.cross_list[i], dbg_count, dbg_kept, err);
}

// ---------------------------------------------------------------------------
// k_row_update: the optimizer step over the compact row list
// ---------------------------------------------------------------------------
constexpr int UPD_THREADS = 256;

// One row's pieces held by a lane: gradient, weights, optimizer state.
template <int NV>
struct RowRegs {
  float g[NV], w[NV], s0[NV], s1[NV];
};

struct RowRef {
  const float* src;
  uint32_t x;
  float den;
  bool act;
};

__device__ __forceinline__ RowRef load_ref(const SegOut& so, int64_t u, uint32_t U) {
  RowRef r{nullptr, 0u, 0.f, false};
  if (u < (int64_t)U) {
    const ulonglong2 v = *reinterpret_cast<const ulonglong2*>(so.desc + u);
    r.src = (const float*)v.x;
    r.x = (uint32_t)v.y;
    r.den = __uint_as_float((uint32_t)(v.y >> 32));
    r.act = r.den > 0.f;
  }
  return r;
}

template <int CH, int CPL>
__device__ __forceinline__ void load_row(const SegTable& tb, const RowRef& r, int l, int L, int C,
                                         bool adam, RowRegs<CH * CPL>& v) {
  if (!r.act) return;
  const int d = tb.d;
#pragma unroll
  for (int c = 0; c < CPL; ++c) {
    const int q = l + c * L;
    if (q < C) {
      const size_t o = (size_t)r.x * d + (size_t)q * CH;
      if constexpr (CH == 4) {
        const float4 g4 = *reinterpret_cast<const float4*>(r.src + q * 4);
        const float4 w4 = *reinterpret_cast<const float4*>(tb.w + o);
        const float4 a4 = *reinterpret_cast<const float4*>(tb.s0 + o);
        v.g[4 * c] = g4.x; v.g[4 * c + 1] = g4.y; v.g[4 * c + 2] = g4.z; v.g[4 * c + 3] = g4.w;
        v.w[4 * c] = w4.x; v.w[4 * c + 1] = w4.y; v.w[4 * c + 2] = w4.z; v.w[4 * c + 3] = w4.w;
        v.s0[4 * c] = a4.x; v.s0[4 * c + 1] = a4.y; v.s0[4 * c + 2] = a4.z; v.s0[4 * c + 3] = a4.w;
        if (adam) {
          const float4 b4 = *reinterpret_cast<const float4*>(tb.s1 + o);
          v.s1[4 * c] = b4.x; v.s1[4 * c + 1] = b4.y; v.s1[4 * c + 2] = b4.z; v.s1[4 * c + 3] = b4.w;
        }
      } else {
        v.g[c] = r.src[q];
        v.w[c] = tb.w[o];
        v.s0[c] = tb.s0[o];
        if (adam) v.s1[c] = tb.s1[o];
      }
    }
  }
}

template <int CH, int CPL>
__device__ __forceinline__ void update_row(const SegTable& tb, const RowRef& r, int l, int L, int C,
                                           bool adam, int32_t tag, RowRegs<CH * CPL>& v,
                                           uint32_t& applied) {
  if (!r.act) return;
  const int d = tb.d;
#pragma unroll
  for (int c = 0; c < CPL; ++c) {
    const int q = l + c * L;
    if (q >= C) continue;
#pragma unroll
    for (int k = 0; k < CH; ++k) {
      const int i = c * CH + k;
      float b = adam ? v.s1[i] : 0.f;
      const float gi = r.den == 1.0f ? v.g[i] : __fdiv_rn(v.g[i], r.den);
      opt_update(tb.opt, v.w[i], v.s0[i], b, gi);
      v.s1[i] = b;
    }
    const size_t o = (size_t)r.x * d + (size_t)q * CH;
    if constexpr (CH == 4) {
      const int i = 4 * c;
      *reinterpret_cast<float4*>(tb.w + o) = make_float4(v.w[i], v.w[i + 1], v.w[i + 2], v.w[i + 3]);
      *reinterpret_cast<float4*>(tb.s0 + o) =
          make_float4(v.s0[i], v.s0[i + 1], v.s0[i + 2], v.s0[i + 3]);
      if (adam)
        *reinterpret_cast<float4*>(tb.s1 + o) =
            make_float4(v.s1[i], v.s1[i + 1], v.s1[i + 2], v.s1[i + 3]);
    } else {
      tb.w[o] = v.w[c];
      tb.s0[o] = v.s0[c];
      if (adam) tb.s1[o] = v.s1[c];
    }
  }
  if (l == 0) {
    tb.ver[r.x] = tag;
    ++applied;
  }
}

// CH floats per piece (4: 16-byte pieces, rows with d % 4 == 0; else 1), at
// most CPL pieces per lane.  Each lane group walks its rows with the next
// row's loads issued before the current row's update (and the list entry two
// rows ahead), so memory latency overlaps the optimizer arithmetic.
template <int CH, int CPL>
__global__ void __launch_bounds__(UPD_THREADS, (CH == 4 && CPL == 1) || (CH == 1 && CPL <= 2) ? 4 : 2)
    k_row_update(StepArgs a, SegTable tb, SegOut so, DevStats* st, ErrSink err) {
  // a failed step changes no row (warp-uniform: the warp reduces at the end)
  if (__any_sync(FULL, ld_volatile_u32(err.step) != 0u)) return;
  const uint32_t U = ld_volatile_u32(so.total);
  const int d = tb.d;
  const int C = d / CH;  // pieces per row
  int L = 1;
  while (L < C && L < 32) L <<= 1;  // lanes per row
  const int lg = __ffs(L) - 1;
  const int G = 32 >> lg;  // rows per warp
  const int lane = threadIdx.x & 31;
  const int g = lane >> lg, l = lane & (L - 1);
  const int64_t gw = (int64_t)blockIdx.x * (UPD_THREADS / 32) + (threadIdx.x >> 5);
  const int64_t TG = (int64_t)gridDim.x * (UPD_THREADS / 32) * G;
  const bool adam = tb.opt.kind == 1;
  const int32_t tag = (int32_t)(a.k + 1);
  uint32_t applied = 0u;
  int64_t u = gw * G + g;
  RowRef cur = load_ref(so, u, U), nxt = load_ref(so, u + TG, U);
  RowRegs<CH * CPL> vc, vn;
  load_row<CH, CPL>(tb, cur, l, L, C, adam, vc);
  for (; u < (int64_t)U; u += TG) {
    const RowRef n2 = load_ref(so, u + 2 * TG, U);
    load_row<CH, CPL>(tb, nxt, l, L, C, adam, vn);
    update_row<CH, CPL>(tb, cur, l, L, C, adam, tag, vc, applied);
    cur = nxt;
    nxt = n2;
    vc = vn;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) applied += __shfl_xor_sync(FULL, applied, o);
  if ((threadIdx.x & 31) == 0 && applied) atomicAdd(&st->rows_applied, (unsigned long long)applied);
}

// ---------------------------------------------------------------------------
// launchers
// ---------------------------------------------------------------------------
template <typename K>
int blocks_per_sm(K kernel, int threads, size_t smem) {
  // static + dynamic shared memory may pass 48 KB: always raise the limit
  cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  int b = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&b, kernel, threads, smem) != cudaSuccess ||
      b < 1)
    b = 1;
  return b;
}

// Window size: one window per resident warp while that keeps windows at 32 to
// 256 positions.
template <int EPL>
int64_t reduce_windows(int64_t Nt, int num_sms, int64_t* wp_out, int* grid_out) {
  using Cfg = ReduceCfg<EPL>;
  static const int bps = blocks_per_sm(k_seg_reduce<EPL>, Cfg::THREADS, Cfg::SMEM);
  const int64_t warps = (int64_t)num_sms * bps * Cfg::WARPS;
  int64_t wp = (Nt + warps - 1) / warps;
  wp = (wp + 31) / 32 * 32;
  wp = wp < 32 ? 32 : (wp > 32 * WIN_ROUNDS ? 32 * WIN_ROUNDS : wp);
  const int64_t n_win = (Nt + wp - 1) / wp;
  const int64_t grid = std::min<int64_t>((int64_t)num_sms * bps, (n_win + Cfg::WARPS - 1) / Cfg::WARPS);
  *wp_out = wp;
  *grid_out = (int)grid;
  return n_win;
}

template <int EPL>
int64_t launch_reduce_epl(const StepArgs& a, const SegTable& tb, const SegOut& so,
                          const uint32_t* keys, const uint32_t* vals, DevStats* stats,
                          uint32_t* dbg_count, uint32_t* dbg_kept, ErrSink err, int num_sms,
                          int64_t wait_ns, cudaStream_t s) {
  using Cfg = ReduceCfg<EPL>;
  int64_t wp = 0;
  int grid = 0;
  const int64_t n_win = reduce_windows<EPL>(tb.pos_end - tb.pos_begin, num_sms, &wp, &grid);
  k_seg_reduce<EPL><<<grid, Cfg::THREADS, Cfg::SMEM, s>>>(a, tb, so, keys, vals, wp, n_win, stats,
                                                          dbg_count, dbg_kept, err, wait_ns);
  return n_win;
}

template <int CH, int CPL>
void launch_update_cfg(const StepArgs& a, const SegTable& tb, const SegOut& so, DevStats* stats,
                       ErrSink err, int num_sms, cudaStream_t s) {
  static const int bps = blocks_per_sm(k_row_update<CH, CPL>, UPD_THREADS, 0);
  const int64_t Nt = tb.pos_end - tb.pos_begin;
  const int C = tb.d / CH;
  int L = 1;
  while (L < C && L < 32) L <<= 1;
  const int64_t rows_per_block = (int64_t)(UPD_THREADS / 32) * (32 / L) * 2;  // two per group at least
  const int64_t grid =
      std::max<int64_t>(1, std::min<int64_t>((int64_t)num_sms * bps, (Nt + rows_per_block - 1) / rows_per_block));
  k_row_update<CH, CPL><<<(unsigned)grid, UPD_THREADS, 0, s>>>(a, tb, so, stats, err);
}

}  // namespace

int64_t seg_window_bound(int64_t N, int num_sms) {
  return (int64_t)num_sms * 64 + (N + 32 * WIN_ROUNDS - 1) / (32 * WIN_ROUNDS) + 1;
}

int64_t launch_seg_reduce(const StepArgs& a, const SegTable& tb, const SegOut& so,
                          const uint32_t* keys, const uint32_t* vals, DevStats* stats,
                          uint32_t* dbg_count, uint32_t* dbg_kept, ErrSink err, int num_sms,
                          int64_t wait_ns, cudaStream_t s) {
  const int d = tb.d;
#define GBA_RED(EP) \
  return launch_reduce_epl<EP>(a, tb, so, keys, vals, stats, dbg_count, dbg_kept, err, num_sms, wait_ns, s)
  if (d <= 32) GBA_RED(1);
  if (d <= 64) GBA_RED(2);
  if (d <= 128) GBA_RED(4);
  GBA_RED(8);
#undef GBA_RED
}

void launch_seg_cross(const StepArgs& a, const SegTable& tb, const SegOut& so, int64_t n_win,
                      uint32_t* dbg_count, uint32_t* dbg_kept, ErrSink err, cudaStream_t s) {
  if (n_win < 2) return;  // one window: no row can cross
  // at most one listed row per window but the last
  const unsigned grid = (unsigned)std::min<int64_t>(n_win - 1, 152 * 8);
  const int d = tb.d;
  if (d <= 32)
    k_seg_cross<1><<<grid, CROSS_THREADS, 0, s>>>(a, tb, so, n_win, dbg_count, dbg_kept, err);
  else if (d <= 64)
    k_seg_cross<2><<<grid, CROSS_THREADS, 0, s>>>(a, tb, so, n_win, dbg_count, dbg_kept, err);
  else if (d <= 128)
    k_seg_cross<4><<<grid, CROSS_THREADS, 0, s>>>(a, tb, so, n_win, dbg_count, dbg_kept, err);
  else
    k_seg_cross<8><<<grid, CROSS_THREADS, 0, s>>>(a, tb, so, n_win, dbg_count, dbg_kept, err);
}

void launch_row_update(const StepArgs& a, const SegTable& tb, const SegOut& so, DevStats* stats,
                       ErrSink err, int num_sms, cudaStream_t s) {
  const int d = tb.d;
  if ((d & 3) == 0) {
    if (d <= 128) return launch_update_cfg<4, 1>(a, tb, so, stats, err, num_sms, s);
    return launch_update_cfg<4, 2>(a, tb, so, stats, err, num_sms, s);
  }
  if (d <= 32) return launch_update_cfg<1, 1>(a, tb, so, stats, err, num_sms, s);
  if (d <= 64) return launch_update_cfg<1, 2>(a, tb, so, stats, err, num_sms, s);
  if (d <= 128) return launch_update_cfg<1, 4>(a, tb, so, stats, err, num_sms, s);
  return launch_update_cfg<1, 8>(a, tb, so, stats, err, num_sms, s);
}

}  // namespace gba
