// K3 + K4 of the GBA aggregate-and-apply step: per unique row of the sorted
// occurrence array, decay each occurrence by the row's step tag against its
// message's token (Eq. (1), Alg. 2), sum the kept gradient rows, divide by the
// number of messages that encountered the row, apply the optimizer to the row
// and its state in place, and set the row's tag to k + 1.
//
// Work is split by occurrences, not by rows, so Zipf-hot rows cost no more per
// occurrence than cold ones.  Each warp owns a contiguous range of the sorted
// array and walks it in rounds of 64 positions; within a round each lane group
// (L lanes, one row-slice of 16-byte vectors per lane) sums a contiguous slice
// of positions sequentially with compensated (TwoSum) float accumulation.
// Rows that start and end inside a slice are applied by their group at once;
// rows crossing slices are stitched in slice order across the warp; rows
// crossing warp ranges leave partial sums in a record that the fixup kernel
// combines in range order.  All orders are fixed, so results are bit-identical
// run to run.
#include "gba_internal.cuh"

namespace gba {

namespace {

constexpr int SEG_THREADS = 256;
constexpr int SEG_WARPS = SEG_THREADS / 32;
constexpr int RS = 64;  // positions per round

constexpr uint32_t F_HEAD = 1u, F_KEEP = 2u, F_NEWMSG = 4u;

// record types
constexpr uint32_t REC_NONE = 0u, REC_PASS = 1u, REC_CLOSED = 2u, REC_OWNER = 3u;
constexpr int REC_META = 6;  // type, x, c_all, c_kept, k_occ, head_pos

struct PosMeta {
  const float* row;  // gradient row of the occurrence
  uint32_t key;
  uint32_t m;        // message index
  uint32_t flags;
  uint32_t pad;
};

__device__ __forceinline__ uint32_t ld_volatile_u32(const uint32_t* p) {
  return *(const volatile uint32_t*)p;
}

// Denominator of the row's weighted sum.
__device__ __forceinline__ float row_denominator(int mode, uint32_t c_all, uint32_t c_kept,
                                                 int M) {
  const uint32_t den = mode == 0 ? c_all : (mode == 1 ? c_kept : (uint32_t)M);
  return (float)den;
}

template <int VEC>
struct Vec;
template <>
struct Vec<4> {
  static __device__ __forceinline__ void load(const float* p, float* v) {
    const float4 q = *reinterpret_cast<const float4*>(p);
    v[0] = q.x; v[1] = q.y; v[2] = q.z; v[3] = q.w;
  }
  static __device__ __forceinline__ void store(float* p, const float* v) {
    *reinterpret_cast<float4*>(p) = make_float4(v[0], v[1], v[2], v[3]);
  }
};
template <>
struct Vec<1> {
  static __device__ __forceinline__ void load(const float* p, float* v) { v[0] = *p; }
  static __device__ __forceinline__ void store(float* p, const float* v) { *p = v[0]; }
};

// Apply the optimizer to this lane's slice of row x: element (e*L + l)*VEC + v.
template <int VEC, int L, int EPL>
__device__ __forceinline__ void apply_slice(const SegTable& tb, uint32_t x, int l,
                                            const CSum* s, float den) {
  const int d = tb.d;
  const size_t rb = (size_t)x * (size_t)d;
#pragma unroll
  for (int e = 0; e < EPL; ++e) {
    const int idx = (e * L + l) * VEC;
    if (idx < d) {
      float w[VEC], s0[VEC], s1[VEC];
      Vec<VEC>::load(tb.w + rb + idx, w);
      Vec<VEC>::load(tb.s0 + rb + idx, s0);
      if (tb.opt.kind == 1) Vec<VEC>::load(tb.s1 + rb + idx, s1);
#pragma unroll
      for (int v = 0; v < VEC; ++v) {
        const float g = __fdiv_rn(csum_value(s[e * VEC + v]), den);
        opt_update(tb.opt, w[v], s0[v], s1[v], g);
      }
      Vec<VEC>::store(tb.w + rb + idx, w);
      Vec<VEC>::store(tb.s0 + rb + idx, s0);
      if (tb.opt.kind == 1) Vec<VEC>::store(tb.s1 + rb + idx, s1);
    }
  }
}

struct RunCounts {
  uint32_t c_all, c_kept, k_occ;
};

// Everything that happens when a row's run is complete.
template <int VEC, int L, int EPL>
__device__ __forceinline__ void finalize_row(const StepArgs& a, const SegTable& tb, uint32_t x,
                                             uint32_t head_pos, const RunCounts& c, int l,
                                             const CSum* s, uint32_t* dbg_count,
                                             uint32_t* dbg_kept, unsigned long long& n_touched,
                                             unsigned long long& n_applied) {
  if (l == 0) {
    ++n_touched;
    if (dbg_count) {
      dbg_count[head_pos] = c.c_all;
      dbg_kept[head_pos] = c.k_occ;
    }
  }
  if (c.k_occ == 0u) return;  // every occurrence excluded: no step, tag unchanged
  if (x >= (uint32_t)tb.rows) return;  // only after a latched consistency error
  apply_slice<VEC, L, EPL>(tb, x, l, s, row_denominator(a.sparse_den, c.c_all, c.c_kept, a.M));
  if (l == 0) {
    tb.ver[x] = (int32_t)(a.k + 1);
    ++n_applied;
  }
}

template <int VEC, int L, int EPL>
__device__ __forceinline__ void write_record(const SegRecords& rec, int64_t wg, int slot, int d,
                                             uint32_t type, uint32_t x, uint32_t head_pos,
                                             const RunCounts& c, int l, const CSum* s) {
  const size_t base = ((size_t)wg * 2 + slot) * (size_t)d;
#pragma unroll
  for (int e = 0; e < EPL; ++e) {
#pragma unroll
    for (int v = 0; v < VEC; ++v) {
      const int idx = (e * L + l) * VEC + v;
      if (idx < d) {
        rec.hi[base + idx] = s[e * VEC + v].hi;
        rec.lo[base + idx] = s[e * VEC + v].lo;
      }
    }
  }
  if (l == 0) {
    uint32_t* m = rec.meta + ((size_t)wg * 2 + slot) * REC_META;
    m[1] = x;
    m[2] = c.c_all;
    m[3] = c.c_kept;
    m[4] = c.k_occ;
    m[5] = head_pos;
    m[0] = type;
  }
}

template <int VEC, int L, int EPL>
__global__ void __launch_bounds__(SEG_THREADS)
    k_segsum_apply(StepArgs a, SegTable tb, const uint32_t* __restrict__ keys,
                   const uint32_t* __restrict__ vals, int64_t range, int64_t n_warps,
                   SegRecords rec, DevStats* st, uint32_t* dbg_count, uint32_t* dbg_kept,
                   ErrSink err) {
  constexpr int G = 32 / L;  // lane groups per warp
  constexpr int E = RS / G;  // positions per group slice
  constexpr int NV = EPL * VEC;
  __shared__ PosMeta s_meta[SEG_WARPS][RS];

  if (ld_volatile_u32(err.dev) & (ERR_ID_RANGE | ERR_TIMEOUT)) return;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int64_t wg = (int64_t)blockIdx.x * SEG_WARPS + warp;
  if (wg >= n_warps) return;
  const int g = lane / L, l = lane % L;
  const int d = tb.d;
  const int M = a.M;
  const int64_t r0 = tb.pos_begin + wg * range;
  const int64_t r1 = (r0 + range < tb.pos_end) ? r0 + range : tb.pos_end;
  const uint32_t* off = a.msg_off + (size_t)tb.t * (M + 1);
  const float* const* rows_ptr = a.rows_ptr + (size_t)tb.t * M;
  const int64_t nbase = a.nbase[tb.t];
  const uint32_t n_t = (uint32_t)(tb.pos_end - tb.pos_begin);
  const uint32_t v_t = (uint32_t)tb.rows;

  unsigned long long n_pairs = 0, n_pairs_dropped = 0, stale_sum = 0, stale_max = 0;
  unsigned long long n_touched = 0, n_applied = 0, n_kept_occ = 0;

  PosMeta* sm = s_meta[warp];

  // State carried between positions: the key and message of the previous one.
  uint32_t prev_key = 0xFFFFFFFFu, prev_m = 0xFFFFFFFFu;
  if (r0 > tb.pos_begin && r0 < r1) {
    prev_key = keys[r0 - 1];
    prev_m = (uint32_t)message_of(off, M, (uint32_t)((int64_t)vals[r0 - 1] - nbase));
  }

  // The run open at the current boundary, replicated across groups.
  CSum carry[NV];
#pragma unroll
  for (int i = 0; i < NV; ++i) carry[i] = CSum{0.f, 0.f};
  RunCounts cc{0u, 0u, 0u};
  uint32_t carry_x = 0u, carry_head = 0u;
  bool carry_active = false, carry_local = false;
  if (r0 < r1 && prev_key == keys[r0]) {  // range starts inside a row owned by an earlier warp
    carry_active = true;
    carry_x = keys[r0] - tb.key_base;
  }
  bool wrote_head_record = false, wrote_tail_record = false;

  for (int64_t rb = r0; rb < r1; rb += RS) {
    const int n_round = (int)((r1 - rb) < RS ? (r1 - rb) : RS);
    // ---- per-position metadata (two positions per lane)
#pragma unroll
    for (int q = 0; q < 2; ++q) {
      const int j = q * 32 + lane;
      if (j < n_round) {
        const uint32_t key = keys[rb + j];
        const uint32_t o_t = (uint32_t)((int64_t)vals[rb + j] - nbase);
        const uint32_t x = key - tb.key_base;
        if (o_t >= n_t || x >= v_t) {
          // cannot happen for a correctly sorted array; never touch memory with it
          raise_error(err, ERR_INTERNAL);
          sm[j].row = nullptr;
          sm[j].key = key;
          sm[j].m = 0u;
          sm[j].pad = 0u;
          sm[j].flags = 0u;
          continue;
        }
        const int m = message_of(off, M, o_t);
        const uint32_t p = o_t - __ldg(off + m);
        const int64_t ref = a.row_staleness == 0 ? (int64_t)tb.ver[x] : a.k;
        const int64_t diff = ref - a.tokens[m];
        const uint64_t s = diff > 0 ? (uint64_t)diff : 0ull;
        const bool keep = s <= (uint64_t)(int64_t)a.iota;
        sm[j].row = rows_ptr[m] + (size_t)p * (size_t)d;
        sm[j].key = key;
        sm[j].m = (uint32_t)m;
        sm[j].pad = (uint32_t)(s > 0xFFFFFFFFull ? 0xFFFFFFFFull : s);
        sm[j].flags = keep ? F_KEEP : 0u;
      }
    }
    __syncwarp();
#pragma unroll
    for (int q = 0; q < 2; ++q) {
      const int j = q * 32 + lane;
      if (j < n_round) {
        const uint32_t pk = j == 0 ? prev_key : sm[j - 1].key;
        const uint32_t pm = j == 0 ? prev_m : sm[j - 1].m;
        if (sm[j].flags & F_KEEP) ++n_kept_occ;
        const bool head = sm[j].key != pk;
        const bool newmsg = head || sm[j].m != pm;
        uint32_t f = sm[j].flags;
        if (head) f |= F_HEAD;
        if (newmsg) {
          f |= F_NEWMSG;
          ++n_pairs;
          if (!(f & F_KEEP)) ++n_pairs_dropped;
          const unsigned long long s = sm[j].pad;
          stale_sum += s;
          stale_max = s > stale_max ? s : stale_max;
        }
        sm[j].flags = f;  // written after all reads of this round's neighbours below
      }
    }
    __syncwarp();
    prev_key = sm[n_round - 1].key;
    prev_m = sm[n_round - 1].m;

    // ---- each group walks its slice sequentially
    const int j0 = g * E;
    CSum acc[NV], cont[NV];
#pragma unroll
    for (int i = 0; i < NV; ++i) acc[i] = cont[i] = CSum{0.f, 0.f};
    RunCounts ac{0u, 0u, 0u}, cn{0u, 0u, 0u};
    uint32_t a_x = 0u, a_head = 0u;
    bool in_cont = (j0 < n_round) && !(sm[j0].flags & F_HEAD);
    bool have_open = false;
    bool any_head = false;
#pragma unroll 4
    for (int jj = 0; jj < E; ++jj) {
      const int j = j0 + jj;
      if (j < n_round) {
        const uint32_t f = sm[j].flags;
        if (f & F_HEAD) {
          any_head = true;
          if (in_cont) {  // the row continued from before ends here
#pragma unroll
            for (int i = 0; i < NV; ++i) cont[i] = acc[i];
            cn = ac;
            in_cont = false;
          } else if (have_open) {  // a row that started in this slice is complete
            finalize_row<VEC, L, EPL>(a, tb, a_x, a_head, ac, l, acc, dbg_count, dbg_kept,
                                      n_touched, n_applied);
          }
#pragma unroll
          for (int i = 0; i < NV; ++i) acc[i] = CSum{0.f, 0.f};
          ac = RunCounts{0u, 0u, 0u};
          a_x = sm[j].key - tb.key_base;
          a_head = (uint32_t)(rb + j);
          have_open = true;
        }
        if (f & F_NEWMSG) {
          ++ac.c_all;
          if (f & F_KEEP) ++ac.c_kept;
        }
        if (f & F_KEEP) {
          ++ac.k_occ;
          const float* row = sm[j].row;
#pragma unroll
          for (int e = 0; e < EPL; ++e) {
            const int idx = (e * L + l) * VEC;
            if (idx < d) {
              float v[VEC];
              Vec<VEC>::load(row + idx, v);
#pragma unroll
              for (int u = 0; u < VEC; ++u) csum_add(acc[e * VEC + u], v[u]);
            }
          }
        }
      }
    }
    // acc: the open run (started at a head in the slice) or, with no head in the
    // slice, the part of the continued row (pass-through).
    const uint32_t head_mask = __ballot_sync(0xffffffffu, any_head && l == 0);

    // ---- stitch the slices of this round in order
    for (int gg = 0; gg < G; ++gg) {
      if (gg * E >= n_round) break;
      const int src = gg * L + l;
      const bool starts_head = (sm[gg * E].flags & F_HEAD) != 0u;
      const bool has_head = (head_mask >> (gg * L)) & 1u;
      if (!starts_head) {
        // continuation of the carried row: its part in slice gg is `cont` if a
        // head closes it inside the slice, else the whole slice (`acc`).
#pragma unroll
        for (int i = 0; i < NV; ++i) {
          const float hi = __shfl_sync(0xffffffffu, has_head ? cont[i].hi : acc[i].hi, src);
          const float lo = __shfl_sync(0xffffffffu, has_head ? cont[i].lo : acc[i].lo, src);
          csum_merge(carry[i], hi, lo);
        }
        cc.c_all += __shfl_sync(0xffffffffu, has_head ? cn.c_all : ac.c_all, gg * L);
        cc.c_kept += __shfl_sync(0xffffffffu, has_head ? cn.c_kept : ac.c_kept, gg * L);
        cc.k_occ += __shfl_sync(0xffffffffu, has_head ? cn.k_occ : ac.k_occ, gg * L);
        if (!has_head) continue;  // the row continues past this slice
      }
      // The carried row (if any) is complete here.
      if (carry_active) {
        if (carry_local) {
          if (g == 0)
            finalize_row<VEC, L, EPL>(a, tb, carry_x, carry_head, cc, l, carry, dbg_count,
                                      dbg_kept, n_touched, n_applied);
        } else {
          if (g == 0)
            write_record<VEC, L, EPL>(rec, wg, 0, d, REC_CLOSED, carry_x, 0u, cc, l, carry);
          wrote_head_record = true;
        }
      }
      // The open run of slice gg becomes the carried row.
#pragma unroll
      for (int i = 0; i < NV; ++i) {
        carry[i].hi = __shfl_sync(0xffffffffu, acc[i].hi, src);
        carry[i].lo = __shfl_sync(0xffffffffu, acc[i].lo, src);
      }
      cc.c_all = __shfl_sync(0xffffffffu, ac.c_all, gg * L);
      cc.c_kept = __shfl_sync(0xffffffffu, ac.c_kept, gg * L);
      cc.k_occ = __shfl_sync(0xffffffffu, ac.k_occ, gg * L);
      carry_x = __shfl_sync(0xffffffffu, a_x, gg * L);
      carry_head = __shfl_sync(0xffffffffu, a_head, gg * L);
      carry_active = true;
      carry_local = true;
    }
    __syncwarp();
  }

  // ---- end of the range: the carried row ends here or continues in the next range
  if (carry_active) {
    const bool closes = (r1 == tb.pos_end) || keys[r1] != keys[r1 - 1];
    if (closes) {
      if (carry_local) {
        if (g == 0)
          finalize_row<VEC, L, EPL>(a, tb, carry_x, carry_head, cc, l, carry, dbg_count,
                                    dbg_kept, n_touched, n_applied);
      } else {
        if (g == 0) write_record<VEC, L, EPL>(rec, wg, 0, d, REC_CLOSED, carry_x, 0u, cc, l, carry);
        wrote_head_record = true;
      }
    } else if (carry_local) {
      if (g == 0)
        write_record<VEC, L, EPL>(rec, wg, 1, d, REC_OWNER, carry_x, carry_head, cc, l, carry);
      wrote_tail_record = true;
    } else {
      if (g == 0) write_record<VEC, L, EPL>(rec, wg, 0, d, REC_PASS, carry_x, 0u, cc, l, carry);
      wrote_head_record = true;
    }
  }
  if (lane == 0) {
    if (!wrote_head_record) rec.meta[((size_t)wg * 2 + 0) * REC_META] = REC_NONE;
    if (!wrote_tail_record) rec.meta[((size_t)wg * 2 + 1) * REC_META] = REC_NONE;
  }

  // ---- counters
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    n_pairs += __shfl_xor_sync(0xffffffffu, n_pairs, o);
    n_pairs_dropped += __shfl_xor_sync(0xffffffffu, n_pairs_dropped, o);
    stale_sum += __shfl_xor_sync(0xffffffffu, stale_sum, o);
    const unsigned long long y = __shfl_xor_sync(0xffffffffu, stale_max, o);
    stale_max = y > stale_max ? y : stale_max;
    n_touched += __shfl_xor_sync(0xffffffffu, n_touched, o);
    n_applied += __shfl_xor_sync(0xffffffffu, n_applied, o);
    n_kept_occ += __shfl_xor_sync(0xffffffffu, n_kept_occ, o);
  }
  if (lane == 0) {
    if (n_pairs) atomicAdd(&st->pairs, n_pairs);
    if (n_pairs_dropped) atomicAdd(&st->pairs_dropped, n_pairs_dropped);
    if (stale_sum) atomicAdd(&st->row_stale_sum, stale_sum);
    if (stale_max) atomicMax(&st->row_stale_max, stale_max);
    if (n_touched) atomicAdd(&st->rows_touched, n_touched);
    if (n_applied) atomicAdd(&st->rows_applied, n_applied);
    if (n_kept_occ) atomicAdd(&st->occ_kept, n_kept_occ);
  }
}

// ---------------------------------------------------------------------------
// Second form, for rows of up to 64 floats: the same walk, but a finished row
// is not updated where it is found.  Its aggregated gradient goes to a
// per-warp shared-memory slot (the row's last position in the round) and,
// once the round's rows are all summed and stitched, the whole warp updates
// them together: each lane group takes a batch of finished rows and issues
// all of their state loads before the first update.  The rows' gradient
// loads of a slice are likewise issued in batches before they are summed.
// ---------------------------------------------------------------------------
constexpr int SEG2_WARPS = 4;
constexpr int SEG2_THREADS = SEG2_WARPS * 32;
constexpr int MSG_CACHE = 256;  // messages whose lookups are cached in shared memory
constexpr int APPLY_BATCH = 4;  // finished rows per lane group per batch
constexpr int SEG2_MIN_BLOCKS = 3;  // 16 warps per SM: at most 128 registers a thread

// The message of table-local occurrence x in the offsets off[0..M] (any memory).
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

template <int VEC, int L, int EPL>
__global__ void __launch_bounds__(SEG2_THREADS, SEG2_MIN_BLOCKS)
    k_segsum_apply2(StepArgs a, SegTable tb, const uint32_t* __restrict__ keys,
                    const uint32_t* __restrict__ vals, int64_t range, int64_t n_warps,
                    SegRecords rec, DevStats* st, uint32_t* dbg_count, uint32_t* dbg_kept,
                    ErrSink err) {
  constexpr int G = 32 / L;
  constexpr int E = RS / G;
  constexpr int NV = EPL * VEC;
  constexpr int DW = L * EPL * VEC;  // floats of a done slot
  constexpr int CH = E < 4 ? E : 4;  // gradient rows loaded per batch
  __shared__ PosMeta s_meta[SEG2_WARPS][RS];
  __shared__ uint8_t s_done[SEG2_WARPS][RS];
  __shared__ uint32_t s_off[MSG_CACHE + 1];
  __shared__ int64_t s_tok[MSG_CACHE];
  __shared__ const float* s_rowp[MSG_CACHE];
  extern __shared__ __align__(16) float s_ghat[];  // [SEG2_WARPS][RS][DW]

  if (ld_volatile_u32(err.dev) & (ERR_ID_RANGE | ERR_TIMEOUT)) return;
  const int M = a.M;
  const uint32_t* off_g = a.msg_off + (size_t)tb.t * (M + 1);
  const float* const* rows_g = a.rows_ptr + (size_t)tb.t * M;
  const bool cached = M <= MSG_CACHE;
  if (cached) {
    for (int i = threadIdx.x; i <= M; i += SEG2_THREADS) s_off[i] = off_g[i];
    for (int i = threadIdx.x; i < M; i += SEG2_THREADS) {
      s_tok[i] = a.tokens[i];
      s_rowp[i] = rows_g[i];
    }
  }
  __syncthreads();
  const uint32_t* off = cached ? s_off : off_g;

  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int64_t wg = (int64_t)blockIdx.x * SEG2_WARPS + warp;
  if (wg >= n_warps) return;
  const int g = lane / L, l = lane % L;
  const int d = tb.d;
  const int64_t r0 = tb.pos_begin + wg * range;
  const int64_t r1 = (r0 + range < tb.pos_end) ? r0 + range : tb.pos_end;
  const int64_t nbase = a.nbase[tb.t];
  const uint32_t n_t = (uint32_t)(tb.pos_end - tb.pos_begin);
  const uint32_t v_t = (uint32_t)tb.rows;

  unsigned long long n_pairs = 0, n_pairs_dropped = 0, stale_sum = 0, stale_max = 0;
  unsigned long long n_touched = 0, n_applied = 0, n_kept_occ = 0;

  PosMeta* sm = s_meta[warp];
  uint8_t* sd = s_done[warp];
  float* gh = s_ghat + (size_t)warp * RS * DW;
  sd[lane] = 0;
  sd[lane + 32] = 0;

  uint32_t prev_key = 0xFFFFFFFFu, prev_m = 0xFFFFFFFFu;
  if (r0 > tb.pos_begin && r0 < r1) {
    prev_key = keys[r0 - 1];
    const uint32_t o_t = (uint32_t)((int64_t)vals[r0 - 1] - nbase);
    prev_m = o_t < n_t ? (uint32_t)message_of_any(off, M, o_t) : 0xFFFFFFFFu;
  }

  CSum carry[NV];
#pragma unroll
  for (int i = 0; i < NV; ++i) carry[i] = CSum{0.f, 0.f};
  RunCounts cc{0u, 0u, 0u};
  uint32_t carry_x = 0u, carry_head = 0u;
  bool carry_active = false, carry_local = false;
  if (r0 < r1 && prev_key == keys[r0]) {
    carry_active = true;
    carry_x = keys[r0] - tb.key_base;
  }
  bool wrote_head_record = false, wrote_tail_record = false;

  // A finished row: counters and debug record, then (if anything was kept)
  // its aggregated gradient into the done slot of position j.  Called by the
  // L lanes of one group.
  auto emit = [&](int j, uint32_t x, uint32_t head_pos, const RunCounts& c, const CSum* s) {
    if (l == 0) {
      ++n_touched;
      if (dbg_count) {
        dbg_count[head_pos] = c.c_all;
        dbg_kept[head_pos] = c.k_occ;
      }
    }
    if (c.k_occ == 0u || x >= v_t) return;
    const float den = row_denominator(a.sparse_den, c.c_all, c.c_kept, M);
#pragma unroll
    for (int e = 0; e < EPL; ++e) {
#pragma unroll
      for (int u = 0; u < VEC; ++u) {
        const int idx = (e * L + l) * VEC + u;
        if (idx < d) gh[j * DW + idx] = __fdiv_rn(csum_value(s[e * VEC + u]), den);
      }
    }
    if (l == 0) {
      sm[j].pad = x;
      sd[j] = 1;
      ++n_applied;
    }
  };

  for (int64_t rb = r0; rb < r1; rb += RS) {
    const int n_round = (int)((r1 - rb) < RS ? (r1 - rb) : RS);
    // ---- per-position metadata
#pragma unroll
    for (int q = 0; q < 2; ++q) {
      const int j = q * 32 + lane;
      if (j < n_round) {
        const uint32_t key = keys[rb + j];
        const uint32_t o_t = (uint32_t)((int64_t)vals[rb + j] - nbase);
        const uint32_t x = key - tb.key_base;
        if (o_t >= n_t || x >= v_t) {
          raise_error(err, ERR_INTERNAL);
          sm[j].row = nullptr;
          sm[j].key = key;
          sm[j].m = 0u;
          sm[j].pad = 0u;
          sm[j].flags = 0u;
          continue;
        }
        const int m = message_of_any(off, M, o_t);
        const uint32_t p = o_t - off[m];
        const int64_t tok = cached ? s_tok[m] : a.tokens[m];
        const float* rowp = cached ? s_rowp[m] : rows_g[m];
        const int64_t ref = a.row_staleness == 0 ? (int64_t)tb.ver[x] : a.k;
        const int64_t diff = ref - tok;
        const uint64_t s = diff > 0 ? (uint64_t)diff : 0ull;
        const bool keep = s <= (uint64_t)(int64_t)a.iota;
        sm[j].row = rowp + (size_t)p * (size_t)d;
        sm[j].key = key;
        sm[j].m = (uint32_t)m;
        sm[j].pad = (uint32_t)(s > 0xFFFFFFFFull ? 0xFFFFFFFFull : s);
        sm[j].flags = keep ? F_KEEP : 0u;
      }
    }
    __syncwarp();
#pragma unroll
    for (int q = 0; q < 2; ++q) {
      const int j = q * 32 + lane;
      if (j < n_round) {
        const uint32_t pk = j == 0 ? prev_key : sm[j - 1].key;
        const uint32_t pm = j == 0 ? prev_m : sm[j - 1].m;
        uint32_t f = sm[j].flags;
        if (f & F_KEEP) ++n_kept_occ;
        const bool head = sm[j].key != pk;
        const bool newmsg = head || sm[j].m != pm;
        if (head) f |= F_HEAD;
        if (newmsg) {
          f |= F_NEWMSG;
          ++n_pairs;
          if (!(f & F_KEEP)) ++n_pairs_dropped;
          const unsigned long long s = sm[j].pad;
          stale_sum += s;
          stale_max = s > stale_max ? s : stale_max;
        }
        sm[j].flags = f;
      }
    }
    __syncwarp();
    prev_key = sm[n_round - 1].key;
    prev_m = sm[n_round - 1].m;

    // ---- each group sums its slice, loading gradient rows in batches of CH
    const int j0 = g * E;
    CSum acc[NV], cont[NV];
#pragma unroll
    for (int i = 0; i < NV; ++i) acc[i] = cont[i] = CSum{0.f, 0.f};
    RunCounts ac{0u, 0u, 0u}, cn{0u, 0u, 0u};
    uint32_t a_x = 0u, a_head = 0u;
    bool in_cont = (j0 < n_round) && !(sm[j0].flags & F_HEAD);
    bool have_open = false;
    int first_head = -1;
#pragma unroll 1
    for (int c0 = 0; c0 < E; c0 += CH) {
      float v[CH][NV];
#pragma unroll
      for (int u = 0; u < CH; ++u) {
        const int j = j0 + c0 + u;
        const bool use = j < n_round && (sm[j].flags & F_KEEP);
        const float* row = use ? sm[j].row : nullptr;
#pragma unroll
        for (int e = 0; e < EPL; ++e) {
          const int idx = (e * L + l) * VEC;
          if (use && idx < d) {
            Vec<VEC>::load(row + idx, &v[u][e * VEC]);
          } else {
#pragma unroll
            for (int w = 0; w < VEC; ++w) v[u][e * VEC + w] = 0.f;
          }
        }
      }
#pragma unroll
      for (int u = 0; u < CH; ++u) {
        const int j = j0 + c0 + u;
        if (j < n_round) {
          const uint32_t f = sm[j].flags;
          if (f & F_HEAD) {
            if (in_cont) {
#pragma unroll
              for (int i = 0; i < NV; ++i) cont[i] = acc[i];
              cn = ac;
              in_cont = false;
              first_head = j;
            } else if (have_open) {
              emit(j - 1, a_x, a_head, ac, acc);
            } else if (first_head < 0) {
              first_head = j;
            }
#pragma unroll
            for (int i = 0; i < NV; ++i) acc[i] = CSum{0.f, 0.f};
            ac = RunCounts{0u, 0u, 0u};
            a_x = sm[j].key - tb.key_base;
            a_head = (uint32_t)(rb + j);
            have_open = true;
          }
          if (f & F_NEWMSG) {
            ++ac.c_all;
            if (f & F_KEEP) ++ac.c_kept;
          }
          if (f & F_KEEP) {
            ++ac.k_occ;
#pragma unroll
            for (int i = 0; i < NV; ++i) csum_add(acc[i], v[u][i]);
          }
        }
      }
    }
    const uint32_t head_mask = __ballot_sync(0xffffffffu, have_open && l == 0);

    // ---- stitch the slices of this round in order
    for (int gg = 0; gg < G; ++gg) {
      if (gg * E >= n_round) break;
      const int src = gg * L + l;
      const bool starts_head = (sm[gg * E].flags & F_HEAD) != 0u;
      const bool has_head = (head_mask >> (gg * L)) & 1u;
      int end_j;  // last position of the carried row, if it completes here
      if (!starts_head) {
#pragma unroll
        for (int i = 0; i < NV; ++i) {
          const float hi = __shfl_sync(0xffffffffu, has_head ? cont[i].hi : acc[i].hi, src);
          const float lo = __shfl_sync(0xffffffffu, has_head ? cont[i].lo : acc[i].lo, src);
          csum_merge(carry[i], hi, lo);
        }
        cc.c_all += __shfl_sync(0xffffffffu, has_head ? cn.c_all : ac.c_all, gg * L);
        cc.c_kept += __shfl_sync(0xffffffffu, has_head ? cn.c_kept : ac.c_kept, gg * L);
        cc.k_occ += __shfl_sync(0xffffffffu, has_head ? cn.k_occ : ac.k_occ, gg * L);
        if (!has_head) continue;
        end_j = __shfl_sync(0xffffffffu, first_head, gg * L) - 1;
      } else {
        end_j = gg * E - 1;
      }
      if (carry_active) {
        if (end_j < 0) {
          raise_error(err, ERR_INTERNAL);  // closed at a round boundary: handled below
        } else if (carry_local) {
          if (g == 0) emit(end_j, carry_x, carry_head, cc, carry);
        } else {
          if (g == 0)
            write_record<VEC, L, EPL>(rec, wg, 0, d, REC_CLOSED, carry_x, 0u, cc, l, carry);
          wrote_head_record = true;
        }
      }
#pragma unroll
      for (int i = 0; i < NV; ++i) {
        carry[i].hi = __shfl_sync(0xffffffffu, acc[i].hi, src);
        carry[i].lo = __shfl_sync(0xffffffffu, acc[i].lo, src);
      }
      cc.c_all = __shfl_sync(0xffffffffu, ac.c_all, gg * L);
      cc.c_kept = __shfl_sync(0xffffffffu, ac.c_kept, gg * L);
      cc.k_occ = __shfl_sync(0xffffffffu, ac.k_occ, gg * L);
      carry_x = __shfl_sync(0xffffffffu, a_x, gg * L);
      carry_head = __shfl_sync(0xffffffffu, a_head, gg * L);
      carry_active = true;
      carry_local = true;
    }

    // ---- does the carried row end with this round?
    const bool last_round = rb + n_round >= r1;
    bool closes;
    if (!last_round)
      closes = keys[rb + n_round] != keys[rb + n_round - 1];
    else
      closes = (r1 == tb.pos_end) || keys[r1] != keys[r1 - 1];
    if (carry_active && closes) {
      if (carry_local) {
        if (g == 0) emit(n_round - 1, carry_x, carry_head, cc, carry);
      } else {
        if (g == 0) write_record<VEC, L, EPL>(rec, wg, 0, d, REC_CLOSED, carry_x, 0u, cc, l, carry);
        wrote_head_record = true;
      }
      carry_active = false;
    }
    if (last_round && carry_active) {
      if (carry_local) {
        if (g == 0)
          write_record<VEC, L, EPL>(rec, wg, 1, d, REC_OWNER, carry_x, carry_head, cc, l, carry);
        wrote_tail_record = true;
      } else {
        if (g == 0) write_record<VEC, L, EPL>(rec, wg, 0, d, REC_PASS, carry_x, 0u, cc, l, carry);
        wrote_head_record = true;
      }
      carry_active = false;
    }
    __syncwarp();

    // ---- update the rows finished in this round, a batch per group at a time
    const uint32_t m0 = __ballot_sync(0xffffffffu, sd[lane] != 0);
    const uint32_t m1 = __ballot_sync(0xffffffffu, sd[lane + 32] != 0);
    const int n0 = __popc(m0);
    const int total = n0 + __popc(m1);
    for (int base = 0; base < total; base += G * APPLY_BATCH) {
      float w[APPLY_BATCH][NV], s0[APPLY_BATCH][NV], s1[APPLY_BATCH][NV];
      int jj[APPLY_BATCH];
      uint32_t xx[APPLY_BATCH];
#pragma unroll
      for (int b = 0; b < APPLY_BATCH; ++b) {
        const int e_i = base + g + G * b;
        jj[b] = -1;
        if (e_i < total) {
          jj[b] = e_i < n0 ? (int)__fns(m0, 0, e_i + 1) : 32 + (int)__fns(m1, 0, e_i - n0 + 1);
          xx[b] = sm[jj[b]].pad;
          const size_t rbase = (size_t)xx[b] * (size_t)d;
#pragma unroll
          for (int e = 0; e < EPL; ++e) {
            const int idx = (e * L + l) * VEC;
            if (idx < d) {
              Vec<VEC>::load(tb.w + rbase + idx, &w[b][e * VEC]);
              Vec<VEC>::load(tb.s0 + rbase + idx, &s0[b][e * VEC]);
              if (tb.opt.kind == 1) Vec<VEC>::load(tb.s1 + rbase + idx, &s1[b][e * VEC]);
            }
          }
        }
      }
#pragma unroll
      for (int b = 0; b < APPLY_BATCH; ++b) {
        if (jj[b] < 0) continue;
        const size_t rbase = (size_t)xx[b] * (size_t)d;
#pragma unroll
        for (int e = 0; e < EPL; ++e) {
          const int idx = (e * L + l) * VEC;
          if (idx < d) {
#pragma unroll
            for (int u = 0; u < VEC; ++u)
              opt_update(tb.opt, w[b][e * VEC + u], s0[b][e * VEC + u], s1[b][e * VEC + u],
                         gh[jj[b] * DW + idx + u]);
            Vec<VEC>::store(tb.w + rbase + idx, &w[b][e * VEC]);
            Vec<VEC>::store(tb.s0 + rbase + idx, &s0[b][e * VEC]);
            if (tb.opt.kind == 1) Vec<VEC>::store(tb.s1 + rbase + idx, &s1[b][e * VEC]);
          }
        }
        if (l == 0) tb.ver[xx[b]] = (int32_t)(a.k + 1);
      }
    }
    __syncwarp();
    sd[lane] = 0;
    sd[lane + 32] = 0;
    __syncwarp();
  }

  if (lane == 0) {
    if (!wrote_head_record) rec.meta[((size_t)wg * 2 + 0) * REC_META] = REC_NONE;
    if (!wrote_tail_record) rec.meta[((size_t)wg * 2 + 1) * REC_META] = REC_NONE;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    n_pairs += __shfl_xor_sync(0xffffffffu, n_pairs, o);
    n_pairs_dropped += __shfl_xor_sync(0xffffffffu, n_pairs_dropped, o);
    stale_sum += __shfl_xor_sync(0xffffffffu, stale_sum, o);
    const unsigned long long y = __shfl_xor_sync(0xffffffffu, stale_max, o);
    stale_max = y > stale_max ? y : stale_max;
    n_touched += __shfl_xor_sync(0xffffffffu, n_touched, o);
    n_applied += __shfl_xor_sync(0xffffffffu, n_applied, o);
    n_kept_occ += __shfl_xor_sync(0xffffffffu, n_kept_occ, o);
  }
  if (lane == 0) {
    if (n_pairs) atomicAdd(&st->pairs, n_pairs);
    if (n_pairs_dropped) atomicAdd(&st->pairs_dropped, n_pairs_dropped);
    if (stale_sum) atomicAdd(&st->row_stale_sum, stale_sum);
    if (stale_max) atomicMax(&st->row_stale_max, stale_max);
    if (n_touched) atomicAdd(&st->rows_touched, n_touched);
    if (n_applied) atomicAdd(&st->rows_applied, n_applied);
    if (n_kept_occ) atomicAdd(&st->occ_kept, n_kept_occ);
  }
}

// Rows that cross warp ranges: the owner (the range where the row starts)
// combines its partial with the following ranges' partials, in range order.
constexpr int FIX_MAX_PER_LANE = 8;  // dims up to 256

__global__ void __launch_bounds__(256)
    k_segsum_fixup(StepArgs a, SegTable tb, int64_t n_warps, SegRecords rec, DevStats* st,
                   uint32_t* dbg_count, uint32_t* dbg_kept, ErrSink err) {
  if (ld_volatile_u32(err.dev) & (ERR_ID_RANGE | ERR_TIMEOUT)) return;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int64_t w = (int64_t)blockIdx.x * 8 + warp;
  if (w >= n_warps) return;
  const uint32_t* m1 = rec.meta + ((size_t)w * 2 + 1) * REC_META;
  if (m1[0] != REC_OWNER) return;
  const int d = tb.d;
  CSum s[FIX_MAX_PER_LANE];
#pragma unroll
  for (int i = 0; i < FIX_MAX_PER_LANE; ++i) {
    const int idx = lane + 32 * i;
    s[i] = CSum{0.f, 0.f};
    if (idx < d) {
      const size_t b = ((size_t)w * 2 + 1) * d + idx;
      s[i] = CSum{rec.hi[b], rec.lo[b]};
    }
  }
  const uint32_t x = m1[1];
  if (x >= (uint32_t)tb.rows) {
    if (lane == 0) raise_error(err, ERR_INTERNAL);
    return;
  }
  RunCounts c{m1[2], m1[3], m1[4]};
  const uint32_t head_pos = m1[5];
  bool closed = false;
  for (int64_t w2 = w + 1; w2 < n_warps; ++w2) {
    const uint32_t* m0 = rec.meta + ((size_t)w2 * 2 + 0) * REC_META;
    const uint32_t type = m0[0];
    if ((type != REC_PASS && type != REC_CLOSED) || m0[1] != x) {
      if (lane == 0) raise_error(err, ERR_INTERNAL);
      return;
    }
#pragma unroll
    for (int i = 0; i < FIX_MAX_PER_LANE; ++i) {
      const int idx = lane + 32 * i;
      if (idx < d) {
        const size_t b = ((size_t)w2 * 2 + 0) * d + idx;
        csum_merge(s[i], rec.hi[b], rec.lo[b]);
      }
    }
    c.c_all += m0[2];
    c.c_kept += m0[3];
    c.k_occ += m0[4];
    if (type == REC_CLOSED) {
      closed = true;
      break;
    }
  }
  if (!closed) {
    if (lane == 0) raise_error(err, ERR_INTERNAL);
    return;
  }
  if (lane == 0) {
    atomicAdd(&st->rows_touched, 1ull);
    if (dbg_count) {
      dbg_count[head_pos] = c.c_all;
      dbg_kept[head_pos] = c.k_occ;
    }
  }
  if (c.k_occ == 0u) return;
  const float den = row_denominator(a.sparse_den, c.c_all, c.c_kept, a.M);
  const size_t rb = (size_t)x * d;
#pragma unroll
  for (int i = 0; i < FIX_MAX_PER_LANE; ++i) {
    const int idx = lane + 32 * i;
    if (idx < d) {
      float w0 = tb.w[rb + idx], s0 = tb.s0[rb + idx];
      float s1 = tb.opt.kind == 1 ? tb.s1[rb + idx] : 0.f;
      opt_update(tb.opt, w0, s0, s1, __fdiv_rn(csum_value(s[i]), den));
      tb.w[rb + idx] = w0;
      tb.s0[rb + idx] = s0;
      if (tb.opt.kind == 1) tb.s1[rb + idx] = s1;
    }
  }
  if (lane == 0) {
    tb.ver[x] = (int32_t)(a.k + 1);
    atomicAdd(&st->rows_applied, 1ull);
  }
}

template <int VEC, int L, int EPL>
void launch_cfg(const StepArgs& a, const SegTable& tb, const uint32_t* keys, const uint32_t* vals,
                int64_t range, int64_t n_warps, SegRecords rec, DevStats* stats,
                uint32_t* dbg_count, uint32_t* dbg_kept, ErrSink err, cudaStream_t s) {
  constexpr int DW = L * EPL * VEC;
  if constexpr (DW <= 64) {
    // rows of up to 64 floats: finished rows are updated in batches per round
    constexpr size_t smem = (size_t)SEG2_WARPS * RS * DW * sizeof(float);
    static bool configured = false;
    if (!configured) {
      cudaFuncSetAttribute(k_segsum_apply2<VEC, L, EPL>,
                           cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
      configured = true;
    }
    const int64_t grid = (n_warps + SEG2_WARPS - 1) / SEG2_WARPS;
    k_segsum_apply2<VEC, L, EPL><<<(unsigned)grid, SEG2_THREADS, smem, s>>>(
        a, tb, keys, vals, range, n_warps, rec, stats, dbg_count, dbg_kept, err);
  } else {
    const int64_t grid = (n_warps + SEG_WARPS - 1) / SEG_WARPS;
    k_segsum_apply<VEC, L, EPL><<<(unsigned)grid, SEG_THREADS, 0, s>>>(
        a, tb, keys, vals, range, n_warps, rec, stats, dbg_count, dbg_kept, err);
  }
}

}  // namespace

// Lane layout for a row width: 16-byte vectors when d is a multiple of 4,
// L lanes per row (a power of two), EPL vectors per lane.
void launch_segsum(const StepArgs& a, const SegTable& tb, const uint32_t* keys,
                   const uint32_t* vals, int64_t range, int64_t n_warps, SegRecords rec,
                   DevStats* stats, uint32_t* dbg_count, uint32_t* dbg_kept, ErrSink err,
                   int /*num_sms*/, cudaStream_t s) {
  const int d = tb.d;
#define GBA_SEG(V, LL, EP) \
  launch_cfg<V, LL, EP>(a, tb, keys, vals, range, n_warps, rec, stats, dbg_count, dbg_kept, err, s)
  if (d % 4 == 0) {
    const int units = d / 4;
    if (units <= 1) GBA_SEG(4, 1, 1);
    else if (units <= 2) GBA_SEG(4, 2, 1);
    else if (units <= 4) GBA_SEG(4, 4, 1);
    else if (units <= 8) GBA_SEG(4, 8, 1);
    else if (units <= 16) GBA_SEG(4, 16, 1);
    else if (units <= 32) GBA_SEG(4, 32, 1);
    else GBA_SEG(4, 32, 2);
  } else {
    if (d <= 2) GBA_SEG(1, 2, 1);
    else if (d <= 4) GBA_SEG(1, 4, 1);
    else if (d <= 8) GBA_SEG(1, 8, 1);
    else if (d <= 16) GBA_SEG(1, 16, 1);
    else if (d <= 32) GBA_SEG(1, 32, 1);
    else if (d <= 64) GBA_SEG(1, 32, 2);
    else if (d <= 128) GBA_SEG(1, 32, 4);
    else GBA_SEG(1, 32, 8);
  }
#undef GBA_SEG
}

void launch_fixup(const StepArgs& a, const SegTable& tb, int64_t n_warps, SegRecords rec,
                  DevStats* stats, uint32_t* dbg_count, uint32_t* dbg_kept, ErrSink err,
                  cudaStream_t s) {
  const int64_t grid = (n_warps + 7) / 8;
  k_segsum_fixup<<<(unsigned)grid, 256, 0, s>>>(a, tb, n_warps, rec, stats, dbg_count, dbg_kept,
                                                err);
}

}  // namespace gba
