// K3 + K4 of the GBA aggregate-and-apply step: per unique row of the sorted
// occurrence array, decay each occurrence by the row's step tag against its
// message's token (Eq. (1), Alg. 2), sum the kept gradient rows, divide by the
// number of messages that encountered the row, apply the optimizer to the row
// and its state in place, and set the row's tag to k + 1.
//
// Work is split by occurrences, not by rows, so Zipf-hot rows cost no more per
// occurrence than cold ones.  Each warp owns a contiguous range of the sorted
// array.  Lane l holds elements [l*EPL, (l+1)*EPL) of the row being summed, so
// the walk over the positions is warp-uniform: the per-position metadata
// (row pointer, head / kept / new-message flags) is computed by all lanes in
// parallel for a round of 64 positions, then the warp streams through the
// round's gradient rows eight at a time (loads issued before they are summed),
// accumulating with compensated (TwoSum) float arithmetic.  A finished row's
// aggregated gradient goes to a small per-warp queue in shared memory; the
// queue is applied eight rows at a time, all state loads issued first.  Rows
// crossing warp ranges leave partial sums in a record that the fixup kernel
// combines in range order.  Every order is fixed, so results are bit-identical
// run to run.
#include "gba_internal.cuh"

namespace gba {

namespace {

constexpr int SEG_WARPS = 4;
constexpr int SEG_THREADS = SEG_WARPS * 32;
constexpr int RS = 32;  // positions per round: one per lane
// finished rows per update batch: 8 rows of up to 64 floats, fewer wider ones
template <int EPL>
__host__ __device__ constexpr int pb_rows() { return EPL <= 2 ? 8 : (EPL == 4 ? 4 : 2); }
template <int EPL>
__host__ __device__ constexpr int queue_rows() { return pb_rows<EPL>(); }
// dynamic shared memory of one block: staged rows and the finished-row queue
template <int EPL>
__host__ __device__ constexpr size_t seg_dyn_smem() {
  return (size_t)SEG_WARPS * (RS + queue_rows<EPL>()) * 32 * EPL * sizeof(float);
}

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}
__device__ __forceinline__ void stage_wait_all() {
  asm volatile("cp.async.commit_group;\n\tcp.async.wait_group 0;" ::: "memory");
}
constexpr int MSG_CACHE = 256;  // messages whose lookups are cached in shared memory

// record types
constexpr uint32_t REC_NONE = 0u, REC_PASS = 1u, REC_CLOSED = 2u, REC_OWNER = 3u;
constexpr int REC_META = 6;  // type, x, c_all, c_kept, k_occ, head_pos


__device__ __forceinline__ uint32_t ld_volatile_u32(const uint32_t* p) {
  return *(const volatile uint32_t*)p;
}

// Denominator of the row's weighted sum.
__device__ __forceinline__ float row_denominator(int mode, uint32_t c_all, uint32_t c_kept,
                                                 int M) {
  const uint32_t den = mode == 0 ? c_all : (mode == 1 ? c_kept : (uint32_t)M);
  return (float)den;
}

// EPL consecutive floats at p (vector access when VECOK: p is EPL*4-aligned).
template <int EPL, bool VECOK>
__device__ __forceinline__ void load_lane(const float* p, int n_valid, float* v) {
  if constexpr (VECOK && EPL == 1) {
    v[0] = *p;
  } else if constexpr (VECOK && EPL == 2) {
    const float2 q = *reinterpret_cast<const float2*>(p);
    v[0] = q.x; v[1] = q.y;
  } else if constexpr (VECOK && EPL % 4 == 0) {
#pragma unroll
    for (int i = 0; i < EPL; i += 4) {
      const float4 q = *reinterpret_cast<const float4*>(p + i);
      v[i] = q.x; v[i + 1] = q.y; v[i + 2] = q.z; v[i + 3] = q.w;
    }
  } else {
#pragma unroll
    for (int i = 0; i < EPL; ++i) v[i] = i < n_valid ? p[i] : 0.f;
  }
}
template <int EPL, bool VECOK>
__device__ __forceinline__ void store_lane(float* p, int n_valid, const float* v) {
  if constexpr (VECOK && EPL == 1) {
    *p = v[0];
  } else if constexpr (VECOK && EPL == 2) {
    *reinterpret_cast<float2*>(p) = make_float2(v[0], v[1]);
  } else if constexpr (VECOK && EPL % 4 == 0) {
#pragma unroll
    for (int i = 0; i < EPL; i += 4)
      *reinterpret_cast<float4*>(p + i) = make_float4(v[i], v[i + 1], v[i + 2], v[i + 3]);
  } else {
#pragma unroll
    for (int i = 0; i < EPL; ++i)
      if (i < n_valid) p[i] = v[i];
  }
}

struct RunCounts {
  uint32_t c_all, c_kept, k_occ;
};

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

// One round's segment (a maximal run of equal keys inside the round).
struct SegInfo {
  uint32_t x;         // row
  uint32_t head_pos;  // sorted position of its first occurrence in the round
  uint32_t c_all, c_kept;
  uint32_t kmask;     // kept positions of the round in this segment
  uint32_t is_head;   // 1 if the row starts here, 0 if it continues from before
};

// Lane j copies gradient row j (d floats) into its staging slot: 16-byte
// copies when d is a multiple of 4 (rows are then 16-byte aligned), else
// 4-byte copies.
__device__ __forceinline__ void stage_row(float* dst, const float* src, int d) {
  if ((d & 3) == 0) {
    for (int i = 0; i < d; i += 4)
      asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_u32(dst + i)),
                   "l"(src + i)
                   : "memory");
  } else {
    for (int i = 0; i < d; ++i)
      asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(smem_u32(dst + i)),
                   "l"(src + i)
                   : "memory");
  }
}

template <int EPL>
__device__ __forceinline__ void write_record(const SegRecords& rec, int64_t wg, int slot, int d,
                                             uint32_t type, uint32_t x, uint32_t head_pos,
                                             const RunCounts& c, int lane, int n_mine,
                                             const CSum* acc) {
  const size_t base = ((size_t)wg * 2 + slot) * (size_t)d + (size_t)lane * EPL;
#pragma unroll
  for (int e = 0; e < EPL; ++e)
    if (e < n_mine) {
      rec.hi[base + e] = acc[e].hi;
      rec.lo[base + e] = acc[e].lo;
    }
  if (lane == 0) {
    uint32_t* m = rec.meta + ((size_t)wg * 2 + slot) * REC_META;
    m[1] = x;
    m[2] = c.c_all;
    m[3] = c.c_kept;
    m[4] = c.k_occ;
    m[5] = head_pos;
    m[0] = type;
  }
}

// A finished row: counters and debug record; if anything was kept, its
// compensated sums go to the warp's queue with the row and the denominator.
template <int EPL>
__device__ __forceinline__ void enqueue_row(uint32_t x, uint32_t head_pos, const RunCounts& rc,
                                            const StepArgs& a, int M, uint32_t v_t, int lane,
                                            const CSum* acc, float* pend, uint32_t* pend_x,
                                            float* pend_den, int& npend, uint32_t& n_touched,
                                            uint32_t& n_applied, uint32_t* dbg_count,
                                            uint32_t* dbg_kept) {
  if (lane == 0) {
    ++n_touched;
    if (dbg_count) {
      dbg_count[head_pos] = rc.c_all;
      dbg_kept[head_pos] = rc.k_occ;
    }
  }
  if (rc.k_occ == 0u || x >= v_t) return;  // nothing kept: no step, tag unchanged
#pragma unroll
  for (int e = 0; e < EPL; ++e) pend[npend * 32 * EPL + lane * EPL + e] = csum_value(acc[e]);
  if (lane == 0) {
    pend_x[npend] = x;
    pend_den[npend] = row_denominator(a.sparse_den, rc.c_all, rc.c_kept, M);
    ++n_applied;
  }
  ++npend;
}

// Applies the queued rows, a batch at a time: all state loads of a batch
// first, then the updates.
template <int EPL, bool VECOK>
__device__ __noinline__ void flush_rows(const StepArgs& a, const SegTable& tb, int lane, int e0,
                                        int n_mine, bool active, const float* pend,
                                        const uint32_t* pend_x, const float* pend_den,
                                        int& npend) {
  constexpr int PB = pb_rows<EPL>();
  const int d = tb.d;
  __syncwarp();
  for (int b0 = 0; b0 < npend; b0 += PB) {
    float w[PB][EPL], s0[PB][EPL], s1[PB][EPL];
#pragma unroll
    for (int i = 0; i < PB; ++i) {
      if (b0 + i < npend && active) {
        const size_t rb = (size_t)pend_x[b0 + i] * (size_t)d + e0;
        load_lane<EPL, VECOK>(tb.w + rb, n_mine, w[i]);
        load_lane<EPL, VECOK>(tb.s0 + rb, n_mine, s0[i]);
        if (tb.opt.kind == 1) load_lane<EPL, VECOK>(tb.s1 + rb, n_mine, s1[i]);
      }
    }
#pragma unroll
    for (int i = 0; i < PB; ++i) {
      if (b0 + i < npend) {
        const uint32_t x = pend_x[b0 + i];
        if (active) {
          const float den = pend_den[b0 + i];
          const size_t rb = (size_t)x * (size_t)d + e0;
#pragma unroll
          for (int e = 0; e < EPL; ++e) {
            const float v = pend[(b0 + i) * 32 * EPL + lane * EPL + e];
            opt_update(tb.opt, w[i][e], s0[i][e], s1[i][e], den == 1.0f ? v : __fdiv_rn(v, den));
          }
          store_lane<EPL, VECOK>(tb.w + rb, n_mine, w[i]);
          store_lane<EPL, VECOK>(tb.s0 + rb, n_mine, s0[i]);
          if (tb.opt.kind == 1) store_lane<EPL, VECOK>(tb.s1 + rb, n_mine, s1[i]);
        }
        if (lane == 0) tb.ver[x] = (int32_t)(a.k + 1);
      }
    }
  }
  npend = 0;
  __syncwarp();
}

template <int EPL, bool VECOK>
__global__ void __launch_bounds__(SEG_THREADS, EPL == 1 ? 4 : (EPL == 2 ? 3 : 1))
    k_segsum_apply(StepArgs a, SegTable tb, const uint32_t* __restrict__ keys,
                   const uint32_t* __restrict__ vals, int64_t range, int64_t n_warps,
                   SegRecords rec, DevStats* st, uint32_t* dbg_count, uint32_t* dbg_kept,
                   ErrSink err) {
  constexpr int PB = pb_rows<EPL>();
  constexpr int QR = queue_rows<EPL>();
  constexpr int DS = 32 * EPL;  // staged row stride (floats)
  __shared__ uint32_t s_off[MSG_CACHE + 1];
  __shared__ int64_t s_tok[MSG_CACHE];
  __shared__ const float* s_rowp[MSG_CACHE];
  __shared__ SegInfo s_seg[SEG_WARPS][RS];
  __shared__ uint32_t s_pend_x[SEG_WARPS][QR];
  __shared__ float s_pend_den[SEG_WARPS][QR];
  extern __shared__ __align__(16) float s_dyn[];  // staged rows, then the queue

  if (ld_volatile_u32(err.step) & (ERR_ID_RANGE | ERR_TIMEOUT)) return;
  const int M = a.M;
  const uint32_t* off_g = a.msg_off + (size_t)tb.t * (M + 1);
  const float* const* rows_g = a.rows_ptr + (size_t)tb.t * M;
  const bool cached = M <= MSG_CACHE;
  if (cached) {
    for (int i = threadIdx.x; i <= M; i += SEG_THREADS) s_off[i] = off_g[i];
    for (int i = threadIdx.x; i < M; i += SEG_THREADS) {
      s_tok[i] = a.tokens[i];
      s_rowp[i] = rows_g[i];
    }
  }
  __syncthreads();
  const uint32_t* off = cached ? s_off : off_g;

  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int64_t wg = (int64_t)blockIdx.x * SEG_WARPS + warp;
  if (wg >= n_warps) return;
  const int d = tb.d;
  const int e0 = lane * EPL;  // first row element of this lane
  const int n_mine = d - e0 < 0 ? 0 : (d - e0 < EPL ? d - e0 : EPL);
  const bool active = n_mine > 0;
  const int64_t r0 = tb.pos_begin + wg * range;
  const int64_t r1 = (r0 + range < tb.pos_end) ? r0 + range : tb.pos_end;
  const int64_t nbase = a.nbase[tb.t];
  const uint32_t n_t = (uint32_t)(tb.pos_end - tb.pos_begin);
  const uint32_t v_t = (uint32_t)tb.rows;
  const uint32_t lt_mask = (1u << lane) - 1u;

  uint32_t n_pairs = 0, n_pairs_dropped = 0, n_touched = 0, n_applied = 0, n_kept_occ = 0;
  unsigned long long stale_sum = 0, stale_max = 0;

  float* stage = s_dyn + (size_t)warp * RS * DS;
  float* pend = s_dyn + (size_t)SEG_WARPS * RS * DS + (size_t)warp * QR * DS;
  uint32_t* pend_x = s_pend_x[warp];
  float* pend_den = s_pend_den[warp];
  SegInfo* seg = s_seg[warp];
  int npend = 0;

  // The row (run) open at the current position; the whole warp holds it,
  // lane l its elements [l*EPL, (l+1)*EPL).
  CSum acc[EPL];
#pragma unroll
  for (int e = 0; e < EPL; ++e) acc[e] = CSum{0.f, 0.f};
  RunCounts rc{0u, 0u, 0u};
  uint32_t run_x = 0u, run_head = 0u;
  bool run_active = false, run_local = false;
  bool wrote_head_record = false, wrote_tail_record = false;

  uint32_t prev_key = 0xFFFFFFFFu, prev_m = 0xFFFFFFFFu;
  if (r0 > tb.pos_begin && r0 < r1) {
    prev_key = keys[r0 - 1];
    const uint32_t o_t = (uint32_t)((int64_t)vals[r0 - 1] - nbase);
    prev_m = o_t < n_t ? (uint32_t)message_of_any(off, M, o_t) : 0xFFFFFFFFu;
    if (prev_key == keys[r0]) {  // the range begins inside a row owned by an earlier range
      run_active = true;
      run_x = keys[r0] - tb.key_base;
    }
  }

  for (int64_t rb = r0; rb < r1; rb += RS) {
    const int n_round = (int)((r1 - rb) < RS ? (r1 - rb) : RS);
    const bool valid = lane < n_round;
    // ---- lane j: metadata of position rb + j; stage its gradient row if kept
    uint32_t key = 0xFFFFFFFFu, m = 0xFFFFFFFEu, stale = 0u;
    bool keep = false;
    if (valid) {
      key = keys[rb + lane];
      const uint32_t o_t = (uint32_t)((int64_t)vals[rb + lane] - nbase);
      const uint32_t x = key - tb.key_base;
      if (o_t >= n_t || x >= v_t) {
        // cannot happen for a correctly sorted array; never touch memory with it
        raise_error(err, ERR_INTERNAL);
      } else {
        m = (uint32_t)message_of_any(off, M, o_t);
        const uint32_t p = o_t - off[m];
        const int64_t tok = cached ? s_tok[m] : a.tokens[m];
        const float* rowp = (cached ? s_rowp[m] : rows_g[m]) + (size_t)p * (size_t)d;
        const int64_t ref = a.row_staleness == 0 ? (int64_t)tb.ver[x] : a.k;
        const int64_t diff = ref - tok;
        const uint64_t sl = diff > 0 ? (uint64_t)diff : 0ull;
        keep = sl <= (uint64_t)(int64_t)a.iota;
        stale = (uint32_t)(sl > 0xFFFFFFFFull ? 0xFFFFFFFFull : sl);
        if (keep) stage_row(stage + lane * DS, rowp, d);
      }
    }
    uint32_t pk = __shfl_up_sync(0xffffffffu, key, 1);
    uint32_t pm = __shfl_up_sync(0xffffffffu, m, 1);
    if (lane == 0) {
      pk = prev_key;
      pm = prev_m;
    }
    const bool head = valid && key != pk;
    const bool newmsg = valid && (head || m != pm);
    if (keep) ++n_kept_occ;
    if (newmsg) {
      ++n_pairs;
      if (!keep) ++n_pairs_dropped;
      stale_sum += stale;
      stale_max = stale > stale_max ? stale : stale_max;
    }
    const uint32_t Hm = __ballot_sync(0xffffffffu, head);
    const uint32_t Km = __ballot_sync(0xffffffffu, keep);
    const uint32_t Nm = __ballot_sync(0xffffffffu, newmsg);
    const uint32_t Vm = __ballot_sync(0xffffffffu, valid);
    // ---- segments of the round (position 0 always starts one): lane-parallel
    const uint32_t Bm = (Hm | 1u) & Vm;
    if ((Bm >> lane) & 1u) {
      const uint32_t above = lane == 31 ? 0u : (Bm & ~((2u << lane) - 1u));
      const int end = above ? __ffs(above) - 1 : n_round;
      const uint32_t rng = (end >= 32 ? 0xFFFFFFFFu : ((1u << end) - 1u)) & ~lt_mask;
      SegInfo& sg = seg[__popc(Bm & lt_mask)];
      sg.x = key - tb.key_base;
      sg.head_pos = (uint32_t)(rb + lane);
      sg.c_all = __popc(Nm & rng);
      sg.c_kept = __popc(Nm & Km & rng);
      sg.kmask = Km & rng;
      sg.is_head = head ? 1u : 0u;
    }
    const int R = __popc(Bm);
    prev_key = __shfl_sync(0xffffffffu, key, n_round - 1);
    prev_m = __shfl_sync(0xffffffffu, m, n_round - 1);
    stage_wait_all();
    __syncwarp();

    // ---- walk the round segment by segment (uniform control flow)
    for (int r = 0; r < R; ++r) {
      const SegInfo sg = seg[r];
      if (sg.is_head) {
        if (run_active) {
          // finish the open row: queue its aggregated gradient (or, for a row
          // that began in an earlier range, leave the partial for the fixup)
          if (!run_local) {
            write_record<EPL>(rec, wg, 0, d, REC_CLOSED, run_x, 0u, rc, lane, n_mine, acc);
            wrote_head_record = true;
          } else {
            enqueue_row<EPL>(run_x, run_head, rc, a, M, v_t, lane, acc, pend, pend_x, pend_den,
                             npend, n_touched, n_applied, dbg_count, dbg_kept);
            if (npend >= PB)
              flush_rows<EPL, VECOK>(a, tb, lane, e0, n_mine, active, pend, pend_x, pend_den,
                                     npend);
          }
        }
#pragma unroll
        for (int e = 0; e < EPL; ++e) acc[e] = CSum{0.f, 0.f};
        rc = RunCounts{sg.c_all, sg.c_kept, (uint32_t)__popc(sg.kmask)};
        run_x = sg.x;
        run_head = sg.head_pos;
        run_active = true;
        run_local = true;
      } else {
        rc.c_all += sg.c_all;
        rc.c_kept += sg.c_kept;
        rc.k_occ += __popc(sg.kmask);
      }
      uint32_t km = sg.kmask;
      while (km) {
        const int j = __ffs(km) - 1;
        km &= km - 1u;
        float v[EPL];
        load_lane<EPL, true>(stage + j * DS + e0, EPL, v);
#pragma unroll
        for (int e = 0; e < EPL; ++e) csum_add(acc[e], v[e]);
      }
    }
    __syncwarp();
  }

  // ---- end of the range: the open row ends here or continues in the next range
  if (run_active) {
    const bool closes = (r1 == tb.pos_end) || keys[r1] != keys[r1 - 1];
    if (closes) {
      if (!run_local) {
        write_record<EPL>(rec, wg, 0, d, REC_CLOSED, run_x, 0u, rc, lane, n_mine, acc);
        wrote_head_record = true;
      } else {
        enqueue_row<EPL>(run_x, run_head, rc, a, M, v_t, lane, acc, pend, pend_x, pend_den,
                         npend, n_touched, n_applied, dbg_count, dbg_kept);
      }
    } else if (run_local) {
      write_record<EPL>(rec, wg, 1, d, REC_OWNER, run_x, run_head, rc, lane, n_mine, acc);
      wrote_tail_record = true;
    } else {
      write_record<EPL>(rec, wg, 0, d, REC_PASS, run_x, 0u, rc, lane, n_mine, acc);
      wrote_head_record = true;
    }
  }
  if (npend > 0)
    flush_rows<EPL, VECOK>(a, tb, lane, e0, n_mine, active, pend, pend_x, pend_den, npend);
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
    n_kept_occ += __shfl_xor_sync(0xffffffffu, n_kept_occ, o);
  }
  if (lane == 0) {
    if (n_pairs) atomicAdd(&st->pairs, (unsigned long long)n_pairs);
    if (n_pairs_dropped) atomicAdd(&st->pairs_dropped, (unsigned long long)n_pairs_dropped);
    if (stale_sum) atomicAdd(&st->row_stale_sum, stale_sum);
    if (stale_max) atomicMax(&st->row_stale_max, stale_max);
    if (n_touched) atomicAdd(&st->rows_touched, (unsigned long long)n_touched);
    if (n_applied) atomicAdd(&st->rows_applied, (unsigned long long)n_applied);
    if (n_kept_occ) atomicAdd(&st->occ_kept, (unsigned long long)n_kept_occ);
  }
}

// ---------------------------------------------------------------------------
// Rows of up to 64 floats: most unique rows of a round occur once, so they are
// handled lane-parallel, and the optimizer runs with one lane per row.
//
// Per round of 32 positions: lane j computes position j's metadata and stages
// its gradient row in shared memory; the round's segments (maximal runs of
// equal keys) are found with ballots.  A segment that starts and ends inside
// the round with at most one kept occurrence is queued by its own lane (its
// row copied, no arithmetic).  The first segment (which may continue the row
// open from the previous round), segments with several kept occurrences, and
// the last segment (which may continue into the next round) are summed by the
// whole warp, lane = element, with compensated arithmetic.  Queued rows are
// applied with lane = row: each lane streams its row's gradient, weights and
// optimizer state in 16-byte pieces.
// ---------------------------------------------------------------------------
constexpr int QCAP = 64;  // queued rows per warp

template <int EPL>
__host__ __device__ constexpr int row_stride() { return 32 * EPL + 4; }  // floats, bank-skewed
template <int EPL>
__host__ __device__ constexpr size_t rows_dyn_smem() {
  return (size_t)SEG_WARPS * (RS + QCAP) * row_stride<EPL>() * sizeof(float);
}

__device__ __forceinline__ void copy_row_smem(float* dst, const float* src, int d) {
  if ((d & 3) == 0) {
    for (int i = 0; i < d; i += 4)
      *reinterpret_cast<float4*>(dst + i) = *reinterpret_cast<const float4*>(src + i);
  } else {
    for (int i = 0; i < d; ++i) dst[i] = src[i];
  }
}

// Applies queued rows [0, npend).  When d is a multiple of 4, L = d/4 lanes
// share a row, each lane one 16-byte piece (so a row is one coalesced access)
// and the warp updates 32/L rows at a time; otherwise one lane per row.
__device__ __noinline__ void apply_queue(const StepArgs& a, const SegTable& tb, int lane,
                                         const float* pend, const uint32_t* pend_x,
                                         const float* pend_den, int qs, int& npend) {
  const int d = tb.d;
  const bool adam = tb.opt.kind == 1;
  __syncwarp();
  if ((d & 3) == 0) {
    const int L = d >> 2;                 // lanes per row (d <= 64: L <= 16)
    const int G = 32 / L;                 // rows per pass
    const int g = lane / L, l = lane - g * L;
    const bool on = g < G;                // lanes past G * L idle (L not a power of two)
    for (int i0 = 0; i0 < npend; i0 += 2 * G) {
      // two rows per lane group in flight
      const int ia = i0 + g, ib = i0 + G + g;
      const bool va = on && ia < npend, vb = on && ib < npend;
      float4 wa, aa, ba, wb, ab, bb;
      uint32_t xa = 0u, xb = 0u;
      if (va) {
        xa = pend_x[ia];
        const size_t r = (size_t)xa * d + 4 * l;
        wa = *reinterpret_cast<const float4*>(tb.w + r);
        aa = *reinterpret_cast<const float4*>(tb.s0 + r);
        if (adam) ba = *reinterpret_cast<const float4*>(tb.s1 + r);
      }
      if (vb) {
        xb = pend_x[ib];
        const size_t r = (size_t)xb * d + 4 * l;
        wb = *reinterpret_cast<const float4*>(tb.w + r);
        ab = *reinterpret_cast<const float4*>(tb.s0 + r);
        if (adam) bb = *reinterpret_cast<const float4*>(tb.s1 + r);
      }
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const bool v = h == 0 ? va : vb;
        if (!v) continue;
        const int i = h == 0 ? ia : ib;
        const uint32_t x = h == 0 ? xa : xb;
        float4 wv = h == 0 ? wa : wb, av = h == 0 ? aa : ab, bv = h == 0 ? ba : bb;
        const float4 gv = *reinterpret_cast<const float4*>(pend + (size_t)i * qs + 4 * l);
        const float den = pend_den[i];
        float* wp = &wv.x;
        float* ap = &av.x;
        float* bp = &bv.x;
        const float* gp = &gv.x;
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          float bk = adam ? bp[k] : 0.f;
          opt_update(tb.opt, wp[k], ap[k], bk, den == 1.0f ? gp[k] : __fdiv_rn(gp[k], den));
          bp[k] = bk;
        }
        const size_t r = (size_t)x * d + 4 * l;
        *reinterpret_cast<float4*>(tb.w + r) = wv;
        *reinterpret_cast<float4*>(tb.s0 + r) = av;
        if (adam) *reinterpret_cast<float4*>(tb.s1 + r) = bv;
        if (l == 0) tb.ver[x] = (int32_t)(a.k + 1);
      }
    }
  } else {
    for (int b0 = 0; b0 < npend; b0 += 32) {
      const int i = b0 + lane;
      if (i < npend) {
        const uint32_t x = pend_x[i];
        const float den = pend_den[i];
        const float* g = pend + (size_t)i * qs;
        float* w = tb.w + (size_t)x * d;
        float* s0 = tb.s0 + (size_t)x * d;
        float* s1 = adam ? tb.s1 + (size_t)x * d : nullptr;
        for (int c = 0; c < d; ++c) {
          float wk = w[c], ak = s0[c], bk = adam ? s1[c] : 0.f;
          opt_update(tb.opt, wk, ak, bk, den == 1.0f ? g[c] : __fdiv_rn(g[c], den));
          w[c] = wk;
          s0[c] = ak;
          if (adam) s1[c] = bk;
        }
        tb.ver[x] = (int32_t)(a.k + 1);
      }
    }
  }
  npend = 0;
  __syncwarp();
}

template <int EPL>
__global__ void __launch_bounds__(SEG_THREADS, EPL == 1 ? 3 : 2)
    k_segsum_rows(StepArgs a, SegTable tb, const uint32_t* __restrict__ keys,
                  const uint32_t* __restrict__ vals, int64_t range, int64_t n_warps,
                  SegRecords rec, DevStats* st, uint32_t* dbg_count, uint32_t* dbg_kept,
                  ErrSink err) {
  constexpr int SS = row_stride<EPL>();
  __shared__ uint32_t s_off[MSG_CACHE + 1];
  __shared__ int64_t s_tok[MSG_CACHE];
  __shared__ const float* s_rowp[MSG_CACHE];
  __shared__ uint4 s_seg[SEG_WARPS][RS];  // by start position: x, head_pos, kmask, counts
  __shared__ uint32_t s_pend_x[SEG_WARPS][QCAP];
  __shared__ float s_pend_den[SEG_WARPS][QCAP];
  extern __shared__ __align__(16) float s_dyn[];  // staged rows, then the queue

  if (ld_volatile_u32(err.step) & (ERR_ID_RANGE | ERR_TIMEOUT)) return;
  const int M = a.M;
  const uint32_t* off_g = a.msg_off + (size_t)tb.t * (M + 1);
  const float* const* rows_g = a.rows_ptr + (size_t)tb.t * M;
  const bool cached = M <= MSG_CACHE;
  if (cached) {
    for (int i = threadIdx.x; i <= M; i += SEG_THREADS) s_off[i] = off_g[i];
    for (int i = threadIdx.x; i < M; i += SEG_THREADS) {
      s_tok[i] = a.tokens[i];
      s_rowp[i] = rows_g[i];
    }
  }
  __syncthreads();
  const uint32_t* off = cached ? s_off : off_g;

  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int64_t wg = (int64_t)blockIdx.x * SEG_WARPS + warp;
  if (wg >= n_warps) return;
  const int d = tb.d;
  const int qs = ((d + 3) & ~3) + 4;  // queued row stride
  const int e0 = lane * EPL;
  const int n_mine = d - e0 < 0 ? 0 : (d - e0 < EPL ? d - e0 : EPL);
  const int64_t r0 = tb.pos_begin + wg * range;
  const int64_t r1 = (r0 + range < tb.pos_end) ? r0 + range : tb.pos_end;
  const int64_t nbase = a.nbase[tb.t];
  const uint32_t n_t = (uint32_t)(tb.pos_end - tb.pos_begin);
  const uint32_t v_t = (uint32_t)tb.rows;
  const uint32_t lt_mask = (1u << lane) - 1u;
  const int mode = a.sparse_den;

  uint32_t n_pairs = 0, n_pairs_dropped = 0, n_touched = 0, n_applied = 0, n_kept_occ = 0;
  unsigned long long stale_sum = 0, stale_max = 0;

  float* stage = s_dyn + (size_t)warp * RS * SS;
  float* pend = s_dyn + (size_t)SEG_WARPS * RS * SS + (size_t)warp * QCAP * SS;
  uint32_t* pend_x = s_pend_x[warp];
  float* pend_den = s_pend_den[warp];
  uint4* seg = s_seg[warp];
  int npend = 0;

  CSum acc[EPL];
#pragma unroll
  for (int e = 0; e < EPL; ++e) acc[e] = CSum{0.f, 0.f};
  RunCounts rc{0u, 0u, 0u};
  uint32_t run_x = 0u, run_head = 0u;
  bool run_active = false, run_local = false;
  bool wrote_head_record = false, wrote_tail_record = false;

  uint32_t prev_key = 0xFFFFFFFFu, prev_m = 0xFFFFFFFFu;
  if (r0 > tb.pos_begin && r0 < r1) {
    prev_key = keys[r0 - 1];
    const uint32_t o_t = (uint32_t)((int64_t)vals[r0 - 1] - nbase);
    prev_m = o_t < n_t ? (uint32_t)message_of_any(off, M, o_t) : 0xFFFFFFFFu;
    if (prev_key == keys[r0]) {  // the range begins inside a row owned by an earlier range
      run_active = true;
      run_x = keys[r0] - tb.key_base;
    }
  }

  // the warp-held row is complete: queue it (or hand it to the fixup kernel)
  auto finish_run = [&]() {
    if (!run_local) {
      write_record<EPL>(rec, wg, 0, d, REC_CLOSED, run_x, 0u, rc, lane, n_mine, acc);
      wrote_head_record = true;
      return;
    }
    if (lane == 0) {
      ++n_touched;
      if (dbg_count) {
        dbg_count[run_head] = rc.c_all;
        dbg_kept[run_head] = rc.k_occ;
      }
    }
    if (rc.k_occ == 0u || run_x >= v_t) return;
#pragma unroll
    for (int e = 0; e < EPL; ++e)
      if (e < n_mine) pend[npend * qs + e0 + e] = csum_value(acc[e]);
    if (lane == 0) {
      pend_x[npend] = run_x;
      pend_den[npend] = row_denominator(mode, rc.c_all, rc.c_kept, M);
      ++n_applied;
    }
    ++npend;
  };

  for (int64_t rb = r0; rb < r1; rb += RS) {
    const int n_round = (int)((r1 - rb) < RS ? (r1 - rb) : RS);
    const bool valid = lane < n_round;
    // ---- lane j: metadata of position rb + j; its gradient row is staged if kept
    uint32_t key = 0xFFFFFFFFu, m = 0xFFFFFFFEu, stale = 0u;
    bool keep = false;
    const float* my_row = nullptr;
    if (valid) {
      key = keys[rb + lane];
      const uint32_t o_t = (uint32_t)((int64_t)vals[rb + lane] - nbase);
      const uint32_t x = key - tb.key_base;
      if (o_t >= n_t || x >= v_t) {
        raise_error(err, ERR_INTERNAL);  // cannot happen for a correctly sorted array
      } else {
        m = (uint32_t)message_of_any(off, M, o_t);
        const uint32_t p = o_t - off[m];
        const int64_t tok = cached ? s_tok[m] : a.tokens[m];
        const float* rowp = (cached ? s_rowp[m] : rows_g[m]) + (size_t)p * (size_t)d;
        const int64_t ref = a.row_staleness == 0 ? (int64_t)tb.ver[x] : a.k;
        const int64_t diff = ref - tok;
        const uint64_t sl = diff > 0 ? (uint64_t)diff : 0ull;
        keep = sl <= (uint64_t)(int64_t)a.iota;
        stale = (uint32_t)(sl > 0xFFFFFFFFull ? 0xFFFFFFFFull : sl);
        my_row = rowp;
      }
    }
    uint32_t pk = __shfl_up_sync(0xffffffffu, key, 1);
    uint32_t pm = __shfl_up_sync(0xffffffffu, m, 1);
    if (lane == 0) {
      pk = prev_key;
      pm = prev_m;
    }
    const bool head = valid && key != pk;
    const bool newmsg = valid && (head || m != pm);
    if (keep) ++n_kept_occ;
    if (newmsg) {
      ++n_pairs;
      if (!keep) ++n_pairs_dropped;
      stale_sum += stale;
      stale_max = stale > stale_max ? stale : stale_max;
    }
    const uint32_t Hm = __ballot_sync(0xffffffffu, head);
    const uint32_t Km = __ballot_sync(0xffffffffu, keep);
    const uint32_t Nm = __ballot_sync(0xffffffffu, newmsg);
    const uint32_t Vm = __ballot_sync(0xffffffffu, valid);
    // ---- stage the kept gradient rows: L = d/4 lanes per row, one 16-byte
    // piece each (a row is one coalesced access); 4-byte copies otherwise
    if ((d & 3) == 0) {
      const int L = d >> 2, G = 32 / L;
      const int g = lane / L, l = lane - g * L;
      for (int j0 = 0; j0 < n_round; j0 += G) {
        const int j = j0 + g;
        const float* src = (const float*)__shfl_sync(0xffffffffu, (unsigned long long)my_row,
                                                     j < 32 ? j : 31);
        if (g < G && j < n_round && ((Km >> j) & 1u))
          asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(
                           smem_u32(stage + j * SS + 4 * l)),
                       "l"(src + 4 * l)
                       : "memory");
      }
    } else if (keep) {
      stage_row(stage + lane * SS, my_row, d);
    }
    const uint32_t Bm = (Hm | 1u) & Vm;  // segment starts (position 0 always starts one)
    const int last_start = 31 - __clz(Bm);
    const bool starts = (Bm >> lane) & 1u;
    bool single = false, single_apply = false;
    uint32_t kmask = 0u, c_all = 0u, c_kept = 0u;
    if (starts) {
      const uint32_t above = lane == 31 ? 0u : (Bm & ~((2u << lane) - 1u));
      const int end = above ? __ffs(above) - 1 : n_round;
      const uint32_t rng = (end >= 32 ? 0xFFFFFFFFu : ((1u << end) - 1u)) & ~lt_mask;
      kmask = Km & rng;
      c_all = __popc(Nm & rng);
      c_kept = __popc(Nm & Km & rng);
      single = lane > 0 && lane < last_start && __popc(kmask) <= 1;
      single_apply = single && kmask != 0u;
      seg[lane] = make_uint4(key - tb.key_base, (uint32_t)(rb + lane), kmask,
                             c_all | (c_kept << 8) | (head ? 1u << 16 : 0u));
    }
    const uint32_t Sm = __ballot_sync(0xffffffffu, single_apply);
    const uint32_t Um = Bm & ~__ballot_sync(0xffffffffu, single);
    prev_key = __shfl_sync(0xffffffffu, key, n_round - 1);
    prev_m = __shfl_sync(0xffffffffu, m, n_round - 1);
    stage_wait_all();
    __syncwarp();
    // a round queues at most one row per segment plus the row it closes
    if (npend > QCAP - 33) apply_queue(a, tb, lane, pend, pend_x, pend_den, qs, npend);

    // ---- rows that occur once in the round, inside it: their own lane queues them
    if (single) {
      ++n_touched;
      if (dbg_count) {
        dbg_count[rb + lane] = c_all;
        dbg_kept[rb + lane] = __popc(kmask);
      }
      if (single_apply) {
        const int slot = npend + __popc(Sm & lt_mask);
        const int pj = __ffs(kmask) - 1;
        copy_row_smem(pend + slot * qs, stage + pj * SS, d);
        pend_x[slot] = key - tb.key_base;
        pend_den[slot] = row_denominator(mode, c_all, c_kept, M);
        ++n_applied;
      }
    }
    npend += __popc(Sm);

    // ---- the other segments, in order, summed by the whole warp
    uint32_t um = Um;
    while (um) {
      const int j = __ffs(um) - 1;
      um &= um - 1u;
      const uint4 sg = seg[j];
      const bool is_head = (sg.w >> 16) & 1u;
      const uint32_t s_call = sg.w & 0xFFu, s_ckept = (sg.w >> 8) & 0xFFu;
      if (!is_head) {  // continues the open row (only at j == 0)
        rc.c_all += s_call;
        rc.c_kept += s_ckept;
        rc.k_occ += __popc(sg.z);
      } else {
        if (run_active) finish_run();  // the open row ended before this head
#pragma unroll
        for (int e = 0; e < EPL; ++e) acc[e] = CSum{0.f, 0.f};
        rc = RunCounts{s_call, s_ckept, (uint32_t)__popc(sg.z)};
        run_x = sg.x;
        run_head = sg.y;
        run_active = true;
        run_local = true;
      }
      uint32_t km = sg.z;
      while (km) {
        const int pj = __ffs(km) - 1;
        km &= km - 1u;
        float v[EPL];
        load_lane<EPL, true>(stage + pj * SS + e0, EPL, v);
#pragma unroll
        for (int e = 0; e < EPL; ++e) csum_add(acc[e], v[e]);
      }
      // a segment before the round's last one ends inside the round
      if (j < last_start) {
        finish_run();
        run_active = false;
      }
    }
    __syncwarp();
  }

  // ---- end of the range: the open row ends here or continues in the next range
  if (run_active) {
    const bool closes = (r1 == tb.pos_end) || keys[r1] != keys[r1 - 1];
    if (closes) {
      finish_run();
    } else if (run_local) {
      write_record<EPL>(rec, wg, 1, d, REC_OWNER, run_x, run_head, rc, lane, n_mine, acc);
      wrote_tail_record = true;
    } else {
      write_record<EPL>(rec, wg, 0, d, REC_PASS, run_x, 0u, rc, lane, n_mine, acc);
      wrote_head_record = true;
    }
  }
  if (npend > 0) apply_queue(a, tb, lane, pend, pend_x, pend_den, qs, npend);
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
    n_kept_occ += __shfl_xor_sync(0xffffffffu, n_kept_occ, o);
    n_touched += __shfl_xor_sync(0xffffffffu, n_touched, o);
    n_applied += __shfl_xor_sync(0xffffffffu, n_applied, o);
  }
  if (lane == 0) {
    if (n_pairs) atomicAdd(&st->pairs, (unsigned long long)n_pairs);
    if (n_pairs_dropped) atomicAdd(&st->pairs_dropped, (unsigned long long)n_pairs_dropped);
    if (stale_sum) atomicAdd(&st->row_stale_sum, stale_sum);
    if (stale_max) atomicMax(&st->row_stale_max, stale_max);
    if (n_touched) atomicAdd(&st->rows_touched, (unsigned long long)n_touched);
    if (n_applied) atomicAdd(&st->rows_applied, (unsigned long long)n_applied);
    if (n_kept_occ) atomicAdd(&st->occ_kept, (unsigned long long)n_kept_occ);
  }
}

// Rows that cross warp ranges: the owner (the range where the row starts)
// combines its partial with the following ranges' partials, in range order.
constexpr int FIX_MAX_PER_LANE = 8;  // dims up to 256

__global__ void __launch_bounds__(256)
    k_segsum_fixup(StepArgs a, SegTable tb, int64_t n_warps, SegRecords rec, DevStats* st,
                   uint32_t* dbg_count, uint32_t* dbg_kept, ErrSink err) {
  if (ld_volatile_u32(err.step) & (ERR_ID_RANGE | ERR_TIMEOUT)) return;
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
  // Walk the following ranges in order; their record headers are read a window
  // at a time (independent loads), then their partial sums are merged in order.
  constexpr int FIX_WIN = 8;
  bool closed = false;
  for (int64_t wb = w + 1; wb < n_warps && !closed; wb += FIX_WIN) {
    uint32_t ty[FIX_WIN], rx[FIX_WIN];
#pragma unroll
    for (int i = 0; i < FIX_WIN; ++i) {
      const int64_t w2 = wb + i;
      ty[i] = REC_NONE;
      rx[i] = 0u;
      if (w2 < n_warps) {
        const uint32_t* m0 = rec.meta + ((size_t)w2 * 2 + 0) * REC_META;
        ty[i] = m0[0];
        rx[i] = m0[1];
      }
    }
#pragma unroll
    for (int i = 0; i < FIX_WIN; ++i) {
      const int64_t w2 = wb + i;
      if (closed || w2 >= n_warps) break;
      if ((ty[i] != REC_PASS && ty[i] != REC_CLOSED) || rx[i] != x) {
        if (lane == 0) raise_error(err, ERR_INTERNAL);
        return;
      }
      const uint32_t* m0 = rec.meta + ((size_t)w2 * 2 + 0) * REC_META;
#pragma unroll
      for (int k = 0; k < FIX_MAX_PER_LANE; ++k) {
        const int idx = lane + 32 * k;
        if (idx < d) {
          const size_t b = ((size_t)w2 * 2 + 0) * d + idx;
          csum_merge(s[k], rec.hi[b], rec.lo[b]);
        }
      }
      c.c_all += m0[2];
      c.c_kept += m0[3];
      c.k_occ += m0[4];
      if (ty[i] == REC_CLOSED) closed = true;
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

template <int EPL, bool VECOK>
int64_t launch_cfg(const StepArgs& a, const SegTable& tb, const uint32_t* keys,
                   const uint32_t* vals, SegRecords rec, int64_t max_warps, DevStats* stats,
                   uint32_t* dbg_count, uint32_t* dbg_kept, ErrSink err, int num_sms,
                   cudaStream_t s) {
  constexpr size_t smem = seg_dyn_smem<EPL>();
  static int blocks_per_sm = 0;  // static + dynamic shared memory may pass 48 KB
  if (blocks_per_sm == 0) {
    cudaFuncSetAttribute(k_segsum_apply<EPL, VECOK>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                         (int)smem);
    int b = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&b, k_segsum_apply<EPL, VECOK>, SEG_THREADS,
                                                      smem) != cudaSuccess || b < 1)
      b = 1;
    blocks_per_sm = b;
  }
  // One wave of resident warps, each owning an equal range of whole rounds.
  const int64_t Nt = tb.pos_end - tb.pos_begin;
  int64_t target = (int64_t)num_sms * blocks_per_sm * SEG_WARPS;
  if (target > max_warps) target = max_warps;
  int64_t range = (Nt + target - 1) / target;
  range = ((range + RS - 1) / RS) * RS;
  if (range < RS) range = RS;
  const int64_t n_warps = (Nt + range - 1) / range;
  const int64_t grid = (n_warps + SEG_WARPS - 1) / SEG_WARPS;
  k_segsum_apply<EPL, VECOK><<<(unsigned)grid, SEG_THREADS, smem, s>>>(
      a, tb, keys, vals, range, n_warps, rec, stats, dbg_count, dbg_kept, err);
  return n_warps;
}


template <int EPL>
int64_t launch_rows(const StepArgs& a, const SegTable& tb, const uint32_t* keys,
                    const uint32_t* vals, SegRecords rec, int64_t max_warps, DevStats* stats,
                    uint32_t* dbg_count, uint32_t* dbg_kept, ErrSink err, int num_sms,
                    cudaStream_t s) {
  constexpr size_t smem = rows_dyn_smem<EPL>();
  static int blocks_per_sm = 0;
  if (blocks_per_sm == 0) {
    cudaFuncSetAttribute(k_segsum_rows<EPL>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                         (int)smem);
    int b = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&b, k_segsum_rows<EPL>, SEG_THREADS,
                                                      smem) != cudaSuccess || b < 1)
      b = 1;
    blocks_per_sm = b;
  }
  const int64_t Nt = tb.pos_end - tb.pos_begin;
  int64_t target = (int64_t)num_sms * blocks_per_sm * SEG_WARPS;
  if (target > max_warps) target = max_warps;
  int64_t range = (Nt + target - 1) / target;
  range = ((range + RS - 1) / RS) * RS;
  if (range < RS) range = RS;
  const int64_t n_warps = (Nt + range - 1) / range;
  const int64_t grid = (n_warps + SEG_WARPS - 1) / SEG_WARPS;
  k_segsum_rows<EPL><<<(unsigned)grid, SEG_THREADS, smem, s>>>(a, tb, keys, vals, range, n_warps,
                                                               rec, stats, dbg_count, dbg_kept,
                                                               err);
  return n_warps;
}

}  // namespace

// Rows of up to 64 floats take the lane-parallel kernel; wider rows the
// warp-per-element one (EPL = elements per lane, vector accesses when d is a
// multiple of EPL).  Returns the number of warp ranges (the fixup kernel's work).
int64_t launch_segsum(const StepArgs& a, const SegTable& tb, const uint32_t* keys,
                      const uint32_t* vals, SegRecords rec, int64_t max_warps, DevStats* stats,
                      uint32_t* dbg_count, uint32_t* dbg_kept, ErrSink err, int num_sms,
                      cudaStream_t s) {
  const int d = tb.d;
  if (d <= 32)
    return launch_rows<1>(a, tb, keys, vals, rec, max_warps, stats, dbg_count, dbg_kept, err,
                          num_sms, s);
  if (d <= 64)
    return launch_rows<2>(a, tb, keys, vals, rec, max_warps, stats, dbg_count, dbg_kept, err,
                          num_sms, s);
#define GBA_SEG(EP, VO)                                                                        \
  return launch_cfg<EP, VO>(a, tb, keys, vals, rec, max_warps, stats, dbg_count, dbg_kept, err, \
                            num_sms, s)
  if (d <= 128) {
    if (d % 4 == 0) GBA_SEG(4, true);
    GBA_SEG(4, false);
  }
  if (d % 8 == 0) GBA_SEG(8, true);
  GBA_SEG(8, false);
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
