// K5 of the GBA aggregate-and-apply step: the dense parameters.
//
// g = (sum over kept messages m of f_m grad_m) / M  (Alg. 2: weighted sum of the
// dense gradients divided by N_a; Appendix A: v_k = (1/M) sum g), then Adagrad
// or Adam in place -- one pass over HBM: every kept gradient is read once, the
// weights and optimizer state are read and written once.
//
// Each persistent CTA walks every gridDim-th tile of DT parameters.  A
// producer warp streams the tile's slice of every kept message into a ring of
// shared-memory stages with 1-D bulk async copies (cp.async.bulk, completion
// counted on an mbarrier per stage); eight consumer warps sum the slices with
// compensated (TwoSum) float arithmetic, release each stage on an "empty"
// mbarrier, and finish the tile with the optimizer.  Every mbarrier wait is
// bounded in time; a wait that gives up latches ERR_TIMEOUT, the CTA stops
// issuing copies, waits (bounded) for the copies it already issued, and exits.
#include "gba_internal.cuh"

namespace gba {

namespace {

#ifndef GBA_DENSE_TILE
#define GBA_DENSE_TILE 2048
#endif
#ifndef GBA_DENSE_STAGES
#define GBA_DENSE_STAGES 8
#endif
constexpr int DT = GBA_DENSE_TILE;       // parameters per tile
constexpr int STAGES = GBA_DENSE_STAGES;  // DT floats each
constexpr int CONSUMER_WARPS = 8;        // 256 threads
constexpr int HALF = CONSUMER_WARPS * 32 * 4;  // floats of one float4 per consumer thread
constexpr int PER = DT / HALF;  // thread c owns [h*HALF + 4c, h*HALF + 4c + 4), h < PER
static_assert(DT % HALF == 0, "a tile is a whole number of float4 rows of the consumers");
constexpr int DENSE_THREADS = (CONSUMER_WARPS + 1) * 32;

__global__ void __launch_bounds__(DENSE_THREADS)
    k_dense_apply(StepArgs a, DenseArgs da, StepScratch sc, ErrSink err, int64_t wait_ns) {
  extern __shared__ __align__(128) unsigned char smem_raw[];
  float* stage_buf = reinterpret_cast<float*>(smem_raw);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem_raw + (size_t)STAGES * DT * sizeof(float));
  uint64_t* empty = full + STAGES;
  __shared__ int s_abort;

  // block-uniform: another kernel may set the word while this block reads it
  if (__syncthreads_or((*(volatile uint32_t*)err.step & (ERR_ID_RANGE | ERR_TIMEOUT)) != 0u)) return;

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  if (tid == 0) {
    for (int i = 0; i < STAGES; ++i) {
      mbar_init(full + i, 1u);
      mbar_init(empty + i, (uint32_t)CONSUMER_WARPS);
    }
    s_abort = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();

  const int n_kept = *sc.n_kept;
  const int64_t D4 = da.D & ~3ll;  // parameters streamed by bulk copies
  // This CTA's tiles of DT parameters (the last one shorter, a multiple of 4
  // so every copy stays 16-byte aligned): blockIdx.x, blockIdx.x + gridDim.x,
  // ...  At any moment the CTAs work on neighbouring tiles, so the copies from
  // the kept messages' buffers touch few DRAM pages and TLB entries.
  const int64_t t0 = (int64_t)blockIdx.x * DT, tstep = (int64_t)gridDim.x * DT;

  if (warp == CONSUMER_WARPS) {
    // ---- producer
    if (lane == 0) {
      uint32_t q = 0;
      bool ok = da.withhold == 0;
      for (int64_t start = t0; start < D4 && ok; start += tstep) {
        const uint32_t bytes = (uint32_t)((D4 - start < DT ? D4 - start : DT) * sizeof(float));
        for (int j = 0; j < n_kept; ++j, ++q) {
          const int stage = (int)(q % STAGES);
          const uint32_t ph = (q / STAGES) & 1u;
          if (!mbar_wait(empty + stage, ph ^ 1u, wait_ns) || *(volatile int*)&s_abort) {
            raise_error(err, ERR_TIMEOUT);
            s_abort = 1;
            ok = false;
            break;
          }
          const float* src = a.dense_ptr[sc.kept_list[j]] + start;
          mbar_arrive_expect_tx(full + stage, bytes);
          bulk_g2s(stage_buf + (size_t)stage * DT, src, bytes, full + stage);
        }
      }
      // Make sure no copy this CTA issued is still landing when it exits.  The
      // copies read valid memory and land within microseconds; this wait has its
      // own one-second bound, independent of the configurable limit.
      const uint32_t n_drain = q < (uint32_t)STAGES ? q : (uint32_t)STAGES;
      for (uint32_t i = 0; i < n_drain; ++i) {
        const uint32_t qq = q - 1 - i;
        mbar_wait(full + (qq % STAGES), (qq / STAGES) & 1u, 1000000000ll);
      }
    }
  } else {
    // ---- consumers: thread c owns parameters [h*HALF + 4c, h*HALF + 4c + 4)
    // of each tile, h < PER
    const int c = tid;
    const float Mf = (float)da.M;
    uint32_t q = 0;
    for (int64_t start = t0; start < D4; start += tstep) {
      const int64_t n = D4 - start < DT ? D4 - start : DT;
      bool mine[PER];
      int64_t e[PER];
      float4 w[PER], s0[PER], s1[PER];
#pragma unroll
      for (int h = 0; h < PER; ++h) {
        const int64_t off = (int64_t)h * HALF + (int64_t)c * 4;
        mine[h] = off < n;
        e[h] = start + off;
        w[h] = s0[h] = s1[h] = make_float4(0.f, 0.f, 0.f, 0.f);
        if (mine[h]) {
          w[h] = *reinterpret_cast<const float4*>(da.w + e[h]);
          s0[h] = *reinterpret_cast<const float4*>(da.s0 + e[h]);
          if (da.opt.kind == 1) s1[h] = *reinterpret_cast<const float4*>(da.s1 + e[h]);
        }
      }
      CSum acc[4 * PER];
#pragma unroll
      for (int i = 0; i < 4 * PER; ++i) acc[i] = CSum{0.f, 0.f};
      bool aborted = false;
      for (int j = 0; j < n_kept; ++j, ++q) {
        const int stage = (int)(q % STAGES);
        const uint32_t ph = (q / STAGES) & 1u;
        // Every lane waits (acquiring the copied bytes); the outcome is made
        // warp-uniform so the warp leaves the loop together.
        const bool ok = __all_sync(0xffffffffu, mbar_wait(full + stage, ph, wait_ns));
        if (!ok) {
          if (lane == 0) {
            raise_error(err, ERR_TIMEOUT);
            s_abort = 1;
          }
          aborted = true;
          break;
        }
        if (a.decay == 0) {
#pragma unroll
          for (int h = 0; h < PER; ++h) {
            if (mine[h]) {
              const float4 v = *reinterpret_cast<const float4*>(stage_buf + (size_t)stage * DT +
                                                                h * HALF + 4 * c);
              csum_add(acc[4 * h + 0], v.x);
              csum_add(acc[4 * h + 1], v.y);
              csum_add(acc[4 * h + 2], v.z);
              csum_add(acc[4 * h + 3], v.w);
            }
          }
        } else {  // weighted: f_m * g with the product's rounding error kept
          const float f = sc.fw[j];
#pragma unroll
          for (int h = 0; h < PER; ++h) {
            if (mine[h]) {
              const float4 v = *reinterpret_cast<const float4*>(stage_buf + (size_t)stage * DT +
                                                                h * HALF + 4 * c);
              csum_add_prod(acc[4 * h + 0], f, v.x);
              csum_add_prod(acc[4 * h + 1], f, v.y);
              csum_add_prod(acc[4 * h + 2], f, v.z);
              csum_add_prod(acc[4 * h + 3], f, v.w);
            }
          }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(empty + stage);
      }
      if (aborted || __shfl_sync(0xffffffffu, *(volatile int*)&s_abort, 0) != 0) break;
#pragma unroll
      for (int h = 0; h < PER; ++h) {
        if (!mine[h]) continue;
        float wv[4] = {w[h].x, w[h].y, w[h].z, w[h].w},
              a0[4] = {s0[h].x, s0[h].y, s0[h].z, s0[h].w},
              a1[4] = {s1[h].x, s1[h].y, s1[h].z, s1[h].w};
#pragma unroll
        for (int i = 0; i < 4; ++i)
          opt_update(da.opt, wv[i], a0[i], a1[i], __fdiv_rn(csum_value(acc[4 * h + i]), Mf));
        *reinterpret_cast<float4*>(da.w + e[h]) = make_float4(wv[0], wv[1], wv[2], wv[3]);
        *reinterpret_cast<float4*>(da.s0 + e[h]) = make_float4(a0[0], a0[1], a0[2], a0[3]);
        if (da.opt.kind == 1)
          *reinterpret_cast<float4*>(da.s1 + e[h]) = make_float4(a1[0], a1[1], a1[2], a1[3]);
      }
    }
    // The last (D mod 4) parameters: plain loads, CTA 0.
    if (blockIdx.x == 0 && c < (int)(da.D - D4)) {
      const int64_t e = D4 + c;
      CSum acc{0.f, 0.f};
      for (int j = 0; j < n_kept; ++j)
        csum_add_prod(acc, a.decay == 0 ? 1.f : sc.fw[j], a.dense_ptr[sc.kept_list[j]][e]);
      float wv = da.w[e], a0 = da.s0[e], a1 = da.opt.kind == 1 ? da.s1[e] : 0.f;
      opt_update(da.opt, wv, a0, a1, __fdiv_rn(csum_value(acc), Mf));
      da.w[e] = wv;
      da.s0[e] = a0;
      if (da.opt.kind == 1) da.s1[e] = a1;
    }
  }
  __syncthreads();
}

// ---------------------------------------------------------------------------
// Eager aggregation (Alg. 2 discussion: because the tokens fix the weights,
// part of the weighted sum may be formed before the step).  Under the FIFO every pushed
// message belongs to a known future step, so its weight is known at push: its
// dense gradient is added to that step's compensated accumulator (hi, lo)
// right away, in push order -- the order the buffered K5 sums in -- and the
// step then reads D accumulators instead of its kept messages.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256)
    k_dense_accumulate(float* __restrict__ hi, float* __restrict__ lo,
                       const float* __restrict__ g, int64_t D, float f, int first) {
  const int64_t D4 = D & ~3ll;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t q = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; q < D4 / 4; q += stride) {
    const float4 v = reinterpret_cast<const float4*>(g)[q];
    const float x[4] = {v.x, v.y, v.z, v.w};
    float4 h4 = make_float4(0.f, 0.f, 0.f, 0.f), l4 = h4;
    if (!first) {
      h4 = reinterpret_cast<const float4*>(hi)[q];
      l4 = reinterpret_cast<const float4*>(lo)[q];
    }
    float hh[4] = {h4.x, h4.y, h4.z, h4.w}, ll[4] = {l4.x, l4.y, l4.z, l4.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      CSum c{hh[i], ll[i]};
      csum_add_prod(c, f, x[i]);
      hh[i] = c.hi;
      ll[i] = c.lo;
    }
    reinterpret_cast<float4*>(hi)[q] = make_float4(hh[0], hh[1], hh[2], hh[3]);
    reinterpret_cast<float4*>(lo)[q] = make_float4(ll[0], ll[1], ll[2], ll[3]);
  }
  if (blockIdx.x == 0 && threadIdx.x < (int)(D - D4)) {
    const int64_t e = D4 + threadIdx.x;
    CSum c{first ? 0.f : hi[e], first ? 0.f : lo[e]};
    csum_add_prod(c, f, g[e]);
    hi[e] = c.hi;
    lo[e] = c.lo;
  }
}

// The step's dense update from its accumulator (has_sum 0: no message was
// kept, the gradient is 0).
__global__ void __launch_bounds__(256)
    k_dense_apply_eager(DenseArgs da, const float* __restrict__ hi, const float* __restrict__ lo,
                        int has_sum, ErrSink err) {
  if (__syncthreads_or((*(volatile uint32_t*)err.step & (ERR_ID_RANGE | ERR_TIMEOUT)) != 0u)) return;
  const float Mf = (float)da.M;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < da.D; e += stride) {
    const float v = has_sum ? __fadd_rn(hi[e], lo[e]) : 0.f;
    float w = da.w[e], s0 = da.s0[e], s1 = da.opt.kind == 1 ? da.s1[e] : 0.f;
    opt_update(da.opt, w, s0, s1, __fdiv_rn(v, Mf));
    da.w[e] = w;
    da.s0[e] = s0;
    if (da.opt.kind == 1) da.s1[e] = s1;
  }
}

}  // namespace

size_t dense_smem_bytes() { return (size_t)STAGES * DT * sizeof(float) + 2 * STAGES * sizeof(uint64_t); }

cudaError_t configure_dense() {
  return cudaFuncSetAttribute(k_dense_apply, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              (int)dense_smem_bytes());
}

void launch_dense(const StepArgs& a, const DenseArgs& da, StepScratch sc, ErrSink err,
                  int64_t wait_ns, int num_sms, cudaStream_t s) {
  const size_t smem = dense_smem_bytes();
  const int64_t n_tiles = ((da.D & ~3ll) + DT - 1) / DT;
  static const int bps = [&]() {  // persistent: as many CTAs as fit on an SM
    int b = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&b, k_dense_apply, DENSE_THREADS, smem) !=
            cudaSuccess ||
        b < 1)
      b = 1;
    return b;
  }();
  int64_t grid = (int64_t)num_sms * bps;
  if (grid > n_tiles) grid = n_tiles;
  if (grid < 1) grid = 1;
  k_dense_apply<<<(unsigned)grid, DENSE_THREADS, smem, s>>>(a, da, sc, err, wait_ns);
}

void launch_dense_accumulate(float* hi, float* lo, const float* g, int64_t D, float f, bool first,
                             int num_sms, cudaStream_t s) {
  int64_t grid = (D / 4 + 255) / 256;
  if (grid > (int64_t)num_sms * 8) grid = (int64_t)num_sms * 8;
  if (grid < 1) grid = 1;
  k_dense_accumulate<<<(unsigned)grid, 256, 0, s>>>(hi, lo, g, D, f, first ? 1 : 0);
}

void launch_dense_eager(const DenseArgs& da, const float* hi, const float* lo, bool has_sum,
                        ErrSink err, int num_sms, cudaStream_t s) {
  int64_t grid = (da.D + 255) / 256;
  if (grid > (int64_t)num_sms * 8) grid = (int64_t)num_sms * 8;
  if (grid < 1) grid = 1;
  k_dense_apply_eager<<<(unsigned)grid, 256, 0, s>>>(da, hi, lo, has_sum ? 1 : 0, err);
}

}  // namespace gba
