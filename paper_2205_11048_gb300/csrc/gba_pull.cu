// Pull responding (Alg. 2): the PS answers a worker with the current embedding
// rows of the IDs it asks for.  One kernel gathers the current rows of one
// table for a list of ids into a caller buffer.
//
// Layout: L lanes per row (the smallest power of two >= d/4, at most 32), each
// lane moving 16-byte pieces when d is a multiple of 4 (rows are then 16-byte
// aligned), one float at a time otherwise; consecutive ids go to consecutive
// lane groups, so the output is written in coalesced runs.  A DIRECT id outside
// [0, V) gets a row of zeros and latches ERR_ID_RANGE in the handle's word.
#include "gba_internal.cuh"

namespace gba {

namespace {

constexpr int PULL_THREADS = 256;

template <bool VEC>
__global__ void __launch_bounds__(PULL_THREADS)
    k_pull_rows(const float* __restrict__ w, int64_t V, int d, int id_mode, uint64_t mod_magic,
                const HashInfo* hinfo, const int64_t* __restrict__ ids, int64_t n,
                float* __restrict__ out, int lg, ErrSink err) {
  const int L = 1 << lg;
  const int lane = threadIdx.x & 31;
  const int l = lane & (L - 1);
  const int64_t groups = (int64_t)gridDim.x * (PULL_THREADS >> lg);
  const int64_t g0 = ((int64_t)blockIdx.x * PULL_THREADS + threadIdx.x) >> lg;
  for (int64_t i = g0; i < n; i += groups) {
    const int64_t id = __ldg(ids + i);
    bool ok = true;
    uint64_t row;
    bool fresh = false;  // HASH: an id never seen gets its initial values
    if (id_mode == 0) {
      ok = id >= 0 && id < V;
      row = ok ? (uint64_t)id : 0ull;
    } else if (id_mode == 1) {
      row = mod_u64((uint64_t)id, (uint64_t)V, mod_magic);
    } else {
      row = hash_find(*hinfo, id);
      fresh = row > hinfo->mask;
      if (fresh) row = 0;
    }
    if (!ok && l == 0) raise_error(err, ERR_ID_RANGE);
    const float* src = w + row * (uint64_t)d;
    float* dst = out + (uint64_t)i * (uint64_t)d;
    if (fresh) {
      for (int q = l; q < d; q += L)
        dst[q] = init_weight(hinfo->seed, hinfo->tag, (uint64_t)id * (uint64_t)d + (uint64_t)q);
      continue;
    }
    if (VEC) {
      const int C = d >> 2;
      for (int q = l; q < C; q += L) {
        float4 v = ok ? __ldg(reinterpret_cast<const float4*>(src) + q)
                      : make_float4(0.f, 0.f, 0.f, 0.f);
        reinterpret_cast<float4*>(dst)[q] = v;
      }
    } else {
      for (int q = l; q < d; q += L) dst[q] = ok ? __ldg(src + q) : 0.f;
    }
  }
}

}  // namespace

void launch_pull_rows(const float* w, int64_t V, int d, int id_mode, uint64_t mod_magic,
                      const HashInfo* hinfo, const int64_t* ids, int64_t n, float* out,
                      ErrSink err, int num_sms, cudaStream_t s) {
  if (n <= 0) return;
  const bool vec = (d & 3) == 0 && ((uintptr_t)out & 15u) == 0;
  const int pieces = vec ? d / 4 : d;
  int lg = 0;
  while ((1 << lg) < pieces && lg < 5) ++lg;
  const int64_t per_block = PULL_THREADS >> lg;
  int64_t grid = (n + per_block - 1) / per_block;
  const int64_t cap = (int64_t)num_sms * 8;
  if (grid > cap) grid = cap;
  if (vec)
    k_pull_rows<true><<<(unsigned)grid, PULL_THREADS, 0, s>>>(w, V, d, id_mode, mod_magic, hinfo, ids, n, out, lg, err);
  else
    k_pull_rows<false><<<(unsigned)grid, PULL_THREADS, 0, s>>>(w, V, d, id_mode, mod_magic, hinfo,
                                                               ids, n, out, lg, err);
}

}  // namespace gba
