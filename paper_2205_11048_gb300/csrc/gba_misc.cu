// Initialisation of parameters and state, and the bounded-wait self test.
#include "gba_internal.cuh"

namespace gba {

namespace {

__global__ void k_init_params(float* __restrict__ w, float* __restrict__ s0,
                              float* __restrict__ s1, int64_t n, int32_t kind, float init_acc,
                              uint64_t seed, uint64_t tag) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const float a0 = kind == 0 ? init_acc : 0.f;
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < n; e += stride) {
    w[e] = init_weight(seed, tag, (uint64_t)e);
    s0[e] = a0;
    if (kind == 1) s1[e] = 0.f;
  }
}

__global__ void k_fill_i32(int32_t* p, int64_t n, int32_t v) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < n; e += stride) p[e] = v;
}

// Waits on a flag that nothing sets, with the library's bounded wait, and
// reports whether the wait gave up.
__global__ void k_wait_selftest(const uint32_t* flag, int64_t limit_ns, uint32_t* result) {
  const uint64_t t0 = globaltimer_ns();
  uint32_t gave_up = 0;
  while (*(const volatile uint32_t*)flag == 0u) {
    if ((int64_t)(globaltimer_ns() - t0) > limit_ns) {
      gave_up = 1;
      break;
    }
  }
  *result = gave_up;
}

int grid_for(int64_t n) {
  int64_t g = (n + 255) / 256;
  if (g > 152 * 16) g = 152 * 16;
  return g < 1 ? 1 : (int)g;
}

}  // namespace

void launch_init_table(float* w, float* s0, float* s1, int32_t* ver, int64_t rows, int32_t d,
                       int32_t kind, float init_acc, uint64_t seed, uint64_t tag,
                       cudaStream_t s) {
  const int64_t n = rows * (int64_t)d;
  k_init_params<<<grid_for(n), 256, 0, s>>>(w, s0, s1, n, kind, init_acc, seed, tag);
  k_fill_i32<<<grid_for(rows), 256, 0, s>>>(ver, rows, 0);
}

void launch_init_dense(float* w, float* s0, float* s1, int64_t D, int32_t kind, float init_acc,
                       uint64_t seed, uint64_t tag, cudaStream_t s) {
  if (D > 0) k_init_params<<<grid_for(D), 256, 0, s>>>(w, s0, s1, D, kind, init_acc, seed, tag);
}

int launch_wait_selftest(int64_t limit_ns, cudaStream_t s, uint32_t* d_word, uint32_t* result) {
  // d_word[0]: the flag (zero, never set); d_word[1]: the kernel's report
  if (cudaMemsetAsync(d_word, 0, 2 * sizeof(uint32_t), s) != cudaSuccess) return -1;
  k_wait_selftest<<<1, 1, 0, s>>>(d_word, limit_ns, d_word + 1);
  if (cudaMemcpyAsync(result, d_word + 1, sizeof(uint32_t), cudaMemcpyDeviceToHost, s) !=
      cudaSuccess)
    return -1;
  if (cudaStreamSynchronize(s) != cudaSuccess) return -1;
  return 0;
}

namespace {

__global__ void k_hash_clear(unsigned long long* keys, uint64_t slots) {
  const uint64_t stride = (uint64_t)gridDim.x * blockDim.x;
  for (uint64_t i = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; i < slots; i += stride)
    keys[i] = HASH_EMPTY;
}

// Every occupied slot of `from` moves to its slot in `to` (no id repeats, so
// the insert never meets its own id), with its row, state and tag.
__global__ void k_hash_rehash(HashInfo from, HashInfo to) {
  const uint64_t stride = (uint64_t)gridDim.x * blockDim.x;
  for (uint64_t i = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; i <= from.mask; i += stride) {
    const unsigned long long key = from.keys[i];
    if (key == HASH_EMPTY) continue;
    uint64_t slot = splitmix64(key) & to.mask;
    for (uint64_t probe = 0; probe <= to.mask; ++probe, slot = (slot + 1) & to.mask)
      if (atomicCAS(to.keys + slot, HASH_EMPTY, key) == HASH_EMPTY) break;
    for (int j = 0; j < from.d; ++j) {
      to.w[slot * from.d + j] = from.w[i * from.d + j];
      to.s0[slot * from.d + j] = from.s0[i * from.d + j];
      if (from.kind == 1) to.s1[slot * from.d + j] = from.s1[i * from.d + j];
    }
    to.ver[slot] = from.ver[i];
  }
}

__global__ void k_hash_lookup(const HashInfo* hinfo, const int64_t* ids, int64_t n, int64_t* slots) {
  const HashInfo hi = *hinfo;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) {
    const uint64_t s = hash_find(hi, ids[i]);
    slots[i] = s > hi.mask ? -1 : (int64_t)s;
  }
}

}  // namespace

void launch_hash_clear(unsigned long long* keys, uint64_t slots, cudaStream_t s) {
  k_hash_clear<<<grid_for((int64_t)slots), 256, 0, s>>>(keys, slots);
}

void launch_hash_rehash(HashInfo from, HashInfo to, cudaStream_t s) {
  k_hash_rehash<<<grid_for((int64_t)from.mask + 1), 256, 0, s>>>(from, to);
}

void launch_hash_lookup(const HashInfo* hinfo, const int64_t* ids, int64_t n, int64_t* slots,
                        cudaStream_t s) {
  if (n > 0) k_hash_lookup<<<grid_for(n), 256, 0, s>>>(hinfo, ids, n, slots);
}

int kernel_binary_version() {
  cudaFuncAttributes attr{};
  if (cudaFuncGetAttributes(&attr, k_init_params) != cudaSuccess) return -1;
  return attr.binaryVersion;
}

}  // namespace gba
