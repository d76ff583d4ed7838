// gba_sort_ids_static: the library's id sort for callers that cannot allocate.
//
// Some callers must not allocate device memory at the point where they need a
// sort: runtimes that reserve all device memory up front and hand none out
// later, or an allocator's own hooks, which cannot re-enter cudaMalloc.  This
// entry point runs the same histogram and onesweep kernels as a global step,
// but takes its scratch from one fixed array in device global memory that is
// part of the library image, so the call itself never allocates.
//
// Properties a caller must know:
//  - The scratch array is file-scope device memory of GBA_STATIC_SORT_BYTES
//    bytes; every GPU that loads the library keeps it until the process exits.
//  - The first call on a device (with that device current) looks up the
//    array's device address with cudaGetSymbolAddress.
//  - The call is synchronous: it waits for its stream before returning.
//  - All calls share the one array and it keeps the previous call's contents.
//    The per-call counters are cleared at the start of each call; calls whose
//    work overlaps on the GPU (two streams, or two host threads) race.
//  - At most GBA_STATIC_SORT_MAX_IDS ids per call; larger inputs are refused.
//  - The outputs hold the sorted result only when GBA_OK is returned.
#include <cuda_runtime.h>

#include <atomic>
#include <mutex>

#include "gba.h"
#include "gba_internal.cuh"

namespace gba {
namespace {

constexpr int64_t kMaxIds = GBA_STATIC_SORT_MAX_IDS;
constexpr int64_t kTile = SORT_TILE_KEYS;  // keys per onesweep tile
constexpr int64_t kMaxTiles = (kMaxIds + kTile - 1) / kTile;
constexpr int kMaxDevices = 64;

// Byte layout of the scratch array.
constexpr size_t kOffKeys = 0;
constexpr size_t kOffVals = kOffKeys + (size_t)kMaxIds * 4;
constexpr size_t kOffStatus = kOffVals + (size_t)kMaxIds * 4;
constexpr size_t kOffHist = kOffStatus + (size_t)kMaxTiles * 256 * 8;
constexpr size_t kOffTiles = kOffHist + 4 * 256 * 4;
constexpr size_t kOffMsgOff = kOffTiles + 16;
constexpr size_t kOffIdsPtr = kOffMsgOff + 16;
constexpr size_t kOffNbase = kOffIdsPtr + 16;
constexpr size_t kOffTinfo = kOffNbase + 16;
constexpr size_t kOffErr = kOffTinfo + 32;  // TableInfo is 24 bytes
static_assert(sizeof(gba::TableInfo) <= 32, "TableInfo outgrew its scratch slot");
constexpr size_t kBytes = kOffErr + 16;
#if GBA_SORT_TILE == 2048
static_assert(kBytes == GBA_STATIC_SORT_BYTES, "scratch size differs from the header");
#else
static_assert(kBytes <= GBA_STATIC_SORT_BYTES, "scratch larger than the header's size");
#endif

static __device__ __align__(256) unsigned char g_sort_scratch[kBytes];

unsigned char* g_scratch_addr[kMaxDevices] = {};
std::mutex g_setup_mutex;
std::atomic<uint32_t> g_epoch[kMaxDevices];

// Writes this call's one-message step description and clears the counters
// and error words that must start at zero.
__global__ void k_static_setup(unsigned char* base, const int64_t* ids, int64_t n, int64_t rows,
                               int32_t id_mode) {
  const int t = threadIdx.x;
  uint32_t* hist = reinterpret_cast<uint32_t*>(base + kOffHist);
  for (int i = t; i < 4 * 256; i += blockDim.x) hist[i] = 0u;
  if (t == 0) {
    uint32_t* tiles = reinterpret_cast<uint32_t*>(base + kOffTiles);
    for (int i = 0; i < 4; ++i) tiles[i] = 0u;
    uint32_t* off = reinterpret_cast<uint32_t*>(base + kOffMsgOff);
    off[0] = 0u;
    off[1] = (uint32_t)n;
    *reinterpret_cast<const int64_t**>(base + kOffIdsPtr) = ids;
    int64_t* nb = reinterpret_cast<int64_t*>(base + kOffNbase);
    nb[0] = 0;
    nb[1] = n;
    TableInfo* ti = reinterpret_cast<TableInfo*>(base + kOffTinfo);
    ti->V = rows;
    ti->key_base = 0u;
    ti->id_mode = id_mode;
    ti->mod_magic = ~0ull / (uint64_t)rows;
    uint32_t* err = reinterpret_cast<uint32_t*>(base + kOffErr);
    err[0] = 0u;
    err[1] = 0u;
  }
}

// The scratch array's device address for the current device (looked up once).
cudaError_t scratch_for_current_device(unsigned char** out, int* dev_out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(g_setup_mutex);
  if (!g_scratch_addr[dev]) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_sort_scratch);
    if (e != cudaSuccess) return e;
    g_scratch_addr[dev] = static_cast<unsigned char*>(p);
    g_epoch[dev].store(0u);
  }
  *out = g_scratch_addr[dev];
  *dev_out = dev;
  return cudaSuccess;
}

}  // namespace
}  // namespace gba

extern "C" gba_status gba_sort_ids_static(const int64_t* ids, int64_t n, int64_t rows,
                                          int32_t id_mode, uint32_t* rows_out,
                                          uint32_t* order_out, void* cuda_stream) {
  using namespace gba;
  if (n < 0 || n > kMaxIds) return GBA_E_ARG;
  if (rows < 1 || rows >= 0xFFFFFFFFll) return GBA_E_ARG;
  if (id_mode != GBA_ID_DIRECT && id_mode != GBA_ID_MODULO) return GBA_E_ARG;
  if (n > 0 && (!ids || !rows_out || !order_out)) return GBA_E_ARG;
  if (n == 0) return GBA_OK;
  // A launch error left by earlier, unrelated work on this thread would be
  // reported (and cleared) by the check after the launches below: refuse to
  // run instead, and leave that error in place for its owner.
  if (cudaPeekAtLastError() != cudaSuccess) return GBA_E_CUDA;
  cudaStream_t s = (cudaStream_t)cuda_stream;
  unsigned char* base = nullptr;
  int dev = 0;
  if (scratch_for_current_device(&base, &dev) != cudaSuccess) return GBA_E_CUDA;

  k_static_setup<<<1, 256, 0, s>>>(base, ids, n, rows, id_mode);

  StepArgs a{};
  a.k = 0;
  a.M = 1;
  a.T = 1;
  a.N = n;
  a.msg_off = reinterpret_cast<const uint32_t*>(base + kOffMsgOff);
  a.ids_ptr = reinterpret_cast<const int64_t* const*>(base + kOffIdsPtr);
  a.nbase = reinterpret_cast<const int64_t*>(base + kOffNbase);
  a.tinfo = reinterpret_cast<const TableInfo*>(base + kOffTinfo);
  StepScratch sc{};
  sc.hist = reinterpret_cast<uint32_t*>(base + kOffHist);
  sc.tile_counter = reinterpret_cast<uint32_t*>(base + kOffTiles);
  uint32_t* err_words = reinterpret_cast<uint32_t*>(base + kOffErr);
  ErrSink err{err_words, err_words, err_words + 1};

  uint64_t kmax = (uint64_t)rows - 1;
  int bits = 1;
  while (bits < 32 && (kmax >> bits) != 0) ++bits;
  const int passes = (bits + 7) / 8;

  int grid = (int)((n + 255) / 256);
  if (grid > 152 * 8) grid = 152 * 8;
  // Ping-pong between the scratch pair and the caller's outputs so that the
  // last pass lands in the outputs; the first pass reads the keys the
  // histogram kernel wrote into the buffer that pass does not write.
  uint32_t* tmp_k = reinterpret_cast<uint32_t*>(base + kOffKeys);
  uint32_t* tmp_v = reinterpret_cast<uint32_t*>(base + kOffVals);
  unsigned long long* status = reinterpret_cast<unsigned long long*>(base + kOffStatus);
  uint32_t* keys0 = ((passes - 1) % 2) == 0 ? tmp_k : rows_out;
  launch_sort_histogram(a, passes, sc, keys0, err, grid, s);
  const uint32_t* kin = keys0;
  const uint32_t* vin = nullptr;
  for (int p = 0; p < passes; ++p) {
    const bool to_out = ((passes - 1 - p) % 2) == 0;
    uint32_t* ko = to_out ? rows_out : tmp_k;
    uint32_t* vo = to_out ? order_out : tmp_v;
    uint32_t ep = g_epoch[dev].fetch_add(1u) + 1u;
    if (ep == 0u) ep = g_epoch[dev].fetch_add(1u) + 1u;
    launch_onesweep(a, p == 0, p, kin, vin, ko, vo, sc, status, ep, err, 2000000000ll, s);
    kin = ko;
    vin = vo;
  }
  if (cudaGetLastError() != cudaSuccess) return GBA_E_CUDA;
  uint32_t word = 0;
  if (cudaMemcpyAsync(&word, err_words, sizeof word, cudaMemcpyDeviceToHost, s) != cudaSuccess)
    return GBA_E_CUDA;
  if (cudaStreamSynchronize(s) != cudaSuccess) return GBA_E_CUDA;
  if (word & ERR_ID_RANGE) return GBA_E_ID_RANGE;
  if (word & ERR_TIMEOUT) return GBA_E_DEVICE_TIMEOUT;
  if (word) return GBA_E_CUDA;
  return GBA_OK;
}
