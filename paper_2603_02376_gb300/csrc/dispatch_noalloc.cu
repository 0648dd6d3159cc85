// moe_dispatch_noalloc: moe_dispatch for callers that cannot allocate device memory.
//
// Some callers can't call cudaMalloc at all: a plugin running inside a host
// framework that owns every byte of device memory and hands out none after
// start-up; a serving loop whose memory was planned once and must not grow or
// fragment; code on a latency-critical path, where cudaMalloc (and cudaFree)
// may implicitly synchronise the whole device. Such a caller may also have no
// workspace to hand over. This variant of moe_dispatch therefore keeps the
// permutation's only scratch -- the per-chunk expert histograms and their
// prefix sums -- in a file-scope __device__ array of fixed size, which every GPU
// that loads this library holds until the process exits.
//
// The array's name in host code is only a host-side stand-in, not a device
// address; a kernel handed the stand-in would fault or, where the GPU can reach
// host memory, silently use the wrong memory. So the first call on each device
// (with that device current) asks the runtime for the real device address with
// cudaGetSymbolAddress and caches it; make that first call before any stream
// capture. Kernels then receive that address. moe_shutdown forgets the cached
// addresses (after cudaDeviceReset the array is loaded again elsewhere).
//
// All calls on a device share the one array and it keeps the previous call's
// contents. Nothing in it needs to start at zero: the histogram kernel writes
// every entry it owns before the scan reads it. Calls whose work overlaps on
// the GPU (different streams without ordering between them) race on the array.
#include <mutex>

#include "common.cuh"

namespace {

// Two halves: chunk histograms, then their per-expert prefix sums.
__device__ __align__(256) int32_t g_dispatch_scratch[2 * MOE_DISPATCH_NOALLOC_MAX_ENTRIES];

constexpr int kMaxDevices = 64;
std::mutex g_scratch_mu;
int32_t* g_scratch_ptr[kMaxDevices] = {};

// Device address of the scratch array on the current device (set up once per device).
moe_status scratch_address(int32_t** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return MOE_ERR_CUDA;
  std::lock_guard<std::mutex> lk(g_scratch_mu);
  if (!g_scratch_ptr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_dispatch_scratch) != cudaSuccess || p == nullptr)
      return MOE_ERR_CUDA;
    g_scratch_ptr[dev] = static_cast<int32_t*>(p);
  }
  *out = g_scratch_ptr[dev];
  return MOE_OK;
}

}  // namespace

namespace moe {
void forget_noalloc_scratch() {
  std::lock_guard<std::mutex> lk(g_scratch_mu);
  for (auto& p : g_scratch_ptr) p = nullptr;
}
}  // namespace moe

extern "C" moe_status moe_dispatch_noalloc(const moe_config* cfg, const uint16_t* x,
                                           const int32_t* topk_idx, int32_t* counts,
                                           int32_t* offsets, int32_t* row_src_token,
                                           int32_t* slot_row, uint16_t* x_perm, void* stream) {
  if (moe_validate_config(cfg) != MOE_OK) return MOE_ERR_INVALID_ARG;
  if (!counts || !offsets || !moe::aligned4(counts) || !moe::aligned4(offsets))
    return MOE_ERR_INVALID_ARG;
  if (cfg->T > 0 && (!topk_idx || !row_src_token || !slot_row || !moe::aligned4(topk_idx) ||
                     !moe::aligned4(row_src_token) || !moe::aligned4(slot_row)))
    return MOE_ERR_INVALID_ARG;
  if (x_perm && (!x || !moe::aligned16(x) || !moe::aligned16(x_perm))) return MOE_ERR_INVALID_ARG;
  // each half of the array holds (chunks + 1) x E histogram entries
  const long entries = (long)(moe::perm_num_chunks(cfg->T) + 1) * cfg->E;
  if (entries > MOE_DISPATCH_NOALLOC_MAX_ENTRIES) return MOE_ERR_UNSUPPORTED;
  int32_t* scratch = nullptr;
  moe_status st = scratch_address(&scratch);
  if (st != MOE_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  st = moe::launch_permutation(*cfg, topk_idx, counts, offsets, row_src_token, slot_row, scratch,
                               scratch + MOE_DISPATCH_NOALLOC_MAX_ENTRIES, s);
  if (st != MOE_OK) return st;
  if (x_perm) return moe::launch_dispatch_rows(cfg->T, cfg->H, cfg->k, x, slot_row, x_perm, s);
  return MOE_OK;
}
