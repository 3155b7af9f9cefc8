// varrate_decode_attn_noalloc: decode attention for callers that cannot allocate device memory.
//
// Some callers only ever receive device pointers for their inputs and outputs and have no way to
// obtain workspace: a plugin inside a host framework that owns every device allocation through its
// own pool, or a latency-critical serving loop that must not allocate after start-up. This entry
// point runs the same decode kernels as varrate_decode_attn, but takes its scratch (the rotated
// queries and the per-split partial results) from a fixed array in device global memory that the
// library itself defines, so the caller passes no workspace and nothing is allocated.
#include <atomic>

#include "common.cuh"
#include "kernels.h"

namespace {

// Scratch for every call of this entry point on a device. Every GPU that loads the library holds
// it until the process exits. Calls share it and it keeps the previous call's contents. It starts
// zero-filled (as a __device__ array without initialiser is); its first part is the decode
// kernel's header (a call count and two alternating sets of arrival counters, each call clearing
// the set the next call uses, so counts left by an overlapping or timed-out call are reported once
// as VARRATE_ERR_CORRUPT and gone one call later), and the decode kernels write every other
// element they later read, so nothing has to be cleared between calls.
constexpr size_t kScratchBytes = size_t(4) << 20;   // 4 MiB
static __device__ __align__(256) unsigned char g_decode_scratch[kScratchBytes];

constexpr int kMaxDevices = 64;
std::atomic<void*> g_scratch_ptr[kMaxDevices];

// Device address of the scratch array on the current device, looked up once per device (with that
// device current) and cached. In host code the symbol is only a host-side handle, never a device
// address, so it must not be passed to a kernel directly. Two threads may both look it up the first
// time; they find the same address. The cache is not told about cudaDeviceReset: after a reset of
// the device the cached address is stale and this entry point must not be used again in the
// process.
void* scratch_on_current_device() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
  void* p = g_scratch_ptr[dev].load(std::memory_order_acquire);
  if (p == nullptr) {
    if (cudaGetSymbolAddress(&p, g_decode_scratch) != cudaSuccess || p == nullptr) return nullptr;
    g_scratch_ptr[dev].store(p, std::memory_order_release);
  }
  return p;
}

}  // namespace

extern "C" varrate_status varrate_decode_attn_noalloc(const varrate_config* cfg,
                                                      const varrate_packed* cache,
                                                      const void* basis_k, const void* basis_v,
                                                      const void* q, int32_t layer,
                                                      const void* tail_k, const void* tail_v,
                                                      int32_t n_tail, void* out,
                                                      int32_t* dev_status, void* stream) {
  const size_t need = varrate_workspace_bytes(cfg, VARRATE_CALL_DECODE);
  if (need == 0) {
    const varrate_status st = varrate_check_config(cfg);
    return st != VARRATE_OK ? st : VARRATE_ERR_ARG;
  }
  if (need > kScratchBytes) return VARRATE_ERR_WORKSPACE;   // shape too large for the fixed scratch
  void* ws = scratch_on_current_device();
  if (ws == nullptr) return VARRATE_ERR_CUDA;
  return varrate_decode_attn(cfg, cache, basis_k, basis_v, q, layer, tail_k, tail_v, n_tail, out,
                             dev_status, ws, kScratchBytes, stream);
}
