// flare_block_softmax_attn_noalloc: the block-query softmax attention call for
// callers that must not allocate device memory.
//
// Some callers cannot hand the library a workspace buffer: a serving engine
// whose memory manager owns every byte of device memory and forbids ad-hoc
// cudaMalloc/cudaFree while requests are in flight (those calls synchronize
// the device and can fail under memory pressure), or a plugin host that only
// passes the tensors of the request itself.  This entry point takes the same
// inputs and outputs as flare_block_softmax_attn but draws its workspace (the
// work order and the split-prefix partials) from one statically sized device
// array owned by this library.
//
// The array lives for as long as the library is loaded and every GPU that
// loads it holds its FLARE_NOALLOC_SCRATCH_BYTES.  In host code the array's
// name is only a host-side stand-in, so its device address is looked up with
// cudaGetSymbolAddress once per device (with that device current) and cached.
// Under CUDA's default lazy module loading, that first lookup is what commits
// the array on the device, so a caller makes its first call at start-up,
// before its own memory pool takes the device and before any stream capture.
// The cached address is tied to the device's primary context and goes stale
// if that context is destroyed (cudaDeviceReset).
// Every call shares the array: calls that overlap on the GPU (other streams,
// other host threads) race on it.  Nothing in it needs to start at zero: each
// call writes every partial it later reads.
#include <cuda_runtime.h>

#include <mutex>

#include "flare.h"

namespace {

static __device__ __align__(256) unsigned char g_softmax_scratch[FLARE_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 256;
std::mutex g_scratch_mu;
void* g_scratch_addr[kMaxDevices] = {};

// Device address of the scratch array on the current device; the first call
// on a device looks it up (no allocation happens here).
flare_status scratch_on_current_device(void** addr) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return FLARE_ERR_CUDA;
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  if (!g_scratch_addr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_softmax_scratch) != cudaSuccess || !p) return FLARE_ERR_CUDA;
    g_scratch_addr[dev] = p;
  }
  *addr = g_scratch_addr[dev];
  return FLARE_OK;
}

}  // namespace

extern "C" flare_status flare_block_softmax_attn_noalloc(
    const flare_softmax_desc* desc, const void* q, const void* k_blk, const void* v_blk,
    const void* k_pool, const void* v_pool, const int32_t* page_table, const int32_t* prefix_len,
    void* out, float* lse, int32_t* dev_status, void* stream) {
  size_t need = 0;
  flare_status st = flare_softmax_workspace_size(desc, &need);
  if (st != FLARE_OK) return st;
  if (need > (size_t)FLARE_NOALLOC_SCRATCH_BYTES) return FLARE_ERR_UNSUPPORTED;
  void* scratch = nullptr;
  if (need > 0) {
    st = scratch_on_current_device(&scratch);
    if (st != FLARE_OK) return st;
  }
  return flare_block_softmax_attn(desc, q, k_blk, v_blk, k_pool, v_pool, page_table, prefix_len,
                                  out, lse, scratch, need > 0 ? (size_t)FLARE_NOALLOC_SCRATCH_BYTES : 0,
                                  dev_status, stream);
}
