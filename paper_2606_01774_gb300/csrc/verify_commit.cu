// Gather-scatter commit of an AR-Trust verify round (serving appendix,
// "Recovering the recurrent state at the accept boundary", path (b)).
//
// Grid (state tile, request, layer): each CTA copies one 64 KiB tile of the
// cached state S^(a) of request r in layer l into the request's pool slot,
// with 16-byte loads, all of a thread's loads issued before its first store.
// A request that accepted every draft (a = K) already has S^(K) in the pool
// and its CTAs return before touching memory.  The cached states are read
// with the streaming hint: each is read at most once.
#include "common.cuh"
#include "kernels.h"

namespace flare {

namespace {
constexpr int kCopyThreads = 256;
constexpr int kVecPerThread = 16;                               // 16 x 16 B in flight
constexpr int kVecPerTile = kCopyThreads * kVecPerThread;       // 64 KiB per CTA
}  // namespace

__global__ void __launch_bounds__(kCopyThreads) verify_commit_kernel(VerifyCommitParams p) {
  const int tile = blockIdx.x, r = blockIdx.y, l = blockIdx.z;
  const int slot = p.state_slot[r], K = p.verify_len[r], a = p.accept[r];
  const bool first = tile == 0 && l == 0 && threadIdx.x == 0;
  if (slot < 0 || slot >= p.nslots) {
    if (first) flag(p.dev_status, FLARE_DEV_BAD_SLOT);
    return;
  }
  if (K < 0 || K > p.max_verify || a < 0 || a > K) {
    if (first) flag(p.dev_status, FLARE_DEV_BAD_VERIFY_LEN);
    return;
  }
  if (a == K) return;
  const size_t n_vec = p.state_elems / 4;
  const uint4* src = reinterpret_cast<const uint4*>(
      p.records[l] + ((size_t)r * p.max_verify + a) * p.state_elems);
  uint4* dst = reinterpret_cast<uint4*>(p.pools[l] + (size_t)slot * p.state_elems);
  const size_t base = (size_t)tile * kVecPerTile + threadIdx.x;
  uint4 buf[kVecPerThread];
#pragma unroll
  for (int i = 0; i < kVecPerThread; ++i) {
    const size_t e = base + (size_t)i * kCopyThreads;
    if (e < n_vec) buf[i] = __ldcs(src + e);
  }
#pragma unroll
  for (int i = 0; i < kVecPerThread; ++i) {
    const size_t e = base + (size_t)i * kCopyThreads;
    if (e < n_vec) dst[e] = buf[i];
  }
}

cudaError_t launch_verify_commit(const VerifyCommitParams& p, cudaStream_t stream) {
  if (p.R == 0 || p.n_layers == 0) return cudaSuccess;
  const size_t n_vec = p.state_elems / 4;
  const unsigned tiles = (unsigned)((n_vec + kVecPerTile - 1) / kVecPerTile);
  verify_commit_kernel<<<dim3(tiles, (unsigned)p.R, (unsigned)p.n_layers), kCopyThreads, 0,
                         stream>>>(p);
  note_launches(1);
  return cudaGetLastError();
}

}  // namespace flare
