// KV append of the state-update pass: the finalized block's keys and values
// become part of the paged prefix.  One CTA per request; 16-byte copies,
// coalesced along the head dimension.  Positions prefix_len[r] + t for the
// first n = append_len[r] (or B) block tokens, through the page table.
#include "common.cuh"
#include "kernels.h"

namespace flare {

__global__ void __launch_bounds__(256) append_kv_kernel(SoftmaxParams p, const int32_t* append_len,
                                                        void* k_pool, void* v_pool, int elem_bytes) {
  const int r = blockIdx.x;
  const int P = p.prefix_len[r];
  const int n = append_len ? append_len[r] : p.B;
  int bad = 0;
  if (n < 0 || n > p.B) bad = FLARE_DEV_BAD_ACCEPT_LEN;
  else if (P < 0 || (long)P + n > (long)p.max_pages * p.page_size) bad = FLARE_DEV_BAD_PREFIX_LEN;
  if (!bad) {
    int badpg = 0;
    for (int t = threadIdx.x; t < n; t += blockDim.x) {
      const int pg = p.page_table[(size_t)r * p.max_pages + (P + t) / p.page_size];
      badpg |= (pg < 0 || pg >= p.num_pages);
    }
    if (__syncthreads_or(badpg)) bad = FLARE_DEV_BAD_PAGE;
  } else {
    __syncthreads_or(0);
  }
  if (bad) {
    if (threadIdx.x == 0) flag(p.dev_status, bad);
    return;
  }
  const int row16 = p.D * elem_bytes / 16;  // 16-byte chunks per (token, head) row
  const size_t total = (size_t)n * p.Hkv * row16;
  const uint4* kb = static_cast<const uint4*>(p.k_blk);
  const uint4* vb = static_cast<const uint4*>(p.v_blk);
  for (size_t e = threadIdx.x; e < total; e += blockDim.x) {
    const int c = (int)(e % row16);
    const int hk = (int)((e / row16) % p.Hkv);
    const int t = (int)(e / ((size_t)row16 * p.Hkv));
    const int pos = P + t;
    const int page = p.page_table[(size_t)r * p.max_pages + pos / p.page_size];
    const size_t dst = (((size_t)page * p.Hkv + hk) * p.page_size + pos % p.page_size) * row16 + c;
    const size_t src = (((size_t)r * p.B + t) * p.Hkv + hk) * row16 + c;
    static_cast<uint4*>(k_pool)[dst] = kb[src];
    static_cast<uint4*>(v_pool)[dst] = vb[src];
  }
}

cudaError_t launch_append_kv(const SoftmaxParams& p, const int32_t* append_len, void* k_pool,
                             void* v_pool, int elem_bytes, cudaStream_t stream) {
  if (p.R == 0) return cudaSuccess;
  append_kv_kernel<<<p.R, 256, 0, stream>>>(p, append_len, k_pool, v_pool, elem_bytes);
  note_launches(1);
  return cudaGetLastError();
}

}  // namespace flare
