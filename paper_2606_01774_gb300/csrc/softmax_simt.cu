// Block-query softmax attention over a paged KV prefix, CUDA-core version.
//
// Serves fp32 activations and any shape the tensor-core kernel does not take.
// Grid (split, request*kv_head, row tile).  The rows of one (request, kv head)
// are its B*G block queries, row m = t*G + g for block position t and query
// head kv_head*G + g (grouped-query attention: the G query heads of a kv head
// share its keys).  The key index space is the prefix (through the page table)
// followed by the block's own keys; a split covers a contiguous range of it.
// Online softmax in base 2 with the logit scale folded into q.
#include <float.h>

#include "common.cuh"
#include "kernels.h"

namespace flare {

namespace {
constexpr int kRows = 16;     // query rows per CTA (4 per warp)
constexpr int kTile = 32;     // keys per smem tile (one per lane)
constexpr int kThreads = 128;

template <typename T>
__device__ __forceinline__ const T* key_row(const SoftmaxParams& p, const T* pool, const T* blk,
                                            int r, int kvh, int P, int idx) {
  if (idx < P) {
    const int page = p.page_table[(size_t)r * p.max_pages + idx / p.page_size];
    return pool + (((size_t)page * p.Hkv + kvh) * p.page_size + idx % p.page_size) * p.D;
  }
  return blk + (((size_t)r * p.B + (idx - P)) * p.Hkv + kvh) * p.D;
}
}  // namespace

template <typename T, int D>
__global__ void __launch_bounds__(kThreads) softmax_simt_kernel(SoftmaxParams p) {
  extern __shared__ float sm[];
  float* Qs = sm;                     // [kRows][D]
  float* Ks = Qs + kRows * D;         // [kTile][D+1]
  float* Vs = Ks + kTile * (D + 1);   // [kTile][D]

  const int split = blockIdx.x, item = blockIdx.y, mt = blockIdx.z;
  const int r = item / p.Hkv, kvh = item % p.Hkv;
  const int M = p.B * p.G;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int P = p.prefix_len[r];
  const int bad = check_request_pages(p.page_table, P, r, p.max_pages, p.page_size, p.num_pages);
  if (bad) {
    if (tid == 0) flag(p.dev_status, bad);
    return;
  }
  const int total = P + p.B;
  const int kv_lo = split * p.split_len;
  const int kv_hi = min(total, kv_lo + p.split_len);

  const T* q = static_cast<const T*>(p.q);
  const T* kpool = static_cast<const T*>(p.k_pool);
  const T* vpool = static_cast<const T*>(p.v_pool);
  const T* kblk = static_cast<const T*>(p.k_blk);
  const T* vblk = static_cast<const T*>(p.v_blk);

  for (int e = tid; e < kRows * D; e += kThreads) {
    const int i = e / D, d = e % D, m = mt * kRows + i;
    float x = 0.f;
    if (m < M) {
      const int t = m / p.G, g = m % p.G;
      x = to_f32(q[(((size_t)r * p.B + t) * p.Hq + kvh * p.G + g) * D + d]) * p.scale_log2;
    }
    Qs[e] = x;
  }

  constexpr int NC = D / 32;
  float acc[4][NC];
  float mrow[4], lrow[4];
#pragma unroll
  for (int w = 0; w < 4; ++w) {
    mrow[w] = -INFINITY;
    lrow[w] = 0.f;
#pragma unroll
    for (int x = 0; x < NC; ++x) acc[w][x] = 0.f;
  }

  for (int lo = kv_lo; lo < kv_hi; lo += kTile) {
    __syncthreads();
    for (int e = tid; e < kTile * D; e += kThreads) {
      const int jj = e / D, d = e % D, idx = lo + jj;
      float kx = 0.f, vx = 0.f;
      if (idx < kv_hi) {
        kx = to_f32(key_row<T>(p, kpool, kblk, r, kvh, P, idx)[d]);
        vx = to_f32(key_row<T>(p, vpool, vblk, r, kvh, P, idx)[d]);
      }
      Ks[jj * (D + 1) + d] = kx;
      Vs[jj * D + d] = vx;
    }
    __syncthreads();
    const int idx = lo + lane;
#pragma unroll
    for (int w = 0; w < 4; ++w) {
      const int i = warp * 4 + w, m = mt * kRows + i;
      if (m >= M) continue;  // warp-uniform
      const int trow = m / p.G;
      const bool causal_row =
          p.row_type ? p.row_type[(size_t)r * p.row_type_stride + trow] == 0 : p.causal != 0;
      const bool vis = idx < kv_hi && (!causal_row || idx < P || idx - P <= trow);
      float s = -INFINITY;
      if (vis) {
        float a = 0.f;
#pragma unroll 8
        for (int d = 0; d < D; ++d) a = fmaf(Qs[i * D + d], Ks[lane * (D + 1) + d], a);
        s = a;
      }
      const float mx = warp_max(s);
      const float mnew = fmaxf(mrow[w], mx);
      if (mnew == -INFINITY) continue;  // nothing visible yet for this row
      const float pj = vis ? exp2f(s - mnew) : 0.f;
      const float corr = exp2f(mrow[w] - mnew);
      lrow[w] = lrow[w] * corr + warp_sum(pj);
#pragma unroll
      for (int x = 0; x < NC; ++x) acc[w][x] *= corr;
      for (int jj = 0; jj < kTile; ++jj) {
        const float pb = __shfl_sync(0xffffffffu, pj, jj);
        if (pb != 0.f) {
#pragma unroll
          for (int x = 0; x < NC; ++x) acc[w][x] = fmaf(pb, Vs[jj * D + lane + 32 * x], acc[w][x]);
        }
      }
      mrow[w] = mnew;
    }
  }

  const float kLn2 = 0.6931471805599453f;
#pragma unroll
  for (int w = 0; w < 4; ++w) {
    const int i = warp * 4 + w, m = mt * kRows + i;
    if (m >= M) continue;
    const float inv = lrow[w] > 0.f ? 1.f / lrow[w] : 0.f;
    const float l2 = lrow[w] > 0.f ? (mrow[w] + log2f(lrow[w])) * kLn2 : -INFINITY;
    if (p.n_split == 1) {
      const int t = m / p.G, g = m % p.G;
      const size_t o = (((size_t)r * p.B + t) * p.Hq + kvh * p.G + g);
#pragma unroll
      for (int x = 0; x < NC; ++x)
        static_cast<T*>(p.out)[o * D + lane + 32 * x] = from_f32<T>(acc[w][x] * inv);
      if (p.lse && lane == 0) p.lse[o] = l2;
    } else {
      const size_t o = ((size_t)item * p.n_split + split) * M + m;
#pragma unroll
      for (int x = 0; x < NC; ++x) p.ws_o[o * D + lane + 32 * x] = acc[w][x] * inv;
      if (lane == 0) p.ws_lse[o] = l2;
    }
  }
}

// Merges the split partials of one (request, kv head, row) into the output:
// lse = log sum_s exp(lse_s), out = sum_s exp(lse_s - lse) out_s.
template <typename T>
__global__ void __launch_bounds__(256) softmax_combine_kernel(SoftmaxParams p) {
  const int item = blockIdx.x, m = blockIdx.y;
  const int r = item / p.Hkv, kvh = item % p.Hkv;
  const int M = p.B * p.G;
  const int P = p.prefix_len[r];
  if (check_request_pages(p.page_table, P, r, p.max_pages, p.page_size, p.num_pages)) return;
  float mx = -INFINITY;
  for (int s = 0; s < p.n_split; ++s)
    mx = fmaxf(mx, p.ws_lse[((size_t)item * p.n_split + s) * M + m]);
  float den = 0.f;
  for (int s = 0; s < p.n_split; ++s) {
    const float l = p.ws_lse[((size_t)item * p.n_split + s) * M + m];
    if (l != -INFINITY) den += expf(l - mx);
  }
  const int t = m / p.G, g = m % p.G;
  const size_t o = (((size_t)r * p.B + t) * p.Hq + kvh * p.G + g);
  for (int d = threadIdx.x; d < p.D; d += blockDim.x) {
    float a = 0.f;
    for (int s = 0; s < p.n_split; ++s) {
      const size_t ps = ((size_t)item * p.n_split + s) * M + m;
      const float l = p.ws_lse[ps];
      if (l != -INFINITY) a += expf(l - mx) * p.ws_o[ps * p.D + d];
    }
    static_cast<T*>(p.out)[o * p.D + d] = from_f32<T>(a / den);
  }
  if (p.lse && threadIdx.x == 0) p.lse[o] = mx + logf(den);
}

template <typename T>
__global__ void gather_prefix_kernel(SoftmaxParams p, int r, T* k_out, T* v_out) {
  const int P = p.prefix_len[r];
  const int bad = check_request_pages(p.page_table, P, r, p.max_pages, p.page_size, p.num_pages);
  if (bad) {
    if (threadIdx.x == 0 && blockIdx.x == 0) flag(p.dev_status, bad);
    return;
  }
  const size_t n = (size_t)P * p.Hkv * p.D;
  for (size_t e = (size_t)blockIdx.x * blockDim.x + threadIdx.x; e < n;
       e += (size_t)gridDim.x * blockDim.x) {
    const int d = e % p.D;
    const int kvh = (e / p.D) % p.Hkv;
    const int j = e / ((size_t)p.D * p.Hkv);
    const int page = p.page_table[(size_t)r * p.max_pages + j / p.page_size];
    const size_t src = (((size_t)page * p.Hkv + kvh) * p.page_size + j % p.page_size) * p.D + d;
    k_out[e] = static_cast<const T*>(p.k_pool)[src];
    v_out[e] = static_cast<const T*>(p.v_pool)[src];
  }
}

namespace {
template <typename T, int D>
cudaError_t launch_simt_d(const SoftmaxParams& p, const SoftmaxPlan& plan, cudaStream_t stream) {
  const size_t smem = sizeof(float) * ((size_t)kRows * D + (size_t)kTile * (D + 1) + kTile * D);
  cudaError_t e = cudaFuncSetAttribute(softmax_simt_kernel<T, D>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  const int M = p.B * p.G;
  dim3 grid(plan.n_split, p.R * p.Hkv, (M + kRows - 1) / kRows);
  softmax_simt_kernel<T, D><<<grid, kThreads, smem, stream>>>(p);
  note_launches(1);
  e = cudaGetLastError();
  if (e != cudaSuccess || plan.n_split == 1) return e;
  return launch_softmax_combine(p, sizeof(T) == 2, stream);
}

template <typename T>
cudaError_t launch_simt(const SoftmaxParams& p, const SoftmaxPlan& plan, cudaStream_t stream) {
  switch (p.D) {
    case 64: return launch_simt_d<T, 64>(p, plan, stream);
    case 128: return launch_simt_d<T, 128>(p, plan, stream);
    case 256: return launch_simt_d<T, 256>(p, plan, stream);
    default: return cudaErrorInvalidValue;
  }
}
}  // namespace

cudaError_t launch_softmax_combine(const SoftmaxParams& p, bool bf16, cudaStream_t stream) {
  const dim3 grid(p.R * p.Hkv, p.B * p.G);
  if (bf16)
    softmax_combine_kernel<__nv_bfloat16><<<grid, 256, 0, stream>>>(p);
  else
    softmax_combine_kernel<float><<<grid, 256, 0, stream>>>(p);
  note_launches(1);
  return cudaGetLastError();
}

cudaError_t launch_softmax_simt(const SoftmaxParams& p, const SoftmaxPlan& plan, bool bf16,
                                cudaStream_t stream) {
  return bf16 ? launch_simt<__nv_bfloat16>(p, plan, stream) : launch_simt<float>(p, plan, stream);
}

cudaError_t launch_gather_prefix(const SoftmaxParams& p, int request, void* k_out, void* v_out,
                                 bool bf16, cudaStream_t stream) {
  const size_t maxn = (size_t)p.max_pages * p.page_size * p.Hkv * p.D;
  const unsigned blocks = (unsigned)((maxn + 255) / 256 > 4096 ? 4096 : (maxn + 255) / 256);
  if (bf16)
    gather_prefix_kernel<__nv_bfloat16><<<blocks ? blocks : 1, 256, 0, stream>>>(
        p, request, (__nv_bfloat16*)k_out, (__nv_bfloat16*)v_out);
  else
    gather_prefix_kernel<float><<<blocks ? blocks : 1, 256, 0, stream>>>(p, request,
                                                                        (float*)k_out,
                                                                        (float*)v_out);
  return cudaGetLastError();
}

}  // namespace flare
