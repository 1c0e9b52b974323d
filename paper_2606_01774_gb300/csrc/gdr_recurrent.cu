// Gated delta rule over one block, token by token, on CUDA cores in fp32.
//
// One CTA per (request, value head).  The state S (dk x dv fp32) lives in
// shared memory; thread (part, c) owns column c of rows [part*dk/np, ...).
// Each block token applies the per-step expansion of the gated delta rule
// (Eq. per-step-fwd):  S_pre = exp(g) S;  u = v - S_pre^T k;  delta = beta u;
// S = S_pre + k delta^T.  The state's columns evolve independently (the
// update acts on S from the left), which is why a column per thread works.
//
// This kernel serves
//   - the denoise pass for fp32 activations (block-end readout, Eq.
//     noisy-block-fwd), and
//   - the commit at an accepted length with optional token-causal outputs
//     (state-update pass), for any activation type.
// The bf16 denoise pass at scale runs on the tensor-core kernel instead.
#include "common.cuh"
#include "kernels.h"

namespace flare {

template <typename T>
__global__ void __launch_bounds__(256) gdr_block_recurrent_kernel(GdrParams p) {
  extern __shared__ float smem[];
  const int dk = p.dk, dv = p.dv;
  const int nparts = blockDim.x / dv;
  float* S = smem;             // [dk][dv]
  float* kvec = S + dk * dv;   // [dk]
  float* qvec = kvec + dk;     // [dk]
  float* red = qvec + dk;      // [nparts][dv]
  float* dlt = red + nparts * dv;  // [dv]

  const int item = blockIdx.x;
  const int r = item / p.Hv, j = item % p.Hv;
  const int h = j / (p.Hv / p.Hk);
  const int tid = threadIdx.x;
  const int c = tid % dv, part = tid / dv;
  const int ilo = part * dk / nparts, ihi = (part + 1) * dk / nparts;

  const int slot = p.state_slot[r];
  if (slot < 0 || slot >= p.nslots) {
    if (tid == 0) flag(p.dev_status, FLARE_DEV_BAD_SLOT);
    return;
  }
  int n = p.B;
  if (p.accept_len) {
    n = p.accept_len[r];
    if (n < 0 || n > p.B) {
      if (tid == 0) flag(p.dev_status, FLARE_DEV_BAD_ACCEPT_LEN);
      return;
    }
  }
  const bool want_state = p.write_state && n > 0;
  const int steps = (p.out_blockend || p.out_causal) ? p.B : (want_state ? n : 0);
  if (steps == 0 && !p.out_blockend) return;

  float* Sg = p.state_pool + ((size_t)slot * p.Hv + j) * dk * dv;
  for (int e = tid; e < dk * dv; e += blockDim.x) S[e] = Sg[e];

  const T* q = static_cast<const T*>(p.q);
  const T* k = static_cast<const T*>(p.k);
  const T* v = static_cast<const T*>(p.v);

  for (int t = 0; t < steps; ++t) {
    const size_t kq = (((size_t)r * p.B + t) * p.Hk + h) * dk;
    const size_t gb = ((size_t)r * p.B + t) * p.Hv + j;
    __syncthreads();
    for (int i = tid; i < dk; i += blockDim.x) {
      kvec[i] = to_f32(k[kq + i]);
      if (q) qvec[i] = to_f32(q[kq + i]);
    }
    __syncthreads();
    const float alpha = expf(p.log_decay[gb]);
    const float bt = p.beta[gb];
    float acc = 0.f;
    for (int i = ilo; i < ihi; ++i) acc = fmaf(S[i * dv + c], kvec[i], acc);
    red[part * dv + c] = acc;
    __syncthreads();
    if (part == 0) {
      float sum = 0.f;
      for (int pp = 0; pp < nparts; ++pp) sum += red[pp * dv + c];
      const float vt = to_f32(v[(((size_t)r * p.B + t) * p.Hv + j) * dv + c]);
      dlt[c] = bt * (vt - alpha * sum);
    }
    __syncthreads();
    const float d = dlt[c];
    for (int i = ilo; i < ihi; ++i) S[i * dv + c] = fmaf(kvec[i], d, alpha * S[i * dv + c]);
    if (want_state && t + 1 == n)
      for (int i = ilo; i < ihi; ++i) Sg[i * dv + c] = S[i * dv + c];
    if (p.out_causal) {
      float a2 = 0.f;
      for (int i = ilo; i < ihi; ++i) a2 = fmaf(S[i * dv + c], qvec[i], a2);
      __syncthreads();  // every thread is done reading red from the delta step
      red[part * dv + c] = a2;
      __syncthreads();
      if (part == 0) {
        float sum = 0.f;
        for (int pp = 0; pp < nparts; ++pp) sum += red[pp * dv + c];
        static_cast<T*>(p.out_causal)[(((size_t)r * p.B + t) * p.Hv + j) * dv + c] =
            from_f32<T>(p.scale * sum);
      }
    }
  }

  if (p.out_blockend) {
    for (int l = 0; l < p.B; ++l) {
      const size_t ql = (((size_t)r * p.B + l) * p.Hk + h) * dk;
      __syncthreads();
      for (int i = tid; i < dk; i += blockDim.x) qvec[i] = to_f32(q[ql + i]);
      __syncthreads();
      float acc = 0.f;
      for (int i = ilo; i < ihi; ++i) acc = fmaf(S[i * dv + c], qvec[i], acc);
      red[part * dv + c] = acc;
      __syncthreads();
      if (part == 0) {
        float sum = 0.f;
        for (int pp = 0; pp < nparts; ++pp) sum += red[pp * dv + c];
        static_cast<T*>(p.out_blockend)[(((size_t)r * p.B + l) * p.Hv + j) * dv + c] =
            from_f32<T>(p.scale * sum);
      }
    }
  }
}

size_t gdr_recurrent_smem_bytes(int dk, int dv, int threads) {
  const int nparts = threads / dv;
  return sizeof(float) * ((size_t)dk * dv + 2 * dk + (size_t)nparts * dv + dv);
}

cudaError_t launch_gdr_recurrent(const GdrParams& p, bool bf16, cudaStream_t stream) {
  const int threads = 256;
  const size_t smem = gdr_recurrent_smem_bytes(p.dk, p.dv, threads);
  const void* fn = bf16 ? (const void*)gdr_block_recurrent_kernel<__nv_bfloat16>
                        : (const void*)gdr_block_recurrent_kernel<float>;
  cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem);
  if (e != cudaSuccess) return e;
  const long items = (long)p.R * p.Hv;
  if (items == 0) return cudaSuccess;
  if (bf16)
    gdr_block_recurrent_kernel<__nv_bfloat16><<<(unsigned)items, threads, smem, stream>>>(p);
  else
    gdr_block_recurrent_kernel<float><<<(unsigned)items, threads, smem, stream>>>(p);
  note_launches(1);
  return cudaGetLastError();
}

}  // namespace flare
