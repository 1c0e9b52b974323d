// State commit at the accepted length (state-update pass), register-resident
// fp32 recurrence.
//
// One CTA per (request, value head) with one thread per value column c: the
// gated delta rule acts on the state from the left, so column c of S evolves
// on its own (Eq. per-step-fwd):
//     u_t[c] = v_t[c] - alpha_t (S^T k_t)[c],   delta_t[c] = beta_t u_t[c],
//     S[:, c] <- alpha_t S[:, c] + k_t delta_t[c].
// Thread c keeps its whole column (d_k floats) in registers; the block's keys
// (and queries, for the optional token-causal outputs) are staged once in
// shared memory as fp32 and read as broadcasts.  After the first n = accept_len
// tokens the column is written back in place (coalesced across threads); n = 0
// leaves the slot untouched.  Exact fp32 arithmetic, no rounding of the state
// to a narrower type, which is what the committed state's accuracy needs.
#include "common.cuh"
#include "kernels.h"

namespace flare {

namespace {
constexpr int kCBmax = 64;
}

template <typename T, int DK, int DV, bool CAUSAL>
__global__ void __launch_bounds__(DV, 2) gdr_commit_kernel(GdrParams p) {
  extern __shared__ float smc[];
  float* Ks = smc;                       // [B][DK]
  float* Qs = Ks + kCBmax * DK;          // [B][DK] (CAUSAL only)
  float* Vs = Qs + (CAUSAL ? kCBmax * DK : 0);  // [B][DV]
  __shared__ float alpha_s[kCBmax], beta_s[kCBmax];

  const int item = blockIdx.x;
  const int r = item / p.Hv, j = item % p.Hv;
  const int h = j / (p.Hv / p.Hk);
  const int c = threadIdx.x;
  const int B = p.B;

  const int slot = p.state_slot[r];
  if (slot < 0 || slot >= p.nslots) {
    if (c == 0) flag(p.dev_status, FLARE_DEV_BAD_SLOT);
    return;
  }
  const int n = p.accept_len[r];
  if (n < 0 || n > B) {
    if (c == 0) flag(p.dev_status, FLARE_DEV_BAD_ACCEPT_LEN);
    return;
  }
  const int steps = CAUSAL ? B : n;
  if (steps == 0) return;

  float* Sg = p.state_pool + ((size_t)slot * p.Hv + j) * DK * DV + c;
  float S[DK];
#pragma unroll
  for (int i = 0; i < DK; ++i) S[i] = Sg[(size_t)i * DV];

  const T* kg = static_cast<const T*>(p.k) + ((size_t)r * B * p.Hk + h) * DK;
  const T* qg = static_cast<const T*>(p.q) + ((size_t)r * B * p.Hk + h) * DK;
  const T* vg = static_cast<const T*>(p.v) + ((size_t)r * B * p.Hv + j) * DV;
  for (int e = c; e < steps * DK; e += DV) {
    const int t = e / DK, i = e % DK;
    Ks[e] = to_f32(kg[(size_t)t * p.Hk * DK + i]);
    if (CAUSAL) Qs[e] = to_f32(qg[(size_t)t * p.Hk * DK + i]);
  }
  for (int e = c; e < steps * DV; e += DV) {
    const int t = e / DV, cc = e % DV;
    Vs[e] = to_f32(vg[(size_t)t * p.Hv * DV + cc]);
  }
  for (int t = c; t < steps; t += DV) {
    const size_t gb = ((size_t)r * B + t) * p.Hv + j;
    alpha_s[t] = expf(p.log_decay[gb]);
    beta_s[t] = p.beta[gb];
  }
  __syncthreads();

#pragma unroll 1
  for (int t = 0; t < steps; ++t) {
    const float4* k4 = reinterpret_cast<const float4*>(Ks + t * DK);
    float d0 = 0.f, d1 = 0.f, d2 = 0.f, d3 = 0.f;
#pragma unroll
    for (int i4 = 0; i4 < DK / 4; ++i4) {
      const float4 kk = k4[i4];
      d0 = fmaf(S[4 * i4], kk.x, d0);
      d1 = fmaf(S[4 * i4 + 1], kk.y, d1);
      d2 = fmaf(S[4 * i4 + 2], kk.z, d2);
      d3 = fmaf(S[4 * i4 + 3], kk.w, d3);
    }
    const float alpha = alpha_s[t];
    const float delta = beta_s[t] * (Vs[t * DV + c] - alpha * ((d0 + d1) + (d2 + d3)));
    __syncwarp();  // re-read k from shared memory below instead of holding it in registers
#pragma unroll
    for (int i4 = 0; i4 < DK / 4; ++i4) {
      const float4 kk = k4[i4];
      S[4 * i4] = fmaf(kk.x, delta, alpha * S[4 * i4]);
      S[4 * i4 + 1] = fmaf(kk.y, delta, alpha * S[4 * i4 + 1]);
      S[4 * i4 + 2] = fmaf(kk.z, delta, alpha * S[4 * i4 + 2]);
      S[4 * i4 + 3] = fmaf(kk.w, delta, alpha * S[4 * i4 + 3]);
    }
    if (t + 1 == n) {
#pragma unroll
      for (int i = 0; i < DK; ++i) Sg[(size_t)i * DV] = S[i];
    }
    if (CAUSAL) {
      const float4* q4 = reinterpret_cast<const float4*>(Qs + t * DK);
      float o0 = 0.f, o1 = 0.f, o2 = 0.f, o3 = 0.f;
#pragma unroll
      for (int i4 = 0; i4 < DK / 4; ++i4) {
        const float4 qq = q4[i4];
        o0 = fmaf(S[4 * i4], qq.x, o0);
        o1 = fmaf(S[4 * i4 + 1], qq.y, o1);
        o2 = fmaf(S[4 * i4 + 2], qq.z, o2);
        o3 = fmaf(S[4 * i4 + 3], qq.w, o3);
      }
      static_cast<T*>(p.out_causal)[(((size_t)r * B + t) * p.Hv + j) * DV + c] =
          from_f32<T>(p.scale * ((o0 + o1) + (o2 + o3)));
    }
  }
}

namespace {

template <typename T, int DK, int DV, bool CAUSAL>
cudaError_t launch_commit_t(const GdrParams& p, cudaStream_t stream) {
  const size_t smem = sizeof(float) * ((size_t)kCBmax * DK * (CAUSAL ? 2 : 1) + (size_t)kCBmax * DV);
  cudaError_t e = cudaFuncSetAttribute(gdr_commit_kernel<T, DK, DV, CAUSAL>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  gdr_commit_kernel<T, DK, DV, CAUSAL><<<p.R * p.Hv, DV, smem, stream>>>(p);
  note_launches(1);
  return cudaGetLastError();
}

template <typename T, bool CAUSAL>
cudaError_t launch_commit_c(const GdrParams& p, cudaStream_t stream) {
  if (p.dk == 128 && p.dv == 128) return launch_commit_t<T, 128, 128, CAUSAL>(p, stream);
  if (p.dk == 128 && p.dv == 64) return launch_commit_t<T, 128, 64, CAUSAL>(p, stream);
  if (p.dk == 64 && p.dv == 128) return launch_commit_t<T, 64, 128, CAUSAL>(p, stream);
  if (p.dk == 64 && p.dv == 64) return launch_commit_t<T, 64, 64, CAUSAL>(p, stream);
  return cudaErrorInvalidValue;
}

}  // namespace

cudaError_t launch_gdr_commit(const GdrParams& p, bool bf16, cudaStream_t stream) {
  if (p.R == 0) return cudaSuccess;
  const bool causal = p.out_causal != nullptr;
  if (bf16)
    return causal ? launch_commit_c<__nv_bfloat16, true>(p, stream)
                  : launch_commit_c<__nv_bfloat16, false>(p, stream);
  return causal ? launch_commit_c<float, true>(p, stream) : launch_commit_c<float, false>(p, stream);
}

}  // namespace flare
