// State commit at the accepted length (state-update pass), register-resident
// fp32 recurrence.
//
// One CTA per (request, value head).  The gated delta rule acts on the state
// from the left, so column c of S evolves on its own (Eq. per-step-fwd):
//     u_t[c] = v_t[c] - alpha_t (S^T k_t)[c],   delta_t[c] = beta_t u_t[c],
//     S[:, c] <- alpha_t S[:, c] + k_t delta_t[c].
// Two threads share column c, each holding half of its d_k rows in registers
// (lanes l and l+16 of a warp, so the two halves of k_t . S[:, c] meet with one
// shuffle).  The block's keys (and queries, for the token-causal outputs) and
// values are staged once in shared memory as fp32 with 16-byte loads issued
// together with the state loads.
//
// The decay is applied lazily: the thread keeps S~ = S / Gam_t with
// Gam_t = alpha_1 ... alpha_t (since the last fold), so a step is
//     u_t = v_t - Gam_t (S~^T k_t),   S~ <- S~ + k_t (beta_t u_t / Gam_t),
// one multiply-add per element for the product and one for the update.  When
// Gam_t would fall below 2^-40 the decay is folded into the state instead
// (S <- Gam_t S~ + k_t delta_t, Gam <- 1), so 1/Gam_t stays bounded.  After the
// first n = accept_len tokens Gam_n S~ is written back in place (coalesced);
// n = 0 leaves the slot untouched.  Exact fp32 arithmetic throughout, which is
// what the committed state's accuracy needs.
#include "common.cuh"
#include "kernels.h"

namespace flare {

namespace {

constexpr int kCBmax = 64;
constexpr float kMinGam = 9.094947017729282e-13f;  // 2^-40

// Rows [row0, row0 + rows) of a [rows_total][n] activation slice (row stride
// `stride` elements) into shared memory as fp32 [rows][n]; 16-byte loads, all
// issued before the first conversion.
template <typename T, int N, int THREADS>
__device__ __forceinline__ void stage_rows(float* dst, const T* src, size_t stride, int rows) {
  constexpr int kPerChunk = 16 / sizeof(T);  // elements per 16-byte chunk
  constexpr int kChunksPerRow = N / kPerChunk;
  constexpr int kMaxIter = (kCBmax * kChunksPerRow + THREADS - 1) / THREADS;
  const int total = rows * kChunksPerRow;
  uint4 buf[kMaxIter];
#pragma unroll
  for (int it = 0; it < kMaxIter; ++it) {
    const int e = threadIdx.x + it * THREADS;
    if (e < total) {
      const int t = e / kChunksPerRow, ch = e % kChunksPerRow;
      buf[it] = *reinterpret_cast<const uint4*>(src + (size_t)t * stride + ch * kPerChunk);
    }
  }
#pragma unroll
  for (int it = 0; it < kMaxIter; ++it) {
    const int e = threadIdx.x + it * THREADS;
    if (e < total) {
      float* d = dst + (size_t)e * kPerChunk;
      if constexpr (sizeof(T) == 2) {
        const __nv_bfloat162* b = reinterpret_cast<const __nv_bfloat162*>(&buf[it]);
        const float2 f0 = __bfloat1622float2(b[0]), f1 = __bfloat1622float2(b[1]);
        const float2 f2 = __bfloat1622float2(b[2]), f3 = __bfloat1622float2(b[3]);
        reinterpret_cast<float4*>(d)[0] = make_float4(f0.x, f0.y, f1.x, f1.y);
        reinterpret_cast<float4*>(d)[1] = make_float4(f2.x, f2.y, f3.x, f3.y);
      } else {
        *reinterpret_cast<float4*>(d) = *reinterpret_cast<const float4*>(&buf[it]);
      }
    }
  }
}

}  // namespace

template <typename T, int DK, int DV, bool CAUSAL>
__global__ void __launch_bounds__(2 * DV, 2) gdr_commit_kernel(GdrParams p) {
  constexpr int kThreads = 2 * DV;
  constexpr int kHalf = DK / 2;  // state rows per thread
  extern __shared__ float smc[];
  __shared__ float alpha_s[kCBmax], beta_s[kCBmax];

  const int item = blockIdx.x;
  const int r = item / p.Hv, j = item % p.Hv;
  const int h = j / (p.Hv / p.Hk);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int half = lane >> 4;               // which half of the rows
  const int c = warp * 16 + (lane & 15);    // value column
  const int B = p.B;

  const int slot = p.state_slot[r];
  if (slot < 0 || slot >= p.nslots) {
    if (threadIdx.x == 0) flag(p.dev_status, FLARE_DEV_BAD_SLOT);
    return;
  }
  const int n = p.accept_len[r];
  if (n < 0 || n > B) {
    if (threadIdx.x == 0) flag(p.dev_status, FLARE_DEV_BAD_ACCEPT_LEN);
    return;
  }
  const int steps = CAUSAL ? B : n;
  if (steps == 0) return;

  float* Ks = smc;                                   // [steps][DK]
  float* Qs = Ks + steps * DK;                       // [steps][DK] (CAUSAL only)
  float* Vs = Qs + (CAUSAL ? steps * DK : 0);        // [steps][DV]

  // state rows half*kHalf .. half*kHalf + kHalf - 1 of column c
  float* Sg = p.state_pool + ((size_t)slot * p.Hv + j) * DK * DV + (size_t)half * kHalf * DV + c;
  float s[kHalf];
#pragma unroll
  for (int m = 0; m < kHalf; ++m) s[m] = Sg[(size_t)m * DV];

  const T* kg = static_cast<const T*>(p.k) + ((size_t)r * B * p.Hk + h) * DK;
  const T* vg = static_cast<const T*>(p.v) + ((size_t)r * B * p.Hv + j) * DV;
  stage_rows<T, DK, kThreads>(Ks, kg, (size_t)p.Hk * DK, steps);
  if (CAUSAL) {
    const T* qg = static_cast<const T*>(p.q) + ((size_t)r * B * p.Hk + h) * DK;
    stage_rows<T, DK, kThreads>(Qs, qg, (size_t)p.Hk * DK, steps);
  }
  stage_rows<T, DV, kThreads>(Vs, vg, (size_t)p.Hv * DV, steps);
  for (int t = threadIdx.x; t < steps; t += kThreads) {
    const size_t gb = ((size_t)r * B + t) * p.Hv + j;
    alpha_s[t] = expf(p.log_decay[gb]);
    beta_s[t] = p.beta[gb];
  }
  __syncthreads();

  float gam = 1.f;  // S = gam * s
#pragma unroll 1
  for (int t = 0; t < steps; ++t) {
    const float4* k4 = reinterpret_cast<const float4*>(Ks + t * DK + half * kHalf);
    float d0 = 0.f, d1 = 0.f, d2 = 0.f, d3 = 0.f;
#pragma unroll
    for (int m4 = 0; m4 < kHalf / 4; ++m4) {
      const float4 kk = k4[m4];
      d0 = fmaf(s[4 * m4], kk.x, d0);
      d1 = fmaf(s[4 * m4 + 1], kk.y, d1);
      d2 = fmaf(s[4 * m4 + 2], kk.z, d2);
      d3 = fmaf(s[4 * m4 + 3], kk.w, d3);
    }
    float dot = (d0 + d1) + (d2 + d3);
    dot += __shfl_xor_sync(0xffffffffu, dot, 16);
    const float gt = gam * alpha_s[t];
    const float delta = beta_s[t] * (Vs[t * DV + c] - gt * dot);
    __syncwarp();  // re-read k from shared memory below instead of holding it in registers
    if (gt >= kMinGam) {  // uniform across the CTA: the gates are per head
      const float w = delta / gt;
#pragma unroll
      for (int m4 = 0; m4 < kHalf / 4; ++m4) {
        const float4 kk = k4[m4];
        s[4 * m4] = fmaf(kk.x, w, s[4 * m4]);
        s[4 * m4 + 1] = fmaf(kk.y, w, s[4 * m4 + 1]);
        s[4 * m4 + 2] = fmaf(kk.z, w, s[4 * m4 + 2]);
        s[4 * m4 + 3] = fmaf(kk.w, w, s[4 * m4 + 3]);
      }
      gam = gt;
    } else {  // fold the decay into the state
#pragma unroll
      for (int m4 = 0; m4 < kHalf / 4; ++m4) {
        const float4 kk = k4[m4];
        s[4 * m4] = fmaf(kk.x, delta, gt * s[4 * m4]);
        s[4 * m4 + 1] = fmaf(kk.y, delta, gt * s[4 * m4 + 1]);
        s[4 * m4 + 2] = fmaf(kk.z, delta, gt * s[4 * m4 + 2]);
        s[4 * m4 + 3] = fmaf(kk.w, delta, gt * s[4 * m4 + 3]);
      }
      gam = 1.f;
    }
    if (t + 1 == n) {
#pragma unroll
      for (int m = 0; m < kHalf; ++m) Sg[(size_t)m * DV] = gam * s[m];
    }
    if (CAUSAL) {
      const float4* q4 = reinterpret_cast<const float4*>(Qs + t * DK + half * kHalf);
      float o0 = 0.f, o1 = 0.f, o2 = 0.f, o3 = 0.f;
#pragma unroll
      for (int m4 = 0; m4 < kHalf / 4; ++m4) {
        const float4 qq = q4[m4];
        o0 = fmaf(s[4 * m4], qq.x, o0);
        o1 = fmaf(s[4 * m4 + 1], qq.y, o1);
        o2 = fmaf(s[4 * m4 + 2], qq.z, o2);
        o3 = fmaf(s[4 * m4 + 3], qq.w, o3);
      }
      float o = (o0 + o1) + (o2 + o3);
      o += __shfl_xor_sync(0xffffffffu, o, 16);
      if (half == 0)
        static_cast<T*>(p.out_causal)[(((size_t)r * B + t) * p.Hv + j) * DV + c] =
            from_f32<T>(p.scale * gam * o);
    }
  }
}

namespace {

template <typename T, int DK, int DV, bool CAUSAL>
cudaError_t launch_commit_t(const GdrParams& p, cudaStream_t stream) {
  auto smem_for = [](int B) {
    return sizeof(float) * ((size_t)B * DK * (CAUSAL ? 2 : 1) + (size_t)B * DV);
  };
  cudaError_t e = cudaFuncSetAttribute(gdr_commit_kernel<T, DK, DV, CAUSAL>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem_for(kCBmax));
  if (e != cudaSuccess) return e;
  gdr_commit_kernel<T, DK, DV, CAUSAL><<<p.R * p.Hv, 2 * DV, smem_for(p.B), stream>>>(p);
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
