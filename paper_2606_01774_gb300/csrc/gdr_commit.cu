// State commit at the accepted length (state-update pass), register-resident
// fp32 recurrence.
//
// One CTA per (request, value head).  The gated delta rule acts on the state
// from the left, so column c of S evolves on its own (Eq. per-step-fwd):
//     u_t[c] = v_t[c] - alpha_t (S^T k_t)[c],   delta_t[c] = beta_t u_t[c],
//     S[:, c] <- alpha_t S[:, c] + k_t delta_t[c].
// Each thread holds a block of 4 columns x d_k/8 rows of S in registers (as
// fp32 pairs, so the multiply-adds run as packed f32x2 instructions): lane
// = 4 * row_group + column_group, so the 8 row groups of a column sit in one
// warp and meet with three shuffles, each loaded key value serves 4 columns,
// and the state moves in 16-byte pieces (a warp covers 16 columns, 8 warps a
// 128-column state).  The block's keys (and queries, for the token-causal
// outputs) and values are staged once in shared memory as fp32 with 16-byte
// loads issued together with the state loads.
//
// The decay is applied lazily: the thread keeps S~ = S / Gam_t with
// Gam_t = alpha_1 ... alpha_t (since the last fold), so a step is
//     u_t = v_t - Gam_t (S~^T k_t),   S~ <- S~ + k_t (beta_t u_t / Gam_t),
// one multiply-add per element for the product and one for the update.  When
// Gam_t would fall below 2^-40 the decay is folded into the state instead
// (S <- Gam_t S~ + k_t delta_t, Gam <- 1), so 1/Gam_t stays bounded.  After the
// first n = accept_len tokens Gam_n S~ is written back in place; n = 0 leaves
// the slot untouched.  Exact fp32 arithmetic throughout, which is what the
// committed state's accuracy needs.
//
// The same kernel runs the AR-Trust verify round (decoding appendix, block
// layout [anchor, d_0 .. d_{K-1}, MASK ...]; serving appendix, cache-and-
// scatter): all L block tokens are stepped, rows 0..K read the state right
// after their own token, the states after the anchor and after each of the
// first K-1 verify tokens are streamed out as S^(0..K-1), the state after
// token K is written to the pool, and the draft rows read the block-end state
// once the loop is done.
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

// MODE 0: commit; 1: commit with token-causal outputs; 2: AR-Trust verify round.
template <typename T, int DK, int DV, int MODE>
__global__ void __launch_bounds__(2 * DV, 2) gdr_commit_kernel(GdrParams p) {
  constexpr bool CAUSAL = MODE != 0;  // queries staged, readouts written
  constexpr bool VERIFY = MODE == 2;
  constexpr int kThreads = 2 * DV;   // DV / 16 warps
  constexpr int kR = DK / 8;         // state rows per thread
  extern __shared__ float smc[];
  // per token: {Gam_t, beta_t, 1/Gam_t (0: fold the decay into the state), Gam after the step}
  __shared__ float4 tok_s[kCBmax];

  const int item = blockIdx.x;
  const int r = item / p.Hv, j = item % p.Hv;
  const int h = j / (p.Hv / p.Hk);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int rg = lane >> 2;                      // row group: rows rg*kR ..
  const int c0 = warp * 16 + (lane & 3) * 4;     // columns c0 .. c0+3
  const int B = p.B;

  const int slot = p.state_slot[r];
  if (slot < 0 || slot >= p.nslots) {
    if (threadIdx.x == 0) flag(p.dev_status, FLARE_DEV_BAD_SLOT);
    return;
  }
  int n, K = 0;
  if constexpr (VERIFY) {
    K = p.verify_len[r];
    if (K < 0 || K > p.max_verify || K > B - 1) {
      if (threadIdx.x == 0) flag(p.dev_status, FLARE_DEV_BAD_VERIFY_LEN);
      return;
    }
    n = K + 1;  // the live state: after the anchor and every verify token
  } else {
    n = p.accept_len[r];
    if (n < 0 || n > B) {
      if (threadIdx.x == 0) flag(p.dev_status, FLARE_DEV_BAD_ACCEPT_LEN);
      return;
    }
  }
  const int steps = CAUSAL ? B : n;
  if (steps == 0) return;

  float* Ks = smc;                                   // [steps][DK]
  float* Qs = Ks + steps * DK;                       // [steps][DK] (CAUSAL only)
  float* Vs = Qs + (CAUSAL ? steps * DK : 0);        // [steps][DV]

  float* Sg = p.state_pool + ((size_t)slot * p.Hv + j) * DK * DV + (size_t)rg * kR * DV + c0;
  // S~[rg*kR + m][c0 .. c0+3] as two fp32 pairs (columns c0, c0+1 and c0+2, c0+3):
  // the products and updates run as packed f32x2 multiply-adds
  uint64_t s[kR][2];
#pragma unroll
  for (int m = 0; m < kR; ++m) {
    const ulonglong2 v = *reinterpret_cast<const ulonglong2*>(Sg + (size_t)m * DV);
    s[m][0] = v.x;
    s[m][1] = v.y;
  }

  const T* kg = static_cast<const T*>(p.k) + ((size_t)r * B * p.Hk + h) * DK;
  const T* vg = static_cast<const T*>(p.v) + ((size_t)r * B * p.Hv + j) * DV;
  stage_rows<T, DK, kThreads>(Ks, kg, (size_t)p.Hk * DK, steps);
  if (CAUSAL) {
    const T* qg = static_cast<const T*>(p.q) + ((size_t)r * B * p.Hk + h) * DK;
    stage_rows<T, DK, kThreads>(Qs, qg, (size_t)p.Hk * DK, steps);
  }
  stage_rows<T, DV, kThreads>(Vs, vg, (size_t)p.Hv * DV, steps);
  // the decay schedule, once per CTA (warp 0): Gam_t = exp(gamma_t) with
  // gamma_t = g_1 + ... + g_t while Gam_t stays >= 2^-40 (the common case, one
  // prefix scan); otherwise thread 0 walks the tokens and folds where needed
  if (warp == 0) {
    const size_t gb = (size_t)r * B * p.Hv + j;
    float g0 = lane < steps ? p.log_decay[gb + (size_t)lane * p.Hv] : 0.f;
    float g1 = lane + 32 < steps ? p.log_decay[gb + (size_t)(lane + 32) * p.Hv] : 0.f;
    const float b0 = lane < steps ? p.beta[gb + (size_t)lane * p.Hv] : 0.f;
    const float b1 = lane + 32 < steps ? p.beta[gb + (size_t)(lane + 32) * p.Hv] : 0.f;
    const float a0 = expf(g0), a1 = expf(g1);
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const float x = __shfl_up_sync(0xffffffffu, g0, o);
      const float y = __shfl_up_sync(0xffffffffu, g1, o);
      if (lane >= o) {
        g0 += x;
        g1 += y;
      }
    }
    g1 += __shfl_sync(0xffffffffu, g0, 31);
    constexpr float kMinLog = -27.725887222397812f;  // ln 2^-40
    const bool fold = __any_sync(0xffffffffu, (lane < steps && g0 < kMinLog) ||
                                                  (lane + 32 < steps && g1 < kMinLog));
    if (!fold) {
      const float e0 = expf(g0), e1 = expf(g1);
      tok_s[lane] = make_float4(e0, b0, expf(-g0), e0);
      tok_s[lane + 32] = make_float4(e1, b1, expf(-g1), e1);
    } else {
      // alpha and beta through shared memory, then the exact running product
      tok_s[lane] = make_float4(a0, b0, 0.f, 0.f);
      tok_s[lane + 32] = make_float4(a1, b1, 0.f, 0.f);
      __syncwarp();
      if (lane == 0) {
        float gam = 1.f;
        for (int t = 0; t < steps; ++t) {
          const float4 e = tok_s[t];
          const float gt = gam * e.x;
          const bool f = gt < kMinGam;
          gam = f ? 1.f : gt;
          tok_s[t] = make_float4(gt, e.y, f ? 0.f : 1.f / gt, gam);
        }
      }
    }
  }
  __syncthreads();

  // out[t] = scale * S^T q_t with S = g * S~ (this thread's 4 columns, the 8
  // row groups of a warp meeting through shuffles)
  auto readout = [&](int t, float g) {
    const float4* q4 = reinterpret_cast<const float4*>(Qs + t * DK + rg * kR);
    uint64_t o01 = 0, o23 = 0;  // fp32 pairs of zero
#pragma unroll
    for (int m4 = 0; m4 < kR / 4; ++m4) {
      const float4 qq = q4[m4];
      const float qv[4] = {qq.x, qq.y, qq.z, qq.w};
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int m = 4 * m4 + e;
        const uint64_t q2 = f2_dup(qv[e]);
        o01 = f2_fma(s[m][0], q2, o01);
        o23 = f2_fma(s[m][1], q2, o23);
      }
    }
    float4 o;
    f2_split(o01, o.x, o.y);
    f2_split(o23, o.z, o.w);
#pragma unroll
    for (int sh = 4; sh < 32; sh <<= 1) {
      o.x += __shfl_xor_sync(0xffffffffu, o.x, sh);
      o.y += __shfl_xor_sync(0xffffffffu, o.y, sh);
      o.z += __shfl_xor_sync(0xffffffffu, o.z, sh);
      o.w += __shfl_xor_sync(0xffffffffu, o.w, sh);
    }
    if (rg == 0) {
      T* out = static_cast<T*>(p.out_causal) + (((size_t)r * B + t) * p.Hv + j) * DV + c0;
      const float sc = p.scale * g;
      out[0] = from_f32<T>(sc * o.x);
      out[1] = from_f32<T>(sc * o.y);
      out[2] = from_f32<T>(sc * o.z);
      out[3] = from_f32<T>(sc * o.w);
    }
  };

  float gam = 1.f;  // S = gam * S~
#pragma unroll 1
  for (int t = 0; t < steps; ++t) {
    float k[kR];
    {
      const float4* k4 = reinterpret_cast<const float4*>(Ks + t * DK + rg * kR);
#pragma unroll
      for (int m4 = 0; m4 < kR / 4; ++m4) {
        const float4 kk = k4[m4];
        k[4 * m4] = kk.x;
        k[4 * m4 + 1] = kk.y;
        k[4 * m4 + 2] = kk.z;
        k[4 * m4 + 3] = kk.w;
      }
    }
    // (S~^T k)[c] over this row group, then over the 8 row groups of the warp
    float4 d;
    {
      // two partial sums per pair keep four independent multiply-add chains
      uint64_t d01[2] = {0, 0}, d23[2] = {0, 0};
#pragma unroll
      for (int m = 0; m < kR; ++m) {
        const uint64_t k2 = f2_dup(k[m]);
        d01[m & 1] = f2_fma(s[m][0], k2, d01[m & 1]);
        d23[m & 1] = f2_fma(s[m][1], k2, d23[m & 1]);
      }
      const uint64_t a01 = f2_add(d01[0], d01[1]), a23 = f2_add(d23[0], d23[1]);
      f2_split(a01, d.x, d.y);
      f2_split(a23, d.z, d.w);
    }
#pragma unroll
    for (int o = 4; o < 32; o <<= 1) {
      d.x += __shfl_xor_sync(0xffffffffu, d.x, o);
      d.y += __shfl_xor_sync(0xffffffffu, d.y, o);
      d.z += __shfl_xor_sync(0xffffffffu, d.z, o);
      d.w += __shfl_xor_sync(0xffffffffu, d.w, o);
    }
    const float4 tp = tok_s[t];
    const float gt = tp.x, bt = tp.y;
    const float4 v = *reinterpret_cast<const float4*>(Vs + t * DV + c0);
    float4 delta;
    delta.x = bt * (v.x - gt * d.x);
    delta.y = bt * (v.y - gt * d.y);
    delta.z = bt * (v.z - gt * d.z);
    delta.w = bt * (v.w - gt * d.w);
    if (tp.z != 0.f) {  // uniform across the CTA: the gates are per head
      const float ig = tp.z;
      const uint64_t w01 = f2(delta.x * ig, delta.y * ig), w23 = f2(delta.z * ig, delta.w * ig);
#pragma unroll
      for (int m = 0; m < kR; ++m) {
        const uint64_t k2 = f2_dup(k[m]);
        s[m][0] = f2_fma(k2, w01, s[m][0]);
        s[m][1] = f2_fma(k2, w23, s[m][1]);
      }
    } else {  // fold the decay into the state
      const uint64_t g2 = f2_dup(gt);
      const uint64_t d01 = f2(delta.x, delta.y), d23 = f2(delta.z, delta.w);
#pragma unroll
      for (int m = 0; m < kR; ++m) {
        const uint64_t k2 = f2_dup(k[m]);
        s[m][0] = f2_fma(k2, d01, f2_mul(g2, s[m][0]));
        s[m][1] = f2_fma(k2, d23, f2_mul(g2, s[m][1]));
      }
    }
    gam = tp.w;
    if constexpr (VERIFY) {
      if (t < K) {  // S^(t), streamed past L2: at most one of them is read back
        float* rec = p.verify_states +
                     (((size_t)r * p.max_verify + t) * p.Hv + j) * DK * DV +
                     (size_t)rg * kR * DV + c0;
        const uint64_t g2 = f2_dup(gam);
#pragma unroll
        for (int m = 0; m < kR; ++m)
          __stcs(reinterpret_cast<ulonglong2*>(rec + (size_t)m * DV),
                 make_ulonglong2(f2_mul(g2, s[m][0]), f2_mul(g2, s[m][1])));
      }
    }
    if (t + 1 == n) {
      const uint64_t g2 = f2_dup(gam);
#pragma unroll
      for (int m = 0; m < kR; ++m)
        *reinterpret_cast<ulonglong2*>(Sg + (size_t)m * DV) =
            make_ulonglong2(f2_mul(g2, s[m][0]), f2_mul(g2, s[m][1]));
    }
    if (CAUSAL && (!VERIFY || t <= K)) readout(t, gam);
  }
  if constexpr (VERIFY) {
    // padding and draft rows read the block-end state
#pragma unroll 1
    for (int t = K + 1; t < B; ++t) readout(t, gam);
  }
}

namespace {

template <typename T, int DK, int DV, int MODE>
cudaError_t launch_commit_t(const GdrParams& p, cudaStream_t stream) {
  auto smem_for = [](int B) {
    return sizeof(float) * ((size_t)B * DK * (MODE != 0 ? 2 : 1) + (size_t)B * DV);
  };
  cudaError_t e = cudaFuncSetAttribute(gdr_commit_kernel<T, DK, DV, MODE>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem_for(kCBmax));
  if (e != cudaSuccess) return e;
  gdr_commit_kernel<T, DK, DV, MODE><<<p.R * p.Hv, 2 * DV, smem_for(p.B), stream>>>(p);
  note_launches(1);
  return cudaGetLastError();
}

template <typename T, int MODE>
cudaError_t launch_commit_c(const GdrParams& p, cudaStream_t stream) {
  if (p.dk == 128 && p.dv == 128) return launch_commit_t<T, 128, 128, MODE>(p, stream);
  if (p.dk == 128 && p.dv == 64) return launch_commit_t<T, 128, 64, MODE>(p, stream);
  if (p.dk == 64 && p.dv == 128) return launch_commit_t<T, 64, 128, MODE>(p, stream);
  if (p.dk == 64 && p.dv == 64) return launch_commit_t<T, 64, 64, MODE>(p, stream);
  return cudaErrorInvalidValue;
}

}  // namespace

cudaError_t launch_gdr_commit(const GdrParams& p, bool bf16, cudaStream_t stream) {
  if (p.R == 0) return cudaSuccess;
  const bool causal = p.out_causal != nullptr;
  if (bf16)
    return causal ? launch_commit_c<__nv_bfloat16, 1>(p, stream)
                  : launch_commit_c<__nv_bfloat16, 0>(p, stream);
  return causal ? launch_commit_c<float, 1>(p, stream) : launch_commit_c<float, 0>(p, stream);
}

cudaError_t launch_gdr_verify(const GdrParams& p, bool bf16, cudaStream_t stream) {
  if (p.R == 0) return cudaSuccess;
  return bf16 ? launch_commit_c<__nv_bfloat16, 2>(p, stream) : launch_commit_c<float, 2>(p, stream);
}

}  // namespace flare
