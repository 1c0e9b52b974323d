// Two-stream training forward of a gated-delta-rule layer, noisy stream
// (appendix "Two-stream recurrence and block-level chain rule",
// Eq. noisy-block-fwd; the Route II fused forward), CUDA-core form in exact
// fp32.  It serves fp32 activations; bf16 activations (d_k = d_v = 128) take
// the chunkwise tensor-core kernel in two_stream_chunk.cu.
//
// One CTA per (sequence, value head, chunk of 64 tokens).  The clean state
// S_[c] at the chunk start (from the clean chunkwise pass) is loaded into
// registers -- each thread holds a 4-column x d_k/8-row block, lane =
// 4 x row group + column group as in the commit kernel -- and the chunk's
// clean and noisy inputs are staged in shared memory once.  Then, block by
// block, with S the clean state before the block:
//   1. every thread forms its rows' share of S^T k_t (clean), S^T k~_t and
//      S^T q~_l (noisy) for the block's tokens; three shuffles finish the
//      column sums, which go to shared memory;
//   2. 2 d_v threads solve the block's two B x B unit-lower-triangular
//      systems, one column each (the chunkwise UT form, Eq. chunk-state):
//        delta_t  = beta_t (v_t - Gam_t S^T k_t) - sum_{i<t} A_ti delta_i,
//        A_ti     = beta_t (Gam_t / Gam_i) (k_t . k_i),
//      the clean ones on the first d_v threads, the noisy ones on the others,
//      which also read the noisy block-end state (Eq. noisy-block-fwd):
//        o~_l = s (Gam~_B S^T q~_l + sum_i (Gam~_B / Gam~_i) (q~_l . k~_i) delta~_i);
//   3. the clean state advances over the block in registers (f_blk of
//      Eq. f-blk): S <- Gam_B S + sum_i (Gam_B / Gam_i) k_i delta_i^T.
// No block-boundary state leaves the chip.  The A matrices and the gate
// prefixes of every block depend only on the inputs, so they are formed for
// the whole chunk before the block loop.  The decay of the clean state is
// applied lazily (S = gam S~, folded back when gam would fall below 2^-40).
// All arithmetic is fp32 (the state products and updates as packed f32x2
// multiply-adds on column pairs); the noisy state is never formed.
#include "common.cuh"
#include "kernels.h"

namespace flare {

namespace {
constexpr int kTsChunk = 64;
constexpr int kTsGroup = 2;  // tokens whose products one pass over the state forms
constexpr float kTsMinGam = 9.094947017729282e-13f;  // 2^-40

template <typename T>
__device__ __forceinline__ void load_vec16(const T* src, float (&f)[16]) {
  if constexpr (sizeof(T) == 2) {
    const uint4 a = *reinterpret_cast<const uint4*>(src);
    const uint4 b = *reinterpret_cast<const uint4*>(src + 8);
    const uint32_t u[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      f[2 * e] = __uint_as_float(u[e] << 16);
      f[2 * e + 1] = __uint_as_float(u[e] & 0xffff0000u);
    }
  } else {
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const float4 v = reinterpret_cast<const float4*>(src)[e];
      f[4 * e] = v.x;
      f[4 * e + 1] = v.y;
      f[4 * e + 2] = v.z;
      f[4 * e + 3] = v.w;
    }
  }
}

// rows [0, rows) of a [.][N] activation slice (row stride `stride` elements) into
// shared memory as [rows][N], 16-byte pieces, all loads issued before the stores
template <typename T, int N, int THREADS>
__device__ __forceinline__ void ts_stage(T* dst, const T* src, size_t stride) {
  constexpr int kPer = 16 / sizeof(T);
  constexpr int kChunks = kTsChunk * N / kPer;
  constexpr int kIt = (kChunks + THREADS - 1) / THREADS;
  uint4 buf[kIt];
#pragma unroll
  for (int it = 0; it < kIt; ++it) {
    const int e = threadIdx.x + it * THREADS;
    if (e < kChunks) {
      const int t = e / (N / kPer), ch = e % (N / kPer);
      buf[it] = __ldg(reinterpret_cast<const uint4*>(src + (size_t)t * stride + ch * kPer));
    }
  }
#pragma unroll
  for (int it = 0; it < kIt; ++it) {
    const int e = threadIdx.x + it * THREADS;
    if (e < kChunks) reinterpret_cast<uint4*>(dst)[e] = buf[it];
  }
}
}  // namespace

template <typename T, int DK, int DV, int B>
__global__ void __launch_bounds__(2 * DV, (B <= 4 && sizeof(T) == 2) ? 2 : 1)
    two_stream_fwd_kernel(TwoStreamParams p) {
  constexpr int kThreads = 2 * DV;
  constexpr int kR = DK / 8;  // state rows per thread
  static_assert(kR % 16 == 0, "a thread's state rows are read 16 at a time");
  constexpr int C = kTsChunk;
  constexpr int M = C / B;    // blocks per chunk
  constexpr int G = B < kTsGroup ? B : kTsGroup;
  extern __shared__ float4 ts_smem[];
  T* ck = reinterpret_cast<T*>(ts_smem);  // clean k   [C][DK]
  T* nk = ck + C * DK;                    // noisy k   [C][DK]
  T* nq = nk + C * DK;                    // noisy q   [C][DK]
  T* cv = nq + C * DK;                    // clean v   [C][DV]
  T* nv = cv + C * DV;                    // noisy v   [C][DV]
  float* lgc = reinterpret_cast<float*>(nv + C * DV);  // clean log-gate, prefix within the block
  float* cb = lgc + C;                                 // clean beta
  float* lgn = cb + C;                                 // noisy log-gate prefix
  float* nb = lgn + C;                                 // noisy beta
  float* Ac = nb + C;                                  // [M][B][B]
  float* An = Ac + M * B * B;                          // [M][B][B]
  float* Aqk = An + M * B * B;                         // [M][B][B]
  float* Y = Aqk + M * B * B;                          // [3][B][DV]: S^T k, S^T k~, S^T q~
  float* Dl = Y + 3 * B * DV;                          // [B][DV] clean deltas

  const int n_chunks = p.L / C;
  const int c = blockIdx.x % n_chunks;
  const int j = (blockIdx.x / n_chunks) % p.Hv;
  const int n = blockIdx.x / (n_chunks * p.Hv);
  const int h = j / (p.Hv / p.Hk);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int rg = lane >> 2;
  const int c0 = warp * 16 + (lane & 3) * 4;
  const size_t tok0 = (size_t)n * p.L + (size_t)c * C;  // first token of the chunk

  // the chunk-start clean state, issued before anything else
  const float* Sg = p.chunk_states + (((size_t)n * p.Hv + j) * n_chunks + c) * DK * DV +
                    (size_t)rg * kR * DV + c0;
  uint64_t s[kR][2];  // fp32 pairs: columns c0, c0+1 and c0+2, c0+3
#pragma unroll
  for (int m = 0; m < kR; ++m) {
    const ulonglong2 v = __ldg(reinterpret_cast<const ulonglong2*>(Sg + (size_t)m * DV));
    s[m][0] = v.x;
    s[m][1] = v.y;
  }

  ts_stage<T, DK, kThreads>(ck, static_cast<const T*>(p.k) + (tok0 * p.Hk + h) * DK,
                            (size_t)p.Hk * DK);
  ts_stage<T, DK, kThreads>(nk, static_cast<const T*>(p.kn) + (tok0 * p.Hk + h) * DK,
                            (size_t)p.Hk * DK);
  ts_stage<T, DK, kThreads>(nq, static_cast<const T*>(p.qn) + (tok0 * p.Hk + h) * DK,
                            (size_t)p.Hk * DK);
  ts_stage<T, DV, kThreads>(cv, static_cast<const T*>(p.v) + (tok0 * p.Hv + j) * DV,
                            (size_t)p.Hv * DV);
  ts_stage<T, DV, kThreads>(nv, static_cast<const T*>(p.vn) + (tok0 * p.Hv + j) * DV,
                            (size_t)p.Hv * DV);
  // gates: the log-gates as prefix sums within each block, and the betas
  if (tid < 2 * C) {
    const bool noisy = tid >= C;
    const int t = noisy ? tid - C : tid;
    const float* g = noisy ? p.gn : p.g;
    const float* bt = noisy ? p.betan : p.beta;
    const size_t gb = (tok0 + t) * p.Hv + j;
    float acc = 0.f;
    for (int i = t - t % B; i <= t; ++i) acc += g[(tok0 + i) * p.Hv + j];
    (noisy ? lgn : lgc)[t] = acc;
    (noisy ? nb : cb)[t] = bt[gb];
  }
  __syncthreads();

  // A matrices of every block of the chunk (inputs only)
  for (int e = tid; e < 3 * M * B * B; e += kThreads) {
    const int kind = e / (M * B * B);
    const int r = e % (M * B * B);
    const int m = r / (B * B), t = (r / B) % B, i = r % B;
    const int tt = m * B + t, ti = m * B + i;
    float val = 0.f;
    if (kind == 2 || i < t) {
      const T* x = kind == 0 ? ck + tt * DK : (kind == 1 ? nk + tt * DK : nq + tt * DK);
      const T* y = kind == 0 ? ck + ti * DK : nk + ti * DK;
      float dot = 0.f;
#pragma unroll 4
      for (int d = 0; d < DK; d += 16) {
        float xf[16], yf[16];
        load_vec16<T>(x + d, xf);
        load_vec16<T>(y + d, yf);
#pragma unroll
        for (int q = 0; q < 16; ++q) dot = fmaf(xf[q], yf[q], dot);
      }
      if (kind == 0) val = cb[tt] * __expf(lgc[tt] - lgc[ti]) * dot;
      else if (kind == 1) val = nb[tt] * __expf(lgn[tt] - lgn[ti]) * dot;
      else val = __expf(lgn[m * B + B - 1] - lgn[ti]) * dot;
    }
    (kind == 0 ? Ac : (kind == 1 ? An : Aqk))[r] = val;
  }
  __syncthreads();

  float gam = 1.f;  // S = gam S~
  T* outg = static_cast<T*>(p.out) + (tok0 * p.Hv + j) * DV;
#pragma unroll 1
  for (int m = 0; m < M; ++m) {
    const int t0 = m * B;
    // 1. products of the state with the block's clean keys, noisy keys, noisy queries
#pragma unroll 1
    for (int tg = 0; tg < B; tg += G) {
      float4 acc[3][G];
#pragma unroll
      for (int kind = 0; kind < 3; ++kind)
#pragma unroll
        for (int u = 0; u < G; ++u) {
          const T* x = (kind == 0 ? ck : (kind == 1 ? nk : nq)) + (t0 + tg + u) * DK + rg * kR;
          uint64_t a01 = 0, a23 = 0;  // fp32 pairs of zero
#pragma unroll
          for (int r0 = 0; r0 < kR; r0 += 16) {
            float xf[16];
            load_vec16<T>(x + r0, xf);
#pragma unroll
            for (int q = 0; q < 16; ++q) {
              const uint64_t x2 = f2_dup(xf[q]);
              a01 = f2_fma(s[r0 + q][0], x2, a01);
              a23 = f2_fma(s[r0 + q][1], x2, a23);
            }
          }
          float4 a4;
          f2_split(a01, a4.x, a4.y);
          f2_split(a23, a4.z, a4.w);
          acc[kind][u] = a4;
        }
#pragma unroll
      for (int kind = 0; kind < 3; ++kind)
#pragma unroll
        for (int u = 0; u < G; ++u) {
          float4 a = acc[kind][u];
#pragma unroll
          for (int o = 4; o < 32; o <<= 1) {
            a.x += __shfl_xor_sync(0xffffffffu, a.x, o);
            a.y += __shfl_xor_sync(0xffffffffu, a.y, o);
            a.z += __shfl_xor_sync(0xffffffffu, a.z, o);
            a.w += __shfl_xor_sync(0xffffffffu, a.w, o);
          }
          if (rg == 0)
            *reinterpret_cast<float4*>(Y + (kind * B + tg + u) * DV + c0) =
                make_float4(gam * a.x, gam * a.y, gam * a.z, gam * a.w);
        }
    }
    __syncthreads();
    // 2. the block's UT systems, one column per thread: clean on the first DV
    //    threads, noisy (and the readout) on the others
    {
      const bool noisy = tid >= DV;
      const int col = noisy ? tid - DV : tid;
      const float* A = (noisy ? An : Ac) + m * B * B;
      const float* lg = noisy ? lgn : lgc;
      const float* bt = noisy ? nb : cb;
      const T* vv = noisy ? nv : cv;
      const float* yk = Y + (noisy ? B : 0) * DV + col;
      float d[B];
#pragma unroll
      for (int t = 0; t < B; ++t) {
        float x = bt[t0 + t] * (to_f32(vv[(t0 + t) * DV + col]) - __expf(lg[t0 + t]) * yk[t * DV]);
#pragma unroll
        for (int i = 0; i < t; ++i) x = fmaf(-A[t * B + i], d[i], x);
        d[t] = x;
      }
      if (!noisy) {
#pragma unroll
        for (int t = 0; t < B; ++t) Dl[t * DV + col] = d[t];
      } else {
        const float gB = __expf(lgn[t0 + B - 1]);
        const float* Aq = Aqk + m * B * B;
        const float* yq = Y + 2 * B * DV + col;
#pragma unroll
        for (int l = 0; l < B; ++l) {
          float o = gB * yq[l * DV];
#pragma unroll
          for (int i = 0; i < B; ++i) o = fmaf(Aq[l * B + i], d[i], o);
          outg[(size_t)(t0 + l) * p.Hv * DV + col] = from_f32<T>(p.scale * o);
        }
      }
    }
    __syncthreads();
    // 3. the clean state advances over the block (f_blk), lazily decayed
    {
      const float gB = __expf(lgc[t0 + B - 1]);
      const bool fold = gam * gB < kTsMinGam;  // uniform: the gates are per head
      if (fold) {
        const uint64_t f = f2_dup(gam * gB);
#pragma unroll
        for (int r = 0; r < kR; ++r) {
          s[r][0] = f2_mul(f, s[r][0]);
          s[r][1] = f2_mul(f, s[r][1]);
        }
      }
#pragma unroll 1
      for (int i = 0; i < B; ++i) {
        // fold: S = Gam_B S + sum_i (Gam_B / Gam_i) k_i delta_i^T with gam = 1;
        // else S~ += k_i delta_i^T / (gam Gam_i) and gam *= Gam_B
        const float coef = fold ? __expf(lgc[t0 + B - 1] - lgc[t0 + i])
                                : __expf(-lgc[t0 + i]) / gam;
        const float4 dd = *reinterpret_cast<const float4*>(Dl + i * DV + c0);
        const uint64_t w01 = f2(dd.x * coef, dd.y * coef), w23 = f2(dd.z * coef, dd.w * coef);
        const T* x = ck + (t0 + i) * DK + rg * kR;
#pragma unroll
        for (int r0 = 0; r0 < kR; r0 += 16) {
          float xf[16];
          load_vec16<T>(x + r0, xf);
#pragma unroll
          for (int q = 0; q < 16; ++q) {
            const uint64_t x2 = f2_dup(xf[q]);
            s[r0 + q][0] = f2_fma(x2, w01, s[r0 + q][0]);
            s[r0 + q][1] = f2_fma(x2, w23, s[r0 + q][1]);
          }
        }
      }
      gam = fold ? 1.f : gam * gB;
    }
  }
}

namespace {
template <typename T, int DK, int DV, int B>
size_t ts_smem_bytes() {
  constexpr int M = kTsChunk / B;
  return (size_t)(3 * kTsChunk * DK + 2 * kTsChunk * DV) * sizeof(T) +
         sizeof(float) * (4 * kTsChunk + 3 * M * B * B + 3 * B * DV + B * DV);
}

template <typename T, int DK, int DV, int B>
cudaError_t launch_ts_t(const TwoStreamParams& p, cudaStream_t stream) {
  const size_t smem = ts_smem_bytes<T, DK, DV, B>();
  cudaError_t e = cudaFuncSetAttribute(two_stream_fwd_kernel<T, DK, DV, B>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  const unsigned grid = (unsigned)((size_t)p.N * p.Hv * (p.L / kTsChunk));
  two_stream_fwd_kernel<T, DK, DV, B><<<grid, 2 * DV, smem, stream>>>(p);
  note_launches(1);
  return cudaGetLastError();
}

template <typename T, int DK, int DV>
cudaError_t launch_ts_b(const TwoStreamParams& p, cudaStream_t stream) {
  switch (p.B) {
    case 1: return launch_ts_t<T, DK, DV, 1>(p, stream);
    case 2: return launch_ts_t<T, DK, DV, 2>(p, stream);
    case 4: return launch_ts_t<T, DK, DV, 4>(p, stream);
    case 8: return launch_ts_t<T, DK, DV, 8>(p, stream);
    case 16: return launch_ts_t<T, DK, DV, 16>(p, stream);
  }
  return cudaErrorInvalidValue;
}

template <typename T>
cudaError_t launch_ts_d(const TwoStreamParams& p, cudaStream_t stream) {
  if (p.dk == 128 && p.dv == 128) return launch_ts_b<T, 128, 128>(p, stream);
  return cudaErrorInvalidValue;
}
}  // namespace

int two_stream_chunk_len() { return kTsChunk; }

cudaError_t launch_two_stream_fwd(const TwoStreamParams& p, bool bf16, cudaStream_t stream) {
  if (p.N == 0) return cudaSuccess;
  // bf16 activations take the chunkwise tensor-core kernel (two_stream_chunk.cu)
  if (bf16 && two_stream_chunk_supported(p.B, p.dk, p.dv)) return launch_two_stream_chunk(p, stream);
  return bf16 ? launch_ts_d<__nv_bfloat16>(p, stream) : launch_ts_d<float>(p, stream);
}

}  // namespace flare
