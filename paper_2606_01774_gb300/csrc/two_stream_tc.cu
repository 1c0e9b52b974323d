// Two-stream training forward of a gated-delta-rule layer on tcgen05 tensor
// cores (appendix "Two-stream recurrence and block-level chain rule",
// Eq. noisy-block-fwd; the Route II fused forward): bf16 activations,
// d_k = d_v = 128.
//
// One CTA per (sequence, value head, chunk of 64 tokens), 256 threads.  The
// clean state lives in tensor memory as the fp32 accumulator S~^T (lane c =
// value column, column i = key dimension; S = gam S~ with the decay applied
// lazily, folded back when gam would fall below 2^-40).  The chunk's clean and
// noisy inputs are staged in shared memory once (bf16); the A matrices and
// gate prefixes of every block depend only on them and are formed up front.
// Then, block by block:
//   1. the block's clean keys k_t, noisy keys k~_t and noisy queries q~_l go
//      to shared memory as the rows of a K-major tf32 operand, and
//      Y = S~^T [k; k~; q~] is one kind::tf32 MMA (A = S~^T read from tensor
//      memory, M = 128, N = 3B rounded up to 16, K = 128);
//   2. each thread reads its lane's row of Y and solves one column of the
//      block's B x B unit-lower-triangular systems (Eq. chunk-state): the
//      clean ones on warps 0-3, the noisy ones on warps 4-7, which also form
//      the noisy block-end readout (Eq. noisy-block-fwd)
//        o~_l = s (Gam~_B S^T q~_l + sum_i (Gam~_B / Gam~_i) (q~_l . k~_i) delta~_i);
//   3. the clean deltas, scaled by 1 / (gam Gam_i), go to tensor memory and
//      the rank-B update S~^T += delta'^T K (f_blk of Eq. f-blk) is a second
//      kind::tf32 MMA accumulating into S~^T (K = B rounded up to 8, the
//      block's keys transposed in shared memory as its B operand).
// The products run with tf32 operands and fp32 accumulation; the state itself
// is never rounded below fp32.  Every wait is bounded: a timeout sets
// FLARE_DEV_WAIT_TIMEOUT and the CTA stops, frees its tensor memory and exits.
#include "common.cuh"
#include "kernels.h"
#include "tc.cuh"

namespace flare {

namespace {
constexpr int kTcChunk = 64;
constexpr int kTcThreads = 256;
constexpr float kTcMinGam = 9.094947017729282e-13f;  // 2^-40

template <int B>
struct TsTcCfg {
  static constexpr int kM = kTcChunk / B;             // blocks per chunk
  static constexpr int kN1 = (3 * B + 15) / 16 * 16;  // rows of the product operand
  static constexpr int kKB = B <= 8 ? 8 : 16;         // K of the update
  static constexpr int kX = 4 * kN1 * 128;            // [k; k~; q~]: 4 chunks of kN1 rows x 128 B
  static constexpr int kKT = 128 * 128;               // keys transposed: 128 rows (i) x 128 B
  static constexpr int kStage = 5 * kTcChunk * 128 * 2;  // k, k~, q~, v, v~ (bf16)
  static constexpr int kSmall = 4 * (4 * kTcChunk + 3 * kM * B * B);
  static constexpr int kSmem = kX + kKT + kStage + kSmall;
};

// the chunk's rows of a [.][128] bf16 activation slice (row stride `stride`
// elements) into shared memory as [64][128], all loads issued before the stores
__device__ __forceinline__ void tc_stage(__nv_bfloat16* dst, const __nv_bfloat16* src,
                                         size_t stride) {
  constexpr int kChunks = kTcChunk * 128 / 8;  // 16-byte pieces
  constexpr int kIt = kChunks / kTcThreads;
  uint4 buf[kIt];
#pragma unroll
  for (int it = 0; it < kIt; ++it) {
    const int e = threadIdx.x + it * kTcThreads;
    buf[it] = __ldg(reinterpret_cast<const uint4*>(src + (size_t)(e / 16) * stride + (e % 16) * 8));
  }
#pragma unroll
  for (int it = 0; it < kIt; ++it)
    reinterpret_cast<uint4*>(dst)[threadIdx.x + it * kTcThreads] = buf[it];
}

__device__ __forceinline__ float bf_lo(uint32_t u) { return __uint_as_float(u << 16); }
__device__ __forceinline__ float bf_hi(uint32_t u) { return __uint_as_float(u & 0xffff0000u); }

// every thread of the CTA waits; the outcome is made CTA-uniform
__device__ __forceinline__ bool tc2_wait(uint64_t* bar, uint32_t parity, int* abort_flag,
                                         int32_t* status) {
  const bool ok = tc::mbar_wait(bar, parity, abort_flag);
  const bool all = __syncthreads_and(ok);
  if (!all && threadIdx.x == 0 && !*abort_flag) {
    *abort_flag = 1;
    flag(status, FLARE_DEV_WAIT_TIMEOUT);
  }
  return all;
}
}  // namespace

template <int B>
__global__ void __launch_bounds__(kTcThreads, B <= 4 ? 2 : 1)
    two_stream_tc_kernel(TwoStreamParams p) {
  using Cfg = TsTcCfg<B>;
  constexpr int DK = 128, DV = 128, C = kTcChunk, M = Cfg::kM, N1 = Cfg::kN1, KB = Cfg::kKB;
  extern __shared__ uint8_t ts2_raw[];
  __shared__ uint64_t bar_p1, bar_upd;
  __shared__ uint32_t tmem_base;
  __shared__ int abort_flag;
  uint8_t* base = (uint8_t*)(((uintptr_t)ts2_raw + 1023) & ~(uintptr_t)1023);
  uint8_t* Xs = base;             // [4][N1][128 B]: rows kind*B + t, column chunks of 32
  uint8_t* KT = Xs + Cfg::kX;     // [128][128 B]: row i holds k_t[i], t < B
  __nv_bfloat16* ck = reinterpret_cast<__nv_bfloat16*>(KT + Cfg::kKT);  // clean k [C][DK]
  __nv_bfloat16* nk = ck + C * DK;                                       // noisy k
  __nv_bfloat16* nq = nk + C * DK;                                       // noisy q
  __nv_bfloat16* cv = nq + C * DK;                                       // clean v [C][DV]
  __nv_bfloat16* nv = cv + C * DV;                                       // noisy v
  float* lgc = reinterpret_cast<float*>(nv + C * DV);  // clean log-gate, prefix within the block
  float* cb = lgc + C;                                 // clean beta
  float* lgn = cb + C;                                 // noisy log-gate prefix
  float* nb = lgn + C;                                 // noisy beta
  float* Ac = nb + C;                                  // [M][B][B]
  float* An = Ac + M * B * B;
  float* Aqk = An + M * B * B;

  const int n_chunks = p.L / C;
  const int c = blockIdx.x % n_chunks;
  const int j = (blockIdx.x / n_chunks) % p.Hv;
  const int n = blockIdx.x / (n_chunks * p.Hv);
  const int h = j / (p.Hv / p.Hk);
  const int tid = threadIdx.x, warp = tid >> 5;
  const int row = tid & 127;  // this thread's tensor-memory lane = value column
  const uint32_t lane_off = (uint32_t)((warp & 3) * 32) << 16;
  const size_t tok0 = (size_t)n * p.L + (size_t)c * C;

  if (tid == 0) {
    abort_flag = 0;
    tc::mbar_init(&bar_p1, 1);
    tc::mbar_init(&bar_upd, 1);
    tc::fence_mbar_init();
  }
  if (warp == 0) tc::tmem_alloc(&tmem_base, 256);
  // the operand tiles start at zero: their padding rows and columns stay so
  for (int e = tid; e < (Cfg::kX + Cfg::kKT) / 16; e += kTcThreads)
    reinterpret_cast<uint4*>(Xs)[e] = make_uint4(0u, 0u, 0u, 0u);
  const __nv_bfloat16* kg = static_cast<const __nv_bfloat16*>(p.k) + (tok0 * p.Hk + h) * DK;
  const __nv_bfloat16* kng = static_cast<const __nv_bfloat16*>(p.kn) + (tok0 * p.Hk + h) * DK;
  const __nv_bfloat16* qng = static_cast<const __nv_bfloat16*>(p.qn) + (tok0 * p.Hk + h) * DK;
  tc_stage(ck, kg, (size_t)p.Hk * DK);
  tc_stage(nk, kng, (size_t)p.Hk * DK);
  tc_stage(nq, qng, (size_t)p.Hk * DK);
  tc_stage(cv, static_cast<const __nv_bfloat16*>(p.v) + (tok0 * p.Hv + j) * DV, (size_t)p.Hv * DV);
  tc_stage(nv, static_cast<const __nv_bfloat16*>(p.vn) + (tok0 * p.Hv + j) * DV, (size_t)p.Hv * DV);
  // gates: the log-gates as prefix sums within each block, and the betas
  if (tid < 2 * C) {
    const bool noisy = tid >= C;
    const int t = noisy ? tid - C : tid;
    const float* g = noisy ? p.gn : p.g;
    const float* bt = noisy ? p.betan : p.beta;
    float acc = 0.f;
    for (int i = t - t % B; i <= t; ++i) acc += g[(tok0 + i) * p.Hv + j];
    (noisy ? lgn : lgc)[t] = acc;
    (noisy ? nb : cb)[t] = bt[(tok0 + t) * p.Hv + j];
  }
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = tmem_base;
  const uint32_t tmS = tmem;        // S~^T                       (128 columns)
  const uint32_t tmY = tmem + 128;  // Y = S~^T [k; k~; q~]       (N1 <= 48 columns)
  const uint32_t tmD = tmem + 192;  // delta'^T, the update's A   (16 columns)

  // the chunk-start clean state: lane `row` holds S[i][row] over i, this
  // thread the half (tid >> 7) of the columns i
  {
    const float* Sg = p.chunk_states + (((size_t)n * p.Hv + j) * n_chunks + c) * DK * DV;
    const int half = tid >> 7;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      uint32_t v[16];
#pragma unroll
      for (int e = 0; e < 16; ++e)
        v[e] = __float_as_uint(__ldg(Sg + (size_t)(half * 64 + q * 16 + e) * DV + row));
      tc::tmem_st16(tmS + lane_off + half * 64 + q * 16, v);
    }
    tc::tmem_st_wait();
  }
  // A matrices of every block of the chunk (inputs only)
  for (int e = tid; e < 3 * M * B * B; e += kTcThreads) {
    const int kind = e / (M * B * B);
    const int r = e % (M * B * B);
    const int m = r / (B * B), t = (r / B) % B, i = r % B;
    const int tt = m * B + t, ti = m * B + i;
    float val = 0.f;
    if (kind == 2 || i < t) {
      const uint4* x = reinterpret_cast<const uint4*>(
          kind == 0 ? ck + tt * DK : (kind == 1 ? nk + tt * DK : nq + tt * DK));
      const uint4* y = reinterpret_cast<const uint4*>(kind == 0 ? ck + ti * DK : nk + ti * DK);
      float dot = 0.f;
#pragma unroll 4
      for (int d = 0; d < DK / 8; ++d) {
        const uint4 a = x[d], b = y[d];
        dot = fmaf(bf_lo(a.x), bf_lo(b.x), dot);
        dot = fmaf(bf_hi(a.x), bf_hi(b.x), dot);
        dot = fmaf(bf_lo(a.y), bf_lo(b.y), dot);
        dot = fmaf(bf_hi(a.y), bf_hi(b.y), dot);
        dot = fmaf(bf_lo(a.z), bf_lo(b.z), dot);
        dot = fmaf(bf_hi(a.z), bf_hi(b.z), dot);
        dot = fmaf(bf_lo(a.w), bf_lo(b.w), dot);
        dot = fmaf(bf_hi(a.w), bf_hi(b.w), dot);
      }
      if (kind == 0) val = cb[tt] * __expf(lgc[tt] - lgc[ti]) * dot;
      else if (kind == 1) val = nb[tt] * __expf(lgn[tt] - lgn[ti]) * dot;
      else val = __expf(lgn[m * B + B - 1] - lgn[ti]) * dot;
    }
    (kind == 0 ? Ac : (kind == 1 ? An : Aqk))[r] = val;
  }

  float gam = 1.f;  // S = gam S~
  __nv_bfloat16* outg = static_cast<__nv_bfloat16*>(p.out) + (tok0 * p.Hv + j) * DV;
  const uint32_t id_p1 = tc::idesc_tf32(128, N1);
  const uint32_t id_up = tc::idesc_tf32(128, 128);
#pragma unroll 1
  for (int m = 0; m < M; ++m) {
    const int t0 = m * B;
    // 1. the product operand: rows kind*B + t of [k; k~; q~] as tf32, K-major,
    //    128-byte swizzle (4 chunks of 32 key dimensions)
    for (int e = tid; e < 3 * B * 16; e += kTcThreads) {
      const int nrow = e >> 4, p8 = e & 15;  // 8 key dimensions per piece
      const int kind = nrow / B, t = nrow % B;
      const uint4 raw = *reinterpret_cast<const uint4*>(
          (kind == 0 ? ck : (kind == 1 ? nk : nq)) + (t0 + t) * DK + p8 * 8);
      uint8_t* dst = Xs + (p8 >> 2) * (N1 * 128) + nrow * 128;
      const int u0 = (p8 & 3) * 2;  // 16-byte unit within the 128-byte row
      *reinterpret_cast<uint4*>(dst + ((u0 ^ (nrow & 7)) << 4)) =
          make_uint4(tc::to_tf32(bf_lo(raw.x)), tc::to_tf32(bf_hi(raw.x)),
                     tc::to_tf32(bf_lo(raw.y)), tc::to_tf32(bf_hi(raw.y)));
      *reinterpret_cast<uint4*>(dst + (((u0 + 1) ^ (nrow & 7)) << 4)) =
          make_uint4(tc::to_tf32(bf_lo(raw.z)), tc::to_tf32(bf_hi(raw.z)),
                     tc::to_tf32(bf_lo(raw.w)), tc::to_tf32(bf_hi(raw.w)));
    }
    tc::fence_async_smem();
    tc::fence_before_sync();
    __syncthreads();
    if (tid == 0) {
      tc::fence_after_sync();
      // MMAs issued by one thread execute in issue order: this product reads
      // S~ after the previous block's update has written it
#pragma unroll
      for (int kk = 0; kk < DK / 8; ++kk) {
        const uint64_t b = tc::sdesc_sw128(
            tc::smem_u32(Xs + (kk >> 2) * (N1 * 128) + (kk & 3) * 32), 16, 1024);
        tc::mma_tf32_ts(tmY, tmS + kk * 8, b, id_p1, kk > 0);
      }
      tc::mma_commit(&bar_p1);
    }
    if (!tc2_wait(&bar_p1, (uint32_t)m & 1u, &abort_flag, p.dev_status)) break;
    tc::fence_after_sync();
    // this lane's row of Y
    uint32_t y[N1];
#pragma unroll
    for (int q = 0; q < N1 / 16; ++q)
      tc::tmem_ld16(tmY + lane_off + q * 16, *reinterpret_cast<uint32_t(*)[16]>(&y[q * 16]));
    tc::tmem_ld_wait();
    // the block's keys transposed, the update's B operand (row i, element t);
    // the previous update has completed (the product above followed it in
    // issue order), so its operands may be overwritten
    for (int e = tid; e < 128 * B; e += kTcThreads) {
      const int i = e / B, t = e % B;
      const float kv = __bfloat162float(ck[(t0 + t) * DK + i]);
      *reinterpret_cast<uint32_t*>(KT + i * 128 + (((t >> 2) ^ (i & 7)) << 4) + (t & 3) * 4) =
          tc::to_tf32(kv);
    }
    const float gB = __expf(lgc[t0 + B - 1]);
    const bool fold = gam * gB < kTcMinGam;  // uniform: the gates are per head
    // 2. the block's UT systems, one column per thread
    {
      const bool noisy = tid >= DV;
      const int col = row;
      const float* A = (noisy ? An : Ac) + m * B * B;
      const float* lg = noisy ? lgn : lgc;
      const float* bt = noisy ? nb : cb;
      const __nv_bfloat16* vv = noisy ? nv : cv;
      float d[B];
#pragma unroll
      for (int t = 0; t < B; ++t) {
        const float yk = __uint_as_float(noisy ? y[B + t] : y[t]);  // S~^T k_t or S~^T k~_t
        float x = bt[t0 + t] * (__bfloat162float(vv[(t0 + t) * DV + col]) -
                                __expf(lg[t0 + t]) * gam * yk);
#pragma unroll
        for (int i = 0; i < t; ++i) x = fmaf(-A[t * B + i], d[i], x);
        d[t] = x;
      }
      if (!noisy) {
        // delta'_i = delta_i (Gam_B / Gam_i) when the decay folds, else
        // delta_i / (gam Gam_i): S~ += k_i delta'_i^T
        uint32_t w[16];
#pragma unroll
        for (int t = 0; t < 16; ++t) {
          float v = 0.f;
          if (t < B) {
            const float coef = fold ? __expf(lgc[t0 + B - 1] - lgc[t0 + t])
                                    : __expf(-lgc[t0 + t]) / gam;
            v = coef * d[t];
          }
          w[t] = tc::to_tf32(v);
        }
        tc::tmem_st16(tmD + lane_off, w);
      } else {
        const float gBn = __expf(lgn[t0 + B - 1]);
        const float* Aq = Aqk + m * B * B;
#pragma unroll
        for (int l = 0; l < B; ++l) {
          float o = gBn * gam * __uint_as_float(y[2 * B + l]);
#pragma unroll
          for (int i = 0; i < B; ++i) o = fmaf(Aq[l * B + i], d[i], o);
          outg[(size_t)(t0 + l) * p.Hv * DV + col] = __float2bfloat16_rn(p.scale * o);
        }
      }
    }
    if (fold) {
      // S~ <- gam Gam_B S~ (the product above has read S~)
      const float f = gam * gB;
      const int half = tid >> 7;
#pragma unroll 1
      for (int q = 0; q < 4; ++q) {
        uint32_t v[16];
        tc::tmem_ld16(tmS + lane_off + half * 64 + q * 16, v);
        tc::tmem_ld_wait();
#pragma unroll
        for (int e = 0; e < 16; ++e) v[e] = __float_as_uint(f * __uint_as_float(v[e]));
        tc::tmem_st16(tmS + lane_off + half * 64 + q * 16, v);
      }
    }
    tc::tmem_st_wait();
    tc::fence_async_smem();
    tc::fence_before_sync();
    __syncthreads();
    // 3. S~^T += delta'^T K
    if (tid == 0) {
      tc::fence_after_sync();
#pragma unroll
      for (int kk = 0; kk < KB / 8; ++kk)
        tc::mma_tf32_ts(tmS, tmD + kk * 8,
                        tc::sdesc_sw128(tc::smem_u32(KT + kk * 32), 16, 1024), id_up, 1u);
      tc::mma_commit(&bar_upd);
    }
    gam = fold ? 1.f : gam * gB;
  }
  // the last update has completed before the tensor memory is freed
  if (tid == 0 && !abort_flag) tc::mbar_wait(&bar_upd, (uint32_t)(M - 1) & 1u, &abort_flag);
  tc::fence_before_sync();
  __syncthreads();
  if (warp == 0) {
    tc::fence_after_sync();
    tc::tmem_dealloc(tmem, 256);
  }
}

namespace {
template <int B>
cudaError_t launch_ts_tc_b(const TwoStreamParams& p, cudaStream_t stream) {
  const int smem = TsTcCfg<B>::kSmem + 1024;
  cudaError_t e = cudaFuncSetAttribute(two_stream_tc_kernel<B>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  const unsigned grid = (unsigned)((size_t)p.N * p.Hv * (p.L / kTcChunk));
  two_stream_tc_kernel<B><<<grid, kTcThreads, smem, stream>>>(p);
  note_launches(1);
  return cudaGetLastError();
}
}  // namespace

bool two_stream_tc_supported(int B, int dk, int dv) {
  return dk == 128 && dv == 128 && (B == 1 || B == 2 || B == 4 || B == 8 || B == 16);
}

cudaError_t launch_two_stream_tc(const TwoStreamParams& p, cudaStream_t stream) {
  if (p.N == 0) return cudaSuccess;
  switch (p.B) {
    case 1: return launch_ts_tc_b<1>(p, stream);
    case 2: return launch_ts_tc_b<2>(p, stream);
    case 4: return launch_ts_tc_b<4>(p, stream);
    case 8: return launch_ts_tc_b<8>(p, stream);
    case 16: return launch_ts_tc_b<16>(p, stream);
  }
  return cudaErrorInvalidValue;
}

}  // namespace flare
