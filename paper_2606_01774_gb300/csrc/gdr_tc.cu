// Denoise pass of a gated-delta-rule layer on tcgen05 tensor cores.
//
// For one (request r, value head j) with q/k head h, block length B <= 64 and
// frozen state S0 (dk x dv, fp32), the block-end readout (Eq. noisy-block-fwd)
// is evaluated through the chunkwise WY/UT form of the block (appendix,
// "Chunk-corrected values", Eq. chunk-state) instead of B sequential steps:
//
//   gamma_t = sum_{i<=t} g_i,  Gam_t = exp(gamma_t)             (cumulative log-gate)
//   A[t][i] = beta_t exp(gamma_t - gamma_i) (k_t . k_i),  i < t
//   X       = diag(beta) (V - diag(Gam) K S0)
//   (I + A) delta = X                                          (per-step delta updates)
//   out[l]  = s (Gam_B S0^T q_l + sum_i exp(gamma_B - gamma_i) (q_l . k_i) delta_i)
//
// Every product with S0 or delta is computed transposed, with the value
// dimension c on the 128 TMEM lanes: column c of the state evolves
// independently of the others (the update acts on S from the left), so thread
// c owns everything about column c from the first MMA to its output.
//
//   MMA 1   G   = [K;Q] K^T          M=128 (BM k rows, BM q rows), N=Bp, K=dk
//   MMA 2   W^T = S0^T [K;Q]^T       M=128 (c),  N=2BM, K=dk   (S0^T is MN-major)
//   solve   (I + A) delta = X        unit lower triangular, 16 rows at a time:
//                                    off-diagonal terms on warp-level tf32 MMA,
//                                    diagonal blocks by fp32 forward substitution
//   MMA 4   O2^T = delta^T M2^T      M=128 (c),  N=Bp,  K=Bp, M2[l][i] = exp(gamma_B-gamma_i) q_l.k_i
//   out[l][c] = s (Gam_B W^T[c][BM+l] + O2^T[c][l])
//
// Bp = B rounded up to 16; BM = 32 for B <= 32, else 64 (the K/Q/V tiles hold
// BM rows).  Inputs bf16, state fp32 read once and rounded to bf16 for the
// MMA, all accumulation fp32.  One CTA per (request, value head), 128
// threads: BM = 64 takes 106 KiB of shared memory and 256 TMEM columns (two
// CTAs per SM), BM = 32 73 KiB and 128 columns (three CTAs per SM).
#include <cudaTypedefs.h>

#include "common.cuh"
#include "kernels.h"
#include "tc.cuh"

namespace flare {

namespace {

constexpr int kLinThreads = 128;
constexpr int kBmax = 64;

// Layout for blocks of up to BM rows (BM = 64, or 32 for B <= 32, which fits
// three CTAs on an SM instead of two).
template <int DK, int DV, int BM>
struct LinCfg {
  static constexpr int kATs = BM + 8;                // row stride of A^T: conflict-free tf32 fragment loads
  static constexpr int kKQ = (DK / 64) * 2 * BM * 128;  // [K;Q]: DK/64 chunks of 2*BM rows x 128 B
  static constexpr int kAT = BM * kATs * 4;          // A^T fp32 [i][t], row stride kATs
  static constexpr int kM2 = BM * 128;               // M2 [l][i] K-major
  // BM = 32: M2 shares the dead [K;Q] region with A^T (1024-byte aligned)
  static constexpr bool kM2InR1 = BM < 64;
  static constexpr int kM2Off = (kAT + 1023) / 1024 * 1024;
  static constexpr int kR1a = kM2InR1 ? kM2Off + kM2 : kAT;
  static constexpr int kR1 = kKQ > kR1a ? kKQ : kR1a;  // [K;Q], then A^T (and M2), then the output stage
  static constexpr int kS0 = (DV / 64) * DK * 128;   // S0^T, MN-major: DV/64 chunks of DK rows x 128 B
  static constexpr int kDs = DV + 8;                 // row stride of delta fp32
  static constexpr int kD32 = BM * kDs * 4;          // delta fp32 [t][c]
  static constexpr int kR2 = kS0 > kD32 ? kS0 : kD32;  // S0^T, then delta
  static constexpr int kV = (DV / 64) * BM * 128;    // V [t][c], DV/64 chunks of BM rows x 128 B
  static constexpr int kD = 128 * 128;               // delta^T [c][t] K-major
  static constexpr int kSmem = kR1 + kR2 + kV + (kM2InR1 ? 0 : kM2) + kD;
  static constexpr int kTmemCols = BM == 64 ? 256 : 128;
  static constexpr int kWCol = BM == 64 ? 128 : 64;  // W^T columns: [K rows | Q rows], 2*BM
  static constexpr int kMinBlocks = BM == 64 ? 2 : 3;
};

struct alignas(16) LinShared {
  uint64_t bar_kq, bar_v, bar_mma;
  uint32_t tmem_base;
  int abort_flag;
  // 16-byte aligned: read as float4 broadcasts
  alignas(16) float gam2[kBmax];  // gamma_t * log2(e)
  alignas(16) float Gam[kBmax];   // exp(gamma_t)
  alignas(16) float beta[kBmax];
};

struct LinMaps {
  CUtensorMap k;  // (dk, Hk, B, R)  box (64, 1, 64, 1), 128-byte swizzle
  CUtensorMap q;
  CUtensorMap v;  // (dv, Hv, B, R)  box (64, 1, 64, 1), no swizzle
};

__device__ __forceinline__ bool lin_wait(uint64_t* bar, uint32_t parity, LinShared& sh,
                                         int32_t* status) {
  const bool ok = tc::mbar_wait(bar, parity, &sh.abort_flag);
  const bool all = __syncthreads_and(ok);
  if (!all && threadIdx.x == 0 && !sh.abort_flag) {
    sh.abort_flag = 1;
    flag(status, FLARE_DEV_WAIT_TIMEOUT);
  }
  return all;
}

__device__ __forceinline__ uint32_t f2tf32(float x) {
  uint32_t r;
  asm("cvt.rna.tf32.f32 %0, %1;" : "=r"(r) : "f"(x));
  return r;
}

// Warp-level D += A B on a 16x8x8 tile, tf32 inputs, fp32 accumulate.
// Fragments (g = lane/4, q = lane%4): a0 A[g][q], a1 A[g+8][q], a2 A[g][q+4],
// a3 A[g+8][q+4]; b0 B[q][g], b1 B[q+4][g]; d0 D[g][2q], d1 D[g][2q+1],
// d2 D[g+8][2q], d3 D[g+8][2q+1].
__device__ __forceinline__ void mma_tf32(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2,
                                         uint32_t a3, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k8.row.col.f32.tf32.tf32.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, "
      "{%8, %9}, {%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// 16 bf16 values (columns c0..c0+15) into row `row` of a K-major SW128 tile.
__device__ __forceinline__ void store16_sw128(uint8_t* tile, int row, int c0, const float (&v)[16]) {
  uint8_t* p = tile + row * 128;
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    uint32_t w[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      __nv_bfloat162 b = __floats2bfloat162_rn(v[8 * h + 2 * e], v[8 * h + 2 * e + 1]);
      w[e] = *reinterpret_cast<uint32_t*>(&b);
    }
    const int g = (c0 >> 3) + h;
    *reinterpret_cast<uint4*>(p + ((g ^ (row & 7)) << 4)) = make_uint4(w[0], w[1], w[2], w[3]);
  }
}

}  // namespace

template <int DK, int DV, int BM>
__global__ void __launch_bounds__(kLinThreads, LinCfg<DK, DV, BM>::kMinBlocks)
    gdr_denoise_tc_kernel(const __grid_constant__ LinMaps maps, GdrParams p) {
  using C = LinCfg<DK, DV, BM>;
  constexpr int kATs = C::kATs;
  extern __shared__ uint8_t smem_raw[];
  __shared__ LinShared sh;
  uint8_t* base = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint8_t* KQs = base;
  uint8_t* S0s = KQs + C::kR1;
  uint8_t* Vs = S0s + C::kR2;
  uint8_t* M2s = C::kM2InR1 ? KQs + C::kM2Off : Vs + C::kV;
  uint8_t* Ds = Vs + C::kV + (C::kM2InR1 ? 0 : C::kM2);
  float* AT = reinterpret_cast<float*>(KQs);   // A^T[i][t], once MMA 1/2 have run
  float* D32 = reinterpret_cast<float*>(S0s);  // delta[t][c], once MMA 2 has run

  const int item = blockIdx.x;
  const int r = item / p.Hv, j = item % p.Hv;
  const int h = j / (p.Hv / p.Hk);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int B = p.B;
  const int Bp = (B + 15) & ~15;

  const int slot = p.state_slot[r];
  if (slot < 0 || slot >= p.nslots) {
    if (tid == 0) flag(p.dev_status, FLARE_DEV_BAD_SLOT);
    return;
  }

  // the state is the long-latency input: its loads go out before the set-up
  constexpr int kPer = DK * DV / 4 / kLinThreads;
  float4 s0buf[kPer];
  {
    const float4* S0g =
        reinterpret_cast<const float4*>(p.state_pool + ((size_t)slot * p.Hv + j) * DK * DV);
#pragma unroll
    for (int n = 0; n < kPer; ++n) {
      // volatile: keep every load issued here, ahead of the set-up below
      const float4* a = S0g + tid + n * kLinThreads;
      asm volatile("ld.global.nc.v4.f32 {%0, %1, %2, %3}, [%4];"
                   : "=f"(s0buf[n].x), "=f"(s0buf[n].y), "=f"(s0buf[n].z), "=f"(s0buf[n].w)
                   : "l"(a));
    }
  }

  if (tid == 0) {
    sh.abort_flag = 0;
    tc::mbar_init(&sh.bar_kq, 1);
    tc::mbar_init(&sh.bar_v, 1);
    tc::mbar_init(&sh.bar_mma, 1);
    tc::fence_mbar_init();
  }
  if (warp == 0) tc::tmem_alloc(&sh.tmem_base, C::kTmemCols);
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = sh.tmem_base;
  const uint32_t tmA = tmem;             // G, then O2^T                 (BM columns)
  const uint32_t tmW = tmem + C::kWCol;  // W^T = S0^T [K;Q]^T           (2*BM columns)
  const uint32_t lane_off = (uint32_t)(warp * 32) << 16;

  if (tid == 0) {
    tc::mbar_expect_tx(&sh.bar_kq, 2 * (DK / 64) * BM * 128);
    for (int c = 0; c < DK / 64; ++c) {
      tc::tma_load_4d(KQs + c * (2 * BM * 128), &maps.k, &sh.bar_kq, c * 64, h, 0, r);
      tc::tma_load_4d(KQs + c * (2 * BM * 128) + BM * 128, &maps.q, &sh.bar_kq, c * 64, h, 0, r);
    }
    tc::mbar_expect_tx(&sh.bar_v, (DV / 64) * BM * 128);
    for (int c = 0; c < DV / 64; ++c)
      tc::tma_load_4d(Vs + c * (BM * 128), &maps.v, &sh.bar_v, c * 64, j, 0, r);
  }

  // S0 (fp32, global) -> bf16 S0^T operand, MN-major 128-byte swizzle:
  // element (c, i) in chunk c/64 at row i, 16-byte group ((c%64)/8) ^ (i%8).
  {
    const float4* buf = s0buf;
#pragma unroll
    for (int n = 0; n < kPer; ++n) {
      const int f = tid + n * kLinThreads;
      const int i = f / (DV / 4), c = (f % (DV / 4)) * 4;
      __nv_bfloat162 lo = __floats2bfloat162_rn(buf[n].x, buf[n].y);
      __nv_bfloat162 hi = __floats2bfloat162_rn(buf[n].z, buf[n].w);
      uint2 w = make_uint2(*reinterpret_cast<uint32_t*>(&lo), *reinterpret_cast<uint32_t*>(&hi));
      const int cc = c & 63;
      uint8_t* dst = S0s + (c >> 6) * (DK * 128) + i * 128 + (((cc >> 3) ^ (i & 7)) << 4) +
                     ((cc & 7) << 1);
      *reinterpret_cast<uint2*>(dst) = w;
    }
  }
  // gates: gamma = inclusive prefix sum of the log-gates over the block
  if (warp == 0) {
    const size_t gb = (size_t)r * B * p.Hv + j;
    float g0 = lane < B ? p.log_decay[gb + (size_t)lane * p.Hv] : 0.f;
    float g1 = lane + 32 < B ? p.log_decay[gb + (size_t)(lane + 32) * p.Hv] : 0.f;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const float a = __shfl_up_sync(0xffffffffu, g0, o);
      const float b = __shfl_up_sync(0xffffffffu, g1, o);
      if (lane >= o) {
        g0 += a;
        g1 += b;
      }
    }
    g1 += __shfl_sync(0xffffffffu, g0, 31);
    sh.gam2[lane] = g0 * 1.4426950408889634f;
    sh.gam2[lane + 32] = g1 * 1.4426950408889634f;
    sh.Gam[lane] = expf(g0);
    sh.Gam[lane + 32] = expf(g1);
    sh.beta[lane] = lane < B ? p.beta[gb + (size_t)lane * p.Hv] : 0.f;
    sh.beta[lane + 32] = lane + 32 < B ? p.beta[gb + (size_t)(lane + 32) * p.Hv] : 0.f;
  }
  tc::fence_async_smem();
  if (!lin_wait(&sh.bar_kq, 0, sh, p.dev_status)) goto done;

  // ---- MMA 1 (Gram) and MMA 2 (state products)
  if (tid == 0) {
    tc::fence_after_sync();
    const uint32_t idG = tc::idesc_bf16(128, Bp, false, false);
    const uint32_t idW = tc::idesc_bf16(128, 2 * BM, true, false);
#pragma unroll
    for (int kk = 0; kk < DK / 16; ++kk) {
      const int c = kk >> 2, off = (kk & 3) * 32;
      // BM = 32: the A operand's rows past the 2*BM of this chunk read the
      // next bytes of shared memory; those rows of G are never read
      const uint64_t kq = tc::sdesc_sw128(tc::smem_u32(KQs + c * (2 * BM * 128) + off), 16, 1024);
      tc::mma_bf16_ss(tmA, kq, kq, idG, kk > 0);
      const uint64_t s0 = tc::sdesc_sw128(tc::smem_u32(S0s + kk * 2048), DK * 128, 1024);
      tc::mma_bf16_ss(tmW, s0, kq, idW, kk > 0);
    }
    tc::mma_commit(&sh.bar_mma);
  }
  if (!lin_wait(&sh.bar_mma, 0, sh, p.dev_status)) goto done;
  tc::fence_after_sync();

  // ---- A^T (from rows 0..BM-1 of G, fp32) and M2 (rows BM..2BM-1, bf16
  // operand); all of a row's G values are loaded from tensor memory before any
  // is used (BM = 32: warps 2 and 3 hold no rows of G)
  if (tid < 2 * BM) {
    const int row = tid & (BM - 1);
    const float gB = sh.gam2[B - 1];
    const float bt = sh.beta[row], gt = sh.gam2[row];
    uint32_t gr[BM];
#pragma unroll
    for (int c0 = 0; c0 < BM; c0 += 16)
      if (c0 < Bp) tc::tmem_ld16(tmA + lane_off + c0, *reinterpret_cast<uint32_t(*)[16]>(&gr[c0]));
    tc::tmem_ld_wait();
#pragma unroll
    for (int c0 = 0; c0 < BM; c0 += 16) {
      if (c0 >= Bp) break;
      // the chunk's log-gates first: the stores below may alias them for the
      // compiler, which would otherwise reload one after every store
      float g2[16];
#pragma unroll
      for (int e = 0; e < 16; ++e) g2[e] = sh.gam2[c0 + e];
      float v[16];
      if (tid < BM) {
#pragma unroll
        for (int e = 0; e < 16; ++e) {
          const int i = c0 + e;
          // A[t][i] = beta_t exp(gamma_t - gamma_i) (k_t . k_i), i < t < B (the
          // exponential taken unconditionally, the mask as a select)
          const float a = bt * tc::ex2(gt - g2[e]) * __uint_as_float(gr[i]);
          v[e] = (i < row && row < B) ? a : 0.f;
        }
#pragma unroll
        for (int e = 0; e < 16; ++e) AT[(c0 + e) * kATs + row] = v[e];
      } else {
#pragma unroll
        for (int e = 0; e < 16; ++e) {
          const int i = c0 + e;
          const float m = tc::ex2(gB - g2[e]) * __uint_as_float(gr[i]);
          v[e] = (i < B && row < B) ? m : 0.f;
        }
        store16_sw128(M2s, row, c0, v);
      }
    }
  }
  if (!lin_wait(&sh.bar_v, 0, sh, p.dev_status)) goto done;  // also publishes A^T

  // ---- delta = (I + A)^{-1} X by forward substitution, X = diag(beta)(V - diag(Gam) K S0).
  // The system acts on each column c on its own; warp w owns columns
  // 32w..32w+31 and walks the rows 16 at a time:
  //   x_b  = X_b - A[b, <b] delta_<b     warp-level tf32 MMA (rows x columns tile)
  //   delta_b = (I + A[b,b])^{-1} x_b    fp32 forward substitution, thread c on column c
  // The two layouts meet in the fp32 delta buffer, inside the warp.
  {
    constexpr int kS = C::kDs;
    const int c = tid;
    const bool col_ok = c < DV;  // warp-uniform
    const int g = lane >> 2, q = lane & 3;
    const uint8_t* vcol = Vs + ((c & (DV - 1)) >> 6) * (BM * 128) + (c & 63) * 2;
#pragma unroll 1
    for (int b0 = 0; b0 < Bp; b0 += 16) {
      uint32_t w[16];
      tc::tmem_ld16(tmW + lane_off + b0, w);  // (K S0)^T[c][t]
      tc::tmem_ld_wait();
      // the block's gates as 16-byte broadcast loads (the solve is bound by
      // shared-memory instruction issue)
      float bb[16], GG[16];
#pragma unroll
      for (int e4 = 0; e4 < 4; ++e4) {
        const float4 b4 = *reinterpret_cast<const float4*>(&sh.beta[b0 + 4 * e4]);
        const float4 g4 = *reinterpret_cast<const float4*>(&sh.Gam[b0 + 4 * e4]);
        bb[4 * e4] = b4.x, bb[4 * e4 + 1] = b4.y, bb[4 * e4 + 2] = b4.z, bb[4 * e4 + 3] = b4.w;
        GG[4 * e4] = g4.x, GG[4 * e4 + 1] = g4.y, GG[4 * e4 + 2] = g4.z, GG[4 * e4 + 3] = g4.w;
      }
      float x[16];
#pragma unroll
      for (int e = 0; e < 16; ++e) {
        const int t = b0 + e;
        const float vt =
            __bfloat162float(*reinterpret_cast<const __nv_bfloat16*>(vcol + t * 128));
        x[e] = (t < B && col_ok) ? bb[e] * (vt - GG[e] * __uint_as_float(w[e])) : 0.f;
      }
      if (col_ok) {
        if (b0 > 0) {
          // x_b -= A[b0.., 0..b0) delta[0..b0, warp's columns]
#pragma unroll
          for (int e = 0; e < 16; ++e) D32[(b0 + e) * kS + c] = x[e];
          __syncwarp();
          const int cw = warp * 32;
          float acc[4][4];
#pragma unroll
          for (int nt = 0; nt < 4; ++nt) {
            const float2 lo = *reinterpret_cast<const float2*>(D32 + (b0 + g) * kS + cw + nt * 8 + 2 * q);
            const float2 hi = *reinterpret_cast<const float2*>(D32 + (b0 + g + 8) * kS + cw + nt * 8 + 2 * q);
            acc[nt][0] = lo.x;
            acc[nt][1] = lo.y;
            acc[nt][2] = hi.x;
            acc[nt][3] = hi.y;
          }
#pragma unroll 2
          for (int i0 = 0; i0 < b0; i0 += 8) {
            // -A[t][i] = -A^T[i][t]
            const float* ar = AT + (i0 + q) * kATs + b0 + g;
            const uint32_t a0 = f2tf32(-ar[0]), a1 = f2tf32(-ar[8]);
            const uint32_t a2 = f2tf32(-ar[4 * kATs]), a3 = f2tf32(-ar[4 * kATs + 8]);
#pragma unroll
            for (int nt = 0; nt < 4; ++nt) {
              const float* br = D32 + (i0 + q) * kS + cw + nt * 8 + g;
              mma_tf32(acc[nt], a0, a1, a2, a3, f2tf32(br[0]), f2tf32(br[4 * kS]));
            }
          }
          __syncwarp();
#pragma unroll
          for (int nt = 0; nt < 4; ++nt) {
            *reinterpret_cast<float2*>(D32 + (b0 + g) * kS + cw + nt * 8 + 2 * q) =
                make_float2(acc[nt][0], acc[nt][1]);
            *reinterpret_cast<float2*>(D32 + (b0 + g + 8) * kS + cw + nt * 8 + 2 * q) =
                make_float2(acc[nt][2], acc[nt][3]);
          }
          __syncwarp();
#pragma unroll
          for (int e = 0; e < 16; ++e) x[e] = D32[(b0 + e) * kS + c];
        }
        // diagonal block: x_t -= A[t][i] delta_i for b0 <= i < t; column i of
        // the block is loaded one step ahead, so the chain through x waits on
        // multiply-adds only
        {
          const float* ad = AT + b0 * kATs + b0;
          float4 an[4];
#pragma unroll
          for (int qq = 0; qq < 4; ++qq) an[qq] = reinterpret_cast<const float4*>(ad)[qq];
#pragma unroll
          for (int e = 0; e < 15; ++e) {
            float4 a[4];
#pragma unroll
            for (int qq = 0; qq < 4; ++qq) a[qq] = an[qq];
            if (e + 1 < 15) {
#pragma unroll
              for (int qq = (e + 1) / 4; qq < 4; ++qq)
                an[qq] = reinterpret_cast<const float4*>(ad + (e + 1) * kATs)[qq];
            }
#pragma unroll
            for (int qq = e / 4; qq < 4; ++qq) {
              if (4 * qq > e) x[4 * qq] = fmaf(-a[qq].x, x[e], x[4 * qq]);
              if (4 * qq + 1 > e) x[4 * qq + 1] = fmaf(-a[qq].y, x[e], x[4 * qq + 1]);
              if (4 * qq + 2 > e) x[4 * qq + 2] = fmaf(-a[qq].z, x[e], x[4 * qq + 2]);
              if (4 * qq + 3 > e) x[4 * qq + 3] = fmaf(-a[qq].w, x[e], x[4 * qq + 3]);
            }
          }
        }
#pragma unroll
        for (int e = 0; e < 16; ++e) D32[(b0 + e) * kS + c] = x[e];
        __syncwarp();  // the next block's MMA reads this block's delta across the warp
      }
      store16_sw128(Ds, c, b0, x);  // delta^T, bf16 operand of MMA 4
    }
  }
  tc::fence_async_smem();
  tc::fence_before_sync();
  __syncthreads();

  // ---- MMA 4: O2^T = delta^T M2^T
  if (tid == 0) {
    tc::fence_after_sync();
    const uint32_t id = tc::idesc_bf16(128, Bp, false, false);
    for (int kk = 0; kk < Bp / 16; ++kk) {
      const uint64_t a = tc::sdesc_sw128(tc::smem_u32(Ds + kk * 32), 16, 1024);
      const uint64_t b = tc::sdesc_sw128(tc::smem_u32(M2s + kk * 32), 16, 1024);
      tc::mma_bf16_ss(tmA, a, b, id, kk > 0);
    }
    tc::mma_commit(&sh.bar_mma);
  }
  if (!lin_wait(&sh.bar_mma, 1, sh, p.dev_status)) goto done;
  tc::fence_after_sync();
  // out[l][c] = s (Gam_B W^T[c][BM+l] + O2^T[c][l]), staged as bf16 [l][c] in the
  // dead [K;Q] region, then written in 16-byte pieces
  {
    const int c = tid;
    const float GB = sh.Gam[B - 1];
    __nv_bfloat16* stage = reinterpret_cast<__nv_bfloat16*>(KQs);
    uint32_t o2[BM], wq[BM];
#pragma unroll
    for (int c0 = 0; c0 < BM; c0 += 16) {
      if (c0 < Bp) {
        tc::tmem_ld16(tmA + lane_off + c0, *reinterpret_cast<uint32_t(*)[16]>(&o2[c0]));
        tc::tmem_ld16(tmW + lane_off + BM + c0, *reinterpret_cast<uint32_t(*)[16]>(&wq[c0]));
      }
    }
    tc::tmem_ld_wait();
    if (c < DV) {
#pragma unroll
      for (int l = 0; l < BM; ++l)
        if (l < B)
          stage[l * DV + c] = __float2bfloat16_rn(
              p.scale * (GB * __uint_as_float(wq[l]) + __uint_as_float(o2[l])));
    }
    __syncthreads();
    constexpr int kPieces = DV / 8;  // 16-byte pieces per output row
    constexpr int kIt = (BM * kPieces + kLinThreads - 1) / kLinThreads;
    __nv_bfloat16* out = static_cast<__nv_bfloat16*>(p.out_blockend);
    uint4 piece[kIt];  // every piece read before the first store
#pragma unroll
    for (int it = 0; it < kIt; ++it) {
      const int e = tid + it * kLinThreads;
      if (e < B * kPieces)
        piece[it] = *reinterpret_cast<const uint4*>(stage + (e / kPieces) * DV + (e % kPieces) * 8);
    }
#pragma unroll
    for (int it = 0; it < kIt; ++it) {
      const int e = tid + it * kLinThreads;
      if (e < B * kPieces) {
        const int l = e / kPieces, pc = e % kPieces;
        *reinterpret_cast<uint4*>(out + (((size_t)r * B + l) * p.Hv + j) * DV + pc * 8) =
            piece[it];
      }
    }
  }

done:
  tc::fence_before_sync();
  __syncthreads();
  if (warp == 0) {
    tc::fence_after_sync();
    tc::tmem_dealloc(tmem, C::kTmemCols);
  }
}

// ------------------------------------------------------------------ host side

namespace {

PFN_cuTensorMapEncodeTiled_v12000 lin_encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void* f = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(f);
  }
  return fn;
}

bool lin_map(CUtensorMap* m, const void* ptr, int d, int H, int B, int R, int box_rows,
             bool swizzle) {
  auto fn = lin_encode_fn();
  if (!fn) return false;
  cuuint64_t gd[4] = {(cuuint64_t)d, (cuuint64_t)H, (cuuint64_t)B, (cuuint64_t)R};
  cuuint64_t gs[3] = {(cuuint64_t)d * 2, (cuuint64_t)H * d * 2, (cuuint64_t)B * H * d * 2};
  cuuint32_t bx[4] = {64, 1, (cuuint32_t)box_rows, 1};
  cuuint32_t es[4] = {1, 1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(ptr), gd, gs, bx, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE,
            swizzle ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_NONE,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) ==
         CUDA_SUCCESS;
}

template <int DK, int DV, int BM>
cudaError_t launch_lin_tc_bm(const GdrParams& p, cudaStream_t stream) {
  using C = LinCfg<DK, DV, BM>;
  LinMaps maps;
  if (!lin_map(&maps.k, p.k, DK, p.Hk, p.B, p.R, BM, true) ||
      !lin_map(&maps.q, p.q, DK, p.Hk, p.B, p.R, BM, true) ||
      !lin_map(&maps.v, p.v, DV, p.Hv, p.B, p.R, BM, false))
    return cudaErrorInvalidValue;
  const int smem = C::kSmem + 1024;
  cudaError_t e = cudaFuncSetAttribute(gdr_denoise_tc_kernel<DK, DV, BM>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  gdr_denoise_tc_kernel<DK, DV, BM><<<p.R * p.Hv, kLinThreads, smem, stream>>>(maps, p);
  note_launches(1);
  return cudaGetLastError();
}

// blocks of up to 32 rows take the smaller layout (three CTAs per SM)
template <int DK, int DV>
cudaError_t launch_lin_tc(const GdrParams& p, cudaStream_t stream) {
  return p.B <= 32 ? launch_lin_tc_bm<DK, DV, 32>(p, stream)
                   : launch_lin_tc_bm<DK, DV, 64>(p, stream);
}

}  // namespace

bool gdr_denoise_tc_supported(int B, int dk, int dv) {
  return B >= 1 && B <= kBmax && (dk == 64 || dk == 128) && (dv == 64 || dv == 128);
}

cudaError_t launch_gdr_denoise_tc(const GdrParams& p, cudaStream_t stream) {
  if (p.dk == 128 && p.dv == 128) return launch_lin_tc<128, 128>(p, stream);
  if (p.dk == 128 && p.dv == 64) return launch_lin_tc<128, 64>(p, stream);
  if (p.dk == 64 && p.dv == 128) return launch_lin_tc<64, 128>(p, stream);
  if (p.dk == 64 && p.dv == 64) return launch_lin_tc<64, 64>(p, stream);
  return cudaErrorInvalidValue;
}

}  // namespace flare
