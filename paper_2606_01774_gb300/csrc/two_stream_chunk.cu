// Two-stream training forward of a gated-delta-rule layer on tcgen05 tensor
// cores, chunkwise: bf16 activations, d_k = d_v = 128, noisy blocks of B = 1,
// 2, 4, 8 or 16 tokens in chunks of 64 (appendix "Two-stream recurrence and
// block-level chain rule", Eq. noisy-block-fwd and Eq. f-blk; the Route II
// fused forward).
//
// Noisy block m of a chunk starts from the clean state after the chunk's
// clean tokens 0 .. mB-1.  Those states are never formed: the clean tokens of
// the whole chunk are one chunkwise delta-rule system (Eq. chunk-state), with
// gamma_t the clean log-gates summed from the chunk start,
//   A[t][i] = beta_t exp(gamma_t - gamma_i) (k_t . k_i),  i < t < 64
//   X_t     = beta_t (v_t - Gam_t S0^T k_t),    (I + A) delta = X
//   S_(m)   = Gam_{mB-1} S0 + sum_{i < mB} exp(gamma_{mB-1} - gamma_i) k_i delta_i^T
// so that for every noisy key and query y of block m
//   S_(m)^T y = Gam_{mB-1} S0^T y + sum_i delta_i P[i][y],
//   P[i][y]   = [i < mB] exp(gamma_{mB-1} - gamma_i) (k_i . y).
// The noisy block then solves its own B x B system on block-local gates and
// reads out every row at the block end (Eq. noisy-block-fwd):
//   X~_t = beta~_t (v~_t - Gam~_t S_(m)^T k~_t),   (I + A~) delta~ = X~
//   o~_l = s (Gam~_end S_(m)^T q~_l + sum_i exp(gamma~_end - gamma~_i) (q~_l . k~_i) delta~_i)
//
// Value column c on tensor-memory lane c.  Per chunk:
//   MMA 1  W^T = S0^T [K; K~; Q~]^T      M=128 (c), N=192, K=128   (A: S0^T bf16, tensor memory)
//          G   = [K; K~] [K; K~; Q~]^T   M=128 (rows), N=192, K=128: every dot product the
//                                         chunk needs (K K^T, K K~^T, K Q~^T, K~ K~^T, K~ Q~^T)
//   T      = (I + A)^{-1}                 fp32, 16 x 16 blocks: the diagonal ones by forward
//                                         substitution, then T_ab = -T_aa sum_c A_ac T_cb by block
//                                         columns, right-looking, within lanes (all warps)
//   MMA d  delta^T = X^T T^T             M=128 (c), N=64, K=64     (X and T as bf16 high + low
//                                         parts, three products: fp32-grade delta)
//   MMA 2  C^T = delta^T P               M=128 (c), N=128, K=64    (A: delta^T bf16, tensor memory)
//   noisy  S_(m)^T y = Gam_{mB-1} W^T + C^T, the B x B solves and the readouts (both groups)
// bf16 operands and fp32 accumulation throughout (the state rounded to bf16
// for its products, as in the denoise kernels).
//
// Persistent CTAs, one per SM (208 KiB of shared memory, 448 tensor-memory
// columns), 256 threads: warps 0-3 and 4-7 are two groups on the same 128
// lanes, which build the tables together and take half of the noisy tokens
// each.  The next chunk's state streams into the state buffer as soon as it
// has been turned into S0^T, its keys and queries once the first MMAs are
// done, its values once this chunk's are read; its gates are loaded into
// registers one chunk ahead.  Every wait is bounded: on a timeout
// the CTA sets FLARE_DEV_WAIT_TIMEOUT, waits (bounded) for its copies and
// MMAs in flight, frees its tensor memory and exits.
#include <cudaTypedefs.h>

#include "common.cuh"
#include "kernels.h"
#include "tc.cuh"
#include "chunk64.cuh"

namespace flare {

namespace {

constexpr int kCkThreads = 256;
constexpr int kCkD = 128;  // d_k = d_v
using namespace chunk64;  // kCkC = 64, the chunk length, and the chunk-system helpers

struct CkCfg {
  static constexpr int kS0 = kCkD * kCkD * 4;     // S0 fp32 [i][c]
  static constexpr int kKX = 2 * 192 * 128;       // [K; K~; Q~]: 2 chunks of 192 rows x 128 B (SW128)
  static constexpr int kV = 2 * kCkC * 128;       // values: 2 chunks of 64 rows x 128 B
  static constexpr int kT = kCkC * kCkC * 4;      // a 64 x 64 fp32 table
  static constexpr int kP = 2 * kCkC * 128;       // P [i][y] bf16 MN-major: 2 chunks of 64 rows
  static constexpr int oS0 = 0;
  static constexpr int oKX = oS0 + kS0;
  static constexpr int oVc = oKX + kKX;
  static constexpr int oVn = oVc + kV;
  static constexpr int oAT = oVn + kV;   // A^T[i][t] (clean)
  static constexpr int oAn = oAT + kT;   // A~[t][i] (noisy, zero outside the block)
  static constexpr int oAq = oAn + kT;   // Aqk^T[i][l] (noisy readout, zero outside the block)
  static constexpr int oP = oAq + kT;
  static constexpr int oT = oP + kP;     // T[t][j] fp32, the lower blocks
  static constexpr int kSmem = oT + kT;
  // once the clean values are read, their buffer holds T as bf16 high and low
  // parts (K-major SW128, rows of 64 elements, 8 KiB each): MMA d's operand
};

struct alignas(16) CkShared {
  uint64_t bar_s0, bar_kx, bar_v, bar_g, bar_mma;
  uint32_t tmem_base;
  int abort_flag;
  alignas(16) float gc2[kCkC];  // clean gamma_t log2(e), from the chunk start
  alignas(16) float Gc[kCkC];   // clean exp(gamma_t)
  alignas(16) float bc[kCkC];   // clean beta
  alignas(16) float gn2[kCkC];  // noisy gamma~_t log2(e), from the block start
  alignas(16) float Gn[kCkC];   // noisy exp(gamma~_t)
  alignas(16) float bn[kCkC];   // noisy beta~
};

struct CkMaps {
  CUtensorMap k, kn, qn;  // (128, Hk, L, N) box (64, 1, 64, 1), 128-byte swizzle
  CUtensorMap v, vn;      // (128, Hv, L, N) box (64, 1, 64, 1), no swizzle
};

}  // namespace

template <int B>
__global__ void __launch_bounds__(kCkThreads, 1)
    two_stream_chunk_kernel(const __grid_constant__ CkMaps maps, TwoStreamParams p) {
  using C = CkCfg;
  constexpr int kIssuer = 32;  // one thread of warp 1 issues every copy and MMA
  extern __shared__ uint8_t smem_raw[];
  __shared__ CkShared sh;
  uint8_t* base = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  float* S0s = reinterpret_cast<float*>(base + C::oS0);
  uint8_t* KX = base + C::oKX;
  uint8_t* Vc = base + C::oVc;
  uint8_t* Vn = base + C::oVn;
  float* AT = reinterpret_cast<float*>(base + C::oAT);
  float* An = reinterpret_cast<float*>(base + C::oAn);
  float* AqT = reinterpret_cast<float*>(base + C::oAq);
  uint8_t* Ps = base + C::oP;
  float* Tf = reinterpret_cast<float*>(base + C::oT);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int col = tid & 127, grp = tid >> 7;  // value column (= lane of tensor memory), group
  const int n_chunks = p.L / kCkC;
  const int total = p.N * p.Hv * n_chunks;

  if (tid == kIssuer) {
    sh.abort_flag = 0;
    tc::mbar_init(&sh.bar_s0, 1);
    tc::mbar_init(&sh.bar_kx, 1);
    tc::mbar_init(&sh.bar_v, 1);
    tc::mbar_init(&sh.bar_g, 1);
    tc::mbar_init(&sh.bar_mma, 1);
    tc::fence_mbar_init();
  }
  if (warp == 0) tc::tmem_alloc(&sh.tmem_base, 512);
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = sh.tmem_base;
  const uint32_t tmS = tmem;        // S0^T bf16 (64 columns); X^T high | low; delta^T (32)
  const uint32_t tmW = tmem + 64;   // W^T: [K | K~ | Q~] parts, 3 x 64 columns
  const uint32_t tmG = tmem + 256;  // G (rows on lanes), 192 columns; then C^T (128)
  const uint32_t tmD = tmem + 448;  // delta^T fp32, 64 columns
  const uint32_t lane_off = (uint32_t)((warp & 3) * 32) << 16;

  struct Loc {
    int n, j, c, h;
    size_t tok0;
  };
  auto loc = [&](int item) {
    Loc l;
    l.c = item % n_chunks;
    l.j = (item / n_chunks) % p.Hv;
    l.n = item / (n_chunks * p.Hv);
    l.h = l.j / (p.Hv / p.Hk);
    l.tok0 = (size_t)l.n * p.L + (size_t)l.c * kCkC;
    return l;
  };
  auto issue_s0 = [&](int item) {
    const Loc l = loc(item);
    const float* src = p.chunk_states + (((size_t)l.n * p.Hv + l.j) * n_chunks + l.c) * kCkD * kCkD;
    tc::mbar_expect_tx(&sh.bar_s0, C::kS0);
    tc::bulk_load(S0s, src, C::kS0, &sh.bar_s0);
  };
  auto issue_kx = [&](int item) {
    const Loc l = loc(item);
    const int t0 = l.c * kCkC;
    tc::mbar_expect_tx(&sh.bar_kx, C::kKX);
#pragma unroll
    for (int d = 0; d < 2; ++d) {
      uint8_t* dst = KX + d * (192 * 128);
      tc::tma_load_4d(dst, &maps.k, &sh.bar_kx, d * 64, l.h, t0, l.n);
      tc::tma_load_4d(dst + 64 * 128, &maps.kn, &sh.bar_kx, d * 64, l.h, t0, l.n);
      tc::tma_load_4d(dst + 128 * 128, &maps.qn, &sh.bar_kx, d * 64, l.h, t0, l.n);
    }
  };
  auto issue_v = [&](int item) {
    const Loc l = loc(item);
    const int t0 = l.c * kCkC;
    tc::mbar_expect_tx(&sh.bar_v, 2 * C::kV);
#pragma unroll
    for (int d = 0; d < 2; ++d) {
      tc::tma_load_4d(Vc + d * (kCkC * 128), &maps.v, &sh.bar_v, d * 64, l.j, t0, l.n);
      tc::tma_load_4d(Vn + d * (kCkC * 128), &maps.vn, &sh.bar_v, d * 64, l.j, t0, l.n);
    }
  };
  // warps 0 (clean) and 4 (noisy) hold the gates of the chunk they process
  // next, loaded one chunk ahead: tokens lane and lane + 32
  float ga = 0.f, gb = 0.f, ba = 0.f, bb = 0.f;
  auto load_gates = [&](int item) {
    const Loc l = loc(item);
    const float* g = grp == 0 ? p.g : p.gn;
    const float* bt = grp == 0 ? p.beta : p.betan;
    ga = g[(l.tok0 + lane) * p.Hv + l.j];
    gb = g[(l.tok0 + lane + 32) * p.Hv + l.j];
    ba = bt[(l.tok0 + lane) * p.Hv + l.j];
    bb = bt[(l.tok0 + lane + 32) * p.Hv + l.j];
  };

  int it = blockIdx.x;
  bool s0_out = false, kx_out = false, v_out = false, mma_out = false;
  uint32_t s0_par = 0, kx_par = 0, v_par = 0;
  if (it < total) {
    if (tid == kIssuer) {
      tc::prefetch_tmap(&maps.k);
      tc::prefetch_tmap(&maps.kn);
      tc::prefetch_tmap(&maps.qn);
      tc::prefetch_tmap(&maps.v);
      tc::prefetch_tmap(&maps.vn);
      issue_s0(it);
      issue_kx(it);
      issue_v(it);
      s0_out = kx_out = v_out = true;
    }
    if ((warp & 3) == 0) load_gates(it);
  }
  bool bad = false;
  uint32_t ph = 0, ph_mma = 0;
  const uint32_t id192 = tc::idesc_bf16(128, 192, false, false);
  const uint32_t id128 = tc::idesc_bf16(128, 128, false, true);
  const uint32_t id64 = tc::idesc_bf16(128, 64, false, false);

#pragma unroll 1
  for (; it < total; it += (int)gridDim.x) {
    const Loc L = loc(it);
    const int it_next = it + (int)gridDim.x < total ? it + (int)gridDim.x : -1;
    // gates: the clean ones summed from the chunk start (warp 0), the noisy
    // ones from each block start (warp 4)
    if ((warp & 3) == 0) {
      float x0 = ga, x1 = gb;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const float u = __shfl_up_sync(0xffffffffu, x0, o);
        const float w = __shfl_up_sync(0xffffffffu, x1, o);
        const bool in0 = grp == 0 ? lane >= o : (lane & (B - 1)) >= o;
        if (in0) {
          x0 += u;
          x1 += w;
        }
      }
      if (grp == 0) {
        x1 += __shfl_sync(0xffffffffu, x0, 31);
        sh.gc2[lane] = x0 * 1.4426950408889634f;
        sh.gc2[lane + 32] = x1 * 1.4426950408889634f;
        sh.Gc[lane] = expf(x0);
        sh.Gc[lane + 32] = expf(x1);
        sh.bc[lane] = ba;
        sh.bc[lane + 32] = bb;
      } else {
        sh.gn2[lane] = x0 * 1.4426950408889634f;
        sh.gn2[lane + 32] = x1 * 1.4426950408889634f;
        sh.Gn[lane] = expf(x0);
        sh.Gn[lane + 32] = expf(x1);
        sh.bn[lane] = ba;
        sh.bn[lane + 32] = bb;
      }
      if (it_next >= 0) load_gates(it_next);
    }

    bad |= !tc::mbar_wait(&sh.bar_s0, ph, &sh.abort_flag);
    if (tid == kIssuer) s0_out = false;
    // S0^T into tensor memory as bf16 pairs, each group half of the rows
#pragma unroll 1
    for (int i0 = grp * 64; i0 < grp * 64 + 64; i0 += 32) {
      uint32_t w[16];
#pragma unroll
      for (int e = 0; e < 16; ++e)
        w[e] = ck_pack(S0s[(i0 + 2 * e) * kCkD + col], S0s[(i0 + 2 * e + 1) * kCkD + col]);
      tc::tmem_st16(tmS + lane_off + i0 / 2, w);
    }
    tc::tmem_st_wait();
    tc::fence_before_sync();
    if (__syncthreads_or(bad)) break;  // S0^T complete, the state buffer read
    if (tid == kIssuer) {
      bad |= !tc::mbar_wait(&sh.bar_kx, ph, &sh.abort_flag);
      kx_out = false;
      tc::fence_after_sync();
      // the Gram first, committed on its own: the tables are built from it
      // while the state products run
#pragma unroll
      for (int kk = 0; kk < kCkD / 16; ++kk) {
        const uint64_t kd = tc::sdesc_sw128(
            tc::smem_u32(KX + (kk >> 2) * (192 * 128) + (kk & 3) * 32), 16, 1024);
        tc::mma_bf16_ss(tmG, kd, kd, id192, kk > 0);  // G = [K; K~] [K; K~; Q~]^T
      }
      tc::mma_commit(&sh.bar_g);
#pragma unroll
      for (int kk = 0; kk < kCkD / 16; ++kk) {
        const uint64_t kd = tc::sdesc_sw128(
            tc::smem_u32(KX + (kk >> 2) * (192 * 128) + (kk & 3) * 32), 16, 1024);
        tc::mma_bf16_ts(tmW, tmS + kk * 8, kd, id192, kk > 0);  // W^T = S0^T [K; K~; Q~]^T
      }
      tc::mma_commit(&sh.bar_mma);
      mma_out = true;
      if (it_next >= 0) {  // the state buffer is free
        issue_s0(it_next);
        s0_out = true;
        s0_par = ph ^ 1u;
      }
    }
    bad |= !tc::mbar_wait(&sh.bar_g, ph, &sh.abort_flag);
    tc::fence_after_sync();

    // ---- tables from G, 32 columns at a time.  Lanes 0..63 hold the rows of
    // K, 64..127 those of K~; every exponential is taken unconditionally and
    // the masks applied as selects (a branch per element would serialise the
    // chains).
    {
      const int row = col & 63;
      const bool krow = col < 64;
      const int m0 = row & ~(B - 1);  // the block start of this row's token
      if (grp == 0) {
        if (krow) {
          // warps 0-1: A^T row i of the clean system
          const float gi = sh.gc2[row];
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            uint32_t gr[32];
            float v[32];
            ck_ld32(tmG + lane_off + 32 * h, gr);
#pragma unroll
            for (int k = 0; k < 32; ++k) {
              const int t = 32 * h + k;
              const float a = sh.bc[t] * tc::ex2(sh.gc2[t] - gi) * __uint_as_float(gr[k]);
              v[k] = t > row ? a : 0.f;
            }
            ck_store32(AT, row, 32 * h, v);
          }
          tc::named_bar_arrive(5, 128);  // A^T to warps 4-5
        } else {
          // warps 2-3: A~ row t
          const float bt = sh.bn[row], gt = sh.gn2[row];
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            uint32_t gr[32];
            float v[32];
            ck_ld32(tmG + lane_off + 64 + 32 * h, gr);
#pragma unroll
            for (int k = 0; k < 32; ++k) {
              const int i = 32 * h + k;
              const float a = bt * tc::ex2(gt - sh.gn2[i]) * __uint_as_float(gr[k]);
              v[k] = (i >= m0 && i < row) ? a : 0.f;
            }
            ck_store32(An, row, 32 * h, v);
          }
        }
      } else {
        if (krow) {
          // warps 4-5: P row i, 128 columns (the noisy keys, then queries),
          // P[i][y] = [i < mB] exp(gamma_{mB-1} - gamma_i) (k_i . y)
          // the factor depends on the row and the block only: one per block
          const float gi = sh.gc2[row];
#pragma unroll 1
          for (int h = 0; h < 4; ++h) {  // columns 32 h .. of the 128: tokens 32 (h % 2) ..
            const int tq = 32 * (h & 1);
            float fm[32 / B];
#pragma unroll
            for (int m = 0; m < 32 / B; ++m) {
              const int mb = tq + m * B;
              const float a = tc::ex2(sh.gc2[mb > 0 ? mb - 1 : 0] - gi);
              fm[m] = row < mb ? a : 0.f;
            }
            uint32_t gr[32];
            ck_ld32(tmG + lane_off + 64 + 32 * h, gr);
#pragma unroll
            for (int u4 = 0; u4 < 4; ++u4) {  // 16-byte units of 8 columns
              const int u = 4 * (h & 1) + u4;   // unit within the 64-column chunk
              uint32_t w[4];
#pragma unroll
              for (int e = 0; e < 4; ++e) {
                float pv[2];
#pragma unroll
                for (int f = 0; f < 2; ++f) {
                  const int k = 8 * u4 + 2 * e + f;  // column within the 32: token tq + k
                  pv[f] = fm[k / B] * __uint_as_float(gr[k]);
                }
                w[e] = ck_pack(pv[0], pv[1]);
              }
              // MN-major SW128: chunk h / 2, row i, 16-byte unit u ^ (i % 8)
              *reinterpret_cast<uint4*>(Ps + (h >> 1) * (kCkC * 128) + row * 128 +
                                        ((u ^ (row & 7)) << 4)) = make_uint4(w[0], w[1], w[2], w[3]);
            }
          }
          tc::fence_async_smem();  // P is the second MMA's operand
          // the diagonal blocks of T once warps 0-1 have written A^T: blocks
          // 2 (warp - 4) and 2 (warp - 4) + 1, a column of one per lane
          tc::named_bar_sync(5, 128);
          ck_diag_inverse(AT, Tf, 2 * (warp - 4) + (lane >> 4), lane & 15);
        } else {
          // warps 6-7: Aqk^T row i (noisy key i): exp(gamma~_end - gamma~_i) (q~_l . k~_i)
          // for the queries l of its block
          const float f = tc::ex2(sh.gn2[m0 + B - 1] - sh.gn2[row]);
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            uint32_t gr[32];
            float v[32];
            ck_ld32(tmG + lane_off + 128 + 32 * h, gr);
#pragma unroll
            for (int k = 0; k < 32; ++k) {
              const int l = 32 * h + k;
              v[k] = (l >= m0 && l < m0 + B) ? f * __uint_as_float(gr[k]) : 0.f;
            }
            ck_store32(AqT, row, 32 * h, v);
          }
        }
      }
    }
    // ---- X = diag(beta) (V - diag(Gam) K S0), tokens 32 grp .. 32 grp + 31,
    // into tensor memory as bf16 high and low parts over S0^T (which the first
    // MMAs have read)
    bad |= !tc::mbar_wait(&sh.bar_mma, ph_mma, &sh.abort_flag);
    ph_mma ^= 1u;
    tc::fence_after_sync();
    if (tid == kIssuer) {
      mma_out = false;
      if (it_next >= 0) {  // the first MMAs, the readers of [K; K~; Q~], are done
        issue_kx(it_next);
        kx_out = true;
        kx_par = ph ^ 1u;
      }
    }
    bad |= !tc::mbar_wait(&sh.bar_v, ph, &sh.abort_flag);
    if (tid == kIssuer) v_out = false;
    {
      const int t0 = 32 * grp;
      uint32_t w0[16], w1[16], hi[16], lo[16];
      tc::tmem_ld16(tmW + lane_off + t0, w0);
      tc::tmem_ld16(tmW + lane_off + t0 + 16, w1);
      tc::tmem_ld_wait();
      const uint8_t* vb = Vc + (col >> 6) * (kCkC * 128) + (col & 63) * 2;
#pragma unroll
      for (int e = 0; e < 16; ++e) {
        float xv[2];
#pragma unroll
        for (int f = 0; f < 2; ++f) {
          const int u = 2 * e + f, t = t0 + u;
          const float vt = __uint_as_float(
              (uint32_t)*reinterpret_cast<const unsigned short*>(vb + t * 128) << 16);
          const float wt = __uint_as_float(u < 16 ? w0[u & 15] : w1[u & 15]);
          xv[f] = sh.bc[t] * (vt - sh.Gc[t] * wt);
        }
        ck_split(xv[0], xv[1], hi[e], lo[e]);
      }
      tc::tmem_st16(tmS + lane_off + 16 * grp, hi);
      tc::tmem_st16(tmS + lane_off + 32 + 16 * grp, lo);
      tc::tmem_st_wait();
    }
    tc::fence_before_sync();
    if (__syncthreads_or(bad)) break;  // tables, T's diagonal blocks, X^T; G and V read

    // ---- T = (I + A)^{-1} below its diagonal blocks: block column 0 on
    // warps 0-3, 1 on warps 4-5, 2 (and the strip of 3) on warps 6-7
    // (columns 1 and 2 share one code path, the block column a run-time
    // value: the groups run at once, so each copy crowds the instruction cache)
    if (warp < 4)
      ck_tcol<128>(AT, Tf, Vc, 0, 1, tid, 1);
    else
      ck_tcol<64>(AT, Tf, Vc, 1 + ((warp - 4) >> 1), warp < 6 ? 1 : 2, tid & 63, warp < 6 ? 2 : 3);
    if (__syncthreads_or(bad)) break;  // T as bf16 high / low parts
    if (tid == kIssuer) {
      const uint32_t tb = tc::smem_u32(Vc);
#pragma unroll
      for (int kk = 0; kk < kCkC / 16; ++kk) {
        const uint64_t bh = tc::sdesc_sw128(tb + kk * 32, 16, 1024);
        const uint64_t bl = tc::sdesc_sw128(tb + 8192 + kk * 32, 16, 1024);
        tc::mma_bf16_ts(tmD, tmS + kk * 8, bh, id64, kk > 0);  // delta^T = X^T T^T
        tc::mma_bf16_ts(tmD, tmS + kk * 8, bl, id64, 1);
        tc::mma_bf16_ts(tmD, tmS + 32 + kk * 8, bh, id64, 1);
      }
      tc::mma_commit(&sh.bar_mma);
      mma_out = true;
    }
    bad |= !tc::mbar_wait(&sh.bar_mma, ph_mma, &sh.abort_flag);
    ph_mma ^= 1u;
    tc::fence_after_sync();
    if (tid == kIssuer) mma_out = false;
    // delta^T as bf16 pairs over X^T's high part, tokens 32 grp .. 32 grp + 31
    {
      uint32_t d0[16], d1[16], w[16];
      tc::tmem_ld16(tmD + lane_off + 32 * grp, d0);
      tc::tmem_ld16(tmD + lane_off + 32 * grp + 16, d1);
      tc::tmem_ld_wait();
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        w[e] = ck_pack(__uint_as_float(d0[2 * e]), __uint_as_float(d0[2 * e + 1]));
        w[8 + e] = ck_pack(__uint_as_float(d1[2 * e]), __uint_as_float(d1[2 * e + 1]));
      }
      tc::tmem_st16(tmS + lane_off + 16 * grp, w);
      tc::tmem_st_wait();
    }
    tc::fence_before_sync();
    if (__syncthreads_or(bad)) break;  // delta^T complete
    if (tid == kIssuer) {
      tc::fence_after_sync();
#pragma unroll
      for (int kk = 0; kk < kCkC / 16; ++kk)
        tc::mma_bf16_ts(tmG, tmS + kk * 8,
                        tc::sdesc_sw128(tc::smem_u32(Ps + kk * 2048), kCkC * 128, 1024), id128,
                        kk > 0);  // C^T = delta^T P, over G
      tc::mma_commit(&sh.bar_mma);
      mma_out = true;
    }
    bad |= !tc::mbar_wait(&sh.bar_mma, ph_mma, &sh.abort_flag);
    ph_mma ^= 1u;
    tc::fence_after_sync();
    if (tid == kIssuer) mma_out = false;

    // ---- noisy blocks, tokens 32 grp .. 32 grp + 31 of the chunk, 16 at a
    // time (whole blocks: B divides 16):
    //   X~_t = beta~_t (v~_t - Gam~_t (Gam_{mB-1} W^T[k~_t] + C^T[k~_t])),
    //   the B x B solves, then
    //   o~_l = s (Gam~_end (Gam_{mB-1} W^T[q~_l] + C^T[q~_l]) + Aqk delta~)
    {
      const uint8_t* vb = Vn + (col >> 6) * (kCkC * 128) + (col & 63) * 2;
      const bool odd = lane & 1;
      __nv_bfloat16* out =
          static_cast<__nv_bfloat16*>(p.out) + (L.tok0 * p.Hv + L.j) * kCkD + (col & ~1);
#pragma unroll 1
      for (int g16 = 0; g16 < 2; ++g16) {
        const int t0 = 32 * grp + 16 * g16;  // the first token of these 16
        float xn[16];
        {
          uint32_t wk[16], ck[16];
          tc::tmem_ld16(tmW + lane_off + 64 + t0, wk);  // W^T, noisy keys
          tc::tmem_ld16(tmG + lane_off + t0, ck);       // C^T, noisy keys
          tc::tmem_ld_wait();
#pragma unroll
          for (int e = 0; e < 16; ++e) {
            const int t = t0 + e;
            const int mb = t0 + (e & ~(B - 1));
            const float am = mb > 0 ? sh.Gc[mb - 1] : 1.f;  // Gam_{mB-1}
            const float vt = __uint_as_float(
                (uint32_t)*reinterpret_cast<const unsigned short*>(vb + t * 128) << 16);
            xn[e] = sh.bn[t] * (vt - sh.Gn[t] * (am * __uint_as_float(wk[e]) +
                                                  __uint_as_float(ck[e])));
          }
        }
        // (I + A~) delta~ = X~ per block, forward substitution
#pragma unroll
        for (int u = 0; u < 16; ++u) {
          const int m0u = u & ~(B - 1);  // block start within the 16 (compile-time)
          float acc = xn[u];
          if constexpr (B >= 4) {  // (t0 + m0u) is then a multiple of 4: 16-byte loads
#pragma unroll
            for (int i4 = 0; 4 * i4 < u - m0u; ++i4) {  // the units holding columns < u
              const float4 a =
                  *reinterpret_cast<const float4*>(An + ck_sw(t0 + u, t0 + m0u + 4 * i4));
              const float av[4] = {a.x, a.y, a.z, a.w};
#pragma unroll
              for (int e = 0; e < 4; ++e) {
                const int i = m0u + 4 * i4 + e;
                if (i < u) acc = fmaf(-av[e], xn[i], acc);
              }
            }
          } else {
#pragma unroll
            for (int e = 0; e < B; ++e)
              if (m0u + e < u) acc = fmaf(-An[ck_sw(t0 + u, t0 + m0u + e)], xn[m0u + e], acc);
          }
          xn[u] = acc;
        }
        // readout, block by block (the block's queries from one AqT row
        // segment per key); adjacent lanes swap one value so that each stores
        // a bf16 pair of two columns
        uint32_t cq[16], wq[16];
        tc::tmem_ld16(tmG + lane_off + 64 + t0, cq);   // C^T, noisy queries
        tc::tmem_ld16(tmW + lane_off + 128 + t0, wq);  // W^T, noisy queries
        tc::tmem_ld_wait();
        // the stores of one pair of queries (u, u + 1)
        auto store_pair = [&](int u, float o0, float o1) {
          o0 *= p.scale;
          o1 *= p.scale;
          const float recv = __shfl_xor_sync(0xffffffffu, odd ? o0 : o1, 1);
          const int l = t0 + (odd ? u + 1 : u);
          *reinterpret_cast<uint32_t*>(out + (size_t)l * p.Hv * kCkD) =
              odd ? ck_pack(recv, o1) : ck_pack(o0, recv);
        };
        if constexpr (B == 1) {
#pragma unroll
          for (int u = 0; u < 16; u += 2) {
            float o[2];
#pragma unroll
            for (int f = 0; f < 2; ++f) {
              const int l = t0 + u + f;
              const float am = l > 0 ? sh.Gc[l - 1] : 1.f;
              o[f] = sh.Gn[l] * (am * __uint_as_float(wq[u + f]) + __uint_as_float(cq[u + f])) +
                     AqT[ck_sw(l, l)] * xn[u + f];
            }
            store_pair(u, o[0], o[1]);
          }
        } else {
#pragma unroll
          for (int mb = 0; mb < 16; mb += B) {
            const int m0 = t0 + mb;  // the block's first token
            const float am = m0 > 0 ? sh.Gc[m0 - 1] : 1.f;
            const float ge = sh.Gn[m0 + B - 1];
            float o[B];
#pragma unroll
            for (int l = 0; l < B; ++l)
              o[l] = ge * (am * __uint_as_float(wq[mb + l]) + __uint_as_float(cq[mb + l]));
#pragma unroll
            for (int e = 0; e < B; ++e) {  // key m0 + e: AqT[m0 + e][m0 .. m0 + B - 1]
              float aq[B];
              if constexpr (B >= 4) {
#pragma unroll
                for (int i4 = 0; i4 < B / 4; ++i4) {
                  const float4 a =
                      *reinterpret_cast<const float4*>(AqT + ck_sw(m0 + e, m0 + 4 * i4));
                  aq[4 * i4] = a.x; aq[4 * i4 + 1] = a.y; aq[4 * i4 + 2] = a.z; aq[4 * i4 + 3] = a.w;
                }
              } else {
                const float2 a = *reinterpret_cast<const float2*>(AqT + ck_sw(m0 + e, m0));
                aq[0] = a.x; aq[1] = a.y;
              }
#pragma unroll
              for (int l = 0; l < B; ++l) o[l] = fmaf(aq[l], xn[mb + e], o[l]);
            }
#pragma unroll
            for (int l = 0; l < B; l += 2) store_pair(mb + l, o[l], o[l + 1]);
          }
        }
      }
    }
    // the next chunk's values: both groups are past their reads of these
    // (the clean ones before the second barrier, the T parts over them by
    // MMA d, the noisy ones just now)
    tc::fence_before_sync();
    if (__syncthreads_or(bad)) break;
    if (tid == kIssuer && it_next >= 0) {
      tc::fence_async_smem();
      issue_v(it_next);
      v_out = true;
      v_par = ph ^ 1u;
    }
    ph ^= 1u;
  }
  bad = __syncthreads_or(bad);
  if (bad && tid == 0 && !sh.abort_flag) {
    sh.abort_flag = 1;
    flag(p.dev_status, FLARE_DEV_WAIT_TIMEOUT);
  }
  if (tid == kIssuer && bad) {
    if (s0_out) tc::mbar_wait(&sh.bar_s0, s0_par, nullptr, 100000000ull);
    if (kx_out) tc::mbar_wait(&sh.bar_kx, kx_par, nullptr, 100000000ull);
    if (v_out) tc::mbar_wait(&sh.bar_v, v_par, nullptr, 100000000ull);
    if (mma_out) tc::mbar_wait(&sh.bar_mma, ph_mma, nullptr, 100000000ull);
  }
  tc::fence_before_sync();
  __syncthreads();
  if (warp == 0) {
    tc::fence_after_sync();
    tc::tmem_dealloc(tmem, 512);
  }
}

// ------------------------------------------------------------------ host side

namespace {

PFN_cuTensorMapEncodeTiled_v12000 ck_encode_fn() {
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

// [N, L, H, 128] bf16 as a 4-D map (128, H, L, N), box (64, 1, 64, 1)
bool ck_map(CUtensorMap* m, const void* x, int H, int L, int N, bool swizzle) {
  auto fn = ck_encode_fn();
  if (!fn) return false;
  cuuint64_t gd[4] = {(cuuint64_t)kCkD, (cuuint64_t)H, (cuuint64_t)L, (cuuint64_t)N};
  cuuint64_t gs[3] = {(cuuint64_t)kCkD * 2, (cuuint64_t)H * kCkD * 2,
                      (cuuint64_t)L * H * kCkD * 2};
  cuuint32_t bx[4] = {64, 1, (cuuint32_t)kCkC, 1};
  cuuint32_t es[4] = {1, 1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(x), gd, gs, bx, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE,
            swizzle ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_NONE,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) ==
         CUDA_SUCCESS;
}

template <int B>
cudaError_t launch_ck(const TwoStreamParams& p, cudaStream_t stream) {
  CkMaps maps;
  if (!ck_map(&maps.k, p.k, p.Hk, p.L, p.N, true) || !ck_map(&maps.kn, p.kn, p.Hk, p.L, p.N, true) ||
      !ck_map(&maps.qn, p.qn, p.Hk, p.L, p.N, true) || !ck_map(&maps.v, p.v, p.Hv, p.L, p.N, false) ||
      !ck_map(&maps.vn, p.vn, p.Hv, p.L, p.N, false))
    return cudaErrorInvalidValue;
  const int smem = CkCfg::kSmem + 1024;
  cudaError_t e = cudaFuncSetAttribute(two_stream_chunk_kernel<B>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  int dev = 0, sms = kNumSMs;
  if (cudaGetDevice(&dev) == cudaSuccess)
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const long items = (long)p.N * p.Hv * (p.L / kCkC);
  const int grid = (int)(items < sms ? items : sms);
  two_stream_chunk_kernel<B><<<grid, kCkThreads, smem, stream>>>(maps, p);
  note_launches(1);
  return cudaGetLastError();
}

}  // namespace

bool two_stream_chunk_supported(int B, int dk, int dv) {
  return dk == kCkD && dv == kCkD && (B == 1 || B == 2 || B == 4 || B == 8 || B == 16);
}

cudaError_t launch_two_stream_chunk(const TwoStreamParams& p, cudaStream_t stream) {
  if (p.N == 0 || p.L == 0) return cudaSuccess;
  switch (p.B) {
    case 1: return launch_ck<1>(p, stream);
    case 2: return launch_ck<2>(p, stream);
    case 4: return launch_ck<4>(p, stream);
    case 8: return launch_ck<8>(p, stream);
    case 16: return launch_ck<16>(p, stream);
  }
  return cudaErrorInvalidValue;
}

}  // namespace flare
