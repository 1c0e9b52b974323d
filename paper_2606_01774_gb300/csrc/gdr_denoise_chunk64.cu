// Denoise pass of a gated-delta-rule layer for the 128 x 128 state on tcgen05
// tensor cores, persistent form for blocks of 33 .. 64 tokens: bf16
// activations, the block as one 64-token chunk.
//
// For one (request r, value head j) with q/k head h and frozen state S0, the
// block-end readout (Eq. noisy-block-fwd) through the chunkwise WY/UT form of
// the block (appendix "Chunk-corrected values", Eq. chunk-state):
//
//   gamma_t = g_0 + ... + g_t,  Gam_t = exp(gamma_t)
//   A[t][i] = beta_t exp(gamma_t - gamma_i) (k_t . k_i),   i < t
//   X       = diag(beta) (V - diag(Gam) K S0),   delta = (I + A)^{-1} X
//   out[l]  = s (Gam_{B-1} S0^T q_l + sum_i exp(gamma_{B-1} - gamma_i) (q_l . k_i) delta_i)
//
// Value column c on tensor-memory lane c; thread c owns column c.  Per item:
//   MMA 1  G   = [K; Q] K^T       M=128 (K rows on lanes 0..63, Q rows on 64..127), N=64, K=128
//          W^T = S0^T [K; Q]^T    M=128 (c), N=128, K=128   (A: S0^T bf16, tensor memory)
//   T      = (I + A)^{-1}          fp32, 16 x 16 blocks: the diagonal ones by forward
//                                  substitution, then block columns
//   MMA d  delta^T = X^T T^T      M=128, N=64, K=64  (X and T as bf16 high + low parts,
//                                  three products: fp32-grade delta)
//   MMA 2  O2^T = delta^T M2^T    M=128, N=64, K=64  (delta^T bf16, tensor memory;
//          M2[l][i] = exp(gamma_{B-1} - gamma_i) (q_l . k_i), bf16 K-major)
//   out[l][c] = s (Gam_{B-1} W^T[c][64 + l] + O2^T[c][l])
// Rows past B read as zero (the block's tensor maps end at B), so A, M2 and X
// vanish there and T is the identity.
//
// Persistent CTAs, two per SM (113 KiB of shared memory, 256 tensor-memory
// columns and 128 threads each), so that each SM holds two items' latency
// chains.  The state arrives in two 32 KiB halves into two buffers: the first
// half's buffer takes the next item's first half as soon as it has been read,
// a whole item ahead; the second half's buffer then holds A^T and T, and takes
// the next item's second half once T is formed.  The key/query buffer holds
// M2 and T's bf16 parts once the first MMAs have read it; delta^T's fp32
// product lands over W^T's key columns, which X has read.  The next item's
// keys and queries are requested once the second MMA has read M2, its values
// once X has read this item's; its gates are loaded into registers one item
// ahead.  Every wait is bounded: on a timeout the CTA sets
// FLARE_DEV_WAIT_TIMEOUT, waits (bounded) for its copies and MMAs in flight,
// frees its tensor memory and exits.
#include <cudaTypedefs.h>

#include "chunk64.cuh"
#include "common.cuh"
#include "kernels.h"
#include "tc.cuh"

namespace flare {

namespace {

constexpr int kD6Threads = 128;
constexpr int kD6D = 128;  // d_k = d_v
using namespace chunk64;   // kCkC = 64 and the chunk-system helpers

struct alignas(16) D6Shared {
  uint64_t bar_s0a, bar_s0b, bar_kq, bar_v, bar_g, bar_mma;
  uint32_t tmem_base;
  int abort_flag;
  alignas(16) float gc2[kCkC];  // gamma_t log2(e)
  alignas(16) float Gc[kCkC];   // exp(gamma_t)
  alignas(16) float bc[kCkC];   // beta (zero past B)
};

struct D6Cfg {
  static constexpr int kS0h = 64 * kD6D * 4;   // half of S0 fp32: rows 64 h .. 64 h + 63
  static constexpr int kKQ = 2 * 128 * 128;    // [K; Q]: 2 chunks of 128 rows x 128 B (SW128)
  static constexpr int kV = 2 * kCkC * 128;    // values: 2 chunks of 64 rows x 128 B
  static constexpr int kT = kCkC * kCkC * 4;   // a 64 x 64 fp32 table
  static constexpr int kM2 = kCkC * 128;       // M2 [l][i] bf16, K-major SW128
  static constexpr int oS0a = 0;               // the state's first half
  static constexpr int oS0b = kS0h;            // its second half; then A^T and T
  static constexpr int oAT = oS0b;
  static constexpr int oT = oS0b + kT;
  static constexpr int oKQ = 2 * kS0h;         // [K; Q]; then M2 and T's bf16 parts
  static constexpr int oM2 = oKQ;
  static constexpr int oTb = oKQ + kM2;        // T high, then low (8 KiB each)
  static constexpr int oV = oKQ + kKQ;
  static constexpr int oSh = oV + kV;          // the barriers and gate factors
  // two CTAs per SM: 2 (kSmem + the 1 KiB the system keeps per CTA) <= 228 KiB
  static constexpr int kSmem = oSh + (int)sizeof(D6Shared);
  static_assert(2 * kT <= kS0h && kM2 + 2 * 8192 <= kKQ, "buffer reuse");
  static_assert(2 * (kSmem + 1024) <= 228 * 1024, "two CTAs per SM");
};

struct D6Maps {
  CUtensorMap k, q;  // (128, Hk, B, R) box (64, 1, 64, 1), 128-byte swizzle
  CUtensorMap v;     // (128, Hv, B, R) box (64, 1, 64, 1), no swizzle
};

// The next item at or after `it` (stride gridDim.x) with a valid slot; bad
// slots are flagged and skipped.  Called by every thread with the same
// arguments.
__device__ __forceinline__ int d6_next(const GdrParams& p, int it, int total, int& slot) {
  for (; it < total; it += gridDim.x) {
    const int s = p.state_slot[it / p.Hv];
    if (s < 0 || s >= p.nslots) {
      if (threadIdx.x == 0) flag(p.dev_status, FLARE_DEV_BAD_SLOT);
      continue;
    }
    slot = s;
    return it;
  }
  return -1;
}

}  // namespace

__global__ void __launch_bounds__(kD6Threads, 2)
    gdr_denoise_chunk64_kernel(const __grid_constant__ D6Maps maps, GdrParams p) {
  using C = D6Cfg;
  constexpr int kIssuer = 32;  // one thread of warp 1 issues every copy and MMA
  // no static shared memory, so that the dynamic window starts 1024-byte
  // aligned (the 128-byte swizzled operands need it): checked below
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* base = smem_raw;
  D6Shared& sh = *reinterpret_cast<D6Shared*>(base + C::oSh);
  float* S0a = reinterpret_cast<float*>(base + C::oS0a);
  float* S0b = reinterpret_cast<float*>(base + C::oS0b);
  float* AT = reinterpret_cast<float*>(base + C::oAT);
  float* Tf = reinterpret_cast<float*>(base + C::oT);
  uint8_t* KQ = base + C::oKQ;
  uint8_t* M2s = base + C::oM2;
  uint8_t* Tb = base + C::oTb;
  uint8_t* Vs = base + C::oV;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int total = p.R * p.Hv;
  const int B = p.B;

  int slot = 0;
  int it = d6_next(p, blockIdx.x, total, slot);
  if (it < 0) return;  // the same answer on every thread
  if (tc::smem_u32(smem_raw) & 1023u) {  // a window the swizzled layout cannot use
    if (tid == 0) flag(p.dev_status, FLARE_DEV_WAIT_TIMEOUT);
    return;
  }

  if (tid == kIssuer) {
    sh.abort_flag = 0;
    tc::mbar_init(&sh.bar_s0a, 1);
    tc::mbar_init(&sh.bar_s0b, 1);
    tc::mbar_init(&sh.bar_kq, 1);
    tc::mbar_init(&sh.bar_v, 1);
    tc::mbar_init(&sh.bar_g, 1);
    tc::mbar_init(&sh.bar_mma, 1);
    tc::fence_mbar_init();
  }
  if (warp == 0) tc::tmem_alloc(&sh.tmem_base, 256);
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = sh.tmem_base;
  const uint32_t tmS = tmem;        // S0^T bf16 (64 columns); X^T high | low; delta^T (32)
  const uint32_t tmW = tmem + 64;   // W^T: [K | Q] parts, 2 x 64 columns; delta^T fp32 over K
  const uint32_t tmG = tmem + 192;  // G (rows on lanes), 64 columns; then O2^T
  const uint32_t lane_off = (uint32_t)(warp * 32) << 16;

  auto issue_s0 = [&](int item, int s, int h) {  // rows 64 h .. 64 h + 63 of the state
    const float* src = p.state_pool + ((size_t)s * p.Hv + item % p.Hv) * kD6D * kD6D +
                       (size_t)h * 64 * kD6D;
    uint64_t* bar = h ? &sh.bar_s0b : &sh.bar_s0a;
    tc::mbar_expect_tx(bar, C::kS0h);
    tc::bulk_load(h ? S0b : S0a, src, C::kS0h, bar);
  };
  auto issue_kq = [&](int item) {
    const int r = item / p.Hv, h = (item % p.Hv) / (p.Hv / p.Hk);
    tc::mbar_expect_tx(&sh.bar_kq, C::kKQ);
#pragma unroll
    for (int d = 0; d < 2; ++d) {
      tc::tma_load_4d(KQ + d * (128 * 128), &maps.k, &sh.bar_kq, d * 64, h, 0, r);
      tc::tma_load_4d(KQ + d * (128 * 128) + 64 * 128, &maps.q, &sh.bar_kq, d * 64, h, 0, r);
    }
  };
  auto issue_v = [&](int item) {
    const int r = item / p.Hv, j = item % p.Hv;
    tc::mbar_expect_tx(&sh.bar_v, C::kV);
#pragma unroll
    for (int d = 0; d < 2; ++d)
      tc::tma_load_4d(Vs + d * (kCkC * 128), &maps.v, &sh.bar_v, d * 64, j, 0, r);
  };
  // warp 0 holds the gates of the item it processes next, loaded one item
  // ahead: tokens lane and lane + 32 (zero past B)
  float ga = 0.f, gb = 0.f, ba = 0.f, bb = 0.f;
  auto load_gates = [&](int item) {
    const size_t g0 = (size_t)(item / p.Hv) * B * p.Hv + item % p.Hv;
    ga = lane < B ? p.log_decay[g0 + (size_t)lane * p.Hv] : 0.f;
    gb = lane + 32 < B ? p.log_decay[g0 + (size_t)(lane + 32) * p.Hv] : 0.f;
    ba = lane < B ? p.beta[g0 + (size_t)lane * p.Hv] : 0.f;
    bb = lane + 32 < B ? p.beta[g0 + (size_t)(lane + 32) * p.Hv] : 0.f;
  };
  auto cand_slot = [&](int c) { return c < total ? p.state_slot[c / p.Hv] : -1; };

  // the issuing thread's record of what is in flight (and the parity its
  // barrier phase completes with), for a clean exit after a timeout
  bool s0a_out = false, s0b_out = false, kq_out = false, v_out = false, mma_out = false;
  uint32_t s0a_par = 0, s0b_par = 0, kq_par = 0, v_par = 0;
  if (tid == kIssuer) {
    tc::prefetch_tmap(&maps.k);
    tc::prefetch_tmap(&maps.q);
    tc::prefetch_tmap(&maps.v);
    issue_s0(it, slot, 0);
    issue_s0(it, slot, 1);
    issue_kq(it);
    issue_v(it);
    s0a_out = s0b_out = kq_out = v_out = true;
  }
  if (warp == 0) load_gates(it);
  int cand = it + gridDim.x;
  int cs = cand_slot(cand);
  bool bad = false;
  uint32_t ph = 0, ph_mma = 0;
  const uint32_t idG = tc::idesc_bf16(128, 64, false, false);
  const uint32_t idW = tc::idesc_bf16(128, 128, false, false);
  const uint32_t id64 = tc::idesc_bf16(128, 64, false, false);

#pragma unroll 1
  while (true) {
    const int r = it / p.Hv, j = it % p.Hv;
    // the block's gates: gamma = inclusive prefix sum of the log-gates over
    // its 64 rows (zero past B)
    if (warp == 0) {
      float x0 = ga, x1 = gb;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const float u = __shfl_up_sync(0xffffffffu, x0, o);
        const float w = __shfl_up_sync(0xffffffffu, x1, o);
        if (lane >= o) {
          x0 += u;
          x1 += w;
        }
      }
      x1 += __shfl_sync(0xffffffffu, x0, 31);
      const float g0 = x0 * 1.4426950408889634f, g1 = x1 * 1.4426950408889634f;
      sh.gc2[lane] = g0;
      sh.gc2[lane + 32] = g1;
      sh.Gc[lane] = expf(x0);
      sh.Gc[lane + 32] = expf(x1);
      sh.bc[lane] = ba;
      sh.bc[lane + 32] = bb;
    }
    // the next item: the candidate when its slot is valid, else the first
    // valid one after it (bad ones flagged on the way)
    int it_next = -1, slot_next = 0;
    if (cand < total) {
      if (cs >= 0 && cs < p.nslots) {
        it_next = cand;
        slot_next = cs;
      } else {
        it_next = d6_next(p, cand, total, slot_next);
      }
    }
    if (it_next >= 0) {
      if (warp == 0) load_gates(it_next);
      cand = it_next + gridDim.x;
      cs = cand_slot(cand);
    }

    // S0^T into tensor memory as bf16 pairs, the state's two halves from
    // their two buffers
#pragma unroll 1
    for (int h = 0; h < 2; ++h) {
      bad |= !tc::mbar_wait(h ? &sh.bar_s0b : &sh.bar_s0a, ph, &sh.abort_flag);
      const float* S0h = h ? S0b : S0a;
#pragma unroll 1
      for (int i0 = 0; i0 < 64; i0 += 32) {
        uint32_t w[16];
#pragma unroll
        for (int e = 0; e < 16; ++e)
          w[e] = ck_pack(S0h[(i0 + 2 * e) * kD6D + tid], S0h[(i0 + 2 * e + 1) * kD6D + tid]);
        tc::tmem_st16(tmS + lane_off + (64 * h + i0) / 2, w);
      }
    }
    if (tid == kIssuer) s0a_out = s0b_out = false;
    tc::tmem_st_wait();
    tc::fence_before_sync();
    if (__syncthreads_or(bad)) break;  // S0^T complete, both halves read
    if (tid == kIssuer && it_next >= 0) {  // the first half's buffer is free
      issue_s0(it_next, slot_next, 0);
      s0a_out = true;
      s0a_par = ph ^ 1u;
    }
    if (tid == kIssuer) {
      bad |= !tc::mbar_wait(&sh.bar_kq, ph, &sh.abort_flag);
      kq_out = false;
      tc::fence_after_sync();
      // the Gram first, committed on its own: the tables are built from it
      // while the state products run
#pragma unroll
      for (int kk = 0; kk < kD6D / 16; ++kk) {
        const uint64_t kd = tc::sdesc_sw128(
            tc::smem_u32(KQ + (kk >> 2) * (128 * 128) + (kk & 3) * 32), 16, 1024);
        tc::mma_bf16_ss(tmG, kd, kd, idG, kk > 0);  // G = [K; Q] K^T
      }
      tc::mma_commit(&sh.bar_g);
#pragma unroll
      for (int kk = 0; kk < kD6D / 16; ++kk) {
        const uint64_t kd = tc::sdesc_sw128(
            tc::smem_u32(KQ + (kk >> 2) * (128 * 128) + (kk & 3) * 32), 16, 1024);
        tc::mma_bf16_ts(tmW, tmS + kk * 8, kd, idW, kk > 0);  // W^T = S0^T [K; Q]^T
      }
      tc::mma_commit(&sh.bar_mma);
      mma_out = true;
    }
    bad |= !tc::mbar_wait(&sh.bar_g, ph, &sh.abort_flag);
    tc::fence_after_sync();

    // ---- tables from G (every exponential taken unconditionally, the masks
    // applied as selects): warps 0-1 A^T (key rows), warps 2-3 M2 (query rows,
    // stored over [K; Q] once the state products have read it) and then T's
    // diagonal blocks
    {
      const int row = tid & 63;
      if (tid < 64) {
        const float gi = sh.gc2[row];
#pragma unroll 1
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
        tc::named_bar_arrive(5, 128);  // A^T to warps 2-3
      } else {
        const bool live = row < B;
        const float gB = sh.gc2[B - 1];
        uint32_t wv[32];  // the row's 64 values as bf16 pairs
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          uint32_t gr[32];
          ck_ld32(tmG + lane_off + 32 * h, gr);
#pragma unroll
          for (int e = 0; e < 16; ++e) {
            // the row factor exp(gamma_{B-1} - gamma_i), zero for i >= B
            const int i = 32 * h + 2 * e;
            const float m0 = tc::ex2(gB - sh.gc2[i]) * __uint_as_float(gr[2 * e]);
            const float m1 = tc::ex2(gB - sh.gc2[i + 1]) * __uint_as_float(gr[2 * e + 1]);
            wv[16 * h + e] =
                ck_pack(live && i < B ? m0 : 0.f, live && i + 1 < B ? m1 : 0.f);
          }
        }
        bad |= !tc::mbar_wait(&sh.bar_mma, ph_mma, &sh.abort_flag);  // [K; Q] read
#pragma unroll
        for (int u = 0; u < 8; ++u)
          *reinterpret_cast<uint4*>(M2s + row * 128 + ((u ^ (row & 7)) << 4)) =
              make_uint4(wv[4 * u], wv[4 * u + 1], wv[4 * u + 2], wv[4 * u + 3]);
        tc::fence_async_smem();  // M2 is the second MMA's operand
        tc::named_bar_sync(5, 128);
        ck_diag_inverse(AT, Tf, 2 * (warp - 2) + (lane >> 4), lane & 15);
      }
    }

    // ---- X = diag(beta) (V - diag(Gam) K S0), all 64 tokens, into tensor
    // memory as bf16 high and low parts over S0^T (which the first MMAs have read)
    bad |= !tc::mbar_wait(&sh.bar_mma, ph_mma, &sh.abort_flag);
    ph_mma ^= 1u;
    tc::fence_after_sync();
    if (tid == kIssuer) mma_out = false;
    bad |= !tc::mbar_wait(&sh.bar_v, ph, &sh.abort_flag);
    if (tid == kIssuer) v_out = false;
    {
      const uint8_t* vb = Vs + (tid >> 6) * (kCkC * 128) + (tid & 63) * 2;
#pragma unroll 1
      for (int h = 0; h < 2; ++h) {
        const int t0 = 32 * h;
        uint32_t w[32], hi[16], lo[16];
        ck_ld32(tmW + lane_off + t0, w);
#pragma unroll
        for (int e = 0; e < 16; ++e) {
          float xv[2];
#pragma unroll
          for (int f = 0; f < 2; ++f) {
            const int u = 2 * e + f, t = t0 + u;
            const float vt = __uint_as_float(
                (uint32_t)*reinterpret_cast<const unsigned short*>(vb + t * 128) << 16);
            xv[f] = sh.bc[t] * (vt - sh.Gc[t] * __uint_as_float(w[u]));
          }
          ck_split(xv[0], xv[1], hi[e], lo[e]);
        }
        tc::tmem_st16(tmS + lane_off + 16 * h, hi);
        tc::tmem_st16(tmS + lane_off + 32 + 16 * h, lo);
      }
      tc::tmem_st_wait();
    }
    tc::fence_before_sync();
    if (__syncthreads_or(bad)) break;  // tables, T's diagonal blocks, X^T; G and V read
    if (tid == kIssuer && it_next >= 0) {
      issue_v(it_next);
      v_out = true;
      v_par = ph ^ 1u;
    }

    // ---- T = (I + A)^{-1} below its diagonal blocks: block column 0 on
    // warps 0-1, 1 on warp 2, 2 (and the strip of 3) on warp 3
    if (warp < 2)
      ck_tcol<64>(AT, Tf, Tb, 0, 1, tid, 1);
    else
      ck_tcol<32>(AT, Tf, Tb, warp - 1, warp == 2 ? 1 : 2, lane, warp);
    if (__syncthreads_or(bad)) break;  // T as bf16 high / low parts; A^T and T read
    if (tid == kIssuer) {
      if (it_next >= 0) {  // A^T and T read: the next item's second half
        issue_s0(it_next, slot_next, 1);
        s0b_out = true;
        s0b_par = ph ^ 1u;
      }
      const uint32_t tb = tc::smem_u32(Tb);
#pragma unroll
      for (int kk = 0; kk < kCkC / 16; ++kk) {
        const uint64_t bh = tc::sdesc_sw128(tb + kk * 32, 16, 1024);
        const uint64_t bl = tc::sdesc_sw128(tb + 8192 + kk * 32, 16, 1024);
        tc::mma_bf16_ts(tmW, tmS + kk * 8, bh, id64, kk > 0);  // delta^T = X^T T^T
        tc::mma_bf16_ts(tmW, tmS + kk * 8, bl, id64, 1);
        tc::mma_bf16_ts(tmW, tmS + 32 + kk * 8, bh, id64, 1);
      }
      tc::mma_commit(&sh.bar_mma);
      mma_out = true;
    }
    bad |= !tc::mbar_wait(&sh.bar_mma, ph_mma, &sh.abort_flag);
    ph_mma ^= 1u;
    tc::fence_after_sync();
    if (tid == kIssuer) mma_out = false;
    // delta^T as bf16 pairs over X^T's high part
#pragma unroll 1
    for (int h = 0; h < 2; ++h) {
      uint32_t d[32], w[16];
      ck_ld32(tmW + lane_off + 32 * h, d);
#pragma unroll
      for (int e = 0; e < 16; ++e) w[e] = ck_pack(__uint_as_float(d[2 * e]), __uint_as_float(d[2 * e + 1]));
      tc::tmem_st16(tmS + lane_off + 16 * h, w);
    }
    tc::tmem_st_wait();
    tc::fence_before_sync();
    if (__syncthreads_or(bad)) break;  // delta^T complete
    if (tid == kIssuer) {
      tc::fence_after_sync();
#pragma unroll
      for (int kk = 0; kk < kCkC / 16; ++kk)
        tc::mma_bf16_ts(tmG, tmS + kk * 8, tc::sdesc_sw128(tc::smem_u32(M2s + kk * 32), 16, 1024),
                        id64, kk > 0);  // O2^T = delta^T M2^T, over G
      tc::mma_commit(&sh.bar_mma);
      mma_out = true;
    }
    bad |= !tc::mbar_wait(&sh.bar_mma, ph_mma, &sh.abort_flag);
    ph_mma ^= 1u;
    tc::fence_after_sync();
    if (tid == kIssuer) {
      mma_out = false;
      if (it_next >= 0) {  // M2 and T's parts read: the buffer takes the next [K; Q]
        tc::fence_async_smem();
        issue_kq(it_next);
        kq_out = true;
        kq_par = ph ^ 1u;
      }
    }

    // ---- out[l][c] = s (Gam_{B-1} W^T[c][64 + l] + O2^T[c][l]); adjacent
    // lanes swap one value so that each stores a bf16 pair of two columns
    {
      const float sG = p.scale * sh.Gc[B - 1];
      const bool odd = lane & 1;
      __nv_bfloat16* out = static_cast<__nv_bfloat16*>(p.out_blockend) +
                           ((size_t)r * B * p.Hv + j) * kD6D + (tid & ~1);
#pragma unroll 1
      for (int h = 0; h < 2; ++h) {
        const int t0 = 32 * h;
        uint32_t o2[32], wq[32];
        tc::tmem_ld16(tmG + lane_off + t0, *reinterpret_cast<uint32_t(*)[16]>(&o2[0]));
        tc::tmem_ld16(tmG + lane_off + t0 + 16, *reinterpret_cast<uint32_t(*)[16]>(&o2[16]));
        tc::tmem_ld16(tmW + lane_off + 64 + t0, *reinterpret_cast<uint32_t(*)[16]>(&wq[0]));
        tc::tmem_ld16(tmW + lane_off + 64 + t0 + 16, *reinterpret_cast<uint32_t(*)[16]>(&wq[16]));
        tc::tmem_ld_wait();
#pragma unroll
        for (int l = 0; l < 32; l += 2) {
          const float a = fmaf(sG, __uint_as_float(wq[l]), p.scale * __uint_as_float(o2[l]));
          const float b =
              fmaf(sG, __uint_as_float(wq[l + 1]), p.scale * __uint_as_float(o2[l + 1]));
          const float recv = __shfl_xor_sync(0xffffffffu, odd ? a : b, 1);
          const int row = t0 + (odd ? l + 1 : l);
          if (row < B)
            *reinterpret_cast<uint32_t*>(out + (size_t)row * p.Hv * kD6D) =
                odd ? ck_pack(recv, b) : ck_pack(a, recv);
        }
      }
    }
    tc::fence_before_sync();
    if (__syncthreads_or(bad)) break;  // the gates and tensor memory free for the next item
    if (it_next < 0) break;
    it = it_next;
    slot = slot_next;
    ph ^= 1u;
  }
  bad = __syncthreads_or(bad);
  if (bad && tid == 0 && !sh.abort_flag) {
    sh.abort_flag = 1;
    flag(p.dev_status, FLARE_DEV_WAIT_TIMEOUT);
  }
  if (tid == kIssuer && bad) {
    if (s0a_out) tc::mbar_wait(&sh.bar_s0a, s0a_par, nullptr, 100000000ull);
    if (s0b_out) tc::mbar_wait(&sh.bar_s0b, s0b_par, nullptr, 100000000ull);
    if (kq_out) tc::mbar_wait(&sh.bar_kq, kq_par, nullptr, 100000000ull);
    if (v_out) tc::mbar_wait(&sh.bar_v, v_par, nullptr, 100000000ull);
    if (mma_out) tc::mbar_wait(&sh.bar_mma, ph_mma, nullptr, 100000000ull);
  }
  tc::fence_before_sync();
  __syncthreads();
  if (warp == 0) {
    tc::fence_after_sync();
    tc::tmem_dealloc(tmem, 256);
  }
}

// ------------------------------------------------------------------ host side

namespace {

PFN_cuTensorMapEncodeTiled_v12000 d6_encode_fn() {
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

// [R, B, H, 128] bf16 activations as a 4-D map (128, H, B, R), box (64, 1,
// 64, 1); rows past B read as zero
bool d6_act_map(CUtensorMap* m, const void* x, int H, int B, int R, bool swizzle) {
  auto fn = d6_encode_fn();
  if (!fn) return false;
  cuuint64_t gd[4] = {(cuuint64_t)kD6D, (cuuint64_t)H, (cuuint64_t)B, (cuuint64_t)R};
  cuuint64_t gs[3] = {(cuuint64_t)kD6D * 2, (cuuint64_t)H * kD6D * 2,
                      (cuuint64_t)B * H * kD6D * 2};
  cuuint32_t bx[4] = {64, 1, (cuuint32_t)kCkC, 1};
  cuuint32_t es[4] = {1, 1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(x), gd, gs, bx, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE,
            swizzle ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_NONE,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) ==
         CUDA_SUCCESS;
}

}  // namespace

bool gdr_denoise_chunk64_supported(int B, int dk, int dv) {
  return B > 32 && B <= kCkC && dk == kD6D && dv == kD6D;
}

cudaError_t launch_gdr_denoise_chunk64(const GdrParams& p, cudaStream_t stream) {
  if (p.R == 0) return cudaSuccess;
  D6Maps maps;
  if (!d6_act_map(&maps.k, p.k, p.Hk, p.B, p.R, true) ||
      !d6_act_map(&maps.q, p.q, p.Hk, p.B, p.R, true) ||
      !d6_act_map(&maps.v, p.v, p.Hv, p.B, p.R, false))
    return cudaErrorInvalidValue;
  const int smem = D6Cfg::kSmem;
  cudaError_t e = cudaFuncSetAttribute(gdr_denoise_chunk64_kernel,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  int dev = 0, sms = kNumSMs;
  if (cudaGetDevice(&dev) == cudaSuccess)
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const long items = (long)p.R * p.Hv;
  const int grid = (int)(items < 2L * sms ? items : 2L * sms);
  gdr_denoise_chunk64_kernel<<<grid, kD6Threads, smem, stream>>>(maps, p);
  note_launches(1);
  return cudaGetLastError();
}

}  // namespace flare
