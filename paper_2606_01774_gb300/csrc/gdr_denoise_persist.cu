// Denoise pass of a gated-delta-rule layer for the 128 x 128 state on tcgen05
// tensor cores, persistent form: bf16 activations, B <= 32.
//
// For one (request r, value head j) with q/k head h and frozen state S0, the
// block-end readout (Eq. noisy-block-fwd) through the chunkwise WY/UT form of
// the block (appendix "Chunk-corrected values", Eq. chunk-state):
//
//   gamma_t = g_0 + ... + g_t,  Gam_t = exp(gamma_t)
//   A[t][i] = beta_t exp(gamma_t - gamma_i) (k_t . k_i),   i < t
//   X       = diag(beta) (V - diag(Gam) K S0)
//   (I + A) delta = X
//   out[l]  = s (Gam_{B-1} S0^T q_l + sum_i exp(gamma_{B-1} - gamma_i) (q_l . k_i) delta_i)
//
// Value column c on tensor-memory lane c; thread c owns column c:
//
//   MMA 1  G   = [K;Q] K^T        M=128 ([K;Q] rows on lanes kG0..), N=Bp, K=128
//          W^T = S0^T [K;Q]^T     M=128 (c), N=2BM, K=128   (A: S0^T, bf16, tensor memory)
//          M2[l][i] = exp(gamma_{B-1} - gamma_i) (q_l . k_i)
//   N      = M2 T, T = (I + A)^{-1}   fp32: T's 16 x 16 diagonal blocks by forward
//          substitution, then (B > 16) N1 = M2_1 T11, N0 = (M2_0 - N1 A10) T00
//   MMA 2  O2^T = X^T N^T         M=128 (c), N=Bp, K=Bp     (X and N as bf16 high + low
//          parts, three products: O2 = delta^T M2^T with delta = T X, never formed)
//   out[l][c] = s (Gam_{B-1} W^T[c][BM + l] + O2^T[c][l])
//
// Bp = B rounded up to 16; the K, Q and V tiles hold BM = 16 or 32 rows (rows
// past B read as zero).  Inputs bf16, the state fp32 in memory and rounded to
// bf16 for the products, all accumulation fp32 (the same precision as the
// one-CTA-per-item kernel in gdr_tc.cu, which serves the other shapes).
//
// Persistent CTAs, two per SM (89-92 KiB of shared memory, 256 tensor-memory
// columns each), 128 threads, each walking the (request, value head) items
// blockIdx.x, blockIdx.x + gridDim.x, ...  The state arrives by bulk copy into
// a 64 KiB buffer that is free again as soon as it has been turned into the
// bf16 S0^T operand, so the next item's state streams in during this item's
// products, solve and readout; the next keys and queries follow this item's
// first MMA, the next values its second CTA barrier, the next gates and slot
// one item ahead into registers.  Three CTA barriers per item (S0^T written,
// A^T, M2, T's diagonal blocks and X^T written, N written); every other wait
// is a thread's own.  A bad slot is flagged in the device status word and
// the item skipped (its output untouched).  Every wait is bounded: on a
// timeout the CTA sets FLARE_DEV_WAIT_TIMEOUT, waits (bounded) for its copies
// and MMAs in flight, frees its tensor memory and exits.
#include <cudaTypedefs.h>

#include "common.cuh"
#include "kernels.h"
#include "tc.cuh"

namespace flare {

namespace {

constexpr int kDpThreads = 128;
constexpr int kDpD = 128;  // d_k = d_v

template <int BM>
struct DpCfg {
  static constexpr int kS0 = kDpD * kDpD * 4;   // S0 fp32 [i][c]
  static constexpr int kATs = BM + 4;           // row stride of A^T (floats)
  static constexpr int kAT = BM * kATs * 4;     // A^T[i][t] = A[t][i]
  static constexpr int kV = 2 * BM * 128;       // values: 2 chunks of BM rows x 128 B
  static constexpr int kG0 = 128 - 2 * BM;      // lane of G's first row
  // the Gram MMA's A operand starts kG0 rows ahead of the [K;Q] tile and
  // reads those bytes from the value and A^T buffers (their rows reach no
  // lane that is read): A^T's buffer is padded so that the two cover them
  static constexpr int kATb0 = (kAT + 1023) / 1024 * 1024;
  static constexpr int kATb = kV + kATb0 >= kG0 * 128 ? kATb0 : kG0 * 128 - kV;
  static constexpr int kKQ = 2 * 2 * BM * 128;  // 2 chunks of [K;Q]: 2BM rows x 128 B (SW128)
  static constexpr int kNb = 2 * BM * 128;      // N [l][j] bf16 high, then low: K-major, SW128
  static constexpr int kMf = BM * kATs * 4;     // an fp32 table: M2 [l][i], T [i][j]
  static constexpr int kSmem = kS0 + kV + kATb + kKQ + kNb + 2 * kMf;
};

struct alignas(16) DpShared {
  uint64_t bar_s0, bar_kq, bar_v, bar_g, bar_mma;
  uint32_t tmem_base;
  int abort_flag;
  // 16-byte aligned: read as float4 broadcasts
  alignas(16) float gam2[32];  // gamma_t log2(e)
  alignas(16) float Gam[32];   // exp(gamma_t)
  alignas(16) float beta[32];
  alignas(16) float eB[32];    // exp(gamma_{B-1} - gamma_i) for i < B, else 0 (the M2 row factor)
};

struct DpMaps {
  CUtensorMap k;  // (128, Hk, B, R) box (64, 1, BM, 1), 128-byte swizzle
  CUtensorMap q;
  CUtensorMap v;  // (128, Hv, B, R) box (64, 1, BM, 1), no swizzle
};

// The next item at or after `it` (stride gridDim.x) with a valid slot; bad
// slots are flagged and skipped.  Called by every thread with the same
// arguments.
__device__ __forceinline__ int dp_next(const GdrParams& p, int it, int total, int& slot) {
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

__device__ __forceinline__ uint32_t dp_pack(float a, float b) {
  __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<uint32_t*>(&h);
}

// x = hi + lo to about 2^-16 relative, each a bf16 pair (a low, b high)
__device__ __forceinline__ void dp_split(float a, float b, uint32_t& hi, uint32_t& lo) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
  const __nv_bfloat162 l = __floats2bfloat162_rn(a - __low2float(h), b - __high2float(h));
  hi = *reinterpret_cast<const uint32_t*>(&h);
  lo = *reinterpret_cast<const uint32_t*>(&l);
}

// Column j of the diagonal block T_aa = (I + A_aa)^{-1} (16 x 16): forward
// substitution, x_t -= A[t][i] x_i for t > i with row i of A^T (A's column i)
// as 16-byte loads; stored whole (zeros above the diagonal) into T[t][j].
template <int kATs>
__device__ __forceinline__ void dp_diag_inverse(const float* AT, float* Tf, int a, int j) {
  float x[16];
#pragma unroll
  for (int t = 0; t < 16; ++t) x[t] = t == j ? 1.f : 0.f;
#pragma unroll
  for (int i = 0; i < 15; ++i) {
    const float xi = x[i];
#pragma unroll
    for (int u = (i + 1) / 4; u < 4; ++u) {
      const float4 q = *reinterpret_cast<const float4*>(AT + (16 * a + i) * kATs + 16 * a + 4 * u);
      const float qv[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
      for (int e = 0; e < 4; ++e)
        if (4 * u + e > i) x[4 * u + e] = fmaf(-qv[e], xi, x[4 * u + e]);
    }
  }
#pragma unroll
  for (int t = 0; t < 16; ++t) Tf[(16 * a + t) * kATs + 16 * a + j] = x[t];
}

}  // namespace

template <int BM>
__global__ void __launch_bounds__(kDpThreads, 2)
    gdr_denoise_persist_kernel(const __grid_constant__ DpMaps maps, GdrParams p) {
  using C = DpCfg<BM>;
  constexpr int kATs = C::kATs;
  constexpr int kG0 = C::kG0;
  // one thread of warp 1 issues every copy and MMA: warp 0 scans the gates,
  // warps 2-3 turn G into A^T and M2
  constexpr int kIssuer = 32;
  extern __shared__ uint8_t smem_raw[];
  __shared__ DpShared sh;
  uint8_t* base = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  float* S0s = reinterpret_cast<float*>(base);
  uint8_t* Vs = base + C::kS0;
  float* AT = reinterpret_cast<float*>(Vs + C::kV);
  uint8_t* KQs = Vs + C::kV + C::kATb;
  uint8_t* Nbs = KQs + C::kKQ;
  float* M2f = reinterpret_cast<float*>(Nbs + C::kNb);
  float* Tf = M2f + BM * kATs;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int total = p.R * p.Hv;
  const int B = p.B;
  const int Bp = (B + 15) & ~15;

  int slot = 0;
  int it = dp_next(p, blockIdx.x, total, slot);
  if (it < 0) return;  // the same answer on every thread

  if (tid == kIssuer) {
    sh.abort_flag = 0;
    tc::mbar_init(&sh.bar_s0, 1);
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
  const uint32_t tmS = tmem;                // S0^T bf16 (64 columns); then X^T high | low
  const uint32_t tmW = tmem + 64;           // W^T: [K part | Q part], 2BM columns
  const uint32_t tmG = tmem + 64 + 2 * BM;  // G (rows on lanes kG0..); then O2^T
  const uint32_t lane_off = (uint32_t)(warp * 32) << 16;

  auto issue_s0 = [&](int item, int s) {
    const float* src = p.state_pool + ((size_t)s * p.Hv + item % p.Hv) * kDpD * kDpD;
    tc::mbar_expect_tx(&sh.bar_s0, C::kS0);
    tc::bulk_load(S0s, src, C::kS0, &sh.bar_s0);
  };
  auto issue_kq = [&](int item) {
    const int r = item / p.Hv, h = (item % p.Hv) / (p.Hv / p.Hk);
    tc::mbar_expect_tx(&sh.bar_kq, C::kKQ);
#pragma unroll
    for (int c = 0; c < 2; ++c) {
      tc::tma_load_4d(KQs + c * (2 * BM * 128), &maps.k, &sh.bar_kq, c * 64, h, 0, r);
      tc::tma_load_4d(KQs + c * (2 * BM * 128) + BM * 128, &maps.q, &sh.bar_kq, c * 64, h, 0, r);
    }
  };
  auto issue_v = [&](int item) {
    const int r = item / p.Hv, j = item % p.Hv;
    tc::mbar_expect_tx(&sh.bar_v, C::kV);
    tc::tma_load_4d(Vs, &maps.v, &sh.bar_v, 0, j, 0, r);
    tc::tma_load_4d(Vs + BM * 128, &maps.v, &sh.bar_v, 64, j, 0, r);
  };
  // warp 0 holds the gates of the item it processes next, loaded one item ahead
  float gq = 0.f, bq = 0.f;
  auto load_gates = [&](int item) {
    const size_t gb = (size_t)(item / p.Hv) * B * p.Hv + item % p.Hv;
    gq = lane < B ? p.log_decay[gb + (size_t)lane * p.Hv] : 0.f;
    bq = lane < B ? p.beta[gb + (size_t)lane * p.Hv] : 0.f;
  };
  auto cand_slot = [&](int c) { return c < total ? p.state_slot[c / p.Hv] : -1; };

  // the issuing thread's record of what is in flight (and the parity its barrier
  // phase completes with), for a clean exit after a timeout
  bool s0_out = false, kq_out = false, v_out = false, mma_out = false;
  uint32_t s0_par = 0, kq_par = 0, v_par = 0;
  if (tid == kIssuer) {
    tc::prefetch_tmap(&maps.k);
    tc::prefetch_tmap(&maps.q);
    tc::prefetch_tmap(&maps.v);
    issue_s0(it, slot);
    issue_kq(it);
    issue_v(it);
    s0_out = kq_out = v_out = true;
  }
  if (warp == 0) load_gates(it);
  int cand = it + gridDim.x;
  int cs = cand_slot(cand);
  bool bad = false;     // this thread gave up on a wait
  uint32_t ph = 0;      // parity of the item's loads
  uint32_t ph_mma = 0;  // parity of the next MMA completion (two per item)
  const uint32_t idG = tc::idesc_bf16(128, Bp, false, false);
  const uint32_t idW = tc::idesc_bf16(128, 2 * BM, false, false);
  const uint32_t idO = tc::idesc_bf16(128, Bp, false, false);

#pragma unroll 1
  while (true) {
    const int r = it / p.Hv, j = it % p.Hv;
    // the block's gates: gamma = inclusive prefix sum of the log-gates
    if (warp == 0) {
      float g = gq;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const float a = __shfl_up_sync(0xffffffffu, g, o);
        if (lane >= o) g += a;
      }
      const float g2 = g * 1.4426950408889634f;
      const float gB2 = __shfl_sync(0xffffffffu, g2, B - 1);
      sh.gam2[lane] = g2;
      sh.Gam[lane] = expf(g);
      sh.beta[lane] = bq;
      sh.eB[lane] = lane < B ? tc::ex2(gB2 - g2) : 0.f;
    }
    // the next item: the candidate when its slot is valid, else the first
    // valid one after it (bad ones flagged on the way)
    int it_next = -1, slot_next = 0;
    if (cand < total) {
      if (cs >= 0 && cs < p.nslots) {
        it_next = cand;
        slot_next = cs;
      } else {
        it_next = dp_next(p, cand, total, slot_next);
      }
    }
    if (it_next >= 0) {
      if (warp == 0) load_gates(it_next);
      cand = it_next + gridDim.x;
      cs = cand_slot(cand);
    }

    // Waits on a copy or an MMA are per thread: a thread that gives up
    // carries `bad` to the next CTA barrier, where the whole CTA stops.
    bad |= !tc::mbar_wait(&sh.bar_s0, ph, &sh.abort_flag);
    if (tid == kIssuer) s0_out = false;
    // S0^T (column c = tid of S0) into tensor memory as bf16 pairs
#pragma unroll 1
    for (int i0 = 0; i0 < kDpD; i0 += 32) {
      uint32_t w[16];
#pragma unroll
      for (int e = 0; e < 16; ++e)
        w[e] = dp_pack(S0s[(i0 + 2 * e) * kDpD + tid], S0s[(i0 + 2 * e + 1) * kDpD + tid]);
      tc::tmem_st16(tmS + lane_off + i0 / 2, w);
    }
    tc::tmem_st_wait();
    tc::fence_before_sync();
    if (__syncthreads_or(bad)) break;  // S0^T complete, the state buffer read
    if (tid == kIssuer) {
      bad |= !tc::mbar_wait(&sh.bar_kq, ph, &sh.abort_flag);
      kq_out = false;
      tc::fence_after_sync();
      // the Gram first, committed on its own: A^T and M2 are built while the
      // state products run
#pragma unroll
      for (int kk = 0; kk < kDpD / 16; ++kk) {
        const uint8_t* kc = KQs + (kk >> 2) * (2 * BM * 128) + (kk & 3) * 32;
        tc::mma_bf16_ss(tmG, tc::sdesc_sw128(tc::smem_u32(kc - kG0 * 128), 16, 1024),
                        tc::sdesc_sw128(tc::smem_u32(kc), 16, 1024), idG, kk > 0);  // G = [K;Q] K^T
      }
      tc::mma_commit(&sh.bar_g);
#pragma unroll
      for (int kk = 0; kk < kDpD / 16; ++kk) {
        const uint8_t* kc = KQs + (kk >> 2) * (2 * BM * 128) + (kk & 3) * 32;
        tc::mma_bf16_ts(tmW, tmS + kk * 8, tc::sdesc_sw128(tc::smem_u32(kc), 16, 1024), idW,
                        kk > 0);  // W^T = S0^T [K;Q]^T
      }
      tc::mma_commit(&sh.bar_mma);
      mma_out = true;
      // the state buffer is free: the next item's state streams in during
      // this item's products, solve and readout (issued after the MMAs, off
      // their path)
      if (it_next >= 0) {
        issue_s0(it_next, slot_next);
        s0_out = true;
        s0_par = ph ^ 1u;
      }
    }
    bad |= !tc::mbar_wait(&sh.bar_v, ph, &sh.abort_flag);
    if (tid == kIssuer) v_out = false;
    // this column of the values as bf16 pairs (rows past B arrive as zeros)
    uint32_t vpk[BM / 2];
    {
      const uint8_t* vb = Vs + (tid >> 6) * (BM * 128) + (tid & 63) * 2;
#pragma unroll
      for (int t2 = 0; t2 < BM / 2; ++t2)
        vpk[t2] = (uint32_t)*reinterpret_cast<const unsigned short*>(vb + (2 * t2) * 128) |
                  ((uint32_t)*reinterpret_cast<const unsigned short*>(vb + (2 * t2 + 1) * 128)
                   << 16);
    }
    // A^T (key rows of G) and M2 (query rows), from the lanes that hold G,
    // once the Gram is in
    if (warp >= kG0 / 32) {
      bad |= !tc::mbar_wait(&sh.bar_g, ph, &sh.abort_flag);
      tc::fence_after_sync();
      uint32_t gr[BM];
#pragma unroll
      for (int c0 = 0; c0 < BM; c0 += 16)
        tc::tmem_ld16(tmG + lane_off + c0, *reinterpret_cast<uint32_t(*)[16]>(&gr[c0]));
      tc::tmem_ld_wait();
      const int row = tid - kG0;
      // the gate factors go to registers first (16-byte loads) and every
      // exponential is taken unconditionally, the masks applied as selects:
      // a branch per element would serialise the load / exponential chains
      if (row >= 0 && row < BM) {
        const int t = row;
        float g2r[BM];
#pragma unroll
        for (int i4 = 0; i4 < BM / 4; ++i4) {
          const float4 q = *reinterpret_cast<const float4*>(&sh.gam2[4 * i4]);
          g2r[4 * i4] = q.x, g2r[4 * i4 + 1] = q.y, g2r[4 * i4 + 2] = q.z, g2r[4 * i4 + 3] = q.w;
        }
        const float bt = sh.beta[t], gt = sh.gam2[t];
        const bool live = t < B;
#pragma unroll
        for (int i = 0; i < BM; ++i) {
          const float a = bt * tc::ex2(gt - g2r[i]) * __uint_as_float(gr[i]);
          AT[i * kATs + t] = (live && i < t) ? a : 0.f;
        }
      } else if (row >= BM) {
        const int l = row - BM;
        float er[BM];
#pragma unroll
        for (int i4 = 0; i4 < BM / 4; ++i4) {
          const float4 q = *reinterpret_cast<const float4*>(&sh.eB[4 * i4]);
          er[4 * i4] = q.x, er[4 * i4 + 1] = q.y, er[4 * i4 + 2] = q.z, er[4 * i4 + 3] = q.w;
        }
#pragma unroll
        for (int i4 = 0; i4 < BM / 4; ++i4) {
          float v[4];
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const int i = 4 * i4 + e;
            const float m = er[i] * __uint_as_float(gr[i]);
            v[e] = (i < B && l < B) ? m : 0.f;
          }
          *reinterpret_cast<float4*>(M2f + l * kATs + 4 * i4) = make_float4(v[0], v[1], v[2], v[3]);
        }
      }
      // T's diagonal blocks from this warp's A^T rows (A's columns), a column
      // of one block per lane
      __syncwarp();
      if (row >= 0 && row < BM) dp_diag_inverse<kATs>(AT, Tf, row >> 4, row & 15);
    }
    bad |= !tc::mbar_wait(&sh.bar_mma, ph_mma, &sh.abort_flag);
    ph_mma ^= 1u;
    tc::fence_after_sync();
    if (tid == kIssuer) {
      mma_out = false;
      if (it_next >= 0) {  // the first MMAs, the only readers of [K;Q], are done
        issue_kq(it_next);
        kq_out = true;
        kq_par = ph ^ 1u;
      }
    }
    // X = diag(beta) (V - diag(Gam) K S0) for this column
    float x[BM];
#pragma unroll
    for (int c0 = 0; c0 < BM; c0 += 16) {
      uint32_t w[16];
      tc::tmem_ld16(tmW + lane_off + c0, w);
      tc::tmem_ld_wait();
#pragma unroll
      for (int e4 = 0; e4 < 4; ++e4) {
        const float4 b4 = *reinterpret_cast<const float4*>(&sh.beta[c0 + 4 * e4]);
        const float4 g4 = *reinterpret_cast<const float4*>(&sh.Gam[c0 + 4 * e4]);
        const float bb[4] = {b4.x, b4.y, b4.z, b4.w}, gg[4] = {g4.x, g4.y, g4.z, g4.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int t = c0 + 4 * e4 + e;
          const uint32_t vp = vpk[t / 2];
          const float vt = __uint_as_float((t & 1) ? (vp & 0xffff0000u) : (vp << 16));
          x[t] = bb[e] * (vt - gg[e] * __uint_as_float(w[4 * e4 + e]));
        }
      }
    }
    // X^T into tensor memory as bf16 high and low parts, over S0^T (read by
    // the first MMAs): high parts in columns 0 .. BM/2 - 1, low parts after
    {
      uint32_t hi[BM / 2], lo[BM / 2];
#pragma unroll
      for (int e = 0; e < BM / 2; ++e) dp_split(x[2 * e], x[2 * e + 1], hi[e], lo[e]);
      if constexpr (BM == 32) {
        tc::tmem_st16(tmS + lane_off, hi);
        tc::tmem_st16(tmS + lane_off + 16, lo);
      } else {
        uint32_t w[16];
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          w[e] = hi[e];
          w[8 + e] = lo[e];
        }
        tc::tmem_st16(tmS + lane_off, w);
      }
      tc::tmem_st_wait();
    }
    // the readout's scale, read here: the gates' buffer is rewritten for the
    // next item once every thread is past the barrier before the second MMA
    const float sG = p.scale * sh.Gam[B - 1];
    tc::fence_before_sync();
    if (__syncthreads_or(bad)) break;  // A^T, M2, T's diagonal and X^T published; the values, W^T's key part and G read
    if (tid == kIssuer && it_next >= 0) {
      tc::fence_async_smem();
      issue_v(it_next);
      v_out = true;
      v_par = ph ^ 1u;
    }

    // N = M2 T with T = (I + A)^{-1} from its diagonal blocks (rows and
    // columns past B: M2 and A are zero there, T the identity).  Four lanes per
    // row l of N, columns 4q .. 4q + 3 of each 16-column half; a row's values
    // travel between its lanes by shuffles.
    {
      const int l = tid >> 2, q = tid & 3, src0 = lane & ~3;
      if (l < BM) {  // every lane of a warp alike
        const float* m2r = M2f + l * kATs;
        float w[16];  // the left factor of N0: Y = M2_0 - N1 A10 (BM = 32) or M2 (BM = 16)
        float n1[4] = {0.f, 0.f, 0.f, 0.f};
        if constexpr (BM == 32) {
          float m1[16];
#pragma unroll
          for (int i4 = 0; i4 < 4; ++i4) {
            const float4 v4 = *reinterpret_cast<const float4*>(m2r + 16 + 4 * i4);
            m1[4 * i4] = v4.x, m1[4 * i4 + 1] = v4.y, m1[4 * i4 + 2] = v4.z, m1[4 * i4 + 3] = v4.w;
          }
#pragma unroll
          for (int i = 0; i < 16; ++i) {  // N1 = M2_1 T11
            const float4 t4 = *reinterpret_cast<const float4*>(Tf + (16 + i) * kATs + 16 + 4 * q);
            n1[0] = fmaf(m1[i], t4.x, n1[0]);
            n1[1] = fmaf(m1[i], t4.y, n1[1]);
            n1[2] = fmaf(m1[i], t4.z, n1[2]);
            n1[3] = fmaf(m1[i], t4.w, n1[3]);
          }
          float v[16];  // N1's row l
#pragma unroll
          for (int i = 0; i < 16; ++i) v[i] = __shfl_sync(0xffffffffu, n1[i & 3], src0 + (i >> 2));
          const float4 m0 = *reinterpret_cast<const float4*>(m2r + 4 * q);
          float y[4] = {m0.x, m0.y, m0.z, m0.w};
#pragma unroll
          for (int e = 0; e < 4; ++e) {  // Y = M2_0 - N1 A10, A[16 + i][4q + e] = A^T row 4q + e
            const float* ar = AT + (4 * q + e) * kATs + 16;
#pragma unroll
            for (int i4 = 0; i4 < 4; ++i4) {
              const float4 a4 = *reinterpret_cast<const float4*>(ar + 4 * i4);
              y[e] = fmaf(-a4.x, v[4 * i4], y[e]);
              y[e] = fmaf(-a4.y, v[4 * i4 + 1], y[e]);
              y[e] = fmaf(-a4.z, v[4 * i4 + 2], y[e]);
              y[e] = fmaf(-a4.w, v[4 * i4 + 3], y[e]);
            }
          }
#pragma unroll
          for (int i = 0; i < 16; ++i) w[i] = __shfl_sync(0xffffffffu, y[i & 3], src0 + (i >> 2));
        } else {
#pragma unroll
          for (int i4 = 0; i4 < 4; ++i4) {
            const float4 v4 = *reinterpret_cast<const float4*>(m2r + 4 * i4);
            w[4 * i4] = v4.x, w[4 * i4 + 1] = v4.y, w[4 * i4 + 2] = v4.z, w[4 * i4 + 3] = v4.w;
          }
        }
        float n0[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int i = 0; i < 16; ++i) {  // N0 = (.) T00
          const float4 t4 = *reinterpret_cast<const float4*>(Tf + i * kATs + 4 * q);
          n0[0] = fmaf(w[i], t4.x, n0[0]);
          n0[1] = fmaf(w[i], t4.y, n0[1]);
          n0[2] = fmaf(w[i], t4.z, n0[2]);
          n0[3] = fmaf(w[i], t4.w, n0[3]);
        }
        // row l of N as bf16 high and low parts, K-major SW128 (columns c ..
        // c + 3 in the 16-byte unit c / 8)
        auto put4 = [&](int c, const float (&v)[4]) {
          uint32_t h0, l0, h1, l1;
          dp_split(v[0], v[1], h0, l0);
          dp_split(v[2], v[3], h1, l1);
          const int off = l * 128 + ((((c >> 3) ^ (l & 7))) << 4) + (c & 7) * 2;
          *reinterpret_cast<uint2*>(Nbs + off) = make_uint2(h0, h1);
          *reinterpret_cast<uint2*>(Nbs + BM * 128 + off) = make_uint2(l0, l1);
        };
        put4(4 * q, n0);
        if constexpr (BM == 32) put4(16 + 4 * q, n1);
        tc::fence_async_smem();  // N is the second MMA's operand
      }
    }
    tc::fence_before_sync();
    if (__syncthreads_or(bad)) break;  // N complete; A^T, M2 and T read
    if (tid == kIssuer) {
      tc::fence_after_sync();
#pragma unroll
      for (int kk = 0; kk < BM / 16; ++kk) {  // O2^T = X^T N^T, over G
        const uint64_t nh = tc::sdesc_sw128(tc::smem_u32(Nbs + kk * 32), 16, 1024);
        const uint64_t nl = tc::sdesc_sw128(tc::smem_u32(Nbs + BM * 128 + kk * 32), 16, 1024);
        tc::mma_bf16_ts(tmG, tmS + kk * 8, nh, idO, kk > 0);
        tc::mma_bf16_ts(tmG, tmS + kk * 8, nl, idO, 1);
        tc::mma_bf16_ts(tmG, tmS + BM / 2 + kk * 8, nh, idO, 1);
      }
      tc::mma_commit(&sh.bar_mma);
      mma_out = true;
    }
    bad |= !tc::mbar_wait(&sh.bar_mma, ph_mma, &sh.abort_flag);
    ph_mma ^= 1u;
    tc::fence_after_sync();
    if (tid == kIssuer) mma_out = false;
    // out[l][c] = s (Gam_{B-1} W^T[c][BM + l] + O2^T[c][l]); adjacent lanes
    // swap one value so that each stores a bf16 pair of two columns
    {
      uint32_t o2[BM], wq[BM];
#pragma unroll
      for (int c0 = 0; c0 < BM; c0 += 16) {
        tc::tmem_ld16(tmG + lane_off + c0, *reinterpret_cast<uint32_t(*)[16]>(&o2[c0]));
        tc::tmem_ld16(tmW + lane_off + BM + c0, *reinterpret_cast<uint32_t(*)[16]>(&wq[c0]));
      }
      tc::tmem_ld_wait();
      const bool odd = lane & 1;
      __nv_bfloat16* out = static_cast<__nv_bfloat16*>(p.out_blockend) +
                           ((size_t)r * B * p.Hv + j) * kDpD + (tid & ~1);
#pragma unroll
      for (int l = 0; l < BM; l += 2) {
        const float a = fmaf(sG, __uint_as_float(wq[l]), p.scale * __uint_as_float(o2[l]));
        const float b = fmaf(sG, __uint_as_float(wq[l + 1]), p.scale * __uint_as_float(o2[l + 1]));
        const float recv = __shfl_xor_sync(0xffffffffu, odd ? a : b, 1);
        const int row = odd ? l + 1 : l;
        if (row < B)
          *reinterpret_cast<uint32_t*>(out + (size_t)row * p.Hv * kDpD) =
              odd ? dp_pack(recv, b) : dp_pack(a, recv);
      }
    }
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
  __syncthreads();

  // after a timeout: let the copies and MMAs in flight land before the
  // shared and tensor memory are given up (bounded waits)
  if (tid == kIssuer && bad) {
    if (s0_out) tc::mbar_wait(&sh.bar_s0, s0_par, nullptr, 100000000ull);
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

PFN_cuTensorMapEncodeTiled_v12000 dp_encode_fn() {
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
// rows, 1); rows past B read as zero
bool dp_act_map(CUtensorMap* m, const void* x, int H, int B, int R, int rows, bool swizzle) {
  auto fn = dp_encode_fn();
  if (!fn) return false;
  cuuint64_t gd[4] = {(cuuint64_t)kDpD, (cuuint64_t)H, (cuuint64_t)B, (cuuint64_t)R};
  cuuint64_t gs[3] = {(cuuint64_t)kDpD * 2, (cuuint64_t)H * kDpD * 2,
                      (cuuint64_t)B * H * kDpD * 2};
  cuuint32_t bx[4] = {64, 1, (cuuint32_t)rows, 1};
  cuuint32_t es[4] = {1, 1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(x), gd, gs, bx, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE,
            swizzle ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_NONE,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) ==
         CUDA_SUCCESS;
}

template <int BM>
cudaError_t launch_dp(const GdrParams& p, cudaStream_t stream) {
  DpMaps maps;
  if (!dp_act_map(&maps.k, p.k, p.Hk, p.B, p.R, BM, true) ||
      !dp_act_map(&maps.q, p.q, p.Hk, p.B, p.R, BM, true) ||
      !dp_act_map(&maps.v, p.v, p.Hv, p.B, p.R, BM, false))
    return cudaErrorInvalidValue;
  const int smem = DpCfg<BM>::kSmem + 1024;
  cudaError_t e = cudaFuncSetAttribute(gdr_denoise_persist_kernel<BM>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  int dev = 0, sms = kNumSMs;
  if (cudaGetDevice(&dev) == cudaSuccess)
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const long items = (long)p.R * p.Hv;
  const int grid = (int)(items < 2L * sms ? items : 2L * sms);
  gdr_denoise_persist_kernel<BM><<<grid, kDpThreads, smem, stream>>>(maps, p);
  note_launches(1);
  return cudaGetLastError();
}

}  // namespace

bool gdr_denoise_persist_supported(int B, int dk, int dv) {
  return B >= 1 && B <= 32 && dk == kDpD && dv == kDpD;
}

cudaError_t launch_gdr_denoise_persist(const GdrParams& p, cudaStream_t stream) {
  if (p.R == 0) return cudaSuccess;
  return p.B <= 16 ? launch_dp<16>(p, stream) : launch_dp<32>(p, stream);
}

}  // namespace flare
