// State commit at the accepted length on tcgen05 tensor cores: bf16
// activations, d_k = d_v = 128, B <= 64, no token-causal outputs.
//
// For one (request r, value head j) with q/k head h, accepted length n > 0 and
// frozen state S0, the committed state is the chunkwise form of the block's
// first n tokens (appendix "Chunk-corrected values", Eq. chunk-state and
// Eq. f-blk; the state-update pass of the serving appendix commits it):
//
//   gamma_t = g_0 + ... + g_t,  Gam_t = exp(gamma_t)
//   A[t][i] = beta_t exp(gamma_t - gamma_i) (k_t . k_i),   i < t < n
//   X_t     = beta_t (v_t - Gam_t S0^T k_t)
//   (I + A) delta = X
//   S^(n)   = Gam_{n-1} S0 + sum_{i<n} exp(gamma_{n-1} - gamma_i) k_i delta_i^T
//
// Everything is computed transposed, value column c on tensor-memory lane c
// (column c of the state evolves on its own, the update acting from the left),
// so thread c owns column c from the state's load to its store:
//
//   MMA 1  G   = K K^T             M=128 (rows t), N=Bp, K=128       bf16
//   MMA 2  W^T = S0^T K^T          M=128 (c),      N=Bp, K=128       S0^T = hi + lo
//   solve  (I + A) delta = X       fp32, thread c on column c, right-looking
//   MMA 3  D  += delta'^T K        M=128 (c),      N=128, K=16 ceil(n/16)   delta' = hi + lo
//
// with D = S^(n)^T accumulating on top of Gam_{n-1} S0^T and delta'_i =
// exp(gamma_{n-1} - gamma_i) delta_i (zero for i >= n).  The keys are bf16, so
// they are exact tensor-core operands; the state and the deltas are fp32 and
// enter as two bf16 terms, x = hi + lo with hi = bf16(x), lo = bf16(x - hi),
// which leaves a relative error of at most 2^-18 per product term, far inside
// what the committed state's fp32-grade accuracy needs.  The Gam_{n-1} S0
// term is formed in fp32 from the loaded state itself.
//
// Persistent CTAs, two per SM (97 KiB of shared memory, 256 tensor-memory
// columns each), 128 threads, each walking the (request, value head) items
// blockIdx.x, blockIdx.x + gridDim.x, ...  The state (64 KiB) arrives by one
// bulk copy, the keys and values by TMA (64-row key boxes with 128-byte
// swizzle, rows past B zero-filled); the next item's state is requested as
// soon as this item's has been read out of shared memory (before its solve),
// its keys and values once this item's update has run, its gates and its
// slot one item ahead into registers, so no global-memory latency sits on a
// CTA's chain.  The committed state is stored straight from tensor memory
// (each warp store covers 128 contiguous bytes of a state row).  Items with
// n = 0 leave the slot untouched; a bad slot or accepted length is flagged in
// the device status word and the item skipped.  Every wait is bounded: on a
// timeout the CTA sets FLARE_DEV_WAIT_TIMEOUT, waits (bounded) for its copies
// and MMAs in flight, frees its tensor memory and exits.
#include <cudaTypedefs.h>

#include "common.cuh"
#include "kernels.h"
#include "tc.cuh"

namespace flare {

namespace {

constexpr int kCtThreads = 128;
constexpr int kCtD = 128;  // d_k = d_v

template <int BM>
struct CtCfg {
  static constexpr int kK = 2 * 64 * 128;          // keys: 2 chunks of 64 rows x 128 B (SW128)
  static constexpr int kS0 = kCtD * kCtD * 4;      // S0 fp32 [i][c]
  static constexpr int kATs = BM + 4;              // row stride of A^T (floats)
  static constexpr int kAT = BM * kATs * 4;        // A^T[i][t] = A[t][i]
  static constexpr int kV = 2 * BM * 128;          // values: 2 chunks of BM rows x 128 B
  // the values, once read into registers, make room for A^T
  static constexpr int kR = kAT > kV ? kAT : kV;
  // tensor-memory columns of each bf16 part of delta'^T (whole 16-column stores)
  static constexpr int kDP = BM / 2 < 16 ? 16 : BM / 2;
  static constexpr int kSmem = kS0 + kK + kR;  // state, keys, values / A^T
};

struct CtMaps {
  CUtensorMap k;  // keys   (128, Hk, B, R) box (64, 1, 64, 1), 128-byte swizzle
  CUtensorMap v;  // values (128, Hv, B, R) box (64, 1, BM, 1), no swizzle
};

struct alignas(16) CtShared {
  uint64_t bar_s0, bar_k, bar_mma;
  uint32_t tmem_base;
  int abort_flag;
  // 16-byte aligned: read as float4 broadcasts
  alignas(16) float gam2[64];  // gamma_t log2(e)
  alignas(16) float Gam[64];   // exp(gamma_t)
  alignas(16) float beta[64];
  alignas(16) float dsc[64];   // exp(gamma_{n-1} - gamma_t) for t < n, else 0 (delta' factor)
};

__device__ __forceinline__ bool ct_wait(uint64_t* bar, uint32_t parity, CtShared& sh,
                                        int32_t* status) {
  const bool ok = tc::mbar_wait(bar, parity, &sh.abort_flag);
  const bool all = __syncthreads_and(ok);
  if (!all && threadIdx.x == 0 && !sh.abort_flag) {
    sh.abort_flag = 1;
    flag(status, FLARE_DEV_WAIT_TIMEOUT);
  }
  return all;
}

// The next item at or after `it` (stride gridDim.x) with a valid slot and
// accepted length n > 0; items with a bad slot or length are flagged and
// skipped.  Called by every thread with the same arguments.
__device__ __forceinline__ int ct_next(const GdrParams& p, int it, int total, int& slot, int& n) {
  for (; it < total; it += gridDim.x) {
    const int r = it / p.Hv;
    const int s = p.state_slot[r];
    if (s < 0 || s >= p.nslots) {
      if (threadIdx.x == 0) flag(p.dev_status, FLARE_DEV_BAD_SLOT);
      continue;
    }
    const int a = p.accept_len ? p.accept_len[r] : p.B;
    if (a < 0 || a > p.B) {
      if (threadIdx.x == 0) flag(p.dev_status, FLARE_DEV_BAD_ACCEPT_LEN);
      continue;
    }
    if (a == 0) continue;
    slot = s;
    n = a;
    return it;
  }
  return -1;
}

__device__ __forceinline__ uint32_t bf2_bits(__nv_bfloat162 b) {
  return *reinterpret_cast<uint32_t*>(&b);
}

// x = hi + lo for the pair (a, b): hi = bf16(x), lo = bf16(x - hi)
__device__ __forceinline__ void split_pair(float a, float b, uint32_t& hi, uint32_t& lo) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
  const float2 hf = __bfloat1622float2(h);
  hi = bf2_bits(h);
  lo = bf2_bits(__floats2bfloat162_rn(a - hf.x, b - hf.y));
}

}  // namespace

template <int BM>
__global__ void __launch_bounds__(kCtThreads, 2)
    gdr_commit_tc_kernel(const __grid_constant__ CtMaps maps, GdrParams p) {
  using C = CtCfg<BM>;
  constexpr int kATs = C::kATs;
  extern __shared__ uint8_t smem_raw[];
  __shared__ CtShared sh;
  uint8_t* base = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  float* S0s = reinterpret_cast<float*>(base);
  uint8_t* Ks = base + C::kS0;
  uint8_t* Rs = Ks + C::kK;  // the values, then A^T
  float* AT = reinterpret_cast<float*>(Rs);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int total = p.R * p.Hv;
  const int B = p.B;
  const int Bp = (B + 15) & ~15;

  int slot = 0, n = 0;
  int it = ct_next(p, blockIdx.x, total, slot, n);
  if (it < 0) return;  // the same answer on every thread

  if (tid == 0) {
    sh.abort_flag = 0;
    tc::mbar_init(&sh.bar_s0, 1);
    tc::mbar_init(&sh.bar_k, 1);
    tc::mbar_init(&sh.bar_mma, 1);
    tc::fence_mbar_init();
  }
  if (warp == 0) tc::tmem_alloc(&sh.tmem_base, 256);
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = sh.tmem_base;
  const uint32_t tmS = tmem;             // S0^T hi [0,64) and lo [64,128); then D
  const uint32_t tmW = tmem + 128;       // W^T; then delta'^T hi [0,kDP) and lo [kDP,2kDP)
  // G: row t on lane kG0 + t, the top BM lanes (warps 2-3), so that warp 0,
  // which also scans the gates and issues the copies and MMAs, is not the
  // one building A^T
  constexpr int kG0 = 128 - BM;
  const uint32_t tmG = tmem + 128 + BM;
  const uint32_t lane_off = (uint32_t)(warp * 32) << 16;

  auto state_of = [&](int item, int s) {
    return p.state_pool + ((size_t)s * p.Hv + item % p.Hv) * kCtD * kCtD;
  };
  auto issue_s0 = [&](int item, int s) {
    const float* src = state_of(item, s);
    tc::mbar_expect_tx(&sh.bar_s0, C::kS0);
#pragma unroll
    for (int q = 0; q < 4; ++q)
      tc::bulk_load(S0s + q * (kCtD * kCtD / 4), src + q * (kCtD * kCtD / 4), C::kS0 / 4,
                    &sh.bar_s0);
  };
  auto issue_kv = [&](int item) {
    const int r = item / p.Hv, j = item % p.Hv, h = j / (p.Hv / p.Hk);
    tc::mbar_expect_tx(&sh.bar_k, C::kK + C::kV);
    tc::tma_load_4d(Ks, &maps.k, &sh.bar_k, 0, h, 0, r);
    tc::tma_load_4d(Ks + 64 * 128, &maps.k, &sh.bar_k, 64, h, 0, r);
    tc::tma_load_4d(Rs, &maps.v, &sh.bar_k, 0, j, 0, r);
    tc::tma_load_4d(Rs + BM * 128, &maps.v, &sh.bar_k, 64, j, 0, r);
  };
  // warp 0 holds the gates of the item it will process next, loaded one item ahead
  float gq0 = 0.f, gq1 = 0.f, bq0 = 0.f, bq1 = 0.f;
  auto load_gates = [&](int item) {
    const size_t gb = (size_t)(item / p.Hv) * B * p.Hv + item % p.Hv;
    gq0 = lane < B ? p.log_decay[gb + (size_t)lane * p.Hv] : 0.f;
    gq1 = lane + 32 < B ? p.log_decay[gb + (size_t)(lane + 32) * p.Hv] : 0.f;
    bq0 = lane < B ? p.beta[gb + (size_t)lane * p.Hv] : 0.f;
    bq1 = lane + 32 < B ? p.beta[gb + (size_t)(lane + 32) * p.Hv] : 0.f;
  };
  // slot and accepted length of the candidate after the next item, one item ahead
  auto cand_slot = [&](int c) { return c < total ? p.state_slot[c / p.Hv] : -1; };
  auto cand_len = [&](int c) {
    return c < total ? (p.accept_len ? p.accept_len[c / p.Hv] : B) : 0;
  };

  // thread 0's record of what is in flight (and the parity its barrier
  // phase completes with), for a clean exit after a timeout
  bool s0_out = false, k_out = false, mma_out = false;
  uint32_t s0_par = 0, k_par = 0;
  if (tid == 0) {
    tc::prefetch_tmap(&maps.k);
    tc::prefetch_tmap(&maps.v);
    issue_s0(it, slot);
    issue_kv(it);
    s0_out = k_out = true;
  }
  if (warp == 0) load_gates(it);
  int cand = it + gridDim.x;
  int cs = cand_slot(cand), ca = cand_len(cand);
  uint32_t ph = 0;      // parity of the item's state and key/value loads
  uint32_t ph_mma = 0;  // parity of the next MMA completion (two per item)
  const uint32_t idN = tc::idesc_bf16(128, Bp, false, false);
  const uint32_t idU = tc::idesc_bf16(128, 128, false, true);

#pragma unroll 1
  while (true) {
    // the block's gates: gamma = inclusive prefix sum of the log-gates
    if (warp == 0) {
      float g0 = gq0, g1 = gq1;
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
      const float g20 = g0 * 1.4426950408889634f, g21 = g1 * 1.4426950408889634f;
      // gamma_{n-1}: lane (n - 1) % 32 of the half holding it
      const float gn0 = __shfl_sync(0xffffffffu, g20, (n - 1) & 31);
      const float gn1 = __shfl_sync(0xffffffffu, g21, (n - 1) & 31);
      const float gn2 = n > 32 ? gn1 : gn0;
      sh.gam2[lane] = g20;
      sh.gam2[lane + 32] = g21;
      sh.Gam[lane] = expf(g0);
      sh.Gam[lane + 32] = expf(g1);
      sh.beta[lane] = bq0;
      sh.beta[lane + 32] = bq1;
      sh.dsc[lane] = lane < n ? tc::ex2(gn2 - g20) : 0.f;
      sh.dsc[lane + 32] = lane + 32 < n ? tc::ex2(gn2 - g21) : 0.f;
    }
    // the next item: the candidate when it is valid and has n > 0, else the
    // first such item after it (bad ones flagged on the way)
    int it_next = -1, slot_next = 0, n_next = 0;
    if (cand < total) {
      if (cs >= 0 && cs < p.nslots && ca > 0 && ca <= B) {
        it_next = cand;
        slot_next = cs;
        n_next = ca;
      } else {
        it_next = ct_next(p, cand, total, slot_next, n_next);
      }
    }
    if (it_next >= 0) {
      if (warp == 0) load_gates(it_next);
      cand = it_next + gridDim.x;
      cs = cand_slot(cand);
      ca = cand_len(cand);
    }

    if (!ct_wait(&sh.bar_s0, ph, sh, p.dev_status)) break;
    if (tid == 0) s0_out = false;
    // S0^T (column c = tid of S0) into tensor memory as bf16 hi and lo parts
#pragma unroll 1
    for (int i0 = 0; i0 < kCtD; i0 += 32) {
      uint32_t hi[16], lo[16];
#pragma unroll
      for (int e = 0; e < 16; ++e)
        split_pair(S0s[(i0 + 2 * e) * kCtD + tid], S0s[(i0 + 2 * e + 1) * kCtD + tid], hi[e],
                   lo[e]);
      tc::tmem_st16(tmS + lane_off + i0 / 2, hi);
      tc::tmem_st16(tmS + lane_off + 64 + i0 / 2, lo);
    }
    tc::tmem_st_wait();
    tc::fence_before_sync();
    if (!ct_wait(&sh.bar_k, ph, sh, p.dev_status)) break;  // also orders the stores above
    if (tid == 0) {
      k_out = false;
      tc::fence_after_sync();
#pragma unroll
      for (int kk = 0; kk < kCtD / 16; ++kk) {
        const uint8_t* kc = Ks + (kk >> 2) * (64 * 128) + (kk & 3) * 32;
        const uint64_t kd = tc::sdesc_sw128(tc::smem_u32(kc), 16, 1024);
        // A operand rows kG0.. are the keys; the rows before read the bytes
        // ahead of the chunk (the state buffer, then the first chunk), which
        // only reach lanes nobody reads
        const uint64_t kg = tc::sdesc_sw128(tc::smem_u32(kc - kG0 * 128), 16, 1024);
        tc::mma_bf16_ss(tmG, kg, kd, idN, kk > 0);                // G = K K^T
        tc::mma_bf16_ts(tmW, tmS + kk * 8, kd, idN, kk > 0);      // W^T = S0hi^T K^T
        tc::mma_bf16_ts(tmW, tmS + 64 + kk * 8, kd, idN, 1u);     //     + S0lo^T K^T
      }
      tc::mma_commit(&sh.bar_mma);
      mma_out = true;
    }
    // this thread's value column (rows past B arrive as zeros)
    uint32_t vraw[BM];
    {
      const uint8_t* vb = Rs + (tid >> 6) * (BM * 128) + (tid & 63) * 2;
#pragma unroll
      for (int t = 0; t < BM; ++t) vraw[t] = *reinterpret_cast<const unsigned short*>(vb + t * 128);
    }
    if (!ct_wait(&sh.bar_mma, ph_mma, sh, p.dev_status)) break;  // the values are read
    ph_mma ^= 1u;
    if (tid == 0) mma_out = false;
    tc::fence_after_sync();

    // the accumulator starts at Gam_{n-1} S0^T (fp32, from the loaded state)
    {
      const float Gn = sh.Gam[n - 1];
#pragma unroll 2
      for (int i0 = 0; i0 < kCtD; i0 += 16) {
        uint32_t d[16];
#pragma unroll
        for (int e = 0; e < 16; ++e) d[e] = __float_as_uint(Gn * S0s[(i0 + e) * kCtD + tid]);
        tc::tmem_st16(tmS + lane_off + i0, d);
      }
    }
    // A^T from the Gram rows t < BM (the warps holding those lanes); rows of
    // A at or past n are zero, so the solve below may run all BM steps
    if (warp >= kG0 / 32) {
      const int t = tid - kG0;
      uint32_t gr[BM];
#pragma unroll
      for (int c0 = 0; c0 < BM; c0 += 16)
        tc::tmem_ld16(tmG + lane_off + c0, *reinterpret_cast<uint32_t(*)[16]>(&gr[c0]));
      tc::tmem_ld_wait();
      if (t >= 0) {
        // the log-gates go to registers first (16-byte loads) and every
        // exponential is taken unconditionally, the mask applied as a
        // select: a branch per element would serialise the chains
        float g2r[BM];
#pragma unroll
        for (int i4 = 0; i4 < BM / 4; ++i4) {
          const float4 q = *reinterpret_cast<const float4*>(&sh.gam2[4 * i4]);
          g2r[4 * i4] = q.x, g2r[4 * i4 + 1] = q.y, g2r[4 * i4 + 2] = q.z, g2r[4 * i4 + 3] = q.w;
        }
        const float bt = sh.beta[t], gt = sh.gam2[t];
        const bool live = t < n;
#pragma unroll
        for (int i = 0; i < BM; ++i) {
          const float a = bt * tc::ex2(gt - g2r[i]) * __uint_as_float(gr[i]);
          AT[i * kATs + t] = (live && i < t) ? a : 0.f;
        }
      }
    }
    // X = diag(beta) (V - diag(Gam) W) for this thread's column
    float x[BM];
#pragma unroll
    for (int c0 = 0; c0 < BM; c0 += 16) {
      uint32_t w[16];
      tc::tmem_ld16(tmW + lane_off + c0, w);  // columns past Bp: stale, used by no kept row
      tc::tmem_ld_wait();
#pragma unroll
      for (int e4 = 0; e4 < 4; ++e4) {
        const float4 b4 = *reinterpret_cast<const float4*>(&sh.beta[c0 + 4 * e4]);
        const float4 g4 = *reinterpret_cast<const float4*>(&sh.Gam[c0 + 4 * e4]);
        const float bb[4] = {b4.x, b4.y, b4.z, b4.w}, gg[4] = {g4.x, g4.y, g4.z, g4.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int t = c0 + 4 * e4 + e;
          x[t] = bb[e] * (__uint_as_float(vraw[t] << 16) - gg[e] * __uint_as_float(w[4 * e4 + e]));
        }
      }
    }
    tc::fence_before_sync();
    __syncthreads();  // A^T published; the state buffer, W^T and G read
    // the next item's state streams in while this one is solved and stored
    if (tid == 0 && it_next >= 0) {
      issue_s0(it_next, slot_next);
      s0_out = true;
      s0_par = ph ^ 1u;
    }

    // (I + A) delta = X, right-looking: once delta_t is final it leaves the
    // remaining rows (A^T row t as 16-byte broadcast loads).  Rows t >= n
    // only touch rows past n (A^T is zero there), which nothing keeps.
#pragma unroll
    for (int t = 0; t < BM; ++t) {
      const float dt = x[t];
      const float* ar = AT + t * kATs;
#pragma unroll
      for (int u4 = (t + 1) / 4; u4 < BM / 4; ++u4) {
        const float4 a = *reinterpret_cast<const float4*>(ar + 4 * u4);
        if (4 * u4 + 0 > t) x[4 * u4 + 0] = fmaf(-a.x, dt, x[4 * u4 + 0]);
        if (4 * u4 + 1 > t) x[4 * u4 + 1] = fmaf(-a.y, dt, x[4 * u4 + 1]);
        if (4 * u4 + 2 > t) x[4 * u4 + 2] = fmaf(-a.z, dt, x[4 * u4 + 2]);
        if (4 * u4 + 3 > t) x[4 * u4 + 3] = fmaf(-a.w, dt, x[4 * u4 + 3]);
      }
    }
    // delta'_t = exp(gamma_{n-1} - gamma_t) delta_t (t < n), as bf16 hi and lo parts
    {
      float dr[BM];
#pragma unroll
      for (int i4 = 0; i4 < BM / 4; ++i4) {
        const float4 q = *reinterpret_cast<const float4*>(&sh.dsc[4 * i4]);
        dr[4 * i4] = q.x, dr[4 * i4 + 1] = q.y, dr[4 * i4 + 2] = q.z, dr[4 * i4 + 3] = q.w;
      }
#pragma unroll
      for (int c0 = 0; c0 < C::kDP; c0 += 16) {
        uint32_t hi[16], lo[16];
#pragma unroll
        for (int e = 0; e < 16; ++e) {
          const int t = 2 * (c0 + e);
          float a = 0.f, b = 0.f;
          if (t < BM) {
            const float xa = x[t] * dr[t], xb = x[t + 1] * dr[t + 1];
            a = t < n ? xa : 0.f;
            b = t + 1 < n ? xb : 0.f;
          }
          split_pair(a, b, hi[e], lo[e]);
        }
        tc::tmem_st16(tmW + lane_off + c0, hi);
        tc::tmem_st16(tmW + lane_off + C::kDP + c0, lo);
      }
    }
    tc::tmem_st_wait();
    tc::fence_before_sync();
    __syncthreads();  // also: A^T read, its region free for the next values
    if (tid == 0) {
      tc::fence_after_sync();
      // D += delta'^T K: the keys [t][i] as an MN-major operand (i contiguous)
      const int ksteps = (n + 15) >> 4;
#pragma unroll 1
      for (int kk = 0; kk < ksteps; ++kk) {
        const uint64_t kb = tc::sdesc_sw128(tc::smem_u32(Ks + kk * 2048), 64 * 128, 1024);
        tc::mma_bf16_ts(tmS, tmW + kk * 8, kb, idU, 1u);
        tc::mma_bf16_ts(tmS, tmW + C::kDP + kk * 8, kb, idU, 1u);
      }
      tc::mma_commit(&sh.bar_mma);
      mma_out = true;
    }
    if (!ct_wait(&sh.bar_mma, ph_mma, sh, p.dev_status)) break;
    ph_mma ^= 1u;
    tc::fence_after_sync();
    if (tid == 0) {
      mma_out = false;
      if (it_next >= 0) {  // the update, the last reader of these keys, is done
        tc::fence_async_smem();
        issue_kv(it_next);
        k_out = true;
        k_par = ph ^ 1u;
      }
    }
    // the committed state: lane c holds S^(n)[i][c] over i
    {
      float* Sg = state_of(it, slot) + tid;
#pragma unroll 1
      for (int i0 = 0; i0 < kCtD; i0 += 32) {
        uint32_t d[32];
        tc::tmem_ld16(tmS + lane_off + i0, *reinterpret_cast<uint32_t(*)[16]>(&d[0]));
        tc::tmem_ld16(tmS + lane_off + i0 + 16, *reinterpret_cast<uint32_t(*)[16]>(&d[16]));
        tc::tmem_ld_wait();
#pragma unroll
        for (int e = 0; e < 32; ++e) Sg[(size_t)(i0 + e) * kCtD] = __uint_as_float(d[e]);
      }
    }
    if (it_next < 0) break;
    it = it_next;
    slot = slot_next;
    n = n_next;
    ph ^= 1u;
  }

  // after a timeout: let the copies and MMAs in flight land before the
  // shared and tensor memory are given up (bounded waits)
  if (tid == 0 && sh.abort_flag) {
    if (s0_out) tc::mbar_wait(&sh.bar_s0, s0_par, nullptr, 100000000ull);
    if (k_out) tc::mbar_wait(&sh.bar_k, k_par, nullptr, 100000000ull);
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

PFN_cuTensorMapEncodeTiled_v12000 ct_encode_fn() {
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
bool ct_act_map(CUtensorMap* m, const void* x, int H, int B, int R, int rows, bool swizzle) {
  auto fn = ct_encode_fn();
  if (!fn) return false;
  cuuint64_t gd[4] = {(cuuint64_t)kCtD, (cuuint64_t)H, (cuuint64_t)B, (cuuint64_t)R};
  cuuint64_t gs[3] = {(cuuint64_t)kCtD * 2, (cuuint64_t)H * kCtD * 2,
                      (cuuint64_t)B * H * kCtD * 2};
  cuuint32_t bx[4] = {64, 1, (cuuint32_t)rows, 1};
  cuuint32_t es[4] = {1, 1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(x), gd, gs, bx, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE,
            swizzle ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_NONE,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) ==
         CUDA_SUCCESS;
}

template <int BM>
cudaError_t launch_ct(const GdrParams& p, cudaStream_t stream) {
  CtMaps maps;
  if (!ct_act_map(&maps.k, p.k, p.Hk, p.B, p.R, 64, true) ||
      !ct_act_map(&maps.v, p.v, p.Hv, p.B, p.R, BM, false))
    return cudaErrorInvalidValue;
  const int smem = CtCfg<BM>::kSmem + 1024;
  cudaError_t e = cudaFuncSetAttribute(gdr_commit_tc_kernel<BM>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  int dev = 0, sms = kNumSMs;
  if (cudaGetDevice(&dev) == cudaSuccess)
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const long items = (long)p.R * p.Hv;
  const int grid = (int)(items < 2L * sms ? items : 2L * sms);
  gdr_commit_tc_kernel<BM><<<grid, kCtThreads, smem, stream>>>(maps, p);
  note_launches(1);
  return cudaGetLastError();
}

}  // namespace

bool gdr_commit_tc_supported(int B, int dk, int dv) {
  return B >= 1 && B <= 64 && dk == kCtD && dv == kCtD;
}

cudaError_t launch_gdr_commit_tc(const GdrParams& p, cudaStream_t stream) {
  if (p.R == 0) return cudaSuccess;
  if (p.B <= 16) return launch_ct<16>(p, stream);
  return p.B <= 32 ? launch_ct<32>(p, stream) : launch_ct<64>(p, stream);
}

}  // namespace flare
