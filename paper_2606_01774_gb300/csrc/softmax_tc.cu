// Block-query softmax attention over a paged KV prefix on the 5th-generation
// tensor cores (tcgen05), bf16 in, fp32 accumulate.
//
// Work item = (request r, kv head, tile of 128 query rows, prefix split).  The
// rows of a (request, kv head) are its B*G block queries, row m = t*G + g
// (grouped-query attention: the G query heads of a kv head share its keys and
// values), so one K/V tile feeds 128 rows of G heads at once.  The key
// sequence of a request is its prefix, 64 tokens per tile read through the
// page table, followed by one tile holding the block's own B keys (the block
// is not in the paged cache during the denoise pass).  Every block row sees
// every prefix token; the mask only touches the ragged prefix end and the
// block tile (bidirectional, or token-causal for the state-update pass).
//
// Tensor memory holds Q (bf16, loaded once), the O accumulator and two S
// buffers; each S buffer is overwritten in place by its bf16 probabilities P,
// which the P.V MMA reads straight from tensor memory.  Shared memory only
// holds a ring of K and V tiles, so per tile the SM moves each K/V byte in
// once (TMA) and out once (MMA operand read).
//
// Warp roles (320 threads):
//   warp 0     TMA producer: K and V tiles (one box per page and 64-column
//              chunk, 128-byte swizzle) in the order the MMA warp consumes
//              them (K runs one tile ahead of V).
//   warp 1     tensor-memory owner and MMA issuer: S_j = Q K_j^T, then
//              O += P_{j-1} V_{j-1}; zeroes V rows past the prefix end so
//              poisoned cache rows never meet a zero probability (0 * NaN).
//              MMAs from this one thread execute in issue order, which is what
//              lets S_{j+2} reuse the buffer P_j lives in.
//   warps 2-9  softmax: two warps per TMEM lane quarter, each thread one query
//              row and half of the tile's 64 key columns; online base-2
//              softmax with a lazily moved running max (O is rescaled only when
//              the max grows by more than 2^8); epilogue divides by the row sum
//              and stores the output (or a split partial).
// Every wait is bounded (tc::mbar_wait); a timeout sets FLARE_DEV_WAIT_TIMEOUT,
// the CTA stops issuing work, writes nothing, frees its TMEM and exits.
#include <cudaTypedefs.h>

#include "common.cuh"
#include "kernels.h"
#include "tc.cuh"

namespace flare {

namespace {

constexpr int kTileN = 64;     // keys per tile
constexpr int kRowsM = 128;    // query rows per CTA (TMEM lanes)
constexpr int kSplit = 1;        // softmax warps per TMEM lane quarter (each takes 64/kSplit keys)
constexpr int kSoftmaxThreads = 128 * kSplit;
constexpr int kThreadsTC = 64 + kSoftmaxThreads;  // producer warp, MMA warp, softmax warps
constexpr float kRescaleThreshold = 8.0f;  // log2 units

struct TcMaps {
  CUtensorMap q;      // (D, Hq, B, R)           box (64, G, 128/G, 1)
  CUtensorMap kblk;   // (D, Hkv, B, R)          box (64, 1, 64, 1)
  CUtensorMap vblk;
  CUtensorMap kpool;  // (D, p, Hkv, num_pages)  box (64, min(p,64), 1, 1)
  CUtensorMap vpool;
};

template <int D>
struct TcCfg {
  static constexpr int kChunks = D / 64;
  static constexpr int kKVBytes = kChunks * kTileN * 128;  // one K (or V) tile
  static constexpr int kQBytes = kChunks * kRowsM * 128;   // Q tile, K-major, 128-byte swizzle
  static constexpr int kKStages = D == 256 ? 3 : (D == 128 ? 6 : 8);  // K ring depth
  static constexpr int kVStages = D == 256 ? 2 : (D == 128 ? 4 : 8);  // V ring depth
  static constexpr int kSmem = kQBytes + (kKStages + kVStages) * kKVBytes;
  // tensor memory: O [0, D), three S/P buffers [D, D + 192)
  static constexpr int kTmemCols = (D + 3 * kTileN) > 256 ? 512 : 256;
  static constexpr int kSCol = D;
};

struct TcShared {
  uint64_t q_full;
  uint64_t k_full[8], v_full[8], k_empty[8], v_empty[8];
  uint64_t s_full[3], p_full[3], pv_done[3];
  uint64_t o_final;
  uint64_t xbar[4];     // row-pair exchange written, one per TMEM lane quarter (64 arrivals)
  uint64_t xread[4];    // row-pair exchange read (64 arrivals)
  float xch[256];       // [half][128 rows]
  uint32_t tmem_base;
  int abort_flag;
};

// All lanes of the warp wait; the outcome is made warp-uniform so that the
// warp-collective instructions that follow are always entered together.
__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, const int* abort) {
  const bool ok = tc::mbar_wait(bar, parity, abort);
  return __all_sync(0xffffffffu, ok);
}

__device__ __forceinline__ bool aborted(const TcShared& sh) {
  return *reinterpret_cast<const volatile int*>(&sh.abort_flag) != 0;
}

__device__ __forceinline__ void set_abort(TcShared& sh, int32_t* status) {
  if (!sh.abort_flag) {
    sh.abort_flag = 1;
    flag(status, FLARE_DEV_WAIT_TIMEOUT);
  }
}

__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, "
      "%11, %12, %13, %14, %15, %16};" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]),
      "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15])
      : "memory");
}

__device__ __forceinline__ void tmem_st_wait() {
  asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

// D[tmem] (+)= A[tmem] * B[smem]^T, bf16, fp32 accumulate; one thread.
__device__ __forceinline__ void mma_bf16_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc,
                                            uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n"
      " .reg .pred p;\n"
      " setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n"
      "}\n" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

}  // namespace

template <int D>
__global__ void __launch_bounds__(kThreadsTC, 1)
    softmax_tc_kernel(const __grid_constant__ TcMaps maps, SoftmaxParams p) {
  using C = TcCfg<D>;
  extern __shared__ uint8_t smem_raw[];
  __shared__ TcShared sh;
  uint8_t* base = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint8_t* Qs = base;
  uint8_t* Ks = Qs + C::kQBytes;
  uint8_t* Vs = Ks + C::kKStages * C::kKVBytes;

  const int mtile = blockIdx.x, split = blockIdx.y, item = blockIdx.z;
  const int r = item / p.Hkv, kvh = item % p.Hkv;
  const int M = p.B * p.G;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

  const int P = p.prefix_len[r];
  const int bad = check_request_pages(p.page_table, P, r, p.max_pages, p.page_size, p.num_pages);
  if (bad) {
    if (tid == 0) flag(p.dev_status, bad);
    return;
  }
  // tiles of this split: prefix tiles [j0, j1) then (last split only) the block tile
  const int n_pref = (P + kTileN - 1) / kTileN;
  const int tps = p.split_len / kTileN;
  const int j0 = split * tps;
  const int j1 = min(n_pref, j0 + tps);
  const int n_pref_here = max(0, j1 - j0);
  const bool has_blk = split == p.n_split - 1;
  const int n_tiles = n_pref_here + (has_blk ? 1 : 0);
  const size_t ws_row0 = ((size_t)item * p.n_split + split) * M;

  if (n_tiles == 0) {  // empty split: mark its partial as empty for the combine pass
    for (int i = tid; i < kRowsM; i += blockDim.x) {
      const int m = mtile * kRowsM + i;
      if (m < M) p.ws_lse[ws_row0 + m] = -INFINITY;
    }
    return;
  }

  if (tid == 0) {
    sh.abort_flag = 0;
    tc::mbar_init(&sh.q_full, 1);
    for (int s = 0; s < C::kKStages; ++s) {
      tc::mbar_init(&sh.k_full[s], 1);
      tc::mbar_init(&sh.k_empty[s], 1);
    }
    for (int s = 0; s < C::kVStages; ++s) {
      tc::mbar_init(&sh.v_full[s], 1);
      tc::mbar_init(&sh.v_empty[s], 1);
    }
    for (int b = 0; b < 3; ++b) {
      tc::mbar_init(&sh.s_full[b], 1);
      tc::mbar_init(&sh.p_full[b], kSoftmaxThreads);
      tc::mbar_init(&sh.pv_done[b], 1);
    }
    tc::mbar_init(&sh.o_final, 1);
    for (int q = 0; q < 4; ++q) {
      tc::mbar_init(&sh.xbar[q], 32 * kSplit);
      tc::mbar_init(&sh.xread[q], 32 * kSplit);
    }
    tc::fence_mbar_init();
  }
  if (warp == 1) tc::tmem_alloc(&sh.tmem_base, C::kTmemCols);
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = sh.tmem_base;
  const uint32_t tmem_o = tmem;
  const uint32_t tmem_s = tmem + C::kSCol;

  // tile index -> (is block tile, prefix tile number)
  auto tile_kind = [&](int j, int& ptile) -> bool {
    if (j < n_pref_here) {
      ptile = j0 + j;
      return false;
    }
    ptile = -1;
    return true;
  };
  // valid key columns of a tile
  auto tile_valid = [&](int j) -> int {
    int pt;
    if (tile_kind(j, pt)) return p.B;
    return min(kTileN, P - pt * kTileN);
  };

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      tc::prefetch_tmap(&maps.kpool);
      tc::prefetch_tmap(&maps.vpool);
      const int Bt = kRowsM / p.G;
      tc::mbar_expect_tx(&sh.q_full, C::kQBytes);
      for (int c = 0; c < C::kChunks; ++c)
        tc::tma_load_4d(Qs + c * (kRowsM * 128), &maps.q, &sh.q_full, c * 64, kvh * p.G,
                        mtile * Bt, r);
      const int box_rows = p.page_size < kTileN ? p.page_size : kTileN;
      // one K or V tile into its ring slot (waits for the slot to be free)
      auto load = [&](int j, int kv) -> bool {
        const int ns = kv ? C::kVStages : C::kKStages;
        const int st = j % ns;
        const uint32_t ph = (uint32_t)(j / ns) & 1u;
        uint64_t* empty = kv ? &sh.v_empty[st] : &sh.k_empty[st];
        uint64_t* full = kv ? &sh.v_full[st] : &sh.k_full[st];
        uint8_t* dst = (kv ? Vs : Ks) + st * C::kKVBytes;
        if (!tc::mbar_wait(empty, ph ^ 1u, &sh.abort_flag)) return false;
        int pt;
        if (tile_kind(j, pt)) {
          tc::mbar_expect_tx(full, C::kKVBytes);
          const CUtensorMap* m = kv ? &maps.vblk : &maps.kblk;
          for (int c = 0; c < C::kChunks; ++c)
            tc::tma_load_4d(dst + c * (kTileN * 128), m, full, c * 64, kvh, 0, r);
        } else {
          const int tok0 = pt * kTileN;
          const int valid = min(kTileN, P - tok0);
          const int nbox = (valid + box_rows - 1) / box_rows;
          tc::mbar_expect_tx(full, (uint32_t)(C::kChunks * nbox * box_rows * 128));
          const CUtensorMap* m = kv ? &maps.vpool : &maps.kpool;
          for (int b = 0; b < nbox; ++b) {
            const int tok = tok0 + b * box_rows;
            const int page = p.page_table[(size_t)r * p.max_pages + tok / p.page_size];
            const int row0 = tok % p.page_size;
            for (int c = 0; c < C::kChunks; ++c)
              tc::tma_load_4d(dst + c * (kTileN * 128) + b * box_rows * 128, m, full, c * 64,
                              row0, kvh, page);
          }
        }
        return true;
      };
      // K runs two tiles ahead of V: K0, K1, K2, V0, K3, V1, ... (the MMA warp
      // consumes K_j at S_j and V_j one step later, at P_j V_j)
      constexpr int kLead = 2;
      bool ok = true;
      for (int j = 0; j < kLead && j < n_tiles && ok; ++j) ok = load(j, 0);
      for (int j = 0; j < n_tiles && ok && !aborted(sh); ++j) {
        if (j + kLead < n_tiles) ok = load(j + kLead, 0);
        if (ok) ok = load(j, 1);
      }
      if (!ok) set_abort(sh, p.dev_status);
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    const uint32_t id_s = tc::idesc_bf16(kRowsM, kTileN, false, false);
    const uint32_t id_o = tc::idesc_bf16(kRowsM, D, false, true);
    bool ok = warp_wait(&sh.q_full, 0, &sh.abort_flag);
    auto issue_pv = [&](int i) -> bool {
      const int st = i % C::kVStages;
      const int pb = i % 3;
      if (!warp_wait(&sh.p_full[pb], (uint32_t)(i / 3) & 1u, &sh.abort_flag)) return false;
      if (!warp_wait(&sh.v_full[st], (uint32_t)(i / C::kVStages) & 1u, &sh.abort_flag))
        return false;
      uint8_t* vst = Vs + st * C::kKVBytes;
      const int valid = tile_valid(i);
      int pt;
      if (!tile_kind(i, pt) && valid < kTileN) {
        // zero the V rows past the prefix end (stale or poisoned cache rows)
        const int nrow = kTileN - valid;
        for (int e = lane; e < C::kChunks * nrow * 8; e += 32) {
          const int c = e / (nrow * 8), rr = valid + (e / 8) % nrow, q16 = e % 8;
          *reinterpret_cast<uint4*>(vst + c * (kTileN * 128) + rr * 128 + q16 * 16) =
              make_uint4(0u, 0u, 0u, 0u);
        }
        tc::fence_async_smem();
      }
      __syncwarp();
      tc::fence_after_sync();
      if (lane == 0) {
#pragma unroll
        for (int kk = 0; kk < kTileN / 16; ++kk) {
          const uint64_t b = tc::sdesc_sw128(tc::smem_u32(vst + kk * 2048), kTileN * 128, 1024);
          mma_bf16_ts(tmem_o, tmem_s + pb * kTileN + kk * 8, b, id_o, (i > 0 || kk > 0) ? 1u : 0u);
        }
        tc::mma_commit(&sh.pv_done[pb]);
        tc::mma_commit(&sh.v_empty[st]);
      }
      __syncwarp();
      return true;
    };
    // S_j = Q K_j^T into S buffer j % 3
    auto issue_s = [&](int j) -> bool {
      const int st = j % C::kKStages;
      const int sb = j % 3;
      if (!warp_wait(&sh.k_full[st], (uint32_t)(j / C::kKStages) & 1u, &sh.abort_flag))
        return false;
      tc::fence_after_sync();
      if (lane == 0) {
        const uint8_t* kst = Ks + st * C::kKVBytes;
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const int c = kk >> 2, off = (kk & 3) * 32;
          const uint64_t a = tc::sdesc_sw128(tc::smem_u32(Qs + c * (kRowsM * 128) + off), 16, 1024);
          const uint64_t b = tc::sdesc_sw128(tc::smem_u32(kst + c * (kTileN * 128) + off), 16, 1024);
          tc::mma_bf16_ss(tmem_s + sb * kTileN, a, b, id_s, kk > 0 ? 1u : 0u);
        }
        tc::mma_commit(&sh.s_full[sb]);
        tc::mma_commit(&sh.k_empty[st]);
      }
      __syncwarp();
      return true;
    };
    // Issue order S0, S1, S2, PV0, S3, PV1, ...: S_{j+2} is queued before the
    // P.V of tile j waits on its probabilities, so the tensor pipe stays fed
    // through the softmax; S_{j+2} reuses the buffer of tile j-1, whose P.V was
    // issued (and, in issue order, executes) before it.
    for (int j = 0; j < 2 && j < n_tiles && ok; ++j) ok = issue_s(j);
    for (int j = 0; j < n_tiles && ok; ++j) {
      if (j + 2 < n_tiles) ok = issue_s(j + 2);
      if (ok) ok = issue_pv(j);
    }
    if (ok && lane == 0) tc::mma_commit(&sh.o_final);
    if (!ok && lane == 0) set_abort(sh, p.dev_status);
  } else {
    // ------------------------------------------------------------ softmax warps
    // Eight warps: warp w reads TMEM lanes 32*(w%4).. (its 32 rows) and key
    // columns 32*half.. of each tile; the two warps of a row pair exchange
    // their tile maxima through shared memory every tile.
    const int quarter = warp & 3;
    const int half = (warp - 2) >> 2;
    const int row = quarter * 32 + lane;
    const int m = mtile * kRowsM + row;
    const int trow = m / p.G;
    const uint32_t lane_off = (uint32_t)(quarter * 32) << 16;
    constexpr int kDh = D / kSplit;       // Q elements / output columns this warp handles
    constexpr int kCols = kTileN / kSplit;  // key columns of each tile this warp handles

    float m_run = -INFINITY, l_run = 0.f;  // l_run: this half's share of the row sum
    bool ok = true;
    for (int j = 0; j < n_tiles; ++j) {
      const int sb = j % 3;
      if (!warp_wait(&sh.s_full[sb], (uint32_t)(j / 3) & 1u, &sh.abort_flag)) {
        ok = false;
        break;
      }
      tc::fence_after_sync();
      const uint32_t sbuf = tmem_s + lane_off + sb * kTileN;
      uint32_t sr[kCols];
#pragma unroll
      for (int c = 0; c < kCols; c += 16)
        tc::tmem_ld16(sbuf + kCols * half + c, *reinterpret_cast<uint32_t(*)[16]>(&sr[c]));
      tc::tmem_ld_wait();

      int pt;
      const bool blk = tile_kind(j, pt);
      const int valid = tile_valid(j);
      const bool full = !blk && valid == kTileN;  // prefix tile: no mask at all
      const int lim = full ? kTileN : ((blk && p.causal) ? min(valid, trow + 1) : valid);
      // tile maximum of the raw scores (scale >= 0 keeps the order)
      float mx[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
      for (int c = 0; c < kCols; ++c)
        if (full || kCols * half + c < lim) mx[c & 3] = fmaxf(mx[c & 3], __uint_as_float(sr[c]));
      float mt = fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3]));
      // the partner has read this slot's previous value before it is overwritten;
      // this exchange also orders both halves' S reads before either writes P.
      if (kSplit > 1) {
        if (j >= 1 && !warp_wait(&sh.xread[quarter], (uint32_t)(j - 1) & 1u, &sh.abort_flag)) {
          ok = false;
          break;
        }
        sh.xch[half * 128 + row] = mt;
        tc::fence_before_sync();
        tc::mbar_arrive(&sh.xbar[quarter]);
        if (!warp_wait(&sh.xbar[quarter], (uint32_t)j & 1u, &sh.abort_flag)) {
          ok = false;
          break;
        }
        tc::fence_after_sync();
        mt = fmaxf(mt, sh.xch[(1 - half) * 128 + row]);
        tc::mbar_arrive(&sh.xread[quarter]);
      }
      const float m_new = fmaxf(m_run, mt * p.scale_log2);
      const bool need = (j == 0) || (m_new > m_run + kRescaleThreshold);
      const bool warp_rescale = __any_sync(0xffffffffu, need);
      float m_use = m_run;
      if (warp_rescale) m_use = (j == 0 || m_new > m_run) ? m_new : m_run;
      const float corr = (j == 0) ? 0.f : tc::ex2(m_run - m_use);
      const float neg_m = -m_use;
      float sum0 = 0.f, sum1 = 0.f;
      uint32_t pk[kCols / 2];
      if (full) {
#pragma unroll
        for (int c = 0; c < kCols; c += 2) {
          const float p0 = tc::ex2(fmaf(__uint_as_float(sr[c]), p.scale_log2, neg_m));
          const float p1 = tc::ex2(fmaf(__uint_as_float(sr[c + 1]), p.scale_log2, neg_m));
          sum0 += p0;
          sum1 += p1;
          __nv_bfloat162 h2 = __floats2bfloat162_rn(p0, p1);
          pk[c / 2] = *reinterpret_cast<uint32_t*>(&h2);
        }
      } else {
#pragma unroll
        for (int c = 0; c < kCols; c += 2) {
          const int col = kCols * half + c;
          const float p0 =
              col < lim ? tc::ex2(fmaf(__uint_as_float(sr[c]), p.scale_log2, neg_m)) : 0.f;
          const float p1 =
              col + 1 < lim ? tc::ex2(fmaf(__uint_as_float(sr[c + 1]), p.scale_log2, neg_m)) : 0.f;
          sum0 += p0;
          sum1 += p1;
          __nv_bfloat162 h2 = __floats2bfloat162_rn(p0, p1);
          pk[c / 2] = *reinterpret_cast<uint32_t*>(&h2);
        }
      }
      const float sum = sum0 + sum1;
      l_run = (j == 0) ? sum : l_run * corr + sum;
      // rescale this half's O columns when the running max moved (P.V of tile j-1 done)
      if (warp_rescale && j >= 1) {
        const int pb = (j - 1) % 3;
        if (!warp_wait(&sh.pv_done[pb], (uint32_t)((j - 1) / 3) & 1u, &sh.abort_flag)) {
          ok = false;
          break;
        }
        tc::fence_after_sync();
#pragma unroll 1
        for (int c = half * kDh; c < (half + 1) * kDh; c += 16) {
          uint32_t o[16];
          tc::tmem_ld16(tmem_o + lane_off + c, o);
          tc::tmem_ld_wait();
#pragma unroll
          for (int i = 0; i < 16; ++i) o[i] = __float_as_uint(__uint_as_float(o[i]) * corr);
          tmem_st16(tmem_o + lane_off + c, o);
        }
      }
      m_run = m_use;
      // P (bf16 pairs) over this warp's kCols / 2 columns of the S buffer
#pragma unroll
      for (int c = 0; c < kCols / 2; c += 16)
        tmem_st16(sbuf + (kCols / 2) * half + c, *reinterpret_cast<uint32_t(*)[16]>(&pk[c]));
      tmem_st_wait();
      tc::fence_before_sync();
      tc::mbar_arrive(&sh.p_full[sb]);
    }
    // row sum = the two halves' shares
    if (kSplit > 1 && ok &&
        !warp_wait(&sh.xread[quarter], (uint32_t)(n_tiles - 1) & 1u, &sh.abort_flag))
      ok = false;
    if (kSplit > 1 && ok) {
      sh.xch[half * 128 + row] = l_run;
      tc::mbar_arrive(&sh.xbar[quarter]);
      if (!warp_wait(&sh.xbar[quarter], (uint32_t)n_tiles & 1u, &sh.abort_flag)) ok = false;
      if (ok) l_run += sh.xch[(1 - half) * 128 + row];
    }
    if (ok && !warp_wait(&sh.o_final, 0, &sh.abort_flag)) ok = false;
    if (!ok) set_abort(sh, p.dev_status);
    tc::fence_after_sync();
    const bool write = ok && m < M && !aborted(sh);
    const float inv = l_run > 0.f ? 1.f / l_run : 0.f;
    const int g = m % p.G;
    const size_t orow = (((size_t)r * p.B + trow) * p.Hq + kvh * p.G + g);
    if (ok) {
#pragma unroll 1
      for (int c = half * kDh; c < (half + 1) * kDh; c += 16) {
        uint32_t o[16];
        tc::tmem_ld16(tmem_o + lane_off + c, o);
        tc::tmem_ld_wait();
        if (!write) continue;
        if (p.n_split == 1) {
          uint32_t pkd[8];
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            __nv_bfloat162 h2 = __floats2bfloat162_rn(__uint_as_float(o[2 * i]) * inv,
                                                      __uint_as_float(o[2 * i + 1]) * inv);
            pkd[i] = *reinterpret_cast<uint32_t*>(&h2);
          }
          uint4* dst = reinterpret_cast<uint4*>(static_cast<__nv_bfloat16*>(p.out) + orow * D + c);
          dst[0] = make_uint4(pkd[0], pkd[1], pkd[2], pkd[3]);
          dst[1] = make_uint4(pkd[4], pkd[5], pkd[6], pkd[7]);
        } else {
          float4* dst = reinterpret_cast<float4*>(p.ws_o + (ws_row0 + m) * D + c);
#pragma unroll
          for (int i = 0; i < 4; ++i)
            dst[i] = make_float4(__uint_as_float(o[4 * i]) * inv, __uint_as_float(o[4 * i + 1]) * inv,
                                 __uint_as_float(o[4 * i + 2]) * inv,
                                 __uint_as_float(o[4 * i + 3]) * inv);
        }
      }
    }
    if (write && half == 0) {
      const float lse = l_run > 0.f ? (m_run + __log2f(l_run)) * 0.6931471805599453f : -INFINITY;
      if (p.n_split == 1) {
        if (p.lse) p.lse[orow] = lse;
      } else {
        p.ws_lse[ws_row0 + m] = lse;
      }
    }
  }
  tc::fence_before_sync();
  __syncthreads();
  if (warp == 1) {
    tc::fence_after_sync();
    tc::tmem_dealloc(tmem, C::kTmemCols);
  }
}

// ------------------------------------------------------------------ host side

namespace {

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
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

bool encode4(CUtensorMap* m, const void* ptr, const uint64_t dims[4], const uint64_t strides[3],
             const uint32_t box[4]) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t gd[4] = {dims[0], dims[1], dims[2], dims[3]};
  cuuint64_t gs[3] = {strides[0], strides[1], strides[2]};
  cuuint32_t bx[4] = {box[0], box[1], box[2], box[3]};
  cuuint32_t es[4] = {1, 1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(ptr), gd, gs, bx, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) ==
         CUDA_SUCCESS;
}

template <int D>
cudaError_t launch_tc_d(const SoftmaxParams& p, const SoftmaxPlan& plan, cudaStream_t stream) {
  using C = TcCfg<D>;
  TcMaps maps;
  const uint64_t e = 2;
  {
    const uint64_t dims[4] = {(uint64_t)D, (uint64_t)p.Hq, (uint64_t)p.B, (uint64_t)p.R};
    const uint64_t str[3] = {D * e, (uint64_t)p.Hq * D * e, (uint64_t)p.B * p.Hq * D * e};
    const uint32_t box[4] = {64, (uint32_t)p.G, (uint32_t)(kRowsM / p.G), 1};
    if (!encode4(&maps.q, p.q, dims, str, box)) return cudaErrorInvalidValue;
  }
  {
    const uint64_t dims[4] = {(uint64_t)D, (uint64_t)p.Hkv, (uint64_t)p.B, (uint64_t)p.R};
    const uint64_t str[3] = {D * e, (uint64_t)p.Hkv * D * e, (uint64_t)p.B * p.Hkv * D * e};
    const uint32_t box[4] = {64, 1, (uint32_t)kTileN, 1};
    if (!encode4(&maps.kblk, p.k_blk, dims, str, box) ||
        !encode4(&maps.vblk, p.v_blk, dims, str, box))
      return cudaErrorInvalidValue;
  }
  {
    const int npages = p.num_pages > 0 ? p.num_pages : 1;
    const uint64_t dims[4] = {(uint64_t)D, (uint64_t)p.page_size, (uint64_t)p.Hkv,
                              (uint64_t)npages};
    const uint64_t str[3] = {D * e, (uint64_t)p.page_size * D * e,
                             (uint64_t)p.Hkv * p.page_size * D * e};
    const uint32_t box[4] = {64, (uint32_t)(p.page_size < kTileN ? p.page_size : kTileN), 1, 1};
    // an empty pool is never read (every prefix is empty); point the map at the block tensor
    const void* kp = p.num_pages > 0 ? p.k_pool : p.k_blk;
    const void* vp = p.num_pages > 0 ? p.v_pool : p.v_blk;
    if (!encode4(&maps.kpool, kp, dims, str, box) || !encode4(&maps.vpool, vp, dims, str, box))
      return cudaErrorInvalidValue;
  }
  const int smem = C::kSmem + 1024;
  cudaError_t err = cudaFuncSetAttribute(softmax_tc_kernel<D>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (err != cudaSuccess) return err;
  const int M = p.B * p.G;
  dim3 grid((M + kRowsM - 1) / kRowsM, plan.n_split, p.R * p.Hkv);
  softmax_tc_kernel<D><<<grid, kThreadsTC, smem, stream>>>(maps, p);
  note_launches(1);
  err = cudaGetLastError();
  if (err != cudaSuccess || plan.n_split == 1) return err;
  return launch_softmax_combine(p, true, stream);
}

}  // namespace

bool softmax_tc_supported(int B, int Hq, int Hkv, int D, int page_size) {
  const int G = Hq / Hkv;
  if (D != 64 && D != 128 && D != 256) return false;
  if (G < 1 || G > kRowsM || (kRowsM % G) != 0) return false;
  if (page_size < 16 || page_size > 128) return false;
  return B >= 1 && B <= kTileN;
}

cudaError_t launch_softmax_tc(const SoftmaxParams& p, const SoftmaxPlan& plan,
                              cudaStream_t stream) {
  switch (p.D) {
    case 64: return launch_tc_d<64>(p, plan, stream);
    case 128: return launch_tc_d<128>(p, plan, stream);
    case 256: return launch_tc_d<256>(p, plan, stream);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace flare
