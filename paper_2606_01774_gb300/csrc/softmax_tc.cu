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
// A one-CTA pre-pass validates every request (prefix length, page ids), drops
// bad ones from the work list and orders the work units longest first.  When
// prefixes are not split, one CTA per SM walks its share of the items (snake
// order over the CTAs), so setup happens once per CTA and the next item's
// loads and S products overlap the current item's epilogue; when they are,
// one CTA runs each item and the last split of a row tile merges the partials.
//
// Tensor memory holds Q (bf16 pairs, loaded per item), the O accumulator and the
// S buffers (three for D <= 128, two for D = 256); each S buffer is
// overwritten in place by its bf16 probabilities P.  Both products read their
// A operand from tensor memory (S = Q K^T and O += P V), so shared memory only
// holds the K and V rings: per tile the SM moves each K/V byte in once (TMA)
// and out once (MMA operand read), and the rings take all of shared memory,
// since a tile load takes about a microsecond from issue to arrival.
//
// Warp roles (256 threads):
//   warp 0     K producer, warp 6 V producer: one TMA box per page and
//              64-column chunk (128-byte swizzle) into their own rings.
//   warp 7     zeroes the V rows past the prefix end once that tile has landed,
//              so poisoned cache rows never meet a zero probability (0 * NaN).
//   warp 1     tensor-memory owner and MMA issuer (one thread): S_j = Q K_j^T,
//              then O += P_j V_j.  MMAs from this one thread execute in issue
//              order, which is what lets an S buffer be reused once the P.V
//              that reads it was issued.
//   warps 2-5  softmax, one per TMEM lane quarter: load the Q rows into tensor
//              memory, then per tile each thread takes one query row and the
//              tile's 64 key columns; online base-2 softmax with a lazily
//              moved running max (O is rescaled only when the max grows by
//              more than 2^8); epilogue divides by the row sum and stores the
//              output (or a split partial).
// Every wait is bounded (tc::mbar_wait); a timeout sets FLARE_DEV_WAIT_TIMEOUT,
// the CTA stops issuing work, writes nothing more, frees its TMEM and exits.
#include <cudaTypedefs.h>

#include "common.cuh"
#include "kernels.h"
#include "tc.cuh"

namespace flare {

namespace {

constexpr int kTileN = 64;     // keys per tile
constexpr int kRowsM = 128;    // query rows per work item (TMEM lanes)
constexpr int kSoftmaxThreads = 128;  // warps 2-5, one per TMEM lane quarter
constexpr int kVWarp = 6;             // V producer
constexpr int kFixWarp = 7;           // zeroes the V rows past a prefix end
constexpr int kThreadsTC = 256;       // K producer, MMA issuer, 4 softmax warps, V producer, fixer
constexpr float kRescaleThreshold = 8.0f;  // log2 units

struct TcMaps {
  CUtensorMap kblk;   // (D, Hkv, B, R)          box (64, 1, 64, 1)
  CUtensorMap vblk;
  CUtensorMap kpool;  // (D, p, Hkv, num_pages)  box (64, min(p,64), 1, 1)
  CUtensorMap vpool;
};

template <int D>
struct TcCfg {
  static constexpr int kChunks = D / 64;
  static constexpr int kKVBytes = kChunks * kTileN * 128;  // one K (or V) tile
  // K and V rings fill shared memory: a tile's load takes about a microsecond
  // from issue to arrival, so the depth of the rings sets the tile rate.
  static constexpr int kKStages = D == 256 ? 3 : (D == 128 ? 6 : 8);  // K ring depth
  static constexpr int kVStages = D == 256 ? 4 : (D == 128 ? 7 : 8);  // V ring depth
  static constexpr int kSmem = (kKStages + kVStages) * kKVBytes;
  // tensor memory: O [0, D), Q as bf16 pairs [D, D + D/2), S/P buffers after
  static constexpr int kQCol = D;
  static constexpr int kSCol = D + D / 2;
  static constexpr int kSBuf = (kSCol + 3 * kTileN) <= 512 ? 3 : 2;  // S/P buffers
  static constexpr int kTmemCols = (kSCol + kSBuf * kTileN) > 256 ? 512 : 256;
};

struct TcShared {
  uint64_t k_full[8], v_full[8], k_empty[8], v_empty[8];
  uint64_t s_full[3], p_full[3], pv_done[3];
  uint64_t q_ready;   // a work item's Q rows are in tensor memory (one phase per item)
  uint64_t o_final;   // a work item's last P.V has completed
  uint64_t o_free;    // a work item's O has been read out (the next item may overwrite it)
  uint64_t v_fix[8];  // per V slot: a partial prefix tile's V rows past the prefix end are zeroed
  uint32_t tmem_base;
  int abort_flag;
  int last_split;     // this CTA merges the split partials of its row tile
  int v_issued;       // V tiles whose loads the V producer has issued (running count)
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

// One work item: query rows mtile*128 .. of (request r, kv head kvh) against
// prefix split `split`: prefix tiles j0 .. j0 + n_pref_here - 1, then (last
// split only) the tile holding the block's own keys.
struct TcWork {
  int r, kvh, mtile, split, item, P;
  int j0, n_pref_here, n_tiles, j_part;
};

// Work item `idx` of the flat list: (row tile, kv head) fastest, then the
// valid work units (request, prefix split) in longest-first order.
__device__ __forceinline__ TcWork tc_work(const SoftmaxParams& p, int n_mt, int idx) {
  TcWork w;
  w.mtile = idx % n_mt;
  w.kvh = (idx / n_mt) % p.Hkv;
  const int unit = p.order[idx / (n_mt * p.Hkv)];
  w.r = unit / p.n_split;
  w.split = unit % p.n_split;
  w.item = w.r * p.Hkv + w.kvh;
  w.P = p.prefix_len[w.r];
  const int n_pref = (w.P + kTileN - 1) / kTileN;
  const int tps = p.split_len / kTileN;
  w.j0 = w.split * tps;
  const int j1 = min(n_pref, w.j0 + tps);
  w.n_pref_here = max(0, j1 - w.j0);
  w.n_tiles = w.n_pref_here + (w.split == p.n_split - 1 ? 1 : 0);
  // the last prefix tile when the prefix ends inside it (its V rows past the
  // end are zeroed), else -1
  w.j_part = (w.n_pref_here > 0 && j1 == n_pref && (w.P % kTileN) != 0) ? w.n_pref_here - 1 : -1;
  return w;
}

}  // namespace

// Merge of the split partials of one row tile (rows mtile*128 ..) of one
// (request, kv head): out = sum_s w_s o_s with w_s = exp(lse_s - lse) and
// lse = log sum_s exp(lse_s) (the splits' partial outputs are already
// normalised by their own row sums).  The weights go to shared memory first
// (one thread per row); then every thread combines 8 (row, 4-column) pieces at
// a time with all their loads in flight.  All threads of the CTA call this;
// `wts` holds 128 * n_split floats.
template <int D>
__device__ void merge_splits(const SoftmaxParams& p, int item, int r, int kvh, int mtile,
                             float* wts) {
  const int M = p.B * p.G;
  const int ns = p.n_split;
  const int m0 = mtile * kRowsM;
  const int rows = min(kRowsM, M - m0);
  const size_t base = (size_t)item * ns * M + m0;  // row i of split s at base + s * M + i
  for (int i = threadIdx.x; i < rows; i += blockDim.x) {
    float mx = -INFINITY;
    for (int s = 0; s < ns; ++s) mx = fmaxf(mx, p.ws_lse[base + (size_t)s * M + i]);
    float den = 0.f;
    for (int s = 0; s < ns; ++s) {
      const float l = p.ws_lse[base + (size_t)s * M + i];
      const float e = l == -INFINITY ? 0.f : expf(l - mx);
      wts[i * ns + s] = e;
      den += e;
    }
    const float inv = 1.f / den;
    for (int s = 0; s < ns; ++s) wts[i * ns + s] *= inv;
    const int m = m0 + i, t = m / p.G, g = m % p.G;
    if (p.lse) p.lse[((size_t)r * p.B + t) * p.Hq + kvh * p.G + g] = mx + logf(den);
  }
  __syncthreads();
  constexpr int kC = D / 4;  // 4-column pieces per row
  constexpr int kBatch = 8;
  const int n_items = rows * kC;
  for (int i0 = threadIdx.x; i0 < n_items; i0 += kBatch * blockDim.x) {
    float4 acc[kBatch];
#pragma unroll
    for (int k = 0; k < kBatch; ++k) acc[k] = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int s = 0; s < ns; ++s) {
      float4 o[kBatch];
#pragma unroll
      for (int k = 0; k < kBatch; ++k) {
        const int it = i0 + k * blockDim.x;
        o[k] = it < n_items ? *reinterpret_cast<const float4*>(
                                  p.ws_o + (base + (size_t)s * M + it / kC) * D + (it % kC) * 4)
                            : make_float4(0.f, 0.f, 0.f, 0.f);
      }
#pragma unroll
      for (int k = 0; k < kBatch; ++k) {
        const int it = i0 + k * blockDim.x;
        const float w = it < n_items ? wts[(it / kC) * ns + s] : 0.f;
        acc[k].x = fmaf(w, o[k].x, acc[k].x);
        acc[k].y = fmaf(w, o[k].y, acc[k].y);
        acc[k].z = fmaf(w, o[k].z, acc[k].z);
        acc[k].w = fmaf(w, o[k].w, acc[k].w);
      }
    }
#pragma unroll
    for (int k = 0; k < kBatch; ++k) {
      const int it = i0 + k * blockDim.x;
      if (it >= n_items) continue;
      const int m = m0 + it / kC, t = m / p.G, g = m % p.G;
      const size_t orow = ((size_t)r * p.B + t) * p.Hq + kvh * p.G + g;
      __nv_bfloat162 lo = __floats2bfloat162_rn(acc[k].x, acc[k].y);
      __nv_bfloat162 hi = __floats2bfloat162_rn(acc[k].z, acc[k].w);
      *reinterpret_cast<uint2*>(static_cast<__nv_bfloat16*>(p.out) + orow * D + (it % kC) * 4) =
          make_uint2(*reinterpret_cast<uint32_t*>(&lo), *reinterpret_cast<uint32_t*>(&hi));
    }
  }
}

// Publishes this CTA's split partial and, if it is the last split of its row
// tile to finish, merges them all (all threads of the CTA call this).
template <int D>
__device__ void finish_split(const SoftmaxParams& p, int item, int r, int kvh, int mtile,
                             int n_mt, int* last_flag, float* wts) {
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0)
    *last_flag = atomicAdd(&p.counters[(size_t)item * n_mt + mtile], 1) == p.n_split - 1;
  __syncthreads();
  if (*last_flag) {
    __threadfence();
    merge_splits<D>(p, item, r, kvh, mtile, wts);
  }
}

// Validation and longest-first order of the work units u = (request r, prefix
// split), on one CTA:
//  - a request whose prefix length is out of range or whose prefix uses a page
//    id outside [0, num_pages) is flagged in the status word and left out of
//    the order (its outputs stay untouched);
//  - the other units are counting-sorted by their tile count (keys capped at
//    4095 tiles), longest first; *n_valid receives their number.
// Units with equal counts come in any order; each unit writes its own
// outputs, so the results do not depend on it.  Also zeroes the split-merge
// counters.
constexpr int kOrderThreads = 1024;
constexpr int kOrderKeys = 4 * kOrderThreads;

__global__ void __launch_bounds__(kOrderThreads) softmax_order_kernel(SoftmaxParams p) {
  __shared__ int start[kOrderKeys];
  __shared__ int wsum[kOrderThreads / 32];
  __shared__ int n_valid;
  const int U = p.R * p.n_split;
  const int tps = p.split_len / kTileN;
  const int t = threadIdx.x;
  const int nw = (p.R + 31) / 32;
  const long long prefix_cap = (long long)p.max_pages * p.page_size;
  for (int i = t; i < kOrderKeys; i += kOrderThreads) start[i] = 0;
  for (int i = t; i < nw; i += kOrderThreads) p.bad_mask[i] = 0u;
  if (p.counters) {
    const int n_cnt = p.R * p.Hkv * ((p.B * p.G + kRowsM - 1) / kRowsM);
    for (int i = t; i < n_cnt; i += kOrderThreads) p.counters[i] = 0;
  }
  if (t == 0) n_valid = 0;
  __syncthreads();
  for (int r = t; r < p.R; r += kOrderThreads) {
    const int P = p.prefix_len[r];
    if (P < 0 || P > prefix_cap) {
      atomicOr(&p.bad_mask[r >> 5], 1u << (r & 31));
      flag(p.dev_status, FLARE_DEV_BAD_PREFIX_LEN);
    }
  }
  // page ids in use: eight table entries per thread in flight at a time
  const long long n_entries = (long long)p.R * p.max_pages;
  constexpr int kIn = 8;
  for (long long i0 = t; i0 < n_entries; i0 += (long long)kIn * kOrderThreads) {
    int id[kIn], rr[kIn];
    bool used[kIn];
#pragma unroll
    for (int u = 0; u < kIn; ++u) {
      const long long i = i0 + (long long)u * kOrderThreads;
      used[u] = false;
      rr[u] = 0;
      id[u] = 0;
      if (i < n_entries) {
        const int r = (int)(i / p.max_pages);
        const int pg = (int)(i - (long long)r * p.max_pages);
        const int P = p.prefix_len[r];
        used[u] = P >= 0 && P <= prefix_cap && (long long)pg * p.page_size < P;
        rr[u] = r;
        id[u] = p.page_table[i];
      }
    }
#pragma unroll
    for (int u = 0; u < kIn; ++u) {
      if (used[u] && (id[u] < 0 || id[u] >= p.num_pages)) {
        atomicOr(&p.bad_mask[rr[u] >> 5], 1u << (rr[u] & 31));
        flag(p.dev_status, FLARE_DEV_BAD_PAGE);
      }
    }
  }
  __syncthreads();
  auto key_of = [&](int u) -> int {
    const int r = u / p.n_split, split = u % p.n_split;
    if (p.bad_mask[r >> 5] & (1u << (r & 31))) return -1;
    const int P = p.prefix_len[r];
    const int n_pref = (P + kTileN - 1) / kTileN;
    const int j0 = split * tps;
    const int here = max(0, min(n_pref, j0 + tps) - j0);
    return min(here + (split == p.n_split - 1 ? 1 : 0), kOrderKeys - 1);
  };
  for (int u = t; u < U; u += kOrderThreads) {
    const int k = key_of(u);
    if (k >= 0) {
      atomicAdd(&start[k], 1);
      atomicAdd(&n_valid, 1);
    }
  }
  __syncthreads();
  // start[k] = number of valid units with a larger key; thread t owns the
  // keys at descending positions 4t .. 4t+3
  int v[4], sum = 0;
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    v[e] = start[kOrderKeys - 1 - (4 * t + e)];
    sum += v[e];
  }
  int incl = sum;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int n = __shfl_up_sync(0xffffffffu, incl, o);
    if ((t & 31) >= o) incl += n;
  }
  if ((t & 31) == 31) wsum[t >> 5] = incl;
  __syncthreads();
  if (t < 32) {
    const int w = wsum[t];
    int wi = w;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int n = __shfl_up_sync(0xffffffffu, wi, o);
      if (t >= o) wi += n;
    }
    wsum[t] = wi - w;
  }
  __syncthreads();
  int run = wsum[t >> 5] + incl - sum;
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    start[kOrderKeys - 1 - (4 * t + e)] = run;
    run += v[e];
  }
  __syncthreads();
  for (int u = t; u < U; u += kOrderThreads) {
    const int k = key_of(u);
    if (k >= 0) p.order[atomicAdd(&start[k], 1)] = u;
  }
  if (t == 0) *p.n_valid = n_valid;
}

// The attention kernel.  Unsplit prefixes (n_split == 1): one CTA per SM walks
// the work items in snake order over the CTAs (round k takes items k*G ..
// k*G + G - 1, in reverse on odd rounds), so that tensor memory, barriers and
// tensor maps are set up once and the next item's loads and S products
// overlap the current item's epilogue.  Split prefixes: one CTA per work item,
// and the last split of a row tile to finish merges the partials.
template <int D>
__global__ void __launch_bounds__(kThreadsTC, 1)
    softmax_tc_kernel(const __grid_constant__ TcMaps maps, SoftmaxParams p) {
  using C = TcCfg<D>;
  constexpr int kSB = C::kSBuf;
  extern __shared__ uint8_t smem_raw[];
  __shared__ TcShared sh;
  uint8_t* base = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint8_t* Ks = base;
  uint8_t* Vs = Ks + C::kKStages * C::kKVBytes;

  const int M = p.B * p.G;
  const int n_mt = (M + kRowsM - 1) / kRowsM;
  const int n_items = n_mt * p.Hkv * *p.n_valid;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const bool split_mode = p.n_split > 1;
  // k-th work item of this CTA, or -1
  auto item_of = [&](int k) -> int {
    const int G = gridDim.x, b = blockIdx.x;
    if (split_mode) return (k == 0 && b < n_items) ? b : -1;
    const int idx = k * G + ((k & 1) ? G - 1 - b : b);
    return idx < n_items ? idx : -1;
  };
  const int idx0 = item_of(0);
  if (idx0 < 0) return;
  if (split_mode) {
    const TcWork w = tc_work(p, n_mt, idx0);
    if (w.n_tiles == 0) {  // empty split: mark its partial as empty for the merge
      const size_t ws_row0 = ((size_t)w.item * p.n_split + w.split) * M;
      for (int i = tid; i < kRowsM; i += blockDim.x) {
        const int m = w.mtile * kRowsM + i;
        if (m < M) p.ws_lse[ws_row0 + m] = -INFINITY;
      }
      finish_split<D>(p, w.item, w.r, w.kvh, w.mtile, n_mt, &sh.last_split,
                      reinterpret_cast<float*>(Ks));
      return;
    }
  }

  if (tid == 0) {
    sh.abort_flag = 0;
    sh.last_split = 0;
    sh.v_issued = 0;
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
    tc::mbar_init(&sh.q_ready, kSoftmaxThreads);
    tc::mbar_init(&sh.o_final, 1);
    tc::mbar_init(&sh.o_free, kSoftmaxThreads);
    for (int s = 0; s < C::kVStages; ++s) tc::mbar_init(&sh.v_fix[s], 1);
    tc::fence_mbar_init();
  }
  if (warp == 1) tc::tmem_alloc(&sh.tmem_base, C::kTmemCols);
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = sh.tmem_base;
  const uint32_t tmem_o = tmem;
  const uint32_t tmem_q = tmem + C::kQCol;
  const uint32_t tmem_s = tmem + C::kSCol;

  if (warp == 0 || warp == kVWarp) {
    // ------------------------------------------------------------ producers
    // warp 0 streams the K tiles and warp kVWarp the V tiles of every work
    // item of this CTA, each into its own ring (slot = running tile count mod
    // ring depth), so neither waits behind the other's slot.
    if (lane == 0) {
      const int kv = warp == 0 ? 0 : 1;
      const CUtensorMap* pool_map = kv ? &maps.vpool : &maps.kpool;
      const CUtensorMap* blk_map = kv ? &maps.vblk : &maps.kblk;
      tc::prefetch_tmap(pool_map);
      tc::prefetch_tmap(blk_map);
      const int box_rows = p.page_size < kTileN ? p.page_size : kTileN;
      const int ns = kv ? C::kVStages : C::kKStages;
      uint8_t* ring = kv ? Vs : Ks;
      bool ok = true;
      int g = 0;  // running tile count
      for (int k = 0; ok && !aborted(sh); ++k) {
        const int idx = item_of(k);
        if (idx < 0) break;
        const TcWork w = tc_work(p, n_mt, idx);
        for (int j = 0; j < w.n_tiles; ++j, ++g) {
          const int st = g % ns;
          const uint32_t ph = (uint32_t)(g / ns) & 1u;
          uint64_t* empty = kv ? &sh.v_empty[st] : &sh.k_empty[st];
          uint64_t* full = kv ? &sh.v_full[st] : &sh.k_full[st];
          uint8_t* dst = ring + st * C::kKVBytes;
          if (!tc::mbar_wait(empty, ph ^ 1u, &sh.abort_flag)) {
            ok = false;
            break;
          }
          if (j >= w.n_pref_here) {  // the block's own keys / values
            tc::mbar_expect_tx(full, C::kKVBytes);
            for (int c = 0; c < C::kChunks; ++c)
              tc::tma_load_4d(dst + c * (kTileN * 128), blk_map, full, c * 64, w.kvh, 0, w.r);
            if (kv) *reinterpret_cast<volatile int*>(&sh.v_issued) = g + 1;
            continue;
          }
          const int tok0 = (w.j0 + j) * kTileN;
          const int valid = min(kTileN, w.P - tok0);
          const int nbox = (valid + box_rows - 1) / box_rows;
          tc::mbar_expect_tx(full, (uint32_t)(C::kChunks * nbox * box_rows * 128));
          for (int bx = 0; bx < nbox; ++bx) {
            const int tok = tok0 + bx * box_rows;
            const int page = p.page_table[(size_t)w.r * p.max_pages + tok / p.page_size];
            const int row0 = tok % p.page_size;
            for (int c = 0; c < C::kChunks; ++c)
              tc::tma_load_4d(dst + c * (kTileN * 128) + bx * box_rows * 128, pool_map, full,
                              c * 64, row0, w.kvh, page);
          }
          if (kv) *reinterpret_cast<volatile int*>(&sh.v_issued) = g + 1;
        }
      }
      if (!ok) set_abort(sh, p.dev_status);
    }
  } else if (warp == kFixWarp) {
    // ------------------------------------------------------------ V fixer
    // The last prefix tile of an item ends inside the tile: its V rows past the
    // prefix end hold stale (possibly poisoned) cache rows.  Once its load has
    // landed they are zeroed, so that a zero probability never meets a NaN
    // (0 * NaN) in P.V; the MMA issuer waits for this instead of the load.
    // A warp of its own, so the V producer never stops to wait for a load.
    bool ok = true;
    int g = 0;  // running tile count
    for (int k = 0; ok && !aborted(sh); ++k) {
      const int idx = item_of(k);
      if (idx < 0) break;
      const TcWork w = tc_work(p, n_mt, idx);
      if (w.j_part >= 0) {
        const int gg = g + w.j_part;
        const int st = gg % C::kVStages;
        // Parity waits are exact only once the tile's load has been issued:
        // then the slot's previous load has been consumed, and its next one
        // needs the P.V that waits for this warp.  Until then, sleep-poll the
        // producer's count (bounded like every wait).
        bool issued = true;
        if (lane == 0) {
          const uint64_t t0 = tc::globaltimer_ns();
          while (*reinterpret_cast<volatile int*>(&sh.v_issued) <= gg) {
            if (aborted(sh) || tc::globaltimer_ns() - t0 > 2000000000ull) {
              issued = false;
              break;
            }
            __nanosleep(64);
          }
        }
        issued = __shfl_sync(0xffffffffu, issued, 0);
        if (!issued ||
            !warp_wait(&sh.v_full[st], (uint32_t)(gg / C::kVStages) & 1u, &sh.abort_flag)) {
          ok = false;
          break;
        }
        uint8_t* dst = Vs + st * C::kKVBytes;
        const int valid = w.P - (w.j0 + w.j_part) * kTileN;  // 1 .. kTileN - 1
        const int n16 = (kTileN - valid) * 8;                 // 16-byte pieces per chunk
        for (int c = 0; c < C::kChunks; ++c)
          for (int e = lane; e < n16; e += 32)
            *reinterpret_cast<uint4*>(dst + c * (kTileN * 128) + (valid + e / 8) * 128 +
                                      (e % 8) * 16) = make_uint4(0u, 0u, 0u, 0u);
        tc::fence_async_smem();
        __syncwarp();
        if (lane == 0) tc::mbar_arrive(&sh.v_fix[st]);
      }
      g += w.n_tiles;
    }
    if (!ok && lane == 0) set_abort(sh, p.dev_status);
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    // One thread waits and issues; operand descriptors advance by adding the
    // byte offset (>> 4) to the start-address field of a base descriptor.
    if (lane == 0) {
      const uint32_t id_s = tc::idesc_bf16(kRowsM, kTileN, false, false);
      const uint32_t id_o = tc::idesc_bf16(kRowsM, D, false, true);
      const uint64_t kdesc0 = tc::sdesc_sw128(tc::smem_u32(Ks), 16, 1024);
      const uint64_t vdesc0 = tc::sdesc_sw128(tc::smem_u32(Vs), kTileN * 128, 1024);
      bool ok = true;
      int g = 0;              // running tile count
      uint32_t fix_par = 0u;  // per V slot: parity of its next zeroed-partial-tile phase
      for (int k = 0; ok && !aborted(sh); ++k) {
        const int idx = item_of(k);
        if (idx < 0) break;
        const TcWork w = tc_work(p, n_mt, idx);
        if (!tc::mbar_wait(&sh.q_ready, (uint32_t)k & 1u, &sh.abort_flag)) {
          ok = false;
          break;
        }
        auto issue_pv = [&](int j) -> bool {
          const int gg = g + j;
          const int st = gg % C::kVStages;
          const int pb = gg % kSB;
          if (!tc::mbar_wait(&sh.p_full[pb], (uint32_t)(gg / kSB) & 1u, &sh.abort_flag))
            return false;
          // the first P.V of an item overwrites O: the previous item's O must be out
          if (j == 0 && k > 0 &&
              !tc::mbar_wait(&sh.o_free, (uint32_t)(k - 1) & 1u, &sh.abort_flag))
            return false;
          // a slot's partial tiles are in order: the next one can only be
          // loaded once the P.V issued after this wait has freed the slot
          bool ready;
          if (j == w.j_part) {
            ready = tc::mbar_wait(&sh.v_fix[st], (fix_par >> st) & 1u, &sh.abort_flag);
            fix_par ^= 1u << st;
          } else {
            ready = tc::mbar_wait(&sh.v_full[st], (uint32_t)(gg / C::kVStages) & 1u,
                                  &sh.abort_flag);
          }
          if (!ready) return false;
          tc::fence_after_sync();
          const uint64_t vd = vdesc0 + (uint64_t)((st * C::kKVBytes) >> 4);
#pragma unroll
          for (int kk = 0; kk < kTileN / 16; ++kk)
            mma_bf16_ts(tmem_o, tmem_s + pb * kTileN + kk * 8, vd + (uint64_t)(kk * (2048 >> 4)),
                        id_o, (j > 0 || kk > 0) ? 1u : 0u);
          tc::mma_commit(&sh.pv_done[pb]);
          tc::mma_commit(&sh.v_empty[st]);
          return true;
        };
        // S_j = Q K_j^T into S buffer (g + j) % kSB (Q from tensor memory)
        auto issue_s = [&](int j) -> bool {
          const int gg = g + j;
          const int st = gg % C::kKStages;
          const int sb = gg % kSB;
          if (!tc::mbar_wait(&sh.k_full[st], (uint32_t)(gg / C::kKStages) & 1u, &sh.abort_flag))
            return false;
          tc::fence_after_sync();
          const uint64_t kd = kdesc0 + (uint64_t)((st * C::kKVBytes) >> 4);
#pragma unroll
          for (int kk = 0; kk < D / 16; ++kk) {
            const int c = kk >> 2, off = (kk & 3) * 32;
            mma_bf16_ts(tmem_s + sb * kTileN, tmem_q + kk * 8,
                        kd + (uint64_t)((c * (kTileN * 128) + off) >> 4), id_s, kk > 0 ? 1u : 0u);
          }
          tc::mma_commit(&sh.s_full[sb]);
          tc::mma_commit(&sh.k_empty[st]);
          return true;
        };
        // Three S buffers: issue order S0, S1, S2, PV0, S3, PV1, ...: S_{j+2}
        // is queued before the P.V of tile j waits on its probabilities and
        // reuses the buffer of tile j-1, whose P.V was issued (and, in issue
        // order, executes) before it.  Two buffers: S0, S1, PV0, S2, PV1, ...:
        // S_{j+2} reuses the buffer of tile j, so it follows P_j V_j.  The
        // running tile count carries the buffers across work items.
        const int n = w.n_tiles;
        for (int j = 0; j < 2 && j < n && ok; ++j) ok = issue_s(j);
        for (int j = 0; j < n && ok; ++j) {
          if (kSB == 3) {
            if (j + 2 < n) ok = issue_s(j + 2);
            if (ok) ok = issue_pv(j);
          } else {
            ok = issue_pv(j);
            if (ok && j + 2 < n) ok = issue_s(j + 2);
          }
        }
        if (ok) tc::mma_commit(&sh.o_final);
        g += n;
      }
      if (!ok) set_abort(sh, p.dev_status);
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------ softmax warps
    // warp w reads TMEM lanes 32*(w%4).. (its 32 query rows) and all 64 key
    // columns of each tile
    const int quarter = warp & 3;
    const int row = quarter * 32 + lane;
    const uint32_t lane_off = (uint32_t)(quarter * 32) << 16;

    // Q row of work item w into tensor memory as bf16 pairs, the A operand of
    // S = Q K^T; rows past the block's B*G are zero
    auto load_q = [&](const TcWork& w) {
      const int m = w.mtile * kRowsM + row;
      const bool live = m < M;
      const int trow = live ? m / p.G : 0, g = m % p.G;
      const uint4* qrow = reinterpret_cast<const uint4*>(
          static_cast<const __nv_bfloat16*>(p.q) +
          (((size_t)w.r * p.B + trow) * p.Hq + w.kvh * p.G + g) * D);
      constexpr int kWords = D / 2;                          // TMEM columns of a row
      constexpr int kBatch = kWords < 64 ? kWords : 64;      // columns per batch of loads
#pragma unroll 1
      for (int c0 = 0; c0 < kWords; c0 += kBatch) {
        uint32_t q[kBatch];
#pragma unroll
        for (int q4 = 0; q4 < kBatch / 4; ++q4) {
          const uint4 v = live ? qrow[(c0 / 4) + q4] : make_uint4(0u, 0u, 0u, 0u);
          q[4 * q4] = v.x;
          q[4 * q4 + 1] = v.y;
          q[4 * q4 + 2] = v.z;
          q[4 * q4 + 3] = v.w;
        }
#pragma unroll
        for (int c = 0; c < kBatch; c += 16)
          tmem_st16(tmem_q + lane_off + c0 + c, *reinterpret_cast<uint32_t(*)[16]>(&q[c]));
      }
      tmem_st_wait();
      tc::fence_before_sync();
      tc::mbar_arrive(&sh.q_ready);
    };

    bool ok = true;
    int g = 0;  // running tile count
    int idx = idx0;
    TcWork w = tc_work(p, n_mt, idx);
    load_q(w);
    for (int k = 0; idx >= 0; ++k) {
      const int m = w.mtile * kRowsM + row;
      const int trow = m / p.G;
      // token-causal block row: the state-update pass, or an anchor / verify
      // row of the per-row encoding (padding rows past the block read none)
      const bool causal_row =
          p.row_type ? (trow < p.B && p.row_type[(size_t)w.r * p.row_type_stride + trow] == 0)
                     : p.causal != 0;
      float m_run = -INFINITY, l_run = 0.f;
      for (int j = 0; j < w.n_tiles; ++j) {
        const int gg = g + j;
        const int sb = gg % kSB;
        if (!warp_wait(&sh.s_full[sb], (uint32_t)(gg / kSB) & 1u, &sh.abort_flag)) {
          ok = false;
          break;
        }
        tc::fence_after_sync();
        const uint32_t sbuf = tmem_s + lane_off + sb * kTileN;
        uint32_t sr[kTileN];
#pragma unroll
        for (int c = 0; c < kTileN; c += 16)
          tc::tmem_ld16(sbuf + c, *reinterpret_cast<uint32_t(*)[16]>(&sr[c]));
        tc::tmem_ld_wait();

        const bool blk = j >= w.n_pref_here;
        const int valid = blk ? p.B : min(kTileN, w.P - (w.j0 + j) * kTileN);
        const bool full = !blk && valid == kTileN;  // prefix tile: no mask at all
        const int lim = full ? kTileN : ((blk && causal_row) ? min(valid, trow + 1) : valid);
        // tile maximum of the raw scores (scale >= 0 keeps the order)
        float mx[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
        for (int c = 0; c < kTileN; ++c)
          if (full || c < lim) mx[c & 3] = fmaxf(mx[c & 3], __uint_as_float(sr[c]));
        const float mt = fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3]));
        const float m_new = fmaxf(m_run, mt * p.scale_log2);
        const bool need = (j == 0) || (m_new > m_run + kRescaleThreshold);
        const bool warp_rescale = __any_sync(0xffffffffu, need);
        float m_use = m_run;
        if (warp_rescale) m_use = (j == 0 || m_new > m_run) ? m_new : m_run;
        const float corr = (j == 0) ? 0.f : tc::ex2(m_run - m_use);
        const float neg_m = -m_use;
        float sum0 = 0.f, sum1 = 0.f;
        uint32_t pk[kTileN / 2];
        if (full) {
#pragma unroll
          for (int c = 0; c < kTileN; c += 2) {
            const float p0 = tc::ex2(fmaf(__uint_as_float(sr[c]), p.scale_log2, neg_m));
            const float p1 = tc::ex2(fmaf(__uint_as_float(sr[c + 1]), p.scale_log2, neg_m));
            sum0 += p0;
            sum1 += p1;
            __nv_bfloat162 h2 = __floats2bfloat162_rn(p0, p1);
            pk[c / 2] = *reinterpret_cast<uint32_t*>(&h2);
          }
        } else {
#pragma unroll
          for (int c = 0; c < kTileN; c += 2) {
            const float p0 =
                c < lim ? tc::ex2(fmaf(__uint_as_float(sr[c]), p.scale_log2, neg_m)) : 0.f;
            const float p1 =
                c + 1 < lim ? tc::ex2(fmaf(__uint_as_float(sr[c + 1]), p.scale_log2, neg_m))
                            : 0.f;
            sum0 += p0;
            sum1 += p1;
            __nv_bfloat162 h2 = __floats2bfloat162_rn(p0, p1);
            pk[c / 2] = *reinterpret_cast<uint32_t*>(&h2);
          }
        }
        const float sum = sum0 + sum1;
        l_run = (j == 0) ? sum : l_run * corr + sum;
        // rescale O when the running max moved (the P.V of the previous tile done)
        if (warp_rescale && j >= 1) {
          const int pb = (gg - 1) % kSB;
          if (!warp_wait(&sh.pv_done[pb], (uint32_t)((gg - 1) / kSB) & 1u, &sh.abort_flag)) {
            ok = false;
            break;
          }
          tc::fence_after_sync();
#pragma unroll 1
          for (int c = 0; c < D; c += 16) {
            uint32_t o[16];
            tc::tmem_ld16(tmem_o + lane_off + c, o);
            tc::tmem_ld_wait();
#pragma unroll
            for (int i = 0; i < 16; ++i) o[i] = __float_as_uint(__uint_as_float(o[i]) * corr);
            tmem_st16(tmem_o + lane_off + c, o);
          }
        }
        m_run = m_use;
        // P (bf16 pairs) over the first 32 columns of the S buffer
#pragma unroll
        for (int c = 0; c < kTileN / 2; c += 16)
          tmem_st16(sbuf + c, *reinterpret_cast<uint32_t(*)[16]>(&pk[c]));
        tmem_st_wait();
        tc::fence_before_sync();
        tc::mbar_arrive(&sh.p_full[sb]);
      }
      g += w.n_tiles;
      if (ok && aborted(sh)) ok = false;
      // the next item's Q can go into tensor memory now: every S product of
      // this item has completed
      const int idx_next = ok ? item_of(k + 1) : -1;
      TcWork wn = w;
      if (idx_next >= 0) {
        wn = tc_work(p, n_mt, idx_next);
        load_q(wn);
      }
      // epilogue: O / l (or the split partial) and the log-sum-exp
      if (ok && !warp_wait(&sh.o_final, (uint32_t)k & 1u, &sh.abort_flag)) ok = false;
      if (!ok) {
        set_abort(sh, p.dev_status);
        break;
      }
      tc::fence_after_sync();
      const bool write = m < M;
      const float inv = l_run > 0.f ? 1.f / l_run : 0.f;
      const int gq = m % p.G;
      const size_t orow = (((size_t)w.r * p.B + trow) * p.Hq + w.kvh * p.G + gq);
      const size_t ws_row = ((size_t)w.item * p.n_split + w.split) * M + m;
#pragma unroll 1
      for (int c = 0; c < D; c += 16) {
        uint32_t o[16];
        tc::tmem_ld16(tmem_o + lane_off + c, o);
        tc::tmem_ld_wait();
        if (!write) continue;
        if (!split_mode) {
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
          float4* dst = reinterpret_cast<float4*>(p.ws_o + ws_row * D + c);
#pragma unroll
          for (int i = 0; i < 4; ++i)
            dst[i] = make_float4(__uint_as_float(o[4 * i]) * inv, __uint_as_float(o[4 * i + 1]) * inv,
                                 __uint_as_float(o[4 * i + 2]) * inv,
                                 __uint_as_float(o[4 * i + 3]) * inv);
        }
      }
      if (write) {
        const float lse = l_run > 0.f ? (m_run + __log2f(l_run)) * 0.6931471805599453f : -INFINITY;
        if (!split_mode) {
          if (p.lse) p.lse[orow] = lse;
        } else {
          p.ws_lse[ws_row] = lse;
        }
      }
      tc::fence_before_sync();
      tc::mbar_arrive(&sh.o_free);
      idx = idx_next;
      w = wn;
    }
    if (!ok) set_abort(sh, p.dev_status);
  }
  tc::fence_before_sync();
  __syncthreads();
  if (warp == 1) {
    tc::fence_after_sync();
    tc::tmem_dealloc(tmem, C::kTmemCols);
  }
  // a CTA that gave up wrote no partial: its row tile is never merged
  if (split_mode && !aborted(sh)) {  // the K/V rings are free: merge weights go there
    const TcWork w = tc_work(p, n_mt, idx0);
    finish_split<D>(p, w.item, w.r, w.kvh, w.mtile, n_mt, &sh.last_split,
                    reinterpret_cast<float*>(Ks));
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
  if (!p.order || !p.n_valid || !p.bad_mask || plan.num_ctas <= 0) return cudaErrorInvalidValue;
  softmax_order_kernel<<<1, kOrderThreads, 0, stream>>>(p);
  note_launches(1);
  err = cudaGetLastError();
  if (err != cudaSuccess) return err;
  softmax_tc_kernel<D><<<(unsigned)plan.num_ctas, kThreadsTC, smem, stream>>>(maps, p);
  note_launches(1);
  return cudaGetLastError();
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
