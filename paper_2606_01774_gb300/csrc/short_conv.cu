// Two-stream causal ShortConv of a block, serving form (appendix "1D Causal
// ShortConv: implementation routes", Eq. short-conv-noisy).
//
// A depthwise causal convolution of width W <= 4: block row l reads its own
// block rows l - i for lags that stay inside the block and the committed conv
// state (the last W - 1 clean tokens before the block, a raw slice of the
// clean stream) for lags that cross the block start; then bias and SiLU.
//
// The kernel is a pure stream (each input byte is used W times from on-chip
// memory), so it is built to keep HBM busy: persistent CTAs, one per SM, walk
// work items (request, 4 KiB channel slab, chunk of up to 8 block rows; small
// items keep the last wave short).  A producer warp stages each item's rows --
// the chunk plus the W - 1 rows before it, from the block or, for the first
// chunk, from the conv state -- in shared memory: when the channels tile by
// 512 bytes as one tensor-map box of (512 bytes x 8) x rows per item (the
// state rows of a first chunk as bulk copies), else one bulk copy per row;
// completion counted on the stage's full barrier (a few large copies keep far
// more bytes in flight per SM than a copy per 4 KiB row); four stages, so three
// items' rows are in flight while 512 compute threads convolve the current
// one, a thread per 8 bytes of channels (4 bf16 or 2 fp32) down the whole
// chunk with its filter taps and a sliding window in registers, writing
// 8-byte outputs coalesced across the slab; they release the stage on its
// empty barrier.
// The arithmetic runs on fp32 pairs (packed f32x2 multiply-add); the SiLU's
// exponentials run on the special-function unit, its reciprocals one per four
// channels (the special-function unit is the busiest pipe here).  With a grid that
// is a multiple of the slab count every CTA keeps one slab, so the filter taps
// are loaded once, while the first rows are on their way.
// The state commit (last W - 1 rows of old state ++ accepted rows) is a bit
// copy done by the threads of each slab's first chunk, the only ones that read
// the old state of those channels, after their reads.
#include <cudaTypedefs.h>
#include <string.h>

#include "common.cuh"
#include "kernels.h"
#include "tc.cuh"

namespace flare {

namespace {
constexpr int kConvThreads = 512;             // a thread per 8-byte column
constexpr int kColBytes = 8;
constexpr int kSlabBytes = kConvThreads * kColBytes;  // 4 KiB of channels per item
constexpr int kChunkRows = 8;                  // block rows per item
constexpr int kMaxStageRows = kChunkRows + 3;  // with the W - 1 <= 3 rows before the chunk
constexpr int kStageBytes = kMaxStageRows * kSlabBytes;
constexpr int kStages = 4;
constexpr size_t kConvSmem = kStages * (size_t)kStageBytes;

struct ConvItem {
  int r, slab, chunk;
};

// The block as (512-byte column blocks, row) tiles: x viewed as
// [R B rows][C / D0 blocks][D0] with D0 = 512 / sizeof(T); boxes of 8 blocks
// (one slab) by kChunkRows + W - 1 rows (a chunk and the rows before it) and
// by kChunkRows rows (a first chunk, whose earlier rows are the conv state).
struct ConvMaps {
  CUtensorMap x_halo, x_first;
  int use;  // 0: the channels do not tile; one bulk copy per row
};

// The slab varies fastest, so that with a grid that is a multiple of the slab
// count every CTA keeps one slab (and its filter taps) for all its items.
__device__ __forceinline__ ConvItem conv_item(int idx, int n_slabs, int n_chunks) {
  ConvItem it;
  it.slab = idx % n_slabs;
  it.chunk = (idx / n_slabs) % n_chunks;
  it.r = idx / (n_slabs * n_chunks);
  return it;
}

__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
__device__ __forceinline__ float rcp_approx(float x) {
  float y;
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// 8 bytes of T as V / 2 fp32 pairs (bf16 widens exactly: its bits are the
// high half of the fp32 pattern)
template <typename T>
__device__ __forceinline__ void unpack8(const uint2& raw, uint64_t* f) {
  if constexpr (sizeof(T) == 2) {
    f[0] = f2(__uint_as_float(raw.x << 16), __uint_as_float(raw.x & 0xffff0000u));
    f[1] = f2(__uint_as_float(raw.y << 16), __uint_as_float(raw.y & 0xffff0000u));
  } else {
    f[0] = f2(__uint_as_float(raw.x), __uint_as_float(raw.y));
  }
}

template <typename T>
__device__ __forceinline__ uint2 pack8(const uint64_t* f) {
  if constexpr (sizeof(T) == 2) {
    uint32_t u[2];
#pragma unroll
    for (int k = 0; k < 2; ++k) {
      float lo, hi;
      f2_split(f[k], lo, hi);
      __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
      u[k] = *reinterpret_cast<uint32_t*>(&h);
    }
    return make_uint2(u[0], u[1]);
  } else {
    float lo, hi;
    f2_split(f[0], lo, hi);
    return make_uint2(__float_as_uint(lo), __float_as_uint(hi));
  }
}

// A request is valid when its slot and (for a committing call) its accepted
// length are in range; otherwise its items are skipped.
__device__ __forceinline__ int conv_check(const ConvParams& p, int r) {
  const int slot = p.state_slot[r];
  if (slot < 0 || slot >= p.nslots) return FLARE_DEV_BAD_SLOT;
  if (p.accept_len) {
    const int n = p.accept_len[r];
    if (n < 0 || n > p.B) return FLARE_DEV_BAD_ACCEPT_LEN;
  }
  return 0;
}
}  // namespace

template <typename T, int W>
__global__ void __launch_bounds__(kConvThreads + 32, 1)
    short_conv_kernel(const __grid_constant__ ConvMaps maps, ConvParams p) {
  constexpr int E = sizeof(T);
  constexpr int V = kColBytes / E;  // channels per thread
  constexpr int P = V / 2;          // fp32 pairs per thread
  constexpr int H = W - 1;          // rows before a chunk
  extern __shared__ __align__(128) uint8_t conv_smem[];
  __shared__ uint64_t full[kStages], empty[kStages];
  __shared__ int st_bad[kStages], st_slot[kStages], st_n[kStages];
  __shared__ int abort_flag, n_issued;

  const int tid = threadIdx.x;
  const size_t row_bytes = (size_t)p.C * E;
  const int n_slabs = (int)((row_bytes + kSlabBytes - 1) / kSlabBytes);
  const int n_chunks = (p.B + kChunkRows - 1) / kChunkRows;
  const int n_items = p.R * n_slabs * n_chunks;
  const char* xg = static_cast<const char*>(p.x);
  char* sg = static_cast<char*>(p.conv_state);

  if (tid == 0) {
    for (int s = 0; s < kStages; ++s) {
      tc::mbar_init(&full[s], 1);
      tc::mbar_init(&empty[s], kConvThreads);
    }
    abort_flag = 0;
    n_issued = 0;
    tc::fence_mbar_init();
  }
  __syncthreads();

  if (tid >= kConvThreads) {
    // producer warp: lane 0 stages every item of this CTA with the request's
    // slot, accepted length and validity
    if (tid == kConvThreads) {
      if (maps.use) {
        tc::prefetch_tmap(&maps.x_halo);
        tc::prefetch_tmap(&maps.x_first);
      }
      int k = 0;
      for (int idx = blockIdx.x; idx < n_items; idx += gridDim.x, ++k) {
        const int st = k % kStages;
        // the stage is free once every compute thread is done with item k - kStages
        if (k >= kStages &&
            !tc::mbar_wait(&empty[st], (uint32_t)((k / kStages) & 1) ^ 1u, &abort_flag)) {
          flag(p.dev_status, FLARE_DEV_WAIT_TIMEOUT);
          abort_flag = 1;
          break;
        }
        const ConvItem it = conv_item(idx, n_slabs, n_chunks);
        const size_t off = (size_t)it.slab * kSlabBytes;
        const uint32_t bytes = (uint32_t)min((size_t)kSlabBytes, row_bytes - off);
        const int l0 = it.chunk * kChunkRows;
        const int rows = min(kChunkRows, p.B - l0);
        uint8_t* dst = conv_smem + (size_t)st * kStageBytes;
        const int bad = conv_check(p, it.r);
        st_bad[st] = bad;
        n_issued = k + 1;
        if (bad) {  // nothing to load; the stage completes empty
          tc::mbar_arrive(&full[st]);
          continue;
        }
        const int slot = p.state_slot[it.r];
        st_slot[st] = slot;
        st_n[st] = p.accept_len ? p.accept_len[it.r] : -1;
        tc::fence_async_smem();
        if (maps.use) {
          // a box always lands whole (rows past the block are read or zero
          // filled and never used); the state rows as bulk copies
          const int row0 = it.r * p.B + l0;
          if (it.chunk == 0) {
            tc::mbar_expect_tx(&full[st], bytes * (uint32_t)H + (uint32_t)(kSlabBytes * kChunkRows));
            for (int j = 0; j < H; ++j)
              tc::bulk_load(dst + (size_t)j * kSlabBytes,
                            sg + ((size_t)slot * H + j) * row_bytes + off, bytes, &full[st]);
            tc::tma_load_3d(dst + (size_t)H * kSlabBytes, &maps.x_first, &full[st], 0,
                            it.slab * 8, row0);
          } else {
            tc::mbar_expect_tx(&full[st], (uint32_t)(kSlabBytes * (kChunkRows + H)));
            tc::tma_load_3d(dst, &maps.x_halo, &full[st], 0, it.slab * 8, row0 - H);
          }
        } else {
          tc::mbar_expect_tx(&full[st], bytes * (uint32_t)(H + rows));
          for (int j = 0; j < H + rows; ++j) {
            const int pos = l0 - H + j;
            const char* src = pos >= 0 ? xg + ((size_t)it.r * p.B + pos) * row_bytes + off
                                       : sg + ((size_t)slot * H + (H + pos)) * row_bytes + off;
            tc::bulk_load(dst + (size_t)j * kSlabBytes, src, bytes, &full[st]);
          }
        }
      }
    }
  } else {
    const int col = tid;
    uint64_t w2[P][W], b2[P];
    int cur_slab = -1;
    // filter taps and bias of this thread's channels, paired (loaded while the
    // first item's rows are on their way, and again only if the slab changes)
    auto load_taps = [&](int slab) {
      cur_slab = slab;
      const size_t off = (size_t)slab * kSlabBytes + (size_t)col * kColBytes;
      if (off >= row_bytes) return;
      const int c0 = (int)(off / E);
      const float2* w2p = reinterpret_cast<const float2*>(p.weight + (size_t)c0 * W);
      float wf[V * W];
#pragma unroll
      for (int q = 0; q < V * W / 2; ++q) {
        const float2 v = __ldg(w2p + q);
        wf[2 * q] = v.x;
        wf[2 * q + 1] = v.y;
      }
      float bf[V];
#pragma unroll
      for (int v = 0; v < V; ++v) bf[v] = 0.f;
      if (p.bias) {
        const float2* b2p = reinterpret_cast<const float2*>(p.bias + c0);
#pragma unroll
        for (int q = 0; q < V / 2; ++q) {
          const float2 v = __ldg(b2p + q);
          bf[2 * q] = v.x;
          bf[2 * q + 1] = v.y;
        }
      }
#pragma unroll
      for (int q = 0; q < P; ++q) {
#pragma unroll
        for (int i = 0; i < W; ++i) w2[q][i] = f2(wf[2 * q * W + i], wf[(2 * q + 1) * W + i]);
        b2[q] = f2(bf[2 * q], bf[2 * q + 1]);
      }
    };
    if ((int)blockIdx.x < n_items) load_taps(conv_item(blockIdx.x, n_slabs, n_chunks).slab);
    const uint64_t neg_log2e = f2(-1.4426950408889634f, -1.4426950408889634f);

    int k = 0;
    for (int idx = blockIdx.x; idx < n_items; idx += gridDim.x, ++k) {
      const int st = k % kStages;
      if (!tc::mbar_wait(&full[st], (uint32_t)(k / kStages) & 1u, &abort_flag)) {
        if (tid == 0) flag(p.dev_status, FLARE_DEV_WAIT_TIMEOUT);
        abort_flag = 1;
        break;
      }
      const ConvItem it = conv_item(idx, n_slabs, n_chunks);
      const size_t off = (size_t)it.slab * kSlabBytes + (size_t)col * kColBytes;
      const int l0 = it.chunk * kChunkRows;
      const int rows = min(kChunkRows, p.B - l0);
      const int bad = st_bad[st];
      if (bad) {
        if (tid == 0 && it.slab == 0 && it.chunk == 0) flag(p.dev_status, bad);
      } else {
        if (it.slab != cur_slab) load_taps(it.slab);
        if (off < row_bytes) {
          const uint8_t* stage = conv_smem + (size_t)st * kStageBytes + (size_t)col * kColBytes;
          // sliding window: win[i] holds row l - i of the current output row l;
          // before the first row it holds the H rows before the chunk (stage rows H - 1 - i)
          uint64_t win[W][P];
#pragma unroll
          for (int i = 0; i < H; ++i)
            unpack8<T>(*reinterpret_cast<const uint2*>(stage + (size_t)(H - 1 - i) * kSlabBytes),
                       win[i]);
          char* outg = static_cast<char*>(p.out) + ((size_t)it.r * p.B + l0) * row_bytes + off;
          // one output row: shift the window, read row j, convolve, SiLU, store
          auto row_out = [&](int j) {
#pragma unroll
            for (int i = W - 1; i > 0; --i)
#pragma unroll
              for (int q = 0; q < P; ++q) win[i][q] = win[i - 1][q];
            unpack8<T>(*reinterpret_cast<const uint2*>(stage + (size_t)(H + j) * kSlabBytes),
                       win[0]);
            uint64_t y[P];
#pragma unroll
            for (int q = 0; q < P; ++q) {
              uint64_t acc = b2[q];
#pragma unroll
              for (int i = 0; i < W; ++i) acc = f2_fma(w2[q][i], win[i][q], acc);
              y[q] = acc;
            }
            if (p.silu) {
              // SiLU u / d with d = 1 + 2^(-u log2 e), the channels of the
              // thread sharing one reciprocal: 1/d_a = (prod_{b != a} d_b) / prod d.
              // The exponent is capped at 30 so the product of four stays below
              // 2^124; that changes only outputs below 2^-25 |u|.
              float u[V], t[V], d[V];
#pragma unroll
              for (int q = 0; q < P; ++q) {
                f2_split(y[q], u[2 * q], u[2 * q + 1]);
                f2_split(f2_mul(y[q], neg_log2e), t[2 * q], t[2 * q + 1]);
              }
#pragma unroll
              for (int e = 0; e < V; ++e) d[e] = 1.f + ex2_approx(fminf(t[e], 30.f));
              if constexpr (V == 4) {
                const float d01 = d[0] * d[1], d23 = d[2] * d[3];
                const float r = rcp_approx(d01 * d23);
                const float r01 = r * d23, r23 = r * d01;  // 1/(d0 d1), 1/(d2 d3)
                y[0] = f2(u[0] * (r01 * d[1]), u[1] * (r01 * d[0]));
                y[1] = f2(u[2] * (r23 * d[3]), u[3] * (r23 * d[2]));
              } else {
                const float r = rcp_approx(d[0] * d[1]);
                y[0] = f2(u[0] * (r * d[1]), u[1] * (r * d[0]));
              }
            }
            *reinterpret_cast<uint2*>(outg + (size_t)j * row_bytes) = pack8<T>(y);
          };
          if (rows == kChunkRows) {
            // a whole chunk: no guards, so the window shifts are renamings
#pragma unroll
            for (int j = 0; j < kChunkRows; ++j) row_out(j);
          } else {
#pragma unroll
            for (int j = 0; j < kChunkRows; ++j)
              if (j < rows) row_out(j);
          }
          // commit: state <- the last H rows of (old state ++ block rows 0..n-1);
          // the old rows of the first chunk are still in the stage
          if constexpr (H > 0) {
            const int n = st_n[st];
            if (n >= 0 && it.chunk == 0) {
              const int slot = st_slot[st];
              uint2 nw[H];
#pragma unroll
              for (int j = 0; j < H; ++j) {
                const int pos = n - H + j;
                nw[j] = pos >= 0 ? __ldg(reinterpret_cast<const uint2*>(
                                       xg + ((size_t)it.r * p.B + pos) * row_bytes + off))
                                 : *reinterpret_cast<const uint2*>(
                                       stage + (size_t)(H + pos) * kSlabBytes);
              }
#pragma unroll
              for (int j = 0; j < H; ++j)
                *reinterpret_cast<uint2*>(sg + ((size_t)slot * H + j) * row_bytes + off) = nw[j];
            }
          }
        }
      }
      tc::mbar_arrive(&empty[st]);  // this thread is done with the stage
    }
  }
  __syncthreads();
  if (tid == kConvThreads && abort_flag) {
    // a wait gave up: give the copies still in flight (the last kStages items
    // issued) a bounded time to land before the shared memory is released
    for (int j = max(n_issued - kStages, 0); j < n_issued; ++j)
      tc::mbar_wait(&full[j % kStages], (uint32_t)(j / kStages) & 1u, nullptr, 100000000ull);
  }
}

namespace {
PFN_cuTensorMapEncodeTiled_v12000 sc_encode_fn() {
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

// x [R B, C] of T as (D0, C / D0, R B) with D0 = 512 / sizeof(T), box (D0, 8, rows)
template <typename T>
bool sc_map(CUtensorMap* m, const void* x, int C, long rows_total, int box_rows) {
  auto fn = sc_encode_fn();
  if (!fn) return false;
  constexpr int D0 = 512 / (int)sizeof(T);
  cuuint64_t gd[3] = {(cuuint64_t)D0, (cuuint64_t)(C / D0), (cuuint64_t)rows_total};
  cuuint64_t gs[2] = {(cuuint64_t)512, (cuuint64_t)C * sizeof(T)};
  cuuint32_t bx[3] = {(cuuint32_t)D0, 8, (cuuint32_t)box_rows};
  cuuint32_t es[3] = {1, 1, 1};
  return fn(m, sizeof(T) == 2 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT32,
            3, const_cast<void*>(x), gd, gs, bx, es, CU_TENSOR_MAP_INTERLEAVE_NONE,
            CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <typename T, int W>
cudaError_t launch_conv_w(const ConvParams& p, int grid, cudaStream_t stream) {
  cudaError_t e = cudaFuncSetAttribute(short_conv_kernel<T, W>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)kConvSmem);
  if (e != cudaSuccess) return e;
  ConvMaps maps;
  memset(&maps, 0, sizeof maps);
  const long rows_total = (long)p.R * p.B;
  if (p.C % (512 / (int)sizeof(T)) == 0 && rows_total < (1l << 31))
    maps.use = sc_map<T>(&maps.x_halo, p.x, p.C, rows_total, kChunkRows + W - 1) &&
               sc_map<T>(&maps.x_first, p.x, p.C, rows_total, kChunkRows);
  short_conv_kernel<T, W><<<grid, kConvThreads + 32, kConvSmem, stream>>>(maps, p);
  note_launches(1);
  return cudaGetLastError();
}

template <typename T>
cudaError_t launch_conv_t(const ConvParams& p, cudaStream_t stream) {
  const size_t row_bytes = (size_t)p.C * sizeof(T);
  const long n_slabs = (long)((row_bytes + kSlabBytes - 1) / kSlabBytes);
  const long items = (long)p.R * n_slabs * ((p.B + kChunkRows - 1) / kChunkRows);
  int dev = 0, sms = kNumSMs;
  if (cudaGetDevice(&dev) == cudaSuccess)
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  int grid = (int)(items < sms ? items : sms);
  if (n_slabs <= grid) grid = grid / (int)n_slabs * (int)n_slabs;  // one slab per CTA
  switch (p.W) {
    case 1: return launch_conv_w<T, 1>(p, grid, stream);
    case 2: return launch_conv_w<T, 2>(p, grid, stream);
    case 3: return launch_conv_w<T, 3>(p, grid, stream);
    case 4: return launch_conv_w<T, 4>(p, grid, stream);
  }
  return cudaErrorInvalidValue;
}
}  // namespace

cudaError_t launch_short_conv(const ConvParams& p, bool bf16, cudaStream_t stream) {
  if (p.R == 0) return cudaSuccess;
  return bf16 ? launch_conv_t<__nv_bfloat16>(p, stream) : launch_conv_t<float>(p, stream);
}

}  // namespace flare
