// Two-stream causal ShortConv of a block, serving form (appendix "1D Causal
// ShortConv: implementation routes", Eq. short-conv-noisy).
//
// A depthwise causal convolution of width W <= 4: block row l reads its own
// block rows l - i for lags that stay inside the block and the committed conv
// state (the last W - 1 clean tokens before the block, a raw slice of the
// clean stream) for lags that cross the block start; then bias and SiLU.
//
// The kernel is a pure stream (each input byte is used W times from on-chip
// memory), so it is built to keep HBM busy: persistent CTAs (two per SM for
// bf16, one for fp32) walk work items (request, channel slab, chunk of up to 8
// block rows).  A slab is 512 columns of a channel pair each: 2 KiB of bf16 or
// 4 KiB of fp32 channels.  A producer warp stages each item's rows -- the
// chunk plus the W - 1 rows before it, from the block or, for the first chunk,
// from the conv state -- in shared memory: when the channels tile by 512 bytes
// as one tensor-map box of (512 bytes x the slab's blocks) x rows per item (the
// state rows of a first chunk as bulk copies), else one bulk copy per row;
// completion counted on the stage's full barrier (a few large copies keep far
// more bytes in flight per SM than a copy per row); four stages, so three
// items' rows are in flight while 512 compute threads convolve the current
// one, a thread per channel pair down the whole chunk with its filter taps
// and a sliding window in registers, writing its pair coalesced across the
// slab; they release the stage on its empty barrier.  The producer also
// leaves each stage's item coordinates in shared memory.
// The arithmetic runs on fp32 pairs (packed f32x2 multiply-add); the SiLU's
// exponentials run on the special-function unit, its reciprocals one per
// channel pair.  With a grid that is a multiple of the slab count every CTA
// keeps one slab, so the filter taps are loaded once, while the first rows are
// on their way.
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
constexpr int kConvThreads = 512;              // compute threads, a channel pair each
constexpr int kChunkRows = 8;                  // block rows per item
constexpr int kMaxStageRows = kChunkRows + 3;  // with the W - 1 <= 3 rows before the chunk
constexpr int kStages = 4;
// A column of the slab is a channel pair: 4 bytes (bf16: 2 KiB slabs, 88 KiB
// of stages, two CTAs per SM) or 8 bytes (fp32: 4 KiB slabs, 176 KiB, one)
template <typename T>
struct ConvCols {
  static constexpr int kColBytes = 2 * (int)sizeof(T);
  static constexpr int kSlabBytes = kConvThreads * kColBytes;
  static constexpr int kBoxBlocks = kSlabBytes / 512;  // 512-byte tensor-map blocks per slab
  static constexpr int kStageBytes = kMaxStageRows * kSlabBytes;
  static constexpr int kSmem = kStages * kStageBytes;
  static constexpr int kCtasPerSM = sizeof(T) == 2 ? 2 : 1;
};

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

// A column (two channels) of T as an fp32 pair, and back; bf16 widens
// exactly (its bits are the high half of the fp32 pattern)
__device__ __forceinline__ uint64_t unpack_col(uint32_t raw) {
  return f2(__uint_as_float(raw << 16), __uint_as_float(raw & 0xffff0000u));
}
__device__ __forceinline__ uint64_t unpack_col(uint2 raw) {
  return f2(__uint_as_float(raw.x), __uint_as_float(raw.y));
}
__device__ __forceinline__ void pack_col(uint64_t f, uint32_t& out) {
  float lo, hi;
  f2_split(f, lo, hi);
  __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
  out = *reinterpret_cast<uint32_t*>(&h);
}
__device__ __forceinline__ void pack_col(uint64_t f, uint2& out) {
  float lo, hi;
  f2_split(f, lo, hi);
  out = make_uint2(__float_as_uint(lo), __float_as_uint(hi));
}
template <typename T>
struct ColWord {
  using type = uint32_t;
};
template <>
struct ColWord<float> {
  using type = uint2;
};

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
__global__ void __launch_bounds__(kConvThreads + 32, ConvCols<T>::kCtasPerSM)
    short_conv_kernel(const __grid_constant__ ConvMaps maps, ConvParams p) {
  constexpr int E = sizeof(T);
  constexpr int kColBytes = ConvCols<T>::kColBytes;
  constexpr int kSlabBytes = ConvCols<T>::kSlabBytes;
  constexpr int kStageBytes = ConvCols<T>::kStageBytes;
  constexpr int H = W - 1;  // rows before a chunk
  using Col = typename ColWord<T>::type;
  extern __shared__ __align__(128) uint8_t conv_smem[];
  __shared__ uint64_t full[kStages], empty[kStages];
  // per stage, written by the producer: the item's request, slab and chunk,
  // the request's slot, accepted length and validity
  __shared__ int st_r[kStages], st_slab[kStages], st_chunk[kStages];
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
        st_r[st] = it.r;
        st_slab[st] = it.slab;
        st_chunk[st] = it.chunk;
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
                            it.slab * ConvCols<T>::kBoxBlocks, row0);
          } else {
            tc::mbar_expect_tx(&full[st], (uint32_t)(kSlabBytes * (kChunkRows + H)));
            tc::tma_load_3d(dst, &maps.x_halo, &full[st], 0, it.slab * ConvCols<T>::kBoxBlocks,
                            row0 - H);
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
    uint64_t w2[W], b2;  // this thread's two channels: taps and bias as fp32 pairs
    int cur_slab = -1;
    // filter taps and bias of this thread's channels (loaded while the first
    // item's rows are on their way, and again only if the slab changes)
    auto load_taps = [&](int slab) {
      cur_slab = slab;
      const size_t off = (size_t)slab * kSlabBytes + (size_t)col * kColBytes;
      if (off >= row_bytes) return;
      const int c0 = (int)(off / E);
      const float2* w2p = reinterpret_cast<const float2*>(p.weight + (size_t)c0 * W);
      float wf[2 * W];
#pragma unroll
      for (int q = 0; q < W; ++q) {
        const float2 v = __ldg(w2p + q);
        wf[2 * q] = v.x;
        wf[2 * q + 1] = v.y;
      }
      float2 bf = make_float2(0.f, 0.f);
      if (p.bias) bf = __ldg(reinterpret_cast<const float2*>(p.bias + c0));
#pragma unroll
      for (int i = 0; i < W; ++i) w2[i] = f2(wf[i], wf[W + i]);
      b2 = f2(bf.x, bf.y);
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
      const int ir = st_r[st], islab = st_slab[st], ichunk = st_chunk[st];
      const size_t off = (size_t)islab * kSlabBytes + (size_t)col * kColBytes;
      const int l0 = ichunk * kChunkRows;
      const int rows = min(kChunkRows, p.B - l0);
      const int bad = st_bad[st];
      if (bad) {
        if (tid == 0 && islab == 0 && ichunk == 0) flag(p.dev_status, bad);
      } else {
        if (islab != cur_slab) load_taps(islab);
        if (off < row_bytes) {
          const uint8_t* stage = conv_smem + (size_t)st * kStageBytes + (size_t)col * kColBytes;
          // sliding window: win[i] holds row l - i of the current output row l;
          // before the first row it holds the H rows before the chunk (stage rows H - 1 - i)
          uint64_t win[W];
#pragma unroll
          for (int i = 0; i < H; ++i)
            win[i] = unpack_col(*reinterpret_cast<const Col*>(stage + (size_t)(H - 1 - i) * kSlabBytes));
          char* outg = static_cast<char*>(p.out) + ((size_t)ir * p.B + l0) * row_bytes + off;
          // one output row: shift the window, read row j, convolve, SiLU, store
          auto row_out = [&](int j) {
#pragma unroll
            for (int i = W - 1; i > 0; --i) win[i] = win[i - 1];
            win[0] = unpack_col(*reinterpret_cast<const Col*>(stage + (size_t)(H + j) * kSlabBytes));
            uint64_t y = b2;
#pragma unroll
            for (int i = 0; i < W; ++i) y = f2_fma(w2[i], win[i], y);
            if (p.silu) {
              // SiLU u / d with d = 1 + 2^(-u log2 e), the two channels sharing
              // one reciprocal: 1/d_a = d_b / (d_a d_b).  The exponent is capped
              // at 60 so the product of two stays below 2^121; that changes only
              // outputs below 2^-60 |u|.
              float u0, u1, t0, t1;
              f2_split(y, u0, u1);
              f2_split(f2_mul(y, neg_log2e), t0, t1);
              const float d0 = 1.f + ex2_approx(fminf(t0, 60.f));
              const float d1 = 1.f + ex2_approx(fminf(t1, 60.f));
              const float r = rcp_approx(d0 * d1);
              y = f2_mul(y, f2_mul(f2_dup(r), f2(d1, d0)));
            }
            Col o;
            pack_col(y, o);
            *reinterpret_cast<Col*>(outg + (size_t)j * row_bytes) = o;
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
            if (n >= 0 && ichunk == 0) {
              const int slot = st_slot[st];
              Col nw[H];
#pragma unroll
              for (int j = 0; j < H; ++j) {
                const int pos = n - H + j;
                nw[j] = pos >= 0 ? *reinterpret_cast<const Col*>(
                                       xg + ((size_t)ir * p.B + pos) * row_bytes + off)
                                 : *reinterpret_cast<const Col*>(
                                       stage + (size_t)(H + pos) * kSlabBytes);
              }
#pragma unroll
              for (int j = 0; j < H; ++j)
                *reinterpret_cast<Col*>(sg + ((size_t)slot * H + j) * row_bytes + off) = nw[j];
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

// x [R B, C] of T as (D0, C / D0, R B) with D0 = 512 / sizeof(T), box (D0, a
// slab's blocks, rows)
template <typename T>
bool sc_map(CUtensorMap* m, const void* x, int C, long rows_total, int box_rows) {
  auto fn = sc_encode_fn();
  if (!fn) return false;
  constexpr int D0 = 512 / (int)sizeof(T);
  cuuint64_t gd[3] = {(cuuint64_t)D0, (cuuint64_t)(C / D0), (cuuint64_t)rows_total};
  cuuint64_t gs[2] = {(cuuint64_t)512, (cuuint64_t)C * sizeof(T)};
  cuuint32_t bx[3] = {(cuuint32_t)D0, (cuuint32_t)ConvCols<T>::kBoxBlocks, (cuuint32_t)box_rows};
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
                                       ConvCols<T>::kSmem);
  if (e != cudaSuccess) return e;
  ConvMaps maps;
  memset(&maps, 0, sizeof maps);
  const long rows_total = (long)p.R * p.B;
  if (p.C % (512 / (int)sizeof(T)) == 0 && rows_total < (1l << 31))
    maps.use = sc_map<T>(&maps.x_halo, p.x, p.C, rows_total, kChunkRows + W - 1) &&
               sc_map<T>(&maps.x_first, p.x, p.C, rows_total, kChunkRows);
  short_conv_kernel<T, W><<<grid, kConvThreads + 32, ConvCols<T>::kSmem, stream>>>(maps, p);
  note_launches(1);
  return cudaGetLastError();
}

template <typename T>
cudaError_t launch_conv_t(const ConvParams& p, cudaStream_t stream) {
  const size_t row_bytes = (size_t)p.C * sizeof(T);
  constexpr int kSlab = ConvCols<T>::kSlabBytes;
  const long n_slabs = (long)((row_bytes + kSlab - 1) / kSlab);
  const long items = (long)p.R * n_slabs * ((p.B + kChunkRows - 1) / kChunkRows);
  int dev = 0, sms = kNumSMs;
  if (cudaGetDevice(&dev) == cudaSuccess)
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const long ctas = (long)ConvCols<T>::kCtasPerSM * sms;
  int grid = (int)(items < ctas ? items : ctas);
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
