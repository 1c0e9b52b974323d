// The 64 x 64 chunk-system helpers of the tcgen05 chunk kernels (the
// two-stream forward, the B = 64 denoise): fp32 tables in shared memory
// swizzled by row, tensor-memory row reads, bf16 high/low splits, and
// T = (I + A)^{-1} of a 64-token chunk (appendix "Chunk-corrected values",
// Eq. chunk-state: the UT/WY system (I + A) delta = X) from its 16 x 16
// diagonal inverses and block columns.
#pragma once

#include <cuda_bf16.h>

#include "tc.cuh"

namespace flare {
namespace chunk64 {

constexpr int kCkC = 64;  // chunk length

__device__ __forceinline__ uint32_t ck_pack(float a, float b) {
  __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<uint32_t*>(&h);
}

// Word offset of element (r, c) of a 64 x 64 fp32 table whose 16-byte units
// are XOR-swizzled by the row (unit c / 4 of row r at unit (c / 4) ^ (r % 16)),
// so that a warp writing one row per lane spreads over every bank.
__device__ __forceinline__ int ck_sw(int r, int c) {
  return r * kCkC + (((c >> 2) ^ (r & 15)) << 2) + (c & 3);
}

// The same for the T table, swizzled by r / 2 (unit c / 4 at (c / 4) ^ (r / 2 % 8)):
// the row groups 2 g .. and 4 g .. that the lanes of a column hold fall in
// distinct banks, and a warp reading one row per lane still spreads over all.
__device__ __forceinline__ int ck_swt(int r, int c) {
  return r * kCkC + (((c >> 2) ^ ((r >> 1) & 7)) << 2) + (c & 3);
}

// 32 table values of row r, columns c0 .. c0 + 31 (c0 a multiple of 4)
__device__ __forceinline__ void ck_store32(float* tbl, int r, int c0, const float (&v)[32]) {
#pragma unroll
  for (int q = 0; q < 8; ++q)
    *reinterpret_cast<float4*>(tbl + ck_sw(r, c0 + 4 * q)) =
        make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
}

// this lane's 32 columns of tensor memory starting at `taddr`
__device__ __forceinline__ void ck_ld32(uint32_t taddr, uint32_t (&r)[32]) {
  tc::tmem_ld16(taddr, *reinterpret_cast<uint32_t(*)[16]>(&r[0]));
  tc::tmem_ld16(taddr + 16, *reinterpret_cast<uint32_t(*)[16]>(&r[16]));
  tc::tmem_ld_wait();
}

// x = hi + lo to about 2^-16 relative, each a bf16 pair (a low, b high)
__device__ __forceinline__ void ck_split(float a, float b, uint32_t& hi, uint32_t& lo) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
  const __nv_bfloat162 l =
      __floats2bfloat162_rn(a - __low2float(h), b - __high2float(h));
  hi = *reinterpret_cast<const uint32_t*>(&h);
  lo = *reinterpret_cast<const uint32_t*>(&l);
}

// Column j of the diagonal block T_aa = (I + A_aa)^{-1}, forward substitution
// (x_t -= A[t][i] x_i for t > i, the A^T rows as 16-byte loads),
// stored whole (zeros above the diagonal) into the swizzled T table.
__device__ __forceinline__ void ck_diag_inverse(const float* AT, float* Tf, int a, int j) {
  float x[16];
#pragma unroll
  for (int t = 0; t < 16; ++t) x[t] = t == j ? 1.f : 0.f;
#pragma unroll
  for (int i = 0; i < 15; ++i) {
    const float xi = x[i];
#pragma unroll
    for (int u = (i + 1) / 4; u < 4; ++u) {
      const float4 q = *reinterpret_cast<const float4*>(AT + ck_sw(16 * a + i, 16 * a + 4 * u));
      const float qv[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
      for (int e = 0; e < 4; ++e)
        if (4 * u + e > i) x[4 * u + e] = fmaf(-qv[e], xi, x[4 * u + e]);
    }
  }
#pragma unroll
  for (int t = 0; t < 16; ++t) Tf[ck_swt(16 * a + t, 16 * a + j)] = x[t];
}

// Block column BC of T below its diagonal block.  Column s of the block
// column lives on R = NT / 16 adjacent lanes (NT = 32, 64 or 128), lane g
// holding rows g RPT .. g RPT + RPT - 1 of every block (RPT = 16 / R), so
// that all of its dependencies travel by shuffles.
// Right-looking (T_c,BC = -T_cc sum_{BC <= d < c} A_cd T_d,BC): once block d
// of the column is known, acc_a += A_ad T_d,BC for every a > d, and the next
// block is T_d+1,BC = -T_d+1,d+1 acc_d+1.  The accumulators are a shift
// register (acc[k] for block row d + 1 + k) so that the loop over d stays a
// loop.  Then the strips BC .. BC + nstrip - 1 (columns 16 BC ..) of T as bf16
// high and low parts into Tb (K-major SW128 rows of 64 elements, zero above
// the diagonal).
template <int NT>
__device__ __forceinline__ void ck_tcol(const float* AT, float* Tf, uint8_t* Tb, int BC, int nstrip,
                                        int q, uint32_t bar_id) {
  constexpr int R = NT / 16, RPT = 16 / R;
  const int s = q / R, g = q % R, lane = q & 31;
  const int src0 = lane & ~(R - 1);  // the first lane of this column
  const int cs = 16 * BC + s;        // the column of T
  float acc[3][RPT];                 // acc[k][e]: row 16 (d + 1 + k) + g RPT + e
#pragma unroll
  for (int k = 0; k < 3; ++k)
#pragma unroll
    for (int e = 0; e < RPT; ++e) acc[k][e] = 0.f;
  float v[16];  // T_d,BC[i][s] of the block d just known
#pragma unroll
  for (int i = 0; i < 16; ++i) v[i] = Tf[ck_swt(16 * BC + i, cs)];
#pragma unroll 1
  for (int d = BC; d < 3; ++d) {
#pragma unroll
    for (int k = 0; k < 3; ++k) {
      const int a = d + 1 + k;
      if (a < 4) {
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          float av[RPT];  // A[16a + g RPT ..][16d + i], 16-byte units addressed one by one
          if constexpr (RPT >= 4) {
#pragma unroll
            for (int e4 = 0; e4 < RPT / 4; ++e4) {
              const float4 v4 = *reinterpret_cast<const float4*>(
                  AT + ck_sw(16 * d + i, 16 * a + g * RPT + 4 * e4));
              av[4 * e4] = v4.x; av[4 * e4 + 1] = v4.y; av[4 * e4 + 2] = v4.z; av[4 * e4 + 3] = v4.w;
            }
          } else {
            const float2 v2 =
                *reinterpret_cast<const float2*>(AT + ck_sw(16 * d + i, 16 * a + g * RPT));
            av[0] = v2.x; av[1] = v2.y;
          }
#pragma unroll
          for (int e = 0; e < RPT; ++e) acc[k][e] = fmaf(av[e], v[i], acc[k][e]);
        }
      }
    }
    // block d + 1: T = -T_cc acc[0], acc[0] gathered from the column's lanes
    const int c = d + 1;
    float w[16];
#pragma unroll
    for (int i = 0; i < 16; ++i) w[i] = __shfl_sync(0xffffffffu, acc[0][i % RPT], src0 + i / RPT);
    float o[RPT];
#pragma unroll
    for (int e = 0; e < RPT; ++e) {
      const int r = 16 * c + g * RPT + e;  // T_cc row
      float x = 0.f;
#pragma unroll
      for (int i4 = 0; i4 < 4; ++i4) {
        const float4 t4 = *reinterpret_cast<const float4*>(Tf + ck_swt(r, 16 * c + 4 * i4));
        x = fmaf(t4.x, w[4 * i4], x);
        x = fmaf(t4.y, w[4 * i4 + 1], x);
        x = fmaf(t4.z, w[4 * i4 + 2], x);
        x = fmaf(t4.w, w[4 * i4 + 3], x);
      }
      o[e] = -x;
      Tf[ck_swt(r, cs)] = o[e];
    }
#pragma unroll
    for (int e = 0; e < RPT; ++e) {
      acc[0][e] = acc[1][e];
      acc[1][e] = acc[2][e];
      acc[2][e] = 0.f;
    }
#pragma unroll
    for (int i = 0; i < 16; ++i) v[i] = __shfl_sync(0xffffffffu, o[i % RPT], src0 + i / RPT);
  }
  tc::named_bar_sync(bar_id, NT);  // the block column complete
  // the strips: 64 rows x 2 units of 8 columns each; zero above the diagonal
#pragma unroll 1
  for (int k = q; k < 128 * nstrip; k += NT) {
    const int u = 2 * BC + (k >> 6);  // 16-byte unit: columns 8u .. 8u + 7
    const int t = k & 63;
    const float4 f0 = *reinterpret_cast<const float4*>(Tf + ck_swt(t, 8 * u));
    const float4 f1 = *reinterpret_cast<const float4*>(Tf + ck_swt(t, 8 * u + 4));
    const float fv[8] = {f0.x, f0.y, f0.z, f0.w, f1.x, f1.y, f1.z, f1.w};
    uint32_t hi[4], lo[4];
#pragma unroll
    for (int e = 0; e < 4; ++e)
      ck_split(8 * u + 2 * e <= t ? fv[2 * e] : 0.f, 8 * u + 2 * e + 1 <= t ? fv[2 * e + 1] : 0.f,
               hi[e], lo[e]);
    const int off = t * 128 + ((u ^ (t & 7)) << 4);
    *reinterpret_cast<uint4*>(Tb + off) = make_uint4(hi[0], hi[1], hi[2], hi[3]);
    *reinterpret_cast<uint4*>(Tb + 8192 + off) = make_uint4(lo[0], lo[1], lo[2], lo[3]);
  }
  tc::fence_async_smem();  // T is MMA d's operand
}

}  // namespace chunk64
}  // namespace flare
