// Shared device helpers of the FLARE CUDA library (sm_103a).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "flare.h"

namespace flare {

template <typename T>
__device__ __forceinline__ float to_f32(T x);
template <>
__device__ __forceinline__ float to_f32<float>(float x) {
  return x;
}
template <>
__device__ __forceinline__ float to_f32<__nv_bfloat16>(__nv_bfloat16 x) {
  return __bfloat162float(x);
}

template <typename T>
__device__ __forceinline__ T from_f32(float x);
template <>
__device__ __forceinline__ float from_f32<float>(float x) {
  return x;
}
template <>
__device__ __forceinline__ __nv_bfloat16 from_f32<__nv_bfloat16>(float x) {
  return __float2bfloat16_rn(x);
}

// Two fp32 lanes in one 64-bit register: the packed f32x2 multiply-add,
// multiply and add of sm_100+ do two channels per instruction.
__device__ __forceinline__ uint64_t f2(float lo, float hi) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}
__device__ __forceinline__ void f2_split(uint64_t v, float& lo, float& hi) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}
__device__ __forceinline__ uint64_t f2_fma(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}
__device__ __forceinline__ uint64_t f2_mul(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
// {x, x}: a scalar operand of a packed instruction
__device__ __forceinline__ uint64_t f2_dup(float x) { return f2(x, x); }
__device__ __forceinline__ uint64_t f2_add(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
__device__ __forceinline__ void flag(int32_t* status, int32_t bits) {
  atomicOr(status, bits);
}

__device__ __forceinline__ float warp_max(float x) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) x = fmaxf(x, __shfl_xor_sync(0xffffffffu, x, o));
  return x;
}

__device__ __forceinline__ float warp_sum(float x) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
  return x;
}

// Checks a request's prefix length and every page id it uses; the whole CTA
// gets the same answer.  Returns 0 if valid, else the FLARE_DEV_* bit.
// Must be called by all threads of the CTA (contains __syncthreads).
__device__ __forceinline__ int check_request_pages(const int32_t* __restrict__ page_table,
                                                   int P, int r, int max_pages, int page_size,
                                                   int num_pages) {
  if (P < 0 || P > max_pages * page_size) return FLARE_DEV_BAD_PREFIX_LEN;
  const int npg = (P + page_size - 1) / page_size;
  int bad = 0;
  for (int i = threadIdx.x; i < npg; i += blockDim.x) {
    const int pg = page_table[(size_t)r * max_pages + i];
    bad |= (pg < 0 || pg >= num_pages);
  }
  return __syncthreads_or(bad) ? FLARE_DEV_BAD_PAGE : 0;
}

}  // namespace flare
