// Internal helpers shared by the VarRate CUDA kernels (not part of the public ABI).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "varrate.h"

namespace vr {

constexpr int kHeadDim = 128;          // the only head width the kernels are built for
constexpr float kLog2e = 1.4426950408889634f;

// Shape of one call, derived once on the host from varrate_config.
struct Shape {
  int B, L, G, grp, H, d, w, pool, r_min, r_max, dtype, mode;
  int64_t N, n_coded, Bc, cap;
};

// Raise the device status word: errors (negative) replace anything larger, a warning only
// replaces VARRATE_OK.
__device__ __forceinline__ void raise_status(int32_t* st, int32_t code) {
  if (st == nullptr) return;
  if (code < 0) atomicMin(st, code);
  else atomicCAS(st, 0, code);
}

template <typename T> __device__ __forceinline__ float to_f(T x);
template <> __device__ __forceinline__ float to_f<float>(float x) { return x; }
template <> __device__ __forceinline__ float to_f<__nv_bfloat16>(__nv_bfloat16 x) {
  return __bfloat162float(x);
}
template <typename T> __device__ __forceinline__ T from_f(float x);
template <> __device__ __forceinline__ float from_f<float>(float x) { return x; }
template <> __device__ __forceinline__ __nv_bfloat16 from_f<__nv_bfloat16>(float x) {
  return __float2bfloat16_rn(x);
}

// Eight consecutive elements starting at a 16-byte (bf16) / 32-byte (fp32) aligned address,
// streamed (read once: evict-first in L2, no L1 allocation).
__device__ __forceinline__ void load8_stream(const __nv_bfloat16* p, float (&f)[8]) {
  uint4 u = __ldcs(reinterpret_cast<const uint4*>(p));
  const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    f[2 * i] = __uint_as_float(w[i] << 16);
    f[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
  }
}
__device__ __forceinline__ void load8_stream(const float* p, float (&f)[8]) {
  float4 a = __ldcs(reinterpret_cast<const float4*>(p));
  float4 b = __ldcs(reinterpret_cast<const float4*>(p) + 1);
  f[0] = a.x; f[1] = a.y; f[2] = a.z; f[3] = a.w;
  f[4] = b.x; f[5] = b.y; f[6] = b.z; f[7] = b.w;
}

__device__ __forceinline__ int64_t pad8(int64_t n) { return (n + 7) & ~int64_t(7); }

}  // namespace vr
