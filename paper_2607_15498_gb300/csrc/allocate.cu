// Step 2 — rank allocation (Sec. 3.2: min-max normalisation, Eq. 4 water-filling, Algorithm 1's
// water level) for every (sequence, layer), one CTA each.
//
// All float arithmetic is IEEE fp32 with explicit round-to-nearest intrinsics (no contraction
// into FMA), so the ranks are a deterministic function of the salience bits:
//   s_hat = (s - min) / (max - min)            (1 if max == min, or in UNIFORM mode)
//   x     = fl(fl(lambda * s_hat) + r_min)
//   rank  = r_max if x >= r_max else max(r_min, floor(x))
// lambda is the largest finite fp32 value >= 0 whose ranks sum to at most B_c, found by bisection
// over the fp32 bit patterns (the sum is non-decreasing in lambda): 31 block-wide counts.
#include "common.cuh"
#include "kernels.h"

namespace vr {

namespace {

constexpr int kThreads = 1024;

__device__ __forceinline__ int rank_of(float lam, float sh, int r_min, int r_max) {
  const float x = __fadd_rn(__fmul_rn(lam, sh), (float)r_min);
  if (x >= (float)r_max) return r_max;          // also catches x = +inf
  const int f = (int)floorf(x);
  return f < r_min ? r_min : f;
}

__device__ __forceinline__ float shat_of(float s, float mn, float den, bool flat) {
  return flat ? 1.0f : __fdiv_rn(__fsub_rn(s, mn), den);
}

// Block-wide sum of one int64 per thread, result returned to every thread.
__device__ int64_t block_sum(int64_t v, int64_t* red) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  __syncthreads();
  if (lane == 0) red[warp] = v;
  __syncthreads();
  if (warp == 0) {
    int64_t x = lane < (int)(blockDim.x >> 5) ? red[lane] : 0;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
    if (lane == 0) red[32] = x;
  }
  __syncthreads();
  return red[32];
}

__global__ void __launch_bounds__(kThreads)
allocate_kernel(const float* __restrict__ sal, uint8_t* __restrict__ ranks,
                int64_t* __restrict__ realized, int32_t* __restrict__ dev_status, Shape s) {
  __shared__ int64_t red[33];
  __shared__ float fred[2][32];
  const int64_t bl = blockIdx.x;
  const int64_t n = s.n_coded;
  const float* sl = sal ? sal + bl * n : nullptr;
  uint8_t* rk = ranks + bl * s.N;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;

  // exact set: full rank
  for (int64_t t = n + tid; t < s.N; t += blockDim.x) rk[t] = (uint8_t)s.r_max;

  // min / max over the coded set (exact in any order)
  float mn = INFINITY, mx = -INFINITY;
  const bool uniform = (s.mode == VARRATE_UNIFORM) || sl == nullptr;
  if (!uniform) {
    for (int64_t t = tid; t < n; t += blockDim.x) {
      const float v = sl[t];
      mn = fminf(mn, v);
      mx = fmaxf(mx, v);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      mn = fminf(mn, __shfl_xor_sync(0xffffffffu, mn, o));
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    }
    if (lane == 0) { fred[0][warp] = mn; fred[1][warp] = mx; }
    __syncthreads();
    mn = INFINITY; mx = -INFINITY;
    for (int i = 0; i < (int)(blockDim.x >> 5); ++i) { mn = fminf(mn, fred[0][i]); mx = fmaxf(mx, fred[1][i]); }
  }
  const bool flat = uniform || !(mx > mn);
  const float den = flat ? 1.0f : __fsub_rn(mx, mn);

  int mode_fixed = -1;    // -1: bisection, otherwise every coded token gets this rank
  if (n == 0) {
    mode_fixed = s.r_max;
  } else if ((int64_t)s.r_min * n > s.Bc) {
    mode_fixed = s.r_min;
    if (tid == 0) raise_status(dev_status, VARRATE_FLOOR_BINDS);
  } else if (s.Bc >= (int64_t)s.r_max * n) {
    mode_fixed = s.r_max;
  }

  float lam = 0.f;
  if (mode_fixed < 0) {
    auto total = [&](uint32_t bits) -> int64_t {
      const float l = __uint_as_float(bits);
      int64_t acc = 0;
      for (int64_t t = tid; t < n; t += blockDim.x)
        acc += rank_of(l, shat_of(sl ? sl[t] : 0.f, mn, den, flat), s.r_min, s.r_max);
      return block_sum(acc, red);
    };
    uint32_t lo;
    if (total(0x7F7FFFFFu) <= s.Bc) {
      lo = 0x7F7FFFFFu;
    } else {
      lo = 0;
      uint32_t hi = 0x7F7FFFFFu;
      while (hi - lo > 1) {
        const uint32_t mid = lo + (hi - lo) / 2;
        if (total(mid) <= s.Bc) lo = mid; else hi = mid;
      }
    }
    lam = __uint_as_float(lo);
  }

  int64_t acc = 0;
  for (int64_t t = tid; t < n; t += blockDim.x) {
    const int r = mode_fixed >= 0 ? mode_fixed
                                  : rank_of(lam, shat_of(sl ? sl[t] : 0.f, mn, den, flat), s.r_min, s.r_max);
    rk[t] = (uint8_t)r;
    acc += r;
  }
  const int64_t sum = block_sum(acc, red);
  if (tid == 0 && realized) realized[bl] = sum;
}

}  // namespace

int launch_allocate(const Shape& s, const float* sal, uint8_t* ranks, int64_t* realized,
                    int32_t* dev_status, cudaStream_t st) {
  allocate_kernel<<<s.B * s.L, kThreads, 0, st>>>(s.mode == VARRATE_UNIFORM ? nullptr : sal, ranks,
                                                  realized, dev_status, s);
  return 1;
}

}  // namespace vr
