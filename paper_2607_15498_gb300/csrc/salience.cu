// Step 1 — salience (Sec. 3.2, Eq. salience): for every window query q (position N - w + q) and
// query head h, alpha_{q,t} = softmax over t <= p of <q, k_t>/sqrt(d); s_t is the mean of alpha over
// the w queries and H heads, kept for the coded set, then averaged over pool_len neighbours.
//
// Two passes over the keys of each KV head g, with the grp*w window rows that read g stacked as
// one row block (row m = local head * w + query):
//   pass 1 (salience_stats): running max and sum of exp per row over a token chunk -> partials;
//   pass 2 (salience_accum): lse per row from the partials, then sum_rows exp(S - lse) per token,
//                            accumulated over every KV head in a fixed order (deterministic).
// Scores are kept in log2 units (scaled by log2(e)/sqrt(d)) so the exponentials are exp2.
#include "common.cuh"
#include "kernels.h"

namespace vr {

namespace {

constexpr int kRows = 128;     // window rows per block
constexpr int kTok = 64;       // tokens per tile
constexpr int kLd = kHeadDim + 4;
constexpr int kThreads = 256;

// Load rows [rb*128, rb*128+128) of the window block of KV head g into smem as fp32.
template <typename T>
__device__ void load_q_rows(float* qs, const T* __restrict__ q_win, const Shape& s, int64_t bl,
                            int g, int rb) {
  const int M = s.grp * s.w;
  for (int idx = threadIdx.x; idx < kRows * kHeadDim; idx += blockDim.x) {
    const int r = idx / kHeadDim, c = idx % kHeadDim;
    const int m = rb * kRows + r;
    float val = 0.f;
    if (m < M) {
      const int h = g * s.grp + m / s.w, q = m % s.w;
      val = to_f(q_win[((bl * s.w + q) * s.H + h) * (int64_t)kHeadDim + c]);
    }
    qs[r * kLd + c] = val;
  }
}

template <typename T>
__device__ void load_k_tile(float* ks, const T* __restrict__ kg, int64_t t0, int64_t t_end) {
  for (int idx = threadIdx.x; idx < kTok * kHeadDim; idx += blockDim.x) {
    const int r = idx / kHeadDim, c = idx % kHeadDim;
    const int64_t t = t0 + r;
    ks[r * kLd + c] = (t < t_end) ? to_f(kg[t * kHeadDim + c]) : 0.f;
  }
}

// acc[4 rows][8 tokens] for rows 4*tr.., tokens tc + 8*i of the tile.
__device__ __forceinline__ void tile_scores(const float* qs, const float* ks, int tr, int tc,
                                            float (&acc)[4][8]) {
#pragma unroll
  for (int a = 0; a < 4; ++a)
#pragma unroll
    for (int i = 0; i < 8; ++i) acc[a][i] = 0.f;
#pragma unroll 4
  for (int c = 0; c < kHeadDim; c += 4) {
    float4 qv[4], kv[8];
#pragma unroll
    for (int a = 0; a < 4; ++a) qv[a] = *reinterpret_cast<const float4*>(&qs[(4 * tr + a) * kLd + c]);
#pragma unroll
    for (int i = 0; i < 8; ++i) kv[i] = *reinterpret_cast<const float4*>(&ks[(tc + 8 * i) * kLd + c]);
#pragma unroll
    for (int a = 0; a < 4; ++a)
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        acc[a][i] = fmaf(qv[a].x, kv[i].x, acc[a][i]);
        acc[a][i] = fmaf(qv[a].y, kv[i].y, acc[a][i]);
        acc[a][i] = fmaf(qv[a].z, kv[i].z, acc[a][i]);
        acc[a][i] = fmaf(qv[a].w, kv[i].w, acc[a][i]);
      }
  }
}

// grid (n_chunks, G * n_row_blocks, B * L); stats[bl][g][m][chunk] = (max, sum exp2(S - max)).
template <typename T>
__global__ void __launch_bounds__(kThreads)
salience_stats_kernel(const T* __restrict__ q_win, const T* __restrict__ k, float2* __restrict__ stats,
                      Shape s, int n_chunks, int64_t chunk, int n_rb) {
  extern __shared__ float smem[];
  float* qs = smem;
  float* ks = smem + kRows * kLd;
  const int64_t bl = blockIdx.z;
  const int g = blockIdx.y / n_rb, rb = blockIdx.y % n_rb;
  const int M = s.grp * s.w;
  const int tid = threadIdx.x, tr = tid / 8, tc = tid % 8;
  const float scale = kLog2e * rsqrtf((float)kHeadDim);

  load_q_rows(qs, q_win, s, bl, g, rb);
  const T* kg = k + (bl * s.G + g) * s.N * kHeadDim;
  const int64_t t_begin = blockIdx.x * chunk;
  const int64_t t_end = min(s.N, t_begin + chunk);

  float run_m[4], run_l[4];
  int64_t pos[4];
#pragma unroll
  for (int a = 0; a < 4; ++a) {
    run_m[a] = -INFINITY;
    run_l[a] = 0.f;
    const int m = rb * kRows + 4 * tr + a;
    pos[a] = s.N - s.w + (m < M ? m % s.w : 0);
  }
  for (int64_t t0 = t_begin; t0 < t_end; t0 += kTok) {
    __syncthreads();
    load_k_tile(ks, kg, t0, t_end);
    __syncthreads();
    float acc[4][8];
    tile_scores(qs, ks, tr, tc, acc);
#pragma unroll
    for (int a = 0; a < 4; ++a) {
      float mx = -INFINITY;
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const int64_t t = t0 + tc + 8 * i;
        acc[a][i] = (t < t_end && t <= pos[a]) ? acc[a][i] * scale : -INFINITY;
        mx = fmaxf(mx, acc[a][i]);
      }
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 4));
      const float nm = fmaxf(run_m[a], mx);
      const float ref = (nm == -INFINITY) ? 0.f : nm;   // a fully masked row keeps l = 0
      float sum = 0.f;
#pragma unroll
      for (int i = 0; i < 8; ++i) sum += exp2f(acc[a][i] - ref);
      sum += __shfl_xor_sync(0xffffffffu, sum, 1);
      sum += __shfl_xor_sync(0xffffffffu, sum, 2);
      sum += __shfl_xor_sync(0xffffffffu, sum, 4);
      run_l[a] = run_l[a] * exp2f(run_m[a] - ref) + sum;
      run_m[a] = nm;
    }
  }
  if (tc == 0) {
#pragma unroll
    for (int a = 0; a < 4; ++a) {
      const int m = rb * kRows + 4 * tr + a;
      if (m < M) stats[((bl * s.G + g) * M + m) * n_chunks + blockIdx.x] = make_float2(run_m[a], run_l[a]);
    }
  }
}

// grid (n_chunks2, B * L); raw[bl][t] = (1/(w H)) sum_g sum_rows exp2(S - lse) for t < N - w.
template <typename T>
__global__ void __launch_bounds__(kThreads)
salience_accum_kernel(const T* __restrict__ q_win, const T* __restrict__ k,
                      const float2* __restrict__ stats, float* __restrict__ raw, Shape s,
                      int n_chunks, int64_t chunk2, int n_rb) {
  extern __shared__ float smem[];
  float* qs = smem;
  float* ks = qs + kRows * kLd;
  float* lse = ks + kTok * kLd;                 // [kRows]
  float* red = lse + kRows;                     // [8 warps][kTok]
  float* col = red + 8 * kTok;                  // [chunk2]
  const int64_t bl = blockIdx.y;
  const int M = s.grp * s.w;
  const int tid = threadIdx.x, tr = tid / 8, tc = tid % 8, warp = tid / 32, lane = tid % 32;
  const float scale = kLog2e * rsqrtf((float)kHeadDim);
  const int64_t t_begin = blockIdx.x * chunk2;
  const int64_t t_end = min(s.n_coded, t_begin + chunk2);
  if (t_begin >= t_end) return;
  for (int64_t i = tid; i < chunk2; i += blockDim.x) col[i] = 0.f;

  for (int g = 0; g < s.G; ++g) {
    const T* kg = k + (bl * s.G + g) * s.N * kHeadDim;
    for (int rb = 0; rb < n_rb; ++rb) {
      __syncthreads();
      load_q_rows(qs, q_win, s, bl, g, rb);
      if (tid < kRows) {
        const int m = rb * kRows + tid;
        float val = INFINITY;   // padding rows contribute exp2(-inf) = 0
        if (m < M) {
          const float2* st = stats + ((bl * s.G + g) * M + m) * n_chunks;
          float mx = -INFINITY;
          for (int c = 0; c < n_chunks; ++c) mx = fmaxf(mx, st[c].x);
          float l = 0.f;
          for (int c = 0; c < n_chunks; ++c)
            if (st[c].x != -INFINITY) l += st[c].y * exp2f(st[c].x - mx);
          val = mx + log2f(l);
        }
        lse[tid] = val;
      }
      for (int64_t t0 = t_begin; t0 < t_end; t0 += kTok) {
        __syncthreads();
        load_k_tile(ks, kg, t0, t_end);
        __syncthreads();
        float acc[4][8];
        tile_scores(qs, ks, tr, tc, acc);
        float part[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          float p = 0.f;
#pragma unroll
          for (int a = 0; a < 4; ++a) p += exp2f(acc[a][i] * scale - lse[4 * tr + a]);
          p += __shfl_xor_sync(0xffffffffu, p, 8);
          p += __shfl_xor_sync(0xffffffffu, p, 16);
          part[i] = p;
        }
        if (lane < 8) {
#pragma unroll
          for (int i = 0; i < 8; ++i) red[warp * kTok + tc + 8 * i] = part[i];
        }
        __syncthreads();
        if (tid < kTok) {
          float sum = 0.f;
#pragma unroll
          for (int wi = 0; wi < 8; ++wi) sum += red[wi * kTok + tid];
          if (t0 + tid < t_end) col[t0 - t_begin + tid] += sum;
        }
      }
    }
  }
  __syncthreads();
  const float inv = 1.0f / (float)(s.w * s.H);
  for (int64_t i = tid; i < t_end - t_begin; i += blockDim.x) raw[bl * s.n_coded + t_begin + i] = col[i] * inv;
}

// grid (ceil(n_coded / 256), B * L): zero-padded moving average of length pool.
__global__ void salience_pool_kernel(const float* __restrict__ raw, float* __restrict__ sal, Shape s) {
  const int64_t bl = blockIdx.y;
  const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= s.n_coded) return;
  const int half = s.pool / 2;
  const float* r = raw + bl * s.n_coded;
  float acc = 0.f;
  for (int i = -half; i <= half; ++i) {
    const int64_t u = t + i;
    if (u >= 0 && u < s.n_coded) acc += r[u];
  }
  sal[bl * s.n_coded + t] = acc / (float)s.pool;
}

}  // namespace

size_t salience_ws_bytes(const Shape& s, int num_sms) {
  if (salience_tc_supported(s)) return salience_tc_ws_bytes(s, num_sms);
  const SalPlan p = salience_plan(s, num_sms);
  const int M = s.grp * s.w;
  size_t b = (size_t)s.B * s.L * s.G * M * p.n_chunks * sizeof(float2);
  b = (b + 255) & ~size_t(255);
  b += (size_t)s.B * s.L * s.n_coded * sizeof(float);
  return (b + 255) & ~size_t(255);
}

SalPlan salience_plan(const Shape& s, int num_sms) {
  SalPlan p;
  p.n_rb = (s.grp * s.w + kRows - 1) / kRows;
  const int64_t units = (int64_t)s.B * s.L * s.G * p.n_rb;
  const int64_t want = (int64_t)4 * num_sms;
  int64_t n = (want + units - 1) / units;
  int64_t chunk = (s.N + n - 1) / n;
  chunk = ((chunk + kTok - 1) / kTok) * kTok;
  if (chunk < 512) chunk = 512;
  p.chunk = chunk;
  p.n_chunks = (int)((s.N + chunk - 1) / chunk);
  const int64_t bl = (int64_t)s.B * s.L;
  int64_t c2 = (s.n_coded * bl + 2 * num_sms - 1) / (2 * num_sms);
  c2 = ((c2 + kTok - 1) / kTok) * kTok;
  p.chunk2 = c2 < kTok ? kTok : (c2 > 2048 ? 2048 : c2);
  p.n_chunks2 = (int)((s.n_coded + p.chunk2 - 1) / p.chunk2);
  return p;
}

int launch_salience(const Shape& s, const void* q_win, const void* k, float* sal_out, void* ws,
                    int32_t* dev_status, int num_sms, cudaStream_t st) {
  if (salience_tc_supported(s)) return launch_salience_tc(s, q_win, k, sal_out, ws, dev_status, num_sms, st);
  const SalPlan p = salience_plan(s, num_sms);
  if (s.n_coded == 0) return 0;
  const int M = s.grp * s.w;
  float2* stats = reinterpret_cast<float2*>(ws);
  size_t off = (size_t)s.B * s.L * s.G * M * p.n_chunks * sizeof(float2);
  off = (off + 255) & ~size_t(255);
  float* raw = reinterpret_cast<float*>(static_cast<char*>(ws) + off);
  const size_t smem1 = (size_t)(kRows + kTok) * kLd * sizeof(float);
  const size_t smem2 = smem1 + (kRows + 8 * kTok + p.chunk2) * sizeof(float);
  dim3 g1(p.n_chunks, s.G * p.n_rb, s.B * s.L);
  dim3 g2(p.n_chunks2, s.B * s.L);
  if (s.dtype == VARRATE_BF16) {
    using T = __nv_bfloat16;
    cudaFuncSetAttribute(salience_stats_kernel<T>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem1);
    cudaFuncSetAttribute(salience_accum_kernel<T>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem2);
    salience_stats_kernel<T><<<g1, kThreads, smem1, st>>>((const T*)q_win, (const T*)k, stats, s, p.n_chunks, p.chunk, p.n_rb);
    salience_accum_kernel<T><<<g2, kThreads, smem2, st>>>((const T*)q_win, (const T*)k, stats, raw, s, p.n_chunks, p.chunk2, p.n_rb);
  } else {
    using T = float;
    cudaFuncSetAttribute(salience_stats_kernel<T>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem1);
    cudaFuncSetAttribute(salience_accum_kernel<T>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem2);
    salience_stats_kernel<T><<<g1, kThreads, smem1, st>>>((const T*)q_win, (const T*)k, stats, s, p.n_chunks, p.chunk, p.n_rb);
    salience_accum_kernel<T><<<g2, kThreads, smem2, st>>>((const T*)q_win, (const T*)k, stats, raw, s, p.n_chunks, p.chunk2, p.n_rb);
  }
  dim3 g3((unsigned)((s.n_coded + 255) / 256), s.B * s.L);
  salience_pool_kernel<<<g3, 256, 0, st>>>(raw, sal_out, s);
  return 3;
}

}  // namespace vr
