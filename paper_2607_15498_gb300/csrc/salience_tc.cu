// Step 1, bf16 — salience on the 5th-generation tensor cores (Sec. 3.2, Eq. salience).
//
// The window rows that read KV head g (row m = local head * w + query, M = group * w of them)
// score every key: S = Q_g K_g^T / sqrt(d), causal inside the window. Two passes over the keys,
// both fed by TMA (128-byte swizzle) and accumulated in TMEM by tcgen05.mma:
//   pass 1  (rows x tokens, M = 128 rows, N = 256 tokens): each epilogue thread owns one row and
//           keeps its running max and sum of 2^(S * log2e / sqrt(d) - max) over the tiles of its
//           epilogue group (two groups take alternate tiles; their partials merge at the end);
//   pass 2  (tokens x rows, M = 128 tokens, N = M rows rounded up to 32): each epilogue thread owns
//           one token and sums 2^(S * log2e / sqrt(d) - lse_row) over the rows of one head; the
//           pool kernel adds the heads in a fixed order (deterministic) and applies the 5-tap mean.
// Warp roles: one TMA producer warp, one MMA-issuing warp, epilogue warps that read TMEM with
// tcgen05.ld (lane quarter = warp % 4). Stages, TMEM buffers and their hand-offs are mbarriers;
// every wait is bounded and a timeout raises VARRATE_ERR_TIMEOUT.
#include <cudaTypedefs.h>

#include "common.cuh"
#include "kernels.h"

namespace vr {

namespace {

constexpr uint32_t kTries = 1u << 22;

// ------------------------------------------------------------------------------- pass 1
constexpr int P1_NGRP = 2;              // epilogue groups of four warps (alternate tiles)
constexpr int P1_EPI = 4 * P1_NGRP;
constexpr int P1_THREADS = (P1_EPI + 2) * 32;
constexpr int P1_TN = 256;              // tokens per tile (MMA N)
constexpr int P1_ST = 3;                // key stages (2 in flight behind the one in use)
constexpr int P1_NACC = 512 / P1_TN;    // TMEM accumulators of P1_TN columns
constexpr int P1_Q = 128 * 256;         // 128 rows x 128 bf16
constexpr int P1_K = P1_TN * 256;       // 128 tokens x 128 bf16

struct P1Smem {
  uint64_t full[P1_ST], empty[P1_ST], tfull[P1_NACC], tempty[P1_NACC];
  uint32_t tmem;
  int err;
};

__global__ void __launch_bounds__(P1_THREADS, 1)
salience_stats_tc_kernel(const __grid_constant__ CUtensorMap tk, const __nv_bfloat16* __restrict__ q_win,
                         float2* __restrict__ stats, int32_t* __restrict__ dev_status, Shape s,
                         int n_chunks, int64_t chunk, int n_rb) {
  extern __shared__ __align__(1024) unsigned char raw_smem[];
  unsigned char* smem = raw_smem + ((1024 - (smem_addr(raw_smem) & 1023)) & 1023);
  unsigned char* qt = smem;
  unsigned char* kst = smem + P1_Q;
  P1Smem& sm = *reinterpret_cast<P1Smem*>(kst + P1_ST * P1_K);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int64_t bl = blockIdx.z;
  const int g = blockIdx.y / n_rb, rb = blockIdx.y % n_rb;
  const int M = s.grp * s.w;
  const int64_t t_begin = (int64_t)blockIdx.x * chunk;
  const int64_t t_end = min(s.N, t_begin + chunk);
  const int n_tiles = (int)((t_end - t_begin + P1_TN - 1) / P1_TN);

  // window rows of this block into shared memory (swizzled K-major), zero rows past M
  if (warp < P1_EPI) {
    for (int idx = tid; idx < 128 * 16; idx += P1_EPI * 32) {
      const int row = idx >> 4, cidx = idx & 15;
      const int m = rb * 128 + row;
      uint4 v = make_uint4(0, 0, 0, 0);
      if (m < M) {
        const int h = g * s.grp + m / s.w, qq = m % s.w;
        v = __ldg(reinterpret_cast<const uint4*>(q_win + ((bl * s.w + qq) * s.H + h) * (int64_t)kHeadDim) + cidx);
      }
      *reinterpret_cast<uint4*>(qt + sw128_offset(row, cidx, 128)) = v;
    }
  }
  if (warp == P1_EPI + 1 && lane == 0) {
    for (int i = 0; i < P1_ST; ++i) { mbar_init(&sm.full[i], 1); mbar_init(&sm.empty[i], 1); }
    for (int i = 0; i < P1_NACC; ++i) { mbar_init(&sm.tfull[i], 1); mbar_init(&sm.tempty[i], 4); }
    sm.err = 0;
    fence_mbar_init();
  }
  if (warp == 0) tmem_alloc(&sm.tmem, 512);
  fence_proxy_async_smem();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = sm.tmem;
  const int64_t row0 = (bl * s.G + g) * s.N + t_begin;
  float rm = -INFINITY, rl = 0.f;   // epilogue: running max and sum of this thread's row

  if (warp == P1_EPI) {
    if (lane == 0) {                                  // TMA producer
      for (int i = 0; i < n_tiles; ++i) {
        const int st = i % P1_ST;
        if (!mbar_wait_bounded(&sm.empty[st], ((i / P1_ST) & 1) ^ 1, kTries)) { sm.err = 1; break; }
        mbar_arrive_expect_tx(&sm.full[st], P1_K);
        const uint32_t dst = smem_addr(kst + st * P1_K);
        tma_load_2d(dst, &tk, 0, (int)(row0 + (int64_t)i * P1_TN), &sm.full[st]);
        tma_load_2d(dst + P1_K / 2, &tk, 64, (int)(row0 + (int64_t)i * P1_TN), &sm.full[st]);
      }
    }
  } else if (warp == P1_EPI + 1) {
    if (lane == 0) {                                  // MMA issuer
      constexpr uint32_t idesc = idesc_bf16_f32(128, P1_TN);
      const uint32_t qa = smem_addr(qt);
      for (int i = 0; i < n_tiles; ++i) {
        const int st = i % P1_ST, b = i % P1_NACC;
        if (!mbar_wait_bounded(&sm.full[st], (i / P1_ST) & 1, kTries) ||
            !mbar_wait_bounded(&sm.tempty[b], ((i / P1_NACC) & 1) ^ 1, kTries)) { sm.err = 1; break; }
        tc_fence_after();
        const uint32_t kb = smem_addr(kst + st * P1_K);
#pragma unroll
        for (int ks = 0; ks < kHeadDim / 16; ++ks) {
          const uint32_t ka = (ks >> 2) * 16384 + (ks & 3) * 32;     // Q panel: 128 rows x 128 B
          const uint32_t kk = (ks >> 2) * (P1_K / 2) + (ks & 3) * 32; // K panel: 128 rows x 128 B
          tc_mma_bf16(tmem + b * P1_TN, sdesc_sw128(qa + ka), sdesc_sw128(kb + kk), idesc, ks > 0);
        }
        tc_commit(&sm.empty[st]);
        tc_commit(&sm.tfull[b]);
      }
    }
  } else {                                            // epilogue: one row, alternate tiles
    const int quarter = warp & 3, eg = warp >> 2;
    const int row = quarter * 32 + lane;
    const int m = rb * 128 + row;
    const int64_t pos = s.N - s.w + (m < M ? m % s.w : 0);   // causal limit of this row
    const float scale = kLog2e * rsqrtf((float)kHeadDim);
    bool bad = false;
    for (int i = eg; i < n_tiles; i += P1_NGRP) {
      const int b = i % P1_NACC;
      if (!bad && !mbar_wait_bounded(&sm.tfull[b], (i / P1_NACC) & 1, kTries)) { sm.err = 1; bad = true; }
      tc_fence_after();
      const int64_t t0 = t_begin + (int64_t)i * P1_TN;
      const uint32_t taddr = tmem + b * P1_TN + ((uint32_t)(quarter * 32) << 16);
      // every token of this tile is a real token before the window, which every window row sees:
      // no mask needed (warp-uniform)
      const bool plain = t0 + P1_TN <= t_end && t0 + P1_TN <= s.N - s.w + 1;
#pragma unroll
      for (int cb = 0; cb < P1_TN / 32; ++cb) {
        float v[32];
        tmem_ld32(taddr + cb * 32, v);
        if (!plain) {
#pragma unroll
          for (int jj = 0; jj < 32; ++jj) {
            const int64_t t = t0 + cb * 32 + jj;
            if (!(t < t_end && t <= pos)) v[jj] = -INFINITY;
          }
        }
        // max as a tree, sums in four interleaved partials (short dependency chains)
        float mx[8];
#pragma unroll
        for (int q = 0; q < 8; ++q) mx[q] = fmaxf(fmaxf(v[4 * q], v[4 * q + 1]), fmaxf(v[4 * q + 2], v[4 * q + 3]));
#pragma unroll
        for (int q = 0; q < 4; ++q) mx[q] = fmaxf(mx[q], mx[q + 4]);
        const float cm = fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3]));
        const float nm = fmaxf(rm, cm * scale);    // scale > 0: max commutes with scaling
        const float ref = nm == -INFINITY ? 0.f : nm;
        float part[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int jj = 0; jj < 32; ++jj) part[jj & 3] += fast_exp2(fmaf(v[jj], scale, -ref));
        rl = rl * fast_exp2(rm - ref) + ((part[0] + part[1]) + (part[2] + part[3]));
        rm = nm;
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&sm.tempty[b]);
    }
  }
  tc_fence_before();
  __syncthreads();
  // every copy and product has landed: the group partials go through the idle key stages
  float* gm = reinterpret_cast<float*>(kst);            // [P1_NGRP][128] maxima
  float* gl = gm + P1_NGRP * 128;                       // [P1_NGRP][128] sums
  if (warp < P1_EPI) {
    gm[(warp >> 2) * 128 + (warp & 3) * 32 + lane] = rm;
    gl[(warp >> 2) * 128 + (warp & 3) * 32 + lane] = rl;
  }
  __syncthreads();
  if (tid < 128) {
    const int m = rb * 128 + tid;
    if (m < M) {
      float mx = -INFINITY;
#pragma unroll
      for (int e = 0; e < P1_NGRP; ++e) mx = fmaxf(mx, gm[e * 128 + tid]);
      float l = 0.f;
      if (mx != -INFINITY) {
#pragma unroll
        for (int e = 0; e < P1_NGRP; ++e)
          if (gm[e * 128 + tid] != -INFINITY) l += gl[e * 128 + tid] * exp2f(gm[e * 128 + tid] - mx);
      }
      stats[((bl * s.G + g) * M + m) * n_chunks + blockIdx.x] = make_float2(mx, l);
    }
  }
  if (warp == 0) tmem_dealloc(tmem, 512);
  if (tid == 0 && sm.err) raise_status(dev_status, VARRATE_ERR_TIMEOUT);
}

// ------------------------------------------------------------------------------- pass 2
constexpr int P2_NGRP = 2;              // epilogue groups of four warps (tiles round-robin)
constexpr int P2_EPI = 4 * P2_NGRP;
constexpr int P2_THREADS = (P2_EPI + 2) * 32;
constexpr int P2_NACC = 4;              // TMEM accumulator slots (npad <= 128: 4 x 128 columns)
constexpr int P2_TM = 128;              // tokens per tile (MMA M)
constexpr int P2_ST = 5;                // key stages (<= 224 KB with a 256-row window block)
constexpr int P2_K = P2_TM * 256;       // 128 tokens x 128 bf16

struct P2Smem {
  uint64_t full[P2_ST], empty[P2_ST], tfull[P2_NACC], tempty[P2_NACC];
  uint32_t tmem;
  int err;
  alignas(16) float nlse[256];   // negated log2-sum-exp per window row (-inf for padding rows)
};

// grid (n_chunks2, G, B * L): raw_g[bl][g][t] = sum over the window rows of head g of
// 2^(S * log2e / sqrt(d) - lse_row) for the coded tokens t of this chunk.
__global__ void __launch_bounds__(P2_THREADS, 1)
salience_accum_tc_kernel(const __grid_constant__ CUtensorMap tk, const __nv_bfloat16* __restrict__ q_win,
                         const float2* __restrict__ stats, float* __restrict__ raw_g,
                         int32_t* __restrict__ dev_status, Shape s, int n_chunks, int64_t chunk2,
                         int npad) {
  extern __shared__ __align__(1024) unsigned char raw_smem[];
  unsigned char* smem = raw_smem + ((1024 - (smem_addr(raw_smem) & 1023)) & 1023);
  unsigned char* kst = smem;                                   // P2_ST x 32 KB
  unsigned char* qb = smem + P2_ST * P2_K;                     // npad rows x 128 bf16
  const int qbytes = (npad * 256 + 1023) & ~1023;
  P2Smem& sm = *reinterpret_cast<P2Smem*>(qb + qbytes);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int g = blockIdx.y;
  const int64_t bl = blockIdx.z;
  const int M = s.grp * s.w;
  const int64_t t_begin = (int64_t)blockIdx.x * chunk2;
  const int64_t t_end = min(s.n_coded, t_begin + chunk2);
  if (t_begin >= t_end) return;
  const int nt = (int)((t_end - t_begin + P2_TM - 1) / P2_TM);
  // accumulators of npad columns: four of 128 columns when npad <= 128, else two of 256
  const int acc_cols = npad <= 128 ? 128 : 256, nacc = 512 / acc_cols;

  if (warp < P2_EPI) {
    // window rows of head g (swizzled K-major) and their negated lse
    for (int idx = tid; idx < npad * 16; idx += P2_EPI * 32) {
      const int row = idx >> 4, cidx = idx & 15;
      uint4 v = make_uint4(0, 0, 0, 0);
      if (row < M) {
        const int h = g * s.grp + row / s.w, qq = row % s.w;
        v = __ldg(reinterpret_cast<const uint4*>(q_win + ((bl * s.w + qq) * s.H + h) * (int64_t)kHeadDim) + cidx);
      }
      *reinterpret_cast<uint4*>(qb + sw128_offset(row, cidx, npad)) = v;
    }
    for (int row = tid; row < npad; row += P2_EPI * 32) {
      float val = -INFINITY;
      if (row < M) {
        const float2* st = stats + ((bl * s.G + g) * M + row) * n_chunks;
        float mx = -INFINITY;
        for (int c = 0; c < n_chunks; ++c) mx = fmaxf(mx, st[c].x);
        float l = 0.f;
        for (int c = 0; c < n_chunks; ++c)
          if (st[c].x != -INFINITY) l += st[c].y * exp2f(st[c].x - mx);
        val = -(mx + log2f(l));
      }
      sm.nlse[row] = val;
    }
  }
  if (warp == P2_EPI + 1 && lane == 0) {
    for (int i = 0; i < P2_ST; ++i) { mbar_init(&sm.full[i], 1); mbar_init(&sm.empty[i], 1); }
    for (int i = 0; i < P2_NACC; ++i) { mbar_init(&sm.tfull[i], 1); mbar_init(&sm.tempty[i], 4); }
    sm.err = 0;
    fence_mbar_init();
  }
  if (warp == 0) tmem_alloc(&sm.tmem, 512);
  fence_proxy_async_smem();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = sm.tmem;
  const int64_t row0 = (bl * s.G + g) * s.N + t_begin;

  if (warp == P2_EPI) {
    if (lane == 0) {                                  // TMA producer
      for (int i = 0; i < nt; ++i) {
        const int st = i % P2_ST;
        if (!mbar_wait_bounded(&sm.empty[st], ((i / P2_ST) & 1) ^ 1, kTries)) { sm.err = 1; break; }
        mbar_arrive_expect_tx(&sm.full[st], P2_K);
        const int y = (int)(row0 + (int64_t)i * P2_TM);
        const uint32_t dst = smem_addr(kst + st * P2_K);
        tma_load_2d(dst, &tk, 0, y, &sm.full[st]);
        tma_load_2d(dst + P2_K / 2, &tk, 64, y, &sm.full[st]);
      }
    }
  } else if (warp == P2_EPI + 1) {
    if (lane == 0) {                                  // MMA issuer
      const uint32_t idesc = idesc_bf16_f32(P2_TM, npad);
      const uint32_t qa = smem_addr(qb);
      for (int i = 0; i < nt; ++i) {
        const int st = i % P2_ST, b = i % nacc;
        if (!mbar_wait_bounded(&sm.full[st], (i / P2_ST) & 1, kTries) ||
            !mbar_wait_bounded(&sm.tempty[b], ((i / nacc) & 1) ^ 1, kTries)) { sm.err = 1; break; }
        tc_fence_after();
        const uint32_t ka = smem_addr(kst + st * P2_K);
#pragma unroll
        for (int ks = 0; ks < kHeadDim / 16; ++ks) {
          const uint32_t offk = (ks >> 2) * (P2_K / 2) + (ks & 3) * 32;   // K panel: 128 rows
          const uint32_t offq = (ks >> 2) * (npad * 128) + (ks & 3) * 32; // Q panel: npad rows
          tc_mma_bf16(tmem + b * acc_cols, sdesc_sw128(ka + offk), sdesc_sw128(qa + offq), idesc, ks > 0);
        }
        tc_commit(&sm.empty[st]);
        tc_commit(&sm.tfull[b]);
      }
    }
  } else {                                            // epilogue: one token per thread
    const float scale = kLog2e * rsqrtf((float)kHeadDim);
    float* out = raw_g + (bl * s.G + g) * s.n_coded;
    const int eg = warp >> 2, row = tid & (P2_TM - 1);   // group eg takes tiles eg, eg + P2_NGRP, ...
    bool bad = false;
    for (int i = eg; i < nt; i += P2_NGRP) {
      const int b = i % nacc;
      if (!bad && !mbar_wait_bounded(&sm.tfull[b], (i / nacc) & 1, kTries)) { sm.err = 1; bad = true; }
      tc_fence_after();
      const uint32_t taddr = tmem + b * acc_cols + ((uint32_t)((warp & 3) * 32) << 16);
      // four partial sums in a fixed order (deterministic), so the adds do not form one chain
      float part[4] = {0.f, 0.f, 0.f, 0.f};
      for (int cb = 0; cb < npad; cb += 32) {
        float v[32];
        tmem_ld32(taddr + cb, v);
        const float4* nl = reinterpret_cast<const float4*>(sm.nlse + cb);
#pragma unroll
        for (int q4 = 0; q4 < 8; ++q4) {
          const float4 n = nl[q4];
          part[0] += fast_exp2(fmaf(v[4 * q4 + 0], scale, n.x));
          part[1] += fast_exp2(fmaf(v[4 * q4 + 1], scale, n.y));
          part[2] += fast_exp2(fmaf(v[4 * q4 + 2], scale, n.z));
          part[3] += fast_exp2(fmaf(v[4 * q4 + 3], scale, n.w));
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&sm.tempty[b]);
      const int64_t t = t_begin + (int64_t)i * P2_TM + row;
      if (t < t_end) out[t] = (part[0] + part[1]) + (part[2] + part[3]);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, 512);
  if (tid == 0 && sm.err) raise_status(dev_status, VARRATE_ERR_TIMEOUT);
}

// s'_t = (1 / pool) sum_{|i| <= pool/2} (1 / (w H)) sum_g raw_g[g][t + i], zero outside the coded set
// (heads summed in a fixed order: deterministic).
__global__ void salience_pool_tc_kernel(const float* __restrict__ raw_g, float* __restrict__ sal, Shape s) {
  const int64_t bl = blockIdx.y;
  const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= s.n_coded) return;
  const int half = s.pool / 2;
  const float* r = raw_g + bl * s.G * s.n_coded;
  const float inv = 1.0f / (float)(s.w * s.H);
  float acc = 0.f;
  for (int i = -half; i <= half; ++i) {
    const int64_t u = t + i;
    if (u < 0 || u >= s.n_coded) continue;
    float sg = 0.f;
    for (int g = 0; g < s.G; ++g) sg += r[(int64_t)g * s.n_coded + u];
    acc += sg * inv;
  }
  sal[bl * s.n_coded + t] = acc / (float)s.pool;
}

int round32(int x) { return (x + 31) & ~31; }

}  // namespace

bool salience_tc_supported(const Shape& s) {
  return s.dtype == VARRATE_BF16 && s.grp * s.w <= 256 &&
         (int64_t)s.B * s.L * s.G * s.N < (int64_t(1) << 31);
}

SalPlan salience_tc_plan(const Shape& s, int num_sms) {
  SalPlan p;
  p.n_rb = (s.grp * s.w + 127) / 128;
  const int64_t units = (int64_t)s.B * s.L * s.G * p.n_rb;
  int64_t n = (2LL * num_sms + units - 1) / units;
  int64_t chunk = (s.N + n - 1) / n;
  chunk = ((chunk + P1_TN - 1) / P1_TN) * P1_TN;
  p.chunk = chunk;
  p.n_chunks = (int)((s.N + chunk - 1) / chunk);
  const int64_t units2 = (int64_t)s.B * s.L * s.G;
  int64_t n2 = (2LL * num_sms + units2 - 1) / units2;
  int64_t c2 = (s.n_coded + n2 - 1) / n2;
  c2 = ((c2 + P2_TM - 1) / P2_TM) * P2_TM;
  p.chunk2 = c2 < P2_TM ? P2_TM : c2;
  p.n_chunks2 = (int)((s.n_coded + p.chunk2 - 1) / p.chunk2);
  return p;
}

size_t salience_tc_ws_bytes(const Shape& s, int num_sms) {
  const SalPlan p = salience_tc_plan(s, num_sms);
  size_t b = (size_t)s.B * s.L * s.G * s.grp * s.w * p.n_chunks * sizeof(float2);
  b = (b + 255) & ~size_t(255);
  b += (size_t)s.B * s.L * s.G * s.n_coded * sizeof(float);   // per-head raw salience
  return (b + 255) & ~size_t(255);
}

bool make_tmap_rows_bf16(CUtensorMap* map, const void* base, uint64_t rows, uint32_t box_rows);

int launch_salience_tc(const Shape& s, const void* q_win, const void* k, float* sal_out, void* ws,
                       int32_t* dev_status, int num_sms, cudaStream_t st) {
  if (s.n_coded == 0) return 0;
  const SalPlan p = salience_tc_plan(s, num_sms);
  const int M = s.grp * s.w;
  const int npad = round32(M);   // every TMEM column the epilogue reads is written by the MMA
  float2* stats = reinterpret_cast<float2*>(ws);
  size_t off = (size_t)s.B * s.L * s.G * M * p.n_chunks * sizeof(float2);
  off = (off + 255) & ~size_t(255);
  float* raw = reinterpret_cast<float*>(static_cast<char*>(ws) + off);
  const uint64_t rows = (uint64_t)s.B * s.L * s.G * s.N;
  CUtensorMap tmap1, tmap2;   // boxes of P1_TN and P2_TM rows
  if (!make_tmap_rows_bf16(&tmap1, k, rows, P1_TN) || !make_tmap_rows_bf16(&tmap2, k, rows, P2_TM)) return -1;
  const size_t smem1 = 1024 + P1_Q + P1_ST * P1_K + sizeof(P1Smem);
  cudaFuncSetAttribute(salience_stats_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem1);
  salience_stats_tc_kernel<<<dim3(p.n_chunks, s.G * p.n_rb, s.B * s.L), P1_THREADS, smem1, st>>>(
      tmap1, (const __nv_bfloat16*)q_win, stats, dev_status, s, p.n_chunks, p.chunk, p.n_rb);
  const size_t qbytes = ((size_t)npad * 256 + 1023) & ~size_t(1023);
  const size_t smem2 = 1024 + P2_ST * P2_K + qbytes + sizeof(P2Smem);
  cudaFuncSetAttribute(salience_accum_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem2);
  salience_accum_tc_kernel<<<dim3(p.n_chunks2, s.G, s.B * s.L), P2_THREADS, smem2, st>>>(
      tmap2, (const __nv_bfloat16*)q_win, stats, raw, dev_status, s, p.n_chunks, p.chunk2, npad);
  salience_pool_tc_kernel<<<dim3((unsigned)((s.n_coded + 255) / 256), s.B * s.L), 256, 0, st>>>(raw, sal_out, s);
  return 3;
}

}  // namespace vr
