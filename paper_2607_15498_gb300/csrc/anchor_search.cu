// Joint codec, nearest-anchor search (Sec. 3.1, Eq. 2), bf16, on the 5th-generation tensor cores.
//
// Every token's joint vector z_t = [k_t of heads 0..G-1 ; v_t of heads 0..G-1] (Eq. 1, D = 2 G d)
// is compared with the anchors z_{a * stride} by squared Euclidean distance,
//   dist(t, a) = |z_t|^2 + |z_a|^2 - 2 z_t . z_a,
// with the bf16 products exact and every sum in fp32 (the paper keeps this search in fp32: its
// bf16 form cancels). Two kernels:
//   anchor_prep_kernel    one pass over K and V: |z_t|^2 of every token (a warp per token, a fixed
//                         shuffle tree, so the value is reproducible), and the anchors copied into a
//                         dense [B L][2][G][n_ap][d] block (n_ap = anchor count rounded up to 256,
//                         padding rows zero with norm +inf, so they are never chosen);
//   anchor_search_tc_kernel  one CTA per 128 tokens of one (sequence, layer): S = Z_tile A^T by
//                         tcgen05.mma (M = 128 tokens x N = 256 anchors per accumulator, K = D in
//                         steps of 64 columns, each step one head half of K or V fed by TMA with a
//                         128-byte swizzle), both TMEM accumulators in use (512 columns) so that the
//                         epilogue of one anchor tile overlaps the products of the next. Epilogue
//                         thread = token row: it turns its 256 scores into distances and keeps the
//                         8 smallest (distance, anchor) pairs in registers, in lexicographic order;
//                         the two epilogue groups (alternate anchor tiles) merge their lists at the
//                         end and the first c pairs are stored.
// A third kernel, anchor_residual_kernel, forms the residuals e_t = z_t - z_bar_t of Eq. 2 from the
// lists (Algorithm 1, third step).
// Warp roles of the search kernel: one TMA producer warp, one MMA-issuing warp, eight epilogue
// warps (lane quarter = warp % 4). Every mbarrier wait is bounded; a timeout raises
// VARRATE_ERR_TIMEOUT.
#include <cudaTypedefs.h>
#include <math.h>

#include "common.cuh"
#include "kernels.h"

namespace vr {

namespace {

constexpr uint32_t kTries = 1u << 22;
constexpr int AS_TM = 128;                  // tokens per CTA (MMA M)
constexpr int AS_TN = 256;                  // anchors per accumulator (MMA N)
constexpr int AS_ST = 4;                    // operand stages
constexpr int AS_ABYTES = AS_TM * 128;      // 128 token rows x 64 bf16
constexpr int AS_BBYTES = AS_TN * 128;      // 256 anchor rows x 64 bf16
constexpr int AS_SBYTES = AS_ABYTES + AS_BBYTES;
constexpr int AS_NGRP = 2;                  // epilogue groups of four warps (alternate anchor tiles)
constexpr int AS_EPI = 4 * AS_NGRP;
constexpr int AS_THREADS = (AS_EPI + 2) * 32;
constexpr int AS_LIST = 8;                  // (distance, anchor) pairs kept per token

struct AsSmem {
  uint64_t full[AS_ST], empty[AS_ST], tfull[AS_NGRP], tempty[AS_NGRP];
  uint32_t tmem;
  int err;
  float md[AS_TM][AS_LIST];                 // group 1's lists, merged by group 0
  int mi[AS_TM][AS_LIST];
};

// ------------------------------------------------------------------------------ prep
// grid (ceil(N / 8), B * L), 256 threads: warp w takes token blockIdx.x * 8 + w.
__global__ void __launch_bounds__(256)
anchor_prep_kernel(const __nv_bfloat16* __restrict__ k, const __nv_bfloat16* __restrict__ v,
                   __nv_bfloat16* __restrict__ anchors, float* __restrict__ anorm,
                   float* __restrict__ tnorm, int G, int64_t N, int stride, int n_a, int n_ap) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t bl = blockIdx.y;
  const int64_t t = (int64_t)blockIdx.x * 8 + warp;
  if (t < N) {
    const bool is_anchor = (t % stride) == 0;
    const int64_t a = t / stride;
    float acc = 0.f;
    for (int kvg = 0; kvg < 2 * G; ++kvg) {
      const int kv = kvg >= G, g = kvg - kv * G;
      const __nv_bfloat16* row = (kv ? v : k) + ((bl * G + g) * N + t) * kHeadDim;
      const uint2 u = __ldg(reinterpret_cast<const uint2*>(row) + lane);   // 4 bf16 per lane
      const float x0 = __uint_as_float(u.x << 16), x1 = __uint_as_float(u.x & 0xffff0000u);
      const float x2 = __uint_as_float(u.y << 16), x3 = __uint_as_float(u.y & 0xffff0000u);
      acc = fmaf(x0, x0, acc);
      acc = fmaf(x1, x1, acc);
      acc = fmaf(x2, x2, acc);
      acc = fmaf(x3, x3, acc);
      if (is_anchor)
        reinterpret_cast<uint2*>(anchors + (((bl * 2 + kv) * G + g) * n_ap + a) * kHeadDim)[lane] = u;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    if (lane == 0) {
      tnorm[bl * N + t] = acc;
      if (is_anchor) anorm[bl * n_ap + a] = acc;
    }
  }
  // padding anchors [n_a, n_ap): zero rows, infinite norm (never among the nearest)
  if (blockIdx.x == 0) {
    const int pad = n_ap - n_a;
    for (int idx = threadIdx.x; idx < pad * 2 * G * 32; idx += blockDim.x) {
      const int ln = idx & 31, rest = idx >> 5;
      const int a = n_a + rest % pad, kvg = rest / pad;
      reinterpret_cast<uint2*>(anchors + ((bl * 2 * G + kvg) * n_ap + a) * kHeadDim)[ln] = make_uint2(0, 0);
    }
    for (int a = n_a + threadIdx.x; a < n_ap; a += blockDim.x) anorm[bl * n_ap + a] = INFINITY;
  }
}

// Insert (d, j) into the sorted list (bd, bi): lexicographic order on (distance, anchor), so equal
// distances keep the lower anchor first whatever order the pairs arrive in.
__device__ __forceinline__ void list_insert(float (&bd)[AS_LIST], int (&bi)[AS_LIST], float d, int j) {
  float cd = d;
  int ci = j;
#pragma unroll
  for (int s = 0; s < AS_LIST; ++s) {
    const bool lt = cd < bd[s] || (cd == bd[s] && ci < bi[s]);
    const float td = bd[s];
    const int ti = bi[s];
    bd[s] = lt ? cd : td;
    bi[s] = lt ? ci : ti;
    cd = lt ? td : cd;
    ci = lt ? ti : ci;
  }
}

// ------------------------------------------------------------------------------ search
// grid (ceil(N / 128), B * L).
__global__ void __launch_bounds__(AS_THREADS, 1)
anchor_search_tc_kernel(const __grid_constant__ CUtensorMap tk, const __grid_constant__ CUtensorMap tv,
                        const __grid_constant__ CUtensorMap ta, const float* __restrict__ tnorm,
                        const float* __restrict__ anorm, int32_t* __restrict__ idx_out,
                        float* __restrict__ dist_out, int32_t* __restrict__ dev_status, int G, int64_t N,
                        int n_ap, int c) {
  extern __shared__ __align__(1024) unsigned char raw_smem[];
  unsigned char* smem = raw_smem + ((1024 - (smem_addr(raw_smem) & 1023)) & 1023);
  AsSmem& sm = *reinterpret_cast<AsSmem*>(smem + AS_ST * AS_SBYTES);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int64_t bl = blockIdx.y;
  const int64_t t0 = (int64_t)blockIdx.x * AS_TM;
  const int n_kb = 4 * G;                    // 64-column steps over D = 2 G d
  const int n_at = n_ap / AS_TN;
  const int total = n_at * n_kb;

  if (warp == AS_EPI + 1 && lane == 0) {
    for (int i = 0; i < AS_ST; ++i) { mbar_init(&sm.full[i], 1); mbar_init(&sm.empty[i], 1); }
    for (int i = 0; i < AS_NGRP; ++i) { mbar_init(&sm.tfull[i], 1); mbar_init(&sm.tempty[i], 4); }
    sm.err = 0;
    fence_mbar_init();
  }
  if (warp == 0) tmem_alloc(&sm.tmem, AS_NGRP * AS_TN);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = sm.tmem;
  const uint32_t stage0 = smem_addr(smem);
  float bd[AS_LIST];
  int bi[AS_LIST];
#pragma unroll
  for (int s = 0; s < AS_LIST; ++s) { bd[s] = INFINITY; bi[s] = -1; }

  if (warp == AS_EPI) {
    if (lane == 0) {                                    // TMA producer
      for (int i = 0; i < total; ++i) {
        const int at = i / n_kb, kb = i - at * n_kb, st = i % AS_ST;
        if (!mbar_wait_bounded(&sm.empty[st], ((i / AS_ST) & 1) ^ 1, kTries)) { sm.err = 1; break; }
        const int kv = kb >= 2 * G;
        const int g = (kb >> 1) - kv * G, half = kb & 1;
        const uint32_t dst = stage0 + st * AS_SBYTES;
        mbar_arrive_expect_tx(&sm.full[st], AS_SBYTES);
        // token rows past N read the next stream's rows (or zeros past the tensor): never stored
        tma_load_2d(dst, kv ? &tv : &tk, 64 * half, (int)((bl * G + g) * N + t0), &sm.full[st]);
        tma_load_2d(dst + AS_ABYTES, &ta, 64 * half, (int)(((bl * 2 + kv) * G + g) * n_ap + at * AS_TN),
                    &sm.full[st]);
      }
    }
  } else if (warp == AS_EPI + 1) {
    if (lane == 0) {                                    // MMA issuer
      constexpr uint32_t idesc = idesc_bf16_f32(AS_TM, AS_TN);
      bool ok = true;
      for (int at = 0; at < n_at && ok; ++at) {
        const int b = at & 1;
        if (!mbar_wait_bounded(&sm.tempty[b], ((at >> 1) & 1) ^ 1, kTries)) { sm.err = 1; break; }
        tc_fence_after();
        for (int kb = 0; kb < n_kb; ++kb) {
          const int i = at * n_kb + kb, st = i % AS_ST;
          if (!mbar_wait_bounded(&sm.full[st], (i / AS_ST) & 1, kTries)) { sm.err = 1; ok = false; break; }
          tc_fence_after();
          const uint32_t a0 = stage0 + st * AS_SBYTES, b0 = a0 + AS_ABYTES;
#pragma unroll
          for (int ks = 0; ks < 4; ++ks)
            tc_mma_bf16(tmem + b * AS_TN, sdesc_sw128(a0 + ks * 32), sdesc_sw128(b0 + ks * 32), idesc,
                        (kb | ks) != 0);
          tc_commit(&sm.empty[st]);
        }
        if (ok) tc_commit(&sm.tfull[b]);
      }
    }
  } else {                                              // epilogue: one token row, alternate tiles
    const int quarter = warp & 3, eg = warp >> 2;
    const int row = quarter * 32 + lane;
    const int64_t t = t0 + row;
    const float nz = t < N ? tnorm[bl * N + t] : 0.f;
    const float* an = anorm + bl * n_ap;
    bool bad = false;
    for (int at = eg; at < n_at; at += AS_NGRP) {
      const int b = at & 1;
      if (!bad && !mbar_wait_bounded(&sm.tfull[b], (at >> 1) & 1, kTries)) { sm.err = 1; bad = true; }
      tc_fence_after();
      const uint32_t taddr = tmem + b * AS_TN + ((uint32_t)(quarter * 32) << 16);
#pragma unroll 1
      for (int cb = 0; cb < AS_TN / 32; ++cb) {
        float sv[32];
        tmem_ld32(taddr + cb * 32, sv);
        const int j0 = at * AS_TN + cb * 32;
        const float4* an4 = reinterpret_cast<const float4*>(an + j0);
#pragma unroll
        for (int q4 = 0; q4 < 8; ++q4) {
          const float4 na = __ldg(an4 + q4);
          const float nav[4] = {na.x, na.y, na.z, na.w};
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const int jj = q4 * 4 + e;
            const float dd = fmaxf(fmaf(-2.f, sv[jj], nz + nav[e]), 0.f);
            if (dd < bd[AS_LIST - 1]) list_insert(bd, bi, dd, j0 + jj);
          }
        }
        __syncwarp();
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&sm.tempty[b]);
    }
    if (eg == 1) {
#pragma unroll
      for (int s = 0; s < AS_LIST; ++s) { sm.md[row][s] = bd[s]; sm.mi[row][s] = bi[s]; }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp < 4) {                                       // group 0 merges and stores
    const int row = warp * 32 + lane;
    const int64_t t = t0 + row;
#pragma unroll
    for (int s = 0; s < AS_LIST; ++s)
      if (sm.mi[row][s] >= 0) list_insert(bd, bi, sm.md[row][s], sm.mi[row][s]);
    if (t < N && !sm.err) {
#pragma unroll
      for (int s = 0; s < AS_LIST; ++s) {
        if (s < c) {
          idx_out[(bl * N + t) * c + s] = bi[s];
          if (dist_out != nullptr) dist_out[(bl * N + t) * c + s] = bd[s];
        }
      }
    }
  }
  if (warp == 0) tmem_dealloc(tmem, AS_NGRP * AS_TN);
  if (tid == 0 && sm.err) raise_status(dev_status, VARRATE_ERR_TIMEOUT);
}

size_t search_smem_bytes() { return 1024 + (size_t)AS_ST * AS_SBYTES + sizeof(AsSmem); }

// ------------------------------------------------------------------------------ residual
// Eq. 2: e_t = z_t - mean of the anchors listed for t. grid (ceil(N / 8), B * L), 256 threads: warp w
// takes token blockIdx.x * 8 + w; lane l owns coordinates 4 l .. 4 l + 3 of every head row. The
// listed anchors are summed in list order in fp32 (bf16 values are exact in fp32), divided by
// their count (IEEE division), subtracted from z_t and rounded to bf16.
__global__ void __launch_bounds__(256)
anchor_residual_kernel(const __nv_bfloat16* __restrict__ k, const __nv_bfloat16* __restrict__ v,
                       const int32_t* __restrict__ idx, __nv_bfloat16* __restrict__ e,
                       int32_t* __restrict__ dev_status, int G, int64_t N, int stride, int c, int n_a) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t bl = blockIdx.y;
  const int64_t t = (int64_t)blockIdx.x * 8 + warp;
  if (t >= N) return;
  int ai[AS_LIST];
  int m = 0;
  bool bad = false;
#pragma unroll
  for (int s = 0; s < AS_LIST; ++s) {
    ai[s] = s < c ? __ldg(idx + (bl * N + t) * c + s) : -1;
    if (ai[s] >= n_a || ai[s] < -1) bad = true;
    if (ai[s] >= 0) ++m;
  }
  if (bad || m == 0) {                               // warp-uniform: every lane read the same list
    if (lane == 0) raise_status(dev_status, VARRATE_ERR_CORRUPT);
    return;
  }
  const float fm = (float)m;
  for (int kvg = 0; kvg < 2 * G; ++kvg) {
    const int kv = kvg >= G, g = kvg - kv * G;
    const __nv_bfloat16* base = (kv ? v : k) + (bl * G + g) * N * kHeadDim;
    const uint2 zu = __ldg(reinterpret_cast<const uint2*>(base + t * kHeadDim) + lane);
    float acc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int s = 0; s < AS_LIST; ++s) {
      if (ai[s] < 0) continue;
      const uint2 u = __ldg(reinterpret_cast<const uint2*>(base + (int64_t)ai[s] * stride * kHeadDim) + lane);
      acc[0] += __uint_as_float(u.x << 16);
      acc[1] += __uint_as_float(u.x & 0xffff0000u);
      acc[2] += __uint_as_float(u.y << 16);
      acc[3] += __uint_as_float(u.y & 0xffff0000u);
    }
    const float z0 = __uint_as_float(zu.x << 16), z1 = __uint_as_float(zu.x & 0xffff0000u);
    const float z2 = __uint_as_float(zu.y << 16), z3 = __uint_as_float(zu.y & 0xffff0000u);
    uint2 o;
    o.x = pack_bf16(__fsub_rn(z0, __fdiv_rn(acc[0], fm)), __fsub_rn(z1, __fdiv_rn(acc[1], fm)));
    o.y = pack_bf16(__fsub_rn(z2, __fdiv_rn(acc[2], fm)), __fsub_rn(z3, __fdiv_rn(acc[3], fm)));
    reinterpret_cast<uint2*>(e + ((bl * N + t) * 2 * G + kvg) * kHeadDim)[lane] = o;
  }
}

}  // namespace

bool make_tmap_rows_bf16(CUtensorMap* map, const void* base, uint64_t rows, uint32_t box_rows);

int anchor_count(int64_t N, int stride) { return (int)((N + stride - 1) / stride); }
int anchor_count_padded(int64_t N, int stride) {
  return (anchor_count(N, stride) + AS_TN - 1) / AS_TN * AS_TN;
}

size_t anchor_search_ws_bytes(const Shape& s, int stride) {
  const size_t n_ap = (size_t)anchor_count_padded(s.N, stride);
  const size_t bl = (size_t)s.B * s.L;
  auto a256 = [](size_t x) { return (x + 255) & ~size_t(255); };
  return a256(bl * 2 * s.G * n_ap * kHeadDim * 2) + a256(bl * n_ap * 4) + a256(bl * (size_t)s.N * 4);
}

bool anchor_residual_supported(const Shape& s, int stride, int c) {
  return s.dtype == VARRATE_BF16 && stride >= 1 && stride <= s.N && c >= 1 && c <= AS_LIST &&
         (int64_t)s.B * s.L <= 65535;
}

int launch_anchor_residual(const Shape& s, const void* k, const void* v, int stride, int c,
                           const int32_t* idx, void* e_out, int32_t* dev_status, cudaStream_t st) {
  anchor_residual_kernel<<<dim3((unsigned)((s.N + 7) / 8), (unsigned)((size_t)s.B * s.L)), 256, 0, st>>>(
      (const __nv_bfloat16*)k, (const __nv_bfloat16*)v, idx, (__nv_bfloat16*)e_out, dev_status, s.G, s.N,
      stride, c, anchor_count(s.N, stride));
  return 1;
}

bool anchor_search_supported(const Shape& s, int stride, int c) {
  if (s.dtype != VARRATE_BF16 || stride < 1 || stride > s.N || c < 1 || c > AS_LIST) return false;
  if ((int64_t)s.B * s.L > 65535 || s.G > 64) return false;
  const uint64_t rows_kv = (uint64_t)s.B * s.L * s.G * s.N;
  const uint64_t rows_a = (uint64_t)s.B * s.L * 2 * s.G * anchor_count_padded(s.N, stride);
  return rows_kv + AS_TM <= (uint64_t)INT32_MAX && rows_a <= (uint64_t)INT32_MAX;
}

int launch_anchor_search(const Shape& s, const void* k, const void* v, int stride, int c, int32_t* idx_out,
                         float* dist_out, int32_t* dev_status, void* ws, cudaStream_t st) {
  const int n_a = anchor_count(s.N, stride), n_ap = anchor_count_padded(s.N, stride);
  const size_t bl = (size_t)s.B * s.L;
  auto a256 = [](size_t x) { return (x + 255) & ~size_t(255); };
  char* w = static_cast<char*>(ws);
  __nv_bfloat16* anchors = reinterpret_cast<__nv_bfloat16*>(w);
  float* anorm = reinterpret_cast<float*>(w + a256(bl * 2 * s.G * n_ap * kHeadDim * 2));
  float* tnorm = reinterpret_cast<float*>(reinterpret_cast<char*>(anorm) + a256(bl * n_ap * 4));
  const uint64_t rows_kv = (uint64_t)s.B * s.L * s.G * s.N;
  const uint64_t rows_a = (uint64_t)bl * 2 * s.G * n_ap;
  CUtensorMap tk, tv, ta;
  if (!make_tmap_rows_bf16(&tk, k, rows_kv, AS_TM) || !make_tmap_rows_bf16(&tv, v, rows_kv, AS_TM) ||
      !make_tmap_rows_bf16(&ta, anchors, rows_a, AS_TN))
    return -1;
  anchor_prep_kernel<<<dim3((unsigned)((s.N + 7) / 8), (unsigned)bl), 256, 0, st>>>(
      (const __nv_bfloat16*)k, (const __nv_bfloat16*)v, anchors, anorm, tnorm, s.G, s.N, stride, n_a, n_ap);
  const size_t smem = search_smem_bytes();
  cudaFuncSetAttribute(anchor_search_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  anchor_search_tc_kernel<<<dim3((unsigned)((s.N + AS_TM - 1) / AS_TM), (unsigned)bl), AS_THREADS, smem, st>>>(
      tk, tv, ta, tnorm, anorm, idx_out, dist_out, dev_status, s.G, s.N, n_ap, c);
  return 2;
}

}  // namespace vr
