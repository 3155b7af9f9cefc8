// Step 3 — rank-bucketed packing (layout tables) and projection (Algorithm 1's projection onto the
// basis; Eq. 5 with the anchor mean at 0).
//
// pack_tables (one CTA per (sequence, layer)):
//   count[r]           tokens of rank r (shared-memory histogram);
//   base[r_min] = 0,   base[r + 1] = base[r] + r * pad8(count[r])  (element offsets);
//   pos[t]             stable position of t among the tokens of its rank, computed 1024 tokens at a
//                      time with warp match/popc and a per-bucket prefix over the 32 warps;
//   perm[slot]         token of each slot, buckets in increasing rank;
//   pad slots          [count[r], pad8(count[r])) of every bucket of every stream set to 0.
// project (grid over slot chunks x (head, K/V) x (sequence, layer)): tokens are visited in
// bucketed slot order, so one coefficient of consecutive slots lands in consecutive addresses of
// its 8-slot group (layout: coef_offset in common.cuh).
#include "common.cuh"
#include "kernels.h"

namespace vr {

namespace {

constexpr int kMaxR = kHeadDim;  // r_max

template <typename T>
__global__ void __launch_bounds__(1024)
pack_tables_kernel(const uint8_t* __restrict__ ranks, int32_t* __restrict__ bucket_count,
                   int64_t* __restrict__ bucket_base, int32_t* __restrict__ perm,
                   int32_t* __restrict__ pos, T* __restrict__ coef, int32_t* __restrict__ dev_status,
                   Shape s) {
  __shared__ int cnt[kMaxR + 1];
  __shared__ int slot_start[kMaxR + 2];
  __shared__ long long base[kMaxR + 2];
  __shared__ int running[kMaxR + 1];
  __shared__ int wcnt[32][kMaxR + 1];
  __shared__ int wpref[32][kMaxR + 1];
  __shared__ int bad;
  const int64_t bl = blockIdx.x;
  const uint8_t* rk = ranks + bl * s.N;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;

  for (int r = tid; r <= kMaxR; r += blockDim.x) { cnt[r] = 0; running[r] = 0; }
  if (tid == 0) bad = 0;
  __syncthreads();
  for (int64_t t = tid; t < s.N; t += blockDim.x) {
    const int r = rk[t];
    if (r < s.r_min || r > s.r_max) bad = 1;
    else atomicAdd(&cnt[r], 1);
  }
  __syncthreads();
  if (bad) {
    if (tid == 0) {
      raise_status(dev_status, VARRATE_ERR_CORRUPT);
      // poison the table so the projection and decode skip this (sequence, layer)
      bucket_base[bl * (kMaxR + 2) + kMaxR + 1] = INT64_MAX;
    }
    return;
  }
  if (tid == 0) {
    long long b = 0;
    int ss = 0;
    for (int r = 0; r <= kMaxR; ++r) {
      base[r] = (r <= s.r_min) ? 0 : b;
      if (r >= s.r_min) b += (long long)r * pad8(cnt[r]);
      slot_start[r] = ss;
      ss += cnt[r];
    }
    base[kMaxR + 1] = b;
    slot_start[kMaxR + 1] = ss;
    if (b > s.cap) raise_status(dev_status, VARRATE_ERR_CORRUPT);
  }
  __syncthreads();
  for (int r = tid; r <= kMaxR + 1; r += blockDim.x) {
    if (r <= kMaxR) bucket_count[bl * (kMaxR + 1) + r] = cnt[r];
    bucket_base[bl * (kMaxR + 2) + r] = base[r];
  }
  if (base[kMaxR + 1] > s.cap) return;

  // stable positions, 1024 tokens per round
  const unsigned lt_mask = (1u << lane) - 1u;
  for (int64_t c0 = 0; c0 < s.N; c0 += blockDim.x) {
    for (int i = tid; i < 32 * (kMaxR + 1); i += blockDim.x) (&wcnt[0][0])[i] = 0;
    __syncthreads();
    const int64_t t = c0 + tid;
    const bool valid = t < s.N;
    const int r = valid ? (int)rk[t] : -1;
    const unsigned peers = __match_any_sync(0xffffffffu, r);
    const int within = __popc(peers & lt_mask);
    if (valid && within == 0) wcnt[warp][r] = __popc(peers);
    __syncthreads();
    if (tid <= kMaxR) {
      int acc = running[tid];
      for (int w = 0; w < 32; ++w) { wpref[w][tid] = acc; acc += wcnt[w][tid]; }
      running[tid] = acc;
    }
    __syncthreads();
    if (valid) {
      const int p = wpref[warp][r] + within;
      pos[bl * s.N + t] = p;
      perm[bl * s.N + slot_start[r] + p] = (int32_t)t;
    }
    __syncthreads();
  }

  // zero the padding slots of every stream of this (sequence, layer)
  const int64_t n_streams = (int64_t)s.G * 2;
  for (int r = s.r_min; r <= s.r_max; ++r) {
    const int n = cnt[r];
    const int npad = (int)(pad8(n) - n);
    if (npad == 0) continue;
    const int64_t per_stream = (int64_t)npad * r;
    const int64_t n8 = pad8(n);
    for (int64_t i = tid; i < n_streams * per_stream; i += blockDim.x) {
      const int64_t st = i / per_stream, rem = i % per_stream;
      const int64_t j = rem / npad, p = n + rem % npad;
      coef[(bl * n_streams + st) * s.cap + base[r] + coef_offset(r, n8, p, (int)j)] = from_f<T>(0.f);
    }
  }
}

constexpr int kTile = 64;
constexpr int kLd = kHeadDim + 4;

// grid (n_chunks, G * 2, B * L), 256 threads.
template <typename T>
__global__ void __launch_bounds__(256)
project_kernel(const T* __restrict__ k, const T* __restrict__ v, const T* __restrict__ basis_k,
               const T* __restrict__ basis_v, const uint8_t* __restrict__ ranks,
               const int32_t* __restrict__ bucket_count, const int64_t* __restrict__ bucket_base,
               const int32_t* __restrict__ perm, const int32_t* __restrict__ pos,
               T* __restrict__ coef, Shape s, int64_t chunk) {
  extern __shared__ float smem[];
  float* us = smem;                         // [128][kLd]  U rows
  float* xs = us + kHeadDim * kLd;          // [64][kLd]   gathered tokens, then coefficients
  __shared__ int stok[kTile], srk[kTile], spos[kTile];
  __shared__ int n8s[kMaxR + 1];
  __shared__ long long bases[kMaxR + 2];
  const int64_t bl = blockIdx.z;
  const int g = blockIdx.y >> 1, kv = blockIdx.y & 1;
  const int64_t l = bl % s.L;
  const int tid = threadIdx.x;

  for (int r = tid; r <= kMaxR + 1; r += blockDim.x) {
    if (r <= kMaxR) n8s[r] = (int)pad8(bucket_count[bl * (kMaxR + 1) + r]);
    bases[r] = bucket_base[bl * (kMaxR + 2) + r];
  }
  const T* U = (kv ? basis_v : basis_k) + (l * s.G + g) * (int64_t)kHeadDim * kHeadDim;
  for (int i = tid; i < kHeadDim * kHeadDim; i += blockDim.x)
    us[(i / kHeadDim) * kLd + (i % kHeadDim)] = to_f(U[i]);
  __syncthreads();
  if (bases[kMaxR + 1] > s.cap) return;   // corrupt tables were reported by pack_tables

  const T* x = (kv ? v : k) + (bl * s.G + g) * s.N * kHeadDim;
  T* out = coef + ((bl * s.G + g) * 2 + kv) * s.cap;
  const int ts = tid / 16, tj = tid % 16;
  const int64_t s_begin = blockIdx.x * chunk;
  const int64_t s_end = min(s.N, s_begin + chunk);
  for (int64_t s0 = s_begin; s0 < s_end; s0 += kTile) {
    __syncthreads();
    if (tid < kTile) {
      const int64_t sl = s0 + tid;
      int t = -1, r = 0, p = 0;
      if (sl < s_end) {
        t = perm[bl * s.N + sl];
        r = ranks[bl * s.N + t];
        p = pos[bl * s.N + t];
      }
      stok[tid] = t; srk[tid] = r; spos[tid] = p;
    }
    __syncthreads();
    for (int i = tid; i < kTile * kHeadDim; i += blockDim.x) {
      const int row = i / kHeadDim, c = i % kHeadDim;
      const int t = stok[row];
      xs[row * kLd + c] = t >= 0 ? to_f(x[(int64_t)t * kHeadDim + c]) : 0.f;
    }
    __syncthreads();
    float acc[4][8];
#pragma unroll
    for (int a = 0; a < 4; ++a)
#pragma unroll
      for (int i = 0; i < 8; ++i) acc[a][i] = 0.f;
#pragma unroll 4
    for (int c = 0; c < kHeadDim; c += 4) {
      float4 xv[4], uv[8];
#pragma unroll
      for (int a = 0; a < 4; ++a) xv[a] = *reinterpret_cast<const float4*>(&xs[(4 * ts + a) * kLd + c]);
#pragma unroll
      for (int i = 0; i < 8; ++i) uv[i] = *reinterpret_cast<const float4*>(&us[(tj + 16 * i) * kLd + c]);
#pragma unroll
      for (int a = 0; a < 4; ++a)
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          acc[a][i] = fmaf(xv[a].x, uv[i].x, acc[a][i]);
          acc[a][i] = fmaf(xv[a].y, uv[i].y, acc[a][i]);
          acc[a][i] = fmaf(xv[a].z, uv[i].z, acc[a][i]);
          acc[a][i] = fmaf(xv[a].w, uv[i].w, acc[a][i]);
        }
    }
    __syncthreads();
#pragma unroll
    for (int a = 0; a < 4; ++a)
#pragma unroll
      for (int i = 0; i < 8; ++i) xs[(4 * ts + a) * kLd + tj + 16 * i] = acc[a][i];
    __syncthreads();
    for (int i = tid; i < kTile * kHeadDim; i += blockDim.x) {
      const int slot = i % kTile, j = i / kTile;
      const int r = srk[slot];
      if (stok[slot] >= 0 && j < r)
        out[bases[r] + coef_offset(r, n8s[r], spos[slot], j)] = from_f<T>(xs[slot * kLd + j]);
    }
  }
}

}  // namespace

int launch_pack(const Shape& s, const void* k, const void* v, const void* basis_k,
                const void* basis_v, const varrate_packed& out, int32_t* dev_status, int num_sms,
                cudaStream_t st) {
  const int64_t units = (int64_t)s.B * s.L * s.G * 2;
  const int64_t want = 4LL * num_sms;
  int64_t n = (want + units - 1) / units;
  int64_t chunk = (s.N + n - 1) / n;
  chunk = ((chunk + kTile - 1) / kTile) * kTile;
  if (chunk < kTile) chunk = kTile;
  const int n_chunks = (int)((s.N + chunk - 1) / chunk);
  const size_t smem = (size_t)(kHeadDim + kTile) * kLd * sizeof(float);
  dim3 grid(n_chunks, s.G * 2, s.B * s.L);
  if (s.dtype == VARRATE_BF16) {
    using T = __nv_bfloat16;
    pack_tables_kernel<T><<<s.B * s.L, 1024, 0, st>>>(out.ranks, out.bucket_count, out.bucket_base,
                                                      out.perm, out.pos, (T*)out.coef, dev_status, s);
    const int np = launch_project_tc(s, k, v, basis_k, basis_v, out, dev_status, num_sms, st);
    return np < 0 ? -1 : 1 + np;
  } else {
    using T = float;
    pack_tables_kernel<T><<<s.B * s.L, 1024, 0, st>>>(out.ranks, out.bucket_count, out.bucket_base,
                                                      out.perm, out.pos, (T*)out.coef, dev_status, s);
    cudaFuncSetAttribute(project_kernel<T>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    project_kernel<T><<<grid, 256, smem, st>>>((const T*)k, (const T*)v, (const T*)basis_k,
                                               (const T*)basis_v, out.ranks, out.bucket_count,
                                               out.bucket_base, out.perm, out.pos, (T*)out.coef, s, chunk);
  }
  return 2;
}

}  // namespace vr
