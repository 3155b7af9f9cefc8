// Step 3, bf16 — projection onto the per-head basis on the 5th-generation tensor cores
// (Algorithm 1's projection c_t = U x_t, Eq. 5 with the anchor mean at 0), written straight into
// the rank-bucketed layout.
//
// One CTA owns a range of tokens (in sequence order) of one (sequence, layer, head, K-or-V) stream
// and runs three warp roles over a 5-stage ring of 128-token tiles:
//   producer (1 thread)  two TMA tile loads per tile (64 columns x 128 rows each, 128-byte swizzle:
//                        the K-major operand layout of the tensor core) of 128 consecutive token
//                        rows; the K / V tensors are read once, front to back;
//   mma (1 thread)       8 x tcgen05.mma (M = 128 tokens, N = 128 coefficients, K = 16) with U
//                        (128 x 128, resident in shared memory) as B, into one of four TMEM
//                        accumulators; tcgen05.commit frees the stage and hands the accumulator on;
//   epilogue (16 warps)  four groups of four take the tiles round-robin (each group covers the 128 TMEM
//                        lanes); thread = token: reads its rank r and in-bucket position p (coalesced),
//                        then its TMEM row 32 columns at a time, and stores coefficient j < r at
//                        its slot of bucket r (coef_offset). Consecutive tokens of one rank hold
//                        consecutive slots, so each store instruction writes a few 16-byte runs.
// Every mbarrier wait is bounded; a timeout raises VARRATE_ERR_TIMEOUT.
#include <cudaTypedefs.h>

#include "common.cuh"
#include "kernels.h"

namespace vr {

namespace {

constexpr int kMaxR = kHeadDim;
constexpr int TM = 128;                    // tokens per tile
constexpr int NST = 5;                     // operand stages
constexpr int TILE_BYTES = TM * kHeadDim * 2;
constexpr int NGRP = 4;                    // epilogue groups of four warps (tiles round-robin)
constexpr int kEpi = 4 * NGRP;             // epilogue warps
constexpr int NACC = 4;                    // TMEM accumulators of 128 columns (all 512 columns)
constexpr int kThreads = (kEpi + 2) * 32;  // + producer warp + MMA warp
constexpr uint32_t kWaitTries = 1u << 22;  // bounded mbarrier polls

struct ProjSmem {
  uint64_t full[NST], empty[NST], tfull[NACC], tempty[NACC];
  uint32_t tmem_base;
  int err;
  int n8[kMaxR + 1];
  long long base[kMaxR + 2];
};

__global__ void __launch_bounds__(kThreads, 1)
project_tc_kernel(const __grid_constant__ CUtensorMap tk, const __grid_constant__ CUtensorMap tv,
                  const __nv_bfloat16* __restrict__ basis_k, const __nv_bfloat16* __restrict__ basis_v,
                  const int32_t* __restrict__ bucket_count, const int64_t* __restrict__ bucket_base,
                  const uint8_t* __restrict__ ranks, const int32_t* __restrict__ pos,
                  __nv_bfloat16* __restrict__ coef, int32_t* __restrict__ dev_status, Shape s,
                  int64_t chunk) {
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  // 1024-byte alignment for the swizzled operand tiles
  unsigned char* smem = smem_raw + ((1024 - (smem_addr(smem_raw) & 1023)) & 1023);
  unsigned char* u_tile = smem;                                   // U, 32 KB
  unsigned char* stages = smem + TILE_BYTES;                      // NST x 32 KB
  ProjSmem& sm = *reinterpret_cast<ProjSmem*>(stages + NST * TILE_BYTES);

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int64_t bl = blockIdx.z;
  const int g = blockIdx.y >> 1, kv = blockIdx.y & 1;
  const int64_t l = bl % s.L;

  for (int r = tid; r <= kMaxR + 1; r += blockDim.x) {
    if (r <= kMaxR) sm.n8[r] = (int)pad8(bucket_count[bl * (kMaxR + 1) + r]);
    sm.base[r] = bucket_base[bl * (kMaxR + 2) + r];
  }
  if (tid == 0) sm.err = 0;
  __syncthreads();
  if (sm.base[kMaxR + 1] > s.cap || sm.base[kMaxR + 1] < 0) return;   // reported by pack_tables

  // U of this head into shared memory (row j = basis vector j), swizzled K-major
  const __nv_bfloat16* U = (kv ? basis_v : basis_k) + (l * s.G + g) * (int64_t)kHeadDim * kHeadDim;
  for (int idx = tid; idx < TM * 16; idx += blockDim.x) {
    const int row = idx >> 4, c = idx & 15;
    *reinterpret_cast<uint4*>(u_tile + sw128_offset(row, c, TM)) =
        __ldg(reinterpret_cast<const uint4*>(U + (int64_t)row * kHeadDim) + c);
  }
  if (warp == kEpi && lane == 0) {
    for (int i = 0; i < NST; ++i) { mbar_init(&sm.full[i], 1); mbar_init(&sm.empty[i], 1); }
    for (int i = 0; i < NACC; ++i) { mbar_init(&sm.tfull[i], 1); mbar_init(&sm.tempty[i], 4); }
    fence_mbar_init();
  }
  if (warp == 0) tmem_alloc(&sm.tmem_base, NACC * kHeadDim);
  fence_proxy_async_smem();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = sm.tmem_base;

  __nv_bfloat16* out = coef + ((bl * s.G + g) * 2 + kv) * s.cap;
  const int64_t t_begin = blockIdx.x * chunk;
  const int64_t t_end = min(s.N, t_begin + chunk);
  const int n_tiles = (int)((t_end - t_begin + TM - 1) / TM);
  const uint32_t stage0 = smem_addr(stages), u_addr = smem_addr(u_tile);

  if (warp == kEpi) {
    // ------------------------------------------------------------------ producer
    if (lane == 0) {
      const CUtensorMap* map = kv ? &tv : &tk;
      const int row0 = (int)((bl * s.G + g) * s.N + t_begin);   // rows of the [B L G N][128] view
      for (int i = 0; i < n_tiles; ++i) {
        const int st = i % NST;
        if (!mbar_wait_bounded(&sm.empty[st], ((i / NST) & 1) ^ 1, kWaitTries)) { sm.err = 1; break; }
        const uint32_t dst = stage0 + st * TILE_BYTES;
        mbar_arrive_expect_tx(&sm.full[st], TILE_BYTES);
        // rows past the stream's end belong to the next stream (or read as zero): their results
        // are never stored
        tma_load_2d(dst, map, 0, row0 + i * TM, &sm.full[st]);
        tma_load_2d(dst + TM * 128, map, 64, row0 + i * TM, &sm.full[st]);
      }
    }
  } else if (warp == kEpi + 1) {
    // ------------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(TM, kHeadDim);
      for (int i = 0; i < n_tiles; ++i) {
        const int st = i % NST, b = i % NACC;
        if (!mbar_wait_bounded(&sm.full[st], (i / NST) & 1, kWaitTries) ||
            !mbar_wait_bounded(&sm.tempty[b], ((i / NACC) & 1) ^ 1, kWaitTries)) { sm.err = 1; break; }
        tc_fence_after();
        const uint32_t a0 = stage0 + st * TILE_BYTES;
        const uint32_t d = tmem + (uint32_t)(b * kHeadDim);
#pragma unroll
        for (int ks = 0; ks < kHeadDim / 16; ++ks) {
          const uint32_t off = (ks >> 2) * (TM * 128) + (ks & 3) * 32;
          tc_mma_bf16(d, sdesc_sw128(a0 + off), sdesc_sw128(u_addr + off), idesc, ks > 0 ? 1u : 0u);
        }
        tc_commit(&sm.empty[st]);
        tc_commit(&sm.tfull[b]);
      }
    }
  } else {
    // ------------------------------------------------------------------ epilogue
    bool bad = false;
    const int eg = warp >> 2, row = tid & (TM - 1);   // epilogue group (tiles eg, eg + NGRP, ...), token row
    // rank and bucket position of this thread's token, one tile of its group ahead of its use
    auto meta = [&](int i, int& r, int& p) {
      const int64_t t = t_begin + (int64_t)i * TM + row;
      const bool ok = i < n_tiles && t < t_end;
      r = ok ? (int)ranks[bl * s.N + t] : 0;
      p = ok ? pos[bl * s.N + t] : 0;
    };
    int r_next, p_next;
    meta(eg, r_next, p_next);
    for (int i = eg; i < n_tiles; i += NGRP) {
      const int b = i % NACC;
      const int r = r_next, p = p_next;
      meta(i + NGRP, r_next, p_next);
      const bool valid = r >= s.r_min && r <= s.r_max;   // a token of this stream, rank in range
      if (!bad && !mbar_wait_bounded(&sm.tfull[b], (i / NACC) & 1, kWaitTries)) { sm.err = 1; bad = true; }
      tc_fence_after();
      const int rmax_w = __reduce_max_sync(0xffffffffu, valid ? r : 0);
      // this slot's position in its 128-slot tile (coef_offset): the row of coefficient j starts at
      // tile + j * tl, the slot's 8-group rotates by one position per row
      const int rr = valid ? r : s.r_min;
      const long long p0 = ((long long)p >> 7) << 7;
      const int tl = (int)min(128LL, (long long)sm.n8[rr] - p0);
      const int ng = max(tl >> 3, 1);
      const int pl = p - (int)p0;
      __nv_bfloat16* tile = out + sm.base[rr] + p0 * rr + (pl & 7);
      const uint32_t taddr = tmem + (uint32_t)(b * kHeadDim) + ((uint32_t)((warp & 3) * 32) << 16);
      int grp = (pl >> 3) % ng;
#pragma unroll
      for (int cb = 0; cb < kHeadDim / 32; ++cb) {
        if (cb * 32 >= rmax_w) break;          // warp-uniform
        float vals[32];
        tmem_ld32(taddr + cb * 32, vals);
#pragma unroll
        for (int jj = 0; jj < 32; ++jj) {
          const int j = cb * 32 + jj;
          if (!bad && valid && j < r) tile[(long long)j * tl + grp * 8] = __float2bfloat16_rn(vals[jj]);
          grp = (grp + 1 == ng) ? 0 : grp + 1;
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&sm.tempty[b]);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, NACC * kHeadDim);
  if (tid == 0 && sm.err) raise_status(dev_status, VARRATE_ERR_TIMEOUT);
}

}  // namespace

size_t project_tc_smem_bytes() { return 1024 + (size_t)(1 + NST) * TILE_BYTES + sizeof(ProjSmem); }

bool make_tmap_rows_bf16(CUtensorMap* map, const void* base, uint64_t rows, uint32_t box_rows);

bool pack_ready(const Shape& s, const void* k, const void* v) {
  if (s.dtype != VARRATE_BF16) return true;
  const uint64_t rows = (uint64_t)s.B * s.L * s.G * s.N;
  CUtensorMap tk, tv;
  return rows <= (uint64_t)INT32_MAX && make_tmap_rows_bf16(&tk, k, rows, TM) &&
         make_tmap_rows_bf16(&tv, v, rows, TM);
}

int launch_project_tc(const Shape& s, const void* k, const void* v, const void* basis_k,
                      const void* basis_v, const varrate_packed& out, int32_t* dev_status,
                      int num_sms, cudaStream_t st) {
  const uint64_t rows = (uint64_t)s.B * s.L * s.G * s.N;
  if (rows > (uint64_t)INT32_MAX) return -1;   // TMA row coordinates are 32-bit
  CUtensorMap tk, tv;
  if (!make_tmap_rows_bf16(&tk, k, rows, TM) || !make_tmap_rows_bf16(&tv, v, rows, TM)) return -1;
  const int64_t units = (int64_t)s.B * s.L * s.G * 2;
  int64_t n = (2LL * num_sms + units - 1) / units;
  int64_t chunk = (s.N + n - 1) / n;
  chunk = ((chunk + TM - 1) / TM) * TM;
  const int n_chunks = (int)((s.N + chunk - 1) / chunk);
  const size_t smem = project_tc_smem_bytes();
  cudaFuncSetAttribute(project_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  project_tc_kernel<<<dim3(n_chunks, s.G * 2, s.B * s.L), kThreads, smem, st>>>(
      tk, tv, (const __nv_bfloat16*)basis_k, (const __nv_bfloat16*)basis_v, out.bucket_count,
      out.bucket_base, out.ranks, out.pos, (__nv_bfloat16*)out.coef, dev_status, s, chunk);
  return 1;
}

}  // namespace vr
