// Step 3, bf16 — projection onto the per-head basis on the 5th-generation tensor cores
// (Algorithm 1's projection c_t = U x_t, Eq. 5 with the anchor mean at 0), written straight into
// the rank-bucketed layout.
//
// One CTA (4 warps) owns a range of bucketed slots of one (sequence, layer, head, K-or-V) stream.
//   gather   token perm[slot0 + i] (256 B) goes to row i of a 128 x 128 bf16 tile with 16-byte
//            cp.async (16 lanes per row, so one warp instruction moves two whole rows), already in
//            the K-major 128-byte-swizzled layout the tensor core reads; 5 stages, 4 tiles in flight. Tokens sit in slot order inside a bucket, so
//            the slot alone gives the rank (prefix search over bucket counts) and the position
//            (slot - bucket start); only perm is read, one tile ahead of its gather.
//   mma      one thread issues 8 x tcgen05.mma (M = 128 slots, N = 128 coefficients, K = 16) with
//            U (128 x 128, resident in shared memory) as B; fp32 accumulator in TMEM, two
//            128-column buffers so tile i's MMA overlaps tile i-1's epilogue; completion through
//            tcgen05.commit on an mbarrier (bounded wait).
//   epilogue warp w reads TMEM lanes 32w..32w+31 (row = slot) 32 columns at a time and stores
//            coefficient j < r_t of the slot's token at base[r] + j * pad8(n_r) + pos: lanes of
//            one bucket write consecutive addresses.
#include "common.cuh"
#include "kernels.h"

namespace vr {

namespace {

constexpr int kMaxR = kHeadDim;
constexpr int TM = 128;                    // slots per tile
constexpr int NST = 5;                     // gather stages
constexpr int TILE_BYTES = TM * kHeadDim * 2;
constexpr uint32_t kWaitTries = 1u << 22;  // bounded mbarrier polls

struct ProjSmem {
  uint64_t mma_bar[2];
  uint32_t tmem_base;
  int err;
  int tok[NST][TM];
  int rk[NST][TM];
  int ps[NST][TM];
  int n8[kMaxR + 1];
  int slot_start[kMaxR + 2];   // first bucketed slot of rank r (exclusive prefix of the counts)
  long long base[kMaxR + 2];
};

__global__ void __launch_bounds__(128, 1)
project_tc_kernel(const __nv_bfloat16* __restrict__ k, const __nv_bfloat16* __restrict__ v,
                  const __nv_bfloat16* __restrict__ basis_k, const __nv_bfloat16* __restrict__ basis_v,
                  const int32_t* __restrict__ bucket_count, const int64_t* __restrict__ bucket_base,
                  const int32_t* __restrict__ perm, __nv_bfloat16* __restrict__ coef,
                  int32_t* __restrict__ dev_status, Shape s, int64_t chunk) {
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  // 1024-byte alignment for the swizzled operand tiles
  unsigned char* smem = smem_raw + ((1024 - (smem_addr(smem_raw) & 1023)) & 1023);
  unsigned char* u_tile = smem;                                   // U, 32 KB
  unsigned char* stages = smem + TILE_BYTES;                      // NST x 32 KB
  ProjSmem& sm = *reinterpret_cast<ProjSmem*>(stages + NST * TILE_BYTES);

  const int tid = threadIdx.x, warp = tid >> 5;
  const int64_t bl = blockIdx.z;
  const int g = blockIdx.y >> 1, kv = blockIdx.y & 1;
  const int64_t l = bl % s.L;

  for (int r = tid; r <= kMaxR + 1; r += blockDim.x) {
    if (r <= kMaxR) sm.n8[r] = (int)pad8(bucket_count[bl * (kMaxR + 1) + r]);
    sm.base[r] = bucket_base[bl * (kMaxR + 2) + r];
  }
  if (tid == 0) {
    sm.err = 0;
    int acc = 0;
    for (int r = 0; r <= kMaxR; ++r) {
      sm.slot_start[r] = acc;
      acc += bucket_count[bl * (kMaxR + 1) + r];
    }
    sm.slot_start[kMaxR + 1] = acc;
  }
  __syncthreads();
  if (sm.base[kMaxR + 1] > s.cap || sm.base[kMaxR + 1] < 0) return;   // reported by pack_tables

  // U of this head into shared memory (row j = basis vector j), swizzled K-major
  const __nv_bfloat16* U = (kv ? basis_v : basis_k) + (l * s.G + g) * (int64_t)kHeadDim * kHeadDim;
  {
    const uint4* src = reinterpret_cast<const uint4*>(U + (int64_t)tid * kHeadDim);
#pragma unroll
    for (int c = 0; c < 16; ++c)
      *reinterpret_cast<uint4*>(u_tile + sw128_offset(tid, c, TM)) = __ldg(src + c);
  }
  if (warp == 0) tmem_alloc(&sm.tmem_base, 256);
  if (tid == 0) {
    mbar_init(&sm.mma_bar[0], 1);
    mbar_init(&sm.mma_bar[1], 1);
    fence_mbar_init();
  }
  fence_proxy_async_smem();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = sm.tmem_base;

  const __nv_bfloat16* x = (kv ? v : k) + (bl * s.G + g) * s.N * kHeadDim;
  __nv_bfloat16* out = coef + ((bl * s.G + g) * 2 + kv) * s.cap;
  const int64_t s_begin = blockIdx.x * chunk;
  const int64_t s_end = min(s.N, s_begin + chunk);
  const int n_tiles = (int)((s_end - s_begin + TM - 1) / TM);
  const uint32_t stage0 = smem_addr(stages), u_addr = smem_addr(u_tile);
  constexpr uint32_t idesc = idesc_bf16_f32(TM, kHeadDim);

  // perm of the next tile to gather, loaded one iteration ahead (-1 past the range)
  auto perm_of = [&](int i) -> int {
    const int64_t slot = s_begin + (int64_t)i * TM + tid;
    return (i < n_tiles && slot < s_end) ? perm[bl * s.N + slot] : -1;
  };
  // slot metadata of row `tid` of tile i (token, rank, position in bucket) into its stage
  auto stage_meta = [&](int i, int t) {
    if (i >= n_tiles) return;
    const int st = i % NST;
    const int slot = (int)(s_begin + (int64_t)i * TM + tid);
    int r = 0, p = 0;
    if (t >= 0) {
      int lo = 0, hi = kMaxR + 1;   // slot_start[lo] <= slot < slot_start[hi]
      while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if (sm.slot_start[mid] <= slot) lo = mid; else hi = mid;
      }
      r = lo;
      p = slot - sm.slot_start[lo];
    }
    sm.tok[st][tid] = t;
    sm.rk[st][tid] = r;
    sm.ps[st][tid] = p;
  };
  // copies of tile i (after its metadata is visible): 16 lanes per 256-byte row, so one warp
  // instruction moves two whole rows
  auto gather = [&](int i) {
    if (i < n_tiles) {
      const int st = i % NST;
      const uint32_t dst = stage0 + st * TILE_BYTES;
      const int c = tid & 15;
#pragma unroll
      for (int q = 0; q < TM / 8; ++q) {
        const int row = (tid >> 4) + 8 * q;
        const int t = sm.tok[st][row];
        const __nv_bfloat16* src = x + (int64_t)(t < 0 ? 0 : t) * kHeadDim + c * 8;
        cp_async16(dst + sw128_offset(row, c, TM), src, t >= 0 ? 16u : 0u);
      }
    }
    cp_async_commit();
  };

  auto epilogue = [&](int i) {
    const bool ok = mbar_wait_bounded(&sm.mma_bar[i & 1], (i >> 1) & 1, kWaitTries);
    if (!ok) sm.err = 1;
    tc_fence_after();
    const int st = i % NST;
    const int t = sm.tok[st][tid], r = sm.rk[st][tid], p = sm.ps[st][tid];
    const int rmax_w = __reduce_max_sync(0xffffffffu, t >= 0 ? r : 0);
    const long long b0 = sm.base[r];
    const int n8 = sm.n8[r];
    const uint32_t taddr = tmem + (uint32_t)((i & 1) * kHeadDim) + ((uint32_t)(warp * 32) << 16);
#pragma unroll
    for (int cb = 0; cb < kHeadDim / 32; ++cb) {
      if (cb * 32 >= rmax_w) break;            // warp-uniform
      float vals[32];
      tmem_ld32(taddr + cb * 32, vals);
      if (ok && t >= 0) {
#pragma unroll
        for (int jj = 0; jj < 32; ++jj) {
          const int j = cb * 32 + jj;
          if (j < r) out[b0 + (long long)j * n8 + p] = __float2bfloat16_rn(vals[jj]);
        }
      }
    }
  };

#pragma unroll
  for (int i = 0; i < NST - 1; ++i) stage_meta(i, perm_of(i));
  int t_next = perm_of(NST - 1);
  __syncthreads();
#pragma unroll
  for (int i = 0; i < NST - 1; ++i) gather(i);
  for (int i = 0; i < n_tiles; ++i) {
    cp_async_wait<NST - 2>();
    fence_proxy_async_smem();
    __syncthreads();
    if (tid == 0) {
      tc_fence_after();
      const uint32_t a0 = stage0 + (i % NST) * TILE_BYTES;
      const uint32_t d = tmem + (uint32_t)((i & 1) * kHeadDim);
#pragma unroll
      for (int ks = 0; ks < kHeadDim / 16; ++ks) {
        const uint32_t off = (ks >> 2) * (TM * 128) + (ks & 3) * 32;
        tc_mma_bf16(d, sdesc_sw128(a0 + off), sdesc_sw128(u_addr + off), idesc, ks > 0 ? 1u : 0u);
      }
      tc_commit(&sm.mma_bar[i & 1]);
    }
    if (i >= 1) epilogue(i - 1);
    // tile i + NST - 1 reuses the stage of tile i - 1, whose MMA and epilogue are complete
    stage_meta(i + NST - 1, t_next);
    t_next = perm_of(i + NST);
    tc_fence_before();
    __syncthreads();
    gather(i + NST - 1);
  }
  if (n_tiles >= 1) epilogue(n_tiles - 1);
  cp_async_wait<0>();
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, 256);
  if (tid == 0 && sm.err) raise_status(dev_status, VARRATE_ERR_TIMEOUT);
}

}  // namespace

size_t project_tc_smem_bytes() { return 1024 + (size_t)(1 + NST) * TILE_BYTES + sizeof(ProjSmem); }

int launch_project_tc(const Shape& s, const void* k, const void* v, const void* basis_k,
                      const void* basis_v, const varrate_packed& out, int32_t* dev_status,
                      int num_sms, cudaStream_t st) {
  const int64_t units = (int64_t)s.B * s.L * s.G * 2;
  int64_t n = (2LL * num_sms + units - 1) / units;
  int64_t chunk = (s.N + n - 1) / n;
  chunk = ((chunk + TM - 1) / TM) * TM;
  const int n_chunks = (int)((s.N + chunk - 1) / chunk);
  const size_t smem = project_tc_smem_bytes();
  cudaFuncSetAttribute(project_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  project_tc_kernel<<<dim3(n_chunks, s.G * 2, s.B * s.L), 128, smem, st>>>(
      (const __nv_bfloat16*)k, (const __nv_bfloat16*)v, (const __nv_bfloat16*)basis_k,
      (const __nv_bfloat16*)basis_v, out.bucket_count, out.bucket_base, out.perm,
      (__nv_bfloat16*)out.coef, dev_status, s, chunk);
  return 1;
}

}  // namespace vr
