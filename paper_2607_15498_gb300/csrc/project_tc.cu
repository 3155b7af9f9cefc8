// Step 3, bf16 — projection onto the per-head basis on the 5th-generation tensor cores
// (Algorithm 1's projection c_t = U x_t, Eq. 5 with the anchor mean at 0), written straight into
// the rank-bucketed layout.
//
// One CTA owns a range of bucketed slots of one (sequence, layer, head, K-or-V) stream and runs
// three warp roles over a 5-stage ring of 128-slot tiles:
//   producers (4 warps)  for tile i: token t = perm[slot]; rank r and in-bucket position p follow
//                        from the slot alone (tokens sit in slot order inside a bucket: r is found
//                        by a prefix search over the bucket counts, p = slot - bucket start). Token
//                        rows (256 B) are gathered with 16-byte cp.async, 16 lanes per row, into a
//                        128 x 128 bf16 tile in the K-major 128-byte-swizzled layout the tensor core
//                        reads; once a tile's copies have landed the producers fence the async proxy
//                        and arrive on the stage's mbarrier (two tiles stay in flight behind it).
//   mma (1 thread)       8 x tcgen05.mma (M = 128 slots, N = 128 coefficients, K = 16) with U
//                        (128 x 128, resident in shared memory) as B, into one of two TMEM
//                        accumulators; tcgen05.commit frees the stage and hands the accumulator on.
//   epilogue (4 warps)   warp w reads TMEM lanes 32w..32w+31 (row = slot) 32 columns at a time and
//                        stores coefficient j < r of the slot's token in the tiled bucket layout
//                        (coef_offset): lanes of one 8-slot group write consecutive addresses.
// Every mbarrier wait is bounded; a timeout raises VARRATE_ERR_TIMEOUT.
#include "common.cuh"
#include "kernels.h"

namespace vr {

namespace {

constexpr int kMaxR = kHeadDim;
constexpr int TM = 128;                    // slots per tile
constexpr int NST = 5;                     // operand stages
constexpr int NMETA = NST + 2;             // metadata ring (outlives the epilogue of its tile)
constexpr int LAG = 2;                     // copy groups kept in flight behind the signalled one
constexpr int TILE_BYTES = TM * kHeadDim * 2;
constexpr int kEpi = 4, kProd = 4;         // warps
constexpr int kThreads = (kEpi + kProd + 1) * 32;
constexpr int kProdThreads = kProd * 32;
constexpr int kRowsPer = TM / kProdThreads;     // metadata rows per producer thread
static_assert(TM % kProdThreads == 0 && kProdThreads % 16 == 0, "producer split");
constexpr uint32_t kWaitTries = 1u << 22;  // bounded mbarrier polls

struct ProjSmem {
  uint64_t full[NST], empty[NST], tfull[2], tempty[2];
  uint32_t tmem_base;
  int err;
  int tok[NMETA][TM];
  int rk[NMETA][TM];
  int ps[NMETA][TM];
  int n8[kMaxR + 1];
  int slot_start[kMaxR + 2];   // first bucketed slot of rank r (exclusive prefix of the counts)
  long long base[kMaxR + 2];
};

__global__ void __launch_bounds__(kThreads, 1)
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

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
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
  for (int idx = tid; idx < TM * 16; idx += blockDim.x) {
    const int row = idx >> 4, c = idx & 15;
    *reinterpret_cast<uint4*>(u_tile + sw128_offset(row, c, TM)) =
        __ldg(reinterpret_cast<const uint4*>(U + (int64_t)row * kHeadDim) + c);
  }
  if (warp == kEpi + kProd && lane == 0) {
    for (int i = 0; i < NST; ++i) { mbar_init(&sm.full[i], kProd * 32); mbar_init(&sm.empty[i], 1); }
    for (int i = 0; i < 2; ++i) { mbar_init(&sm.tfull[i], 1); mbar_init(&sm.tempty[i], kEpi); }
    fence_mbar_init();
  }
  if (warp == 0) tmem_alloc(&sm.tmem_base, 256);
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

  if (warp >= kEpi && warp < kEpi + kProd) {
    // ------------------------------------------------------------------ producers
    const int pt = tid - kEpi * 32;            // 0 .. kProdThreads - 1
    bool bad = false;
    auto signal = [&](int j) {                 // this thread's copies of tile j have landed
      fence_proxy_async_smem();
      mbar_arrive(&sm.full[j % NST]);
    };
    // perm of this thread's two rows, one tile ahead of its use
    auto perm_of = [&](int i, int row) -> int {
      const int64_t slot = s_begin + (int64_t)i * TM + row;
      return (i < n_tiles && slot < s_end) ? perm[bl * s.N + slot] : -1;
    };
    int t_next[kRowsPer];
#pragma unroll
    for (int h = 0; h < kRowsPer; ++h) t_next[h] = perm_of(0, pt + kProdThreads * h);
    for (int i = 0; i < n_tiles; ++i) {
      const int st = i % NST, mt = i % NMETA;
      int t_cur[kRowsPer];
#pragma unroll
      for (int h = 0; h < kRowsPer; ++h) {
        t_cur[h] = t_next[h];
        t_next[h] = perm_of(i + 1, pt + kProdThreads * h);
      }
      if (!bad && !mbar_wait_bounded(&sm.empty[st], ((i / NST) & 1) ^ 1, kWaitTries)) { sm.err = 1; bad = true; }
      // bucket of the tile's first slot (same search in every lane: broadcast reads), then a short
      // forward scan per row: buckets are in slot order
      const int slot0 = (int)(s_begin + (int64_t)i * TM);
      int r0 = 0;
      {
        int lo = 0, hi = kMaxR + 1;            // slot_start[lo] <= slot0 < slot_start[hi]
        while (hi - lo > 1) {
          const int mid = (lo + hi) >> 1;
          if (sm.slot_start[mid] <= slot0) lo = mid; else hi = mid;
        }
        r0 = lo;
      }
#pragma unroll
      for (int h = 0; h < kRowsPer; ++h) {
        const int row = pt + kProdThreads * h;
        const int slot = slot0 + row;
        const int t = t_cur[h];
        int r = 0, p = 0;
        if (t >= 0) {
          r = r0;
          while (sm.slot_start[r + 1] <= slot) ++r;
          p = slot - sm.slot_start[r];
        }
        sm.tok[mt][row] = t;
        sm.rk[mt][row] = r;
        sm.ps[mt][row] = p;
      }
      named_sync(1, kProd * 32);               // metadata of every row of the tile is visible
      const uint32_t dst = stage0 + st * TILE_BYTES;
      const int c = pt & 15;
#pragma unroll
      for (int q = 0; q < TM * 16 / kProdThreads; ++q) {
        const int row = (pt >> 4) + (kProdThreads / 16) * q;
        const int t = sm.tok[mt][row];
        const __nv_bfloat16* src = x + (int64_t)(t < 0 ? 0 : t) * kHeadDim + c * 8;
        cp_async16(dst + sw128_offset(row, c, TM), src, t >= 0 ? 16u : 0u);
      }
      cp_async_commit();
      if (i >= LAG) {
        cp_async_wait<LAG>();
        signal(i - LAG);
      }
    }
    cp_async_wait<0>();
    for (int j = max(0, n_tiles - LAG); j < n_tiles; ++j) signal(j);
  } else if (warp == kEpi + kProd) {
    // ------------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(TM, kHeadDim);
      for (int i = 0; i < n_tiles; ++i) {
        const int st = i % NST, b = i & 1;
        if (!mbar_wait_bounded(&sm.full[st], (i / NST) & 1, kWaitTries) ||
            !mbar_wait_bounded(&sm.tempty[b], ((i >> 1) & 1) ^ 1, kWaitTries)) { sm.err = 1; break; }
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
    for (int i = 0; i < n_tiles; ++i) {
      const int b = i & 1, mt = i % NMETA;
      if (!bad && !mbar_wait_bounded(&sm.tfull[b], (i >> 1) & 1, kWaitTries)) { sm.err = 1; bad = true; }
      tc_fence_after();
      const int t = sm.tok[mt][tid], r = sm.rk[mt][tid], p = sm.ps[mt][tid];
      const int rmax_w = __reduce_max_sync(0xffffffffu, t >= 0 ? r : 0);
      // this slot's position in its 128-slot tile (coef_offset): the row of coefficient j starts at
      // tile + j * tl, the slot's 8-group rotates by one position per row
      const long long p0 = ((long long)p >> 7) << 7;
      const int tl = (int)min(128LL, (long long)sm.n8[r] - p0);
      const int ng = max(tl >> 3, 1);
      const int pl = p - (int)p0;
      __nv_bfloat16* tile = out + sm.base[r] + p0 * r + (pl & 7);
      const uint32_t taddr = tmem + (uint32_t)(b * kHeadDim) + ((uint32_t)(warp * 32) << 16);
      int grp = (pl >> 3) % ng;
#pragma unroll
      for (int cb = 0; cb < kHeadDim / 32; ++cb) {
        if (cb * 32 >= rmax_w) break;          // warp-uniform
        float vals[32];
        tmem_ld32(taddr + cb * 32, vals);
#pragma unroll
        for (int jj = 0; jj < 32; ++jj) {
          const int j = cb * 32 + jj;
          if (!bad && t >= 0 && j < r) tile[(long long)j * tl + grp * 8] = __float2bfloat16_rn(vals[jj]);
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
  project_tc_kernel<<<dim3(n_chunks, s.G * 2, s.B * s.L), kThreads, smem, st>>>(
      (const __nv_bfloat16*)k, (const __nv_bfloat16*)v, (const __nv_bfloat16*)basis_k,
      (const __nv_bfloat16*)basis_v, out.bucket_count, out.bucket_base, out.perm,
      (__nv_bfloat16*)out.coef, dev_status, s, chunk);
  return 1;
}

}  // namespace vr
