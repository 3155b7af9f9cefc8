// Step 4 for a window of new tokens, bf16 — decode attention of n_q consecutive queries per
// sequence in one call, on the packed coefficients (Sec. 3.1: attention over the cache of Eq. 5,
// with the most recent tokens kept exact; causal within the window).
//
// Query i of the window (0 <= i < n_q) is the token at position n_tail - n_q + i of the exact tail;
// it attends to every coded token and to the tail tokens 0 .. n_tail - n_q + i. Rows of one
// (sequence, KV head) are rho = i * group + h (R = n_q * group <= 128), taken in 8-row n-tiles.
//
// Three launches per call, each scheduled while its predecessor drains (programmatic dependent
// launch):
//  1. window_qfrag_kernel: q~[rho] = U_K q[rho] * log2(e)/sqrt(d) per (sequence, KV head), written
//     as the score-MMA B fragments (bf16 hi + lo) of each row group (the 16 rows one warp holds).
//  2. decode_window_kernel<RG>: the coded part. The cost line of decode_common.cuh cuts every
//     (sequence, head) stream into equal ranges over a persistent grid. The 8 warps of a CTA form
//     8 / RG teams of RG warps; a team takes every (8 / RG)-th 128-slot item of the CTA's range and
//     streams it once into its own shared-memory ring (1-D bulk copies, one per chunk of up to
//     8 KB, completing on per-stage mbarriers). Every warp of the team reads each chunk and computes
//     its own row group on it (warp rg of a team: n-tiles rg and rg + RG), so the coefficients are
//     read from HBM once whatever the number of query rows. The last warp of the team to release a
//     stage (a per-stage shared-memory count) refills it with the chunk SPT ahead.
//        scores  S^T[slot][row] += K^T[slot][j] Q~^T[j][row]   (m16n8k16, q~ split hi + lo)
//        softmax online per row, as in the single-query kernel (lazy max with kSlack headroom)
//        values  O~^T[j][row] += V[j][slot] P^T[slot][row]      (P in bf16)
//     The teams' states merge in shared memory into one partial (m, l, o~[128]) per row, per
//     (segment, CTA).
//  3. window_combine_kernel: per (sequence, KV head) and 8 rows, merges the partials of the CTAs
//     that shared the segment, adds the causal exact tail (scores and values in fp32 on CUDA
//     cores, 64 tokens at a time, online), rotates o~ back with U_V^T and normalises.
//
// Every bounded wait that gives up raises VARRATE_ERR_TIMEOUT; the CTA then streams nothing more,
// writes empty partials and waits (bounded) for its copies in flight before it exits.
#include <stddef.h>

#include <atomic>

#include "common.cuh"
#include "decode_common.cuh"
#include "kernels.h"

namespace vr {

namespace {

constexpr int NW = 8;                                      // warps per CTA
constexpr int kQfBytes = (kHeadDim / 16) * 2 * 32 * 16;    // one row group's q~ fragments (8 KB)
constexpr int kQfWords = kQfBytes / 16;                    // in uint4
constexpr int kPartStride = kHeadDim + 4;                  // o~[128], m, l, pad
constexpr int kAccStride = kHeadDim + 4;                   // merge buffer rows (bank spread)

template <int RG>
struct WinCfg {
  static constexpr int NTEAM = NW / RG;
  // ring stages per team: about 160-192 KB of ring in all, next to RG * 8 KB of q~ fragments
  static constexpr int SPT = RG == 1 ? 3 : (RG == 2 ? 5 : (RG == 4 ? 10 : 16));
  static constexpr int RING = NTEAM * SPT * STAGE;
  static constexpr int NBAR = NTEAM * SPT;
  static constexpr int ROWS = 16 * RG;                     // query rows a CTA can hold
};

struct WinTables {
  long long base[kMaxR + 2];
  int cnt[kMaxR + 1];
  int it_lo[kMaxR + 1];
  int it_pref[kMaxR + 2];
};

template <int RG>
struct WinMerge {   // aliases the ring once every warp has finished a segment
  float M[WinCfg<RG>::NTEAM][WinCfg<RG>::ROWS];
  float L[WinCfg<RG>::NTEAM][WinCfg<RG>::ROWS];
  float F[WinCfg<RG>::NTEAM][WinCfg<RG>::ROWS];
  float mx[WinCfg<RG>::ROWS], l[WinCfg<RG>::ROWS];
  float acc[WinCfg<RG>::NTEAM][WinCfg<RG>::ROWS][kAccStride];
};

template <int RG>
constexpr size_t win_smem_bytes() {
  return (size_t)WinCfg<RG>::RING + (size_t)RG * kQfBytes + sizeof(WinTables);
}

// ------------------------------------------------------------------ 1. rotated query fragments

// grid (B G, RG, 4), 256 threads. CTA (seg, rg, z) computes q~[rho][j] for the 16 rows of row group
// rg (n-tiles rg and rg + RG; rows past R are zero) and the 32 coefficients j in [32 z, 32 z + 32),
// and writes them as fragments
//   qf[seg][rg][jc][u][lane] = {hi(b0), hi(b1), lo(b0), lo(b1)}   (uint4, jc = 2 z, 2 z + 1)
// with b0 = (q~[rho][16 jc + 2c], q~[rho][16 jc + 2c + 1]), b1 the same 8 columns later,
// rho = 8 n-tile(u) + lane / 4, c = lane % 4: the B operand of m16n8k16 for k = 16 jc .. 16 jc + 15.
constexpr int kQfJ = 32;   // coefficients per CTA
__global__ void __launch_bounds__(256)
window_qfrag_kernel(const __nv_bfloat16* __restrict__ basis_k, const __nv_bfloat16* __restrict__ q,
                    uint4* __restrict__ qf, Shape s, int layer, int n_q, int rg_count, int ntt) {
  __shared__ float ut[kHeadDim][kQfJ + 1];   // U_K rows 32 z .. 32 z + 31, transposed
  __shared__ float qs[16][kHeadDim];         // query rows
  __shared__ float qt[16][kQfJ + 1];         // rotated rows
  const int tid = threadIdx.x;
  const long long seg = blockIdx.x;
  const int rg = blockIdx.y, z = blockIdx.z;
  const int b = (int)(seg / s.G), g = (int)(seg % s.G);
  const int R = n_q * s.grp;
  pdl_trigger();
  pdl_wait();
  const __nv_bfloat16* U = basis_k + ((long long)layer * s.G + g) * kHeadDim * kHeadDim + (long long)z * kQfJ * kHeadDim;
  // 32 rows x 128 bf16 = 512 uint4: two per thread, both loads in flight
  {
    const uint4* u4 = reinterpret_cast<const uint4*>(U);
    const uint4 v0 = __ldg(u4 + tid), v1 = __ldg(u4 + tid + 256);
    const uint4 vv[2] = {v0, v1};
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int e = tid + 256 * h, j = e >> 4, i0 = (e & 15) * 8;
      const uint32_t w[4] = {vv[h].x, vv[h].y, vv[h].z, vv[h].w};
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        ut[i0 + 2 * k][j] = __uint_as_float(w[k] << 16);
        ut[i0 + 2 * k + 1][j] = __uint_as_float(w[k] & 0xffff0000u);
      }
    }
  }
  // local row l: n-tile rg (l < 8) or rg + RG, row 8 * nt + l % 8; 16 rows x 16 uint4
  {
    const int l = tid >> 4, c4 = tid & 15;
    const int nt = l < 8 ? rg : rg + rg_count;
    const int rho = 8 * nt + (l & 7);
    uint4 v = make_uint4(0u, 0u, 0u, 0u);
    if (nt < ntt && rho < R) {
      const int iq = rho / s.grp, h = rho % s.grp;
      v = __ldg(reinterpret_cast<const uint4*>(q + (((long long)b * n_q + iq) * s.H + (long long)g * s.grp + h) * kHeadDim) + c4);
    }
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      qs[l][c4 * 8 + 2 * k] = __uint_as_float(w[k] << 16);
      qs[l][c4 * 8 + 2 * k + 1] = __uint_as_float(w[k] & 0xffff0000u);
    }
  }
  __syncthreads();
  {   // thread: coefficient j = tid % 32, rows l0 .. l0 + 1 (l0 = 2 (tid / 32))
    const int j = tid & (kQfJ - 1), l0 = (tid >> 5) * 2;
    float a0 = 0.f, a1 = 0.f;
#pragma unroll 8
    for (int i = 0; i < kHeadDim; ++i) {
      const float u = ut[i][j];
      a0 = fmaf(u, qs[l0][i], a0);
      a1 = fmaf(u, qs[l0 + 1][i], a1);
    }
    const float scale = kLog2e * rsqrtf((float)kHeadDim);
    qt[l0][j] = a0 * scale;
    qt[l0 + 1][j] = a1 * scale;
  }
  __syncthreads();
  uint4* dst = qf + (seg * rg_count + rg) * kQfWords + (long long)z * 2 * 2 * 32;
  if (tid < 2 * 2 * 32) {
    const int jl = tid / 64, u = (tid / 32) & 1, lane = tid & 31;   // jc = 2 z + jl
    const int l = u * 8 + (lane >> 2), j = jl * 16 + 2 * (lane & 3);
    uint32_t h0, l0, h1, l1;
    split_bf16(qt[l][j], qt[l][j + 1], h0, l0);
    split_bf16(qt[l][j + 8], qt[l][j + 9], h1, l1);
    dst[tid] = make_uint4(h0, h1, l0, l1);
  }
}

// ------------------------------------------------------------------ 2. coded part

// Producer cursor of a team: the next chunk of its item stream (items k, k + NTEAM, ...).
struct WProd {
  int k;
  Item item;
  int phase;   // 0 = K rows, 1 = V rows
  int jc;      // chunk index inside the phase
};

// Geometry of the cursor's chunk (element offset in its stream, bytes, K or V), then advance the
// cursor. Every warp of a team runs the same cursor; only the warp that refills a stage issues.
template <int NTEAM>
__device__ __forceinline__ bool take_chunk(WProd& p, const WinTables& sm, int total, long long& off,
                                           uint32_t& bytes, int& kv) {
  if (p.k >= total) return false;
  const int r = p.item.r;
  const long long n8 = pad8(sm.cnt[r]);
  const long long t0 = (long long)p.item.it * ISL;
  const long long tl = min((long long)ISL, n8 - t0);
  const int lgc = chunk_lg((int)tl);
  const int j0 = p.jc << lgc;
  const int rows = min(1 << lgc, r - j0);
  bytes = (uint32_t)(rows * tl * 2);
  off = sm.base[r] + t0 * r + (long long)j0 * tl;
  kv = p.phase;
  const int nj = (r + (1 << lgc) - 1) >> lgc;
  if (++p.jc == nj) {
    p.jc = 0;
    if (++p.phase == 2) {
      p.phase = 0;
      p.k += NTEAM;
      if (p.k < total) p.item = next_rr<NTEAM>(sm, p.item, p.k);
    }
  }
  return true;
}

template <int RG>
__global__ void __launch_bounds__(NW * 32, 1)
decode_window_kernel(const __nv_bfloat16* __restrict__ coef, const int32_t* __restrict__ bucket_count,
                     const int64_t* __restrict__ bucket_base, const uint4* __restrict__ qf,
                     float* __restrict__ part, int32_t* __restrict__ dev_status, Shape s, int layer,
                     int ntt) {
  using Cf = WinCfg<RG>;
  constexpr int NTEAM = Cf::NTEAM, SPT = Cf::SPT;
  extern __shared__ __align__(128) unsigned char smem[];
  const uint32_t ring = smem_addr(smem);
  const uint4* qfs = reinterpret_cast<const uint4*>(smem + Cf::RING);
  static_assert(Cf::RING % 16 == 0 && kQfBytes % 16 == 0, "aligned shared-memory regions");
  WinTables& sm = *reinterpret_cast<WinTables*>(smem + Cf::RING + RG * kQfBytes);
  static_assert(sizeof(WinMerge<RG>) <= (size_t)Cf::RING, "merge buffers fit in the ring");
  WinMerge<RG>& mg = *reinterpret_cast<WinMerge<RG>*>(smem);
  __shared__ long long segW[64];
  __shared__ long long segP[65];
  __shared__ long long cuts[kMaxCtas + 1];
  __shared__ uint64_t bar[Cf::NBAR];   // full barrier per ring stage
  __shared__ uint32_t relc[Cf::NBAR];  // releases of each stage (monotonic; RG per refill)
  __shared__ uint32_t iss[Cf::NBAR];   // copies issued into each stage
  __shared__ uint64_t bar_q;           // q~ fragments of the segment

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int g8 = lane >> 2, c = lane & 3;
  const int rg = warp % RG, team = warp / RG;
  const int C = gridDim.x, cta = blockIdx.x;
  const bool has_b = rg + RG < ntt;   // warp-uniform: the warp's second n-tile holds rows
  const uint64_t policy = l2_evict_first_policy();

  pdl_trigger();
  if (tid < Cf::NBAR) { mbar_init(&bar[tid], 1); relc[tid] = 0u; iss[tid] = 0u; }
  if (tid == Cf::NBAR) mbar_init(&bar_q, 1);
  fence_mbar_init();
  fence_proxy_async_smem();
  pdl_wait();
  seg_lengths(bucket_base, s, layer, segW, segP, tid);
  const long long T = segP[64];
  for (int c2 = tid; c2 <= C; c2 += blockDim.x) cuts[c2] = cut_at(T, c2, C);
  __syncthreads();
  const long long lo_g = cuts[cta], hi_g = cuts[cta + 1];
  int b, g;
  segment_at(segP, segW, s.B, s.G, lo_g, b, g);
  auto seg_start = [&](int bb, int gg) { return segP[bb] + gg * (segW[bb] + kSegCost + kSegEnd) + kSegCost; };
  bool more = b < s.B && seg_start(b, g) < hi_g;

  const uint32_t ring_t = ring + team * SPT * STAGE;
  uint64_t* bars = &bar[team * SPT];
  uint32_t* rel = &relc[team * SPT];
  uint32_t* issc = &iss[team * SPT];
  uint32_t n_cons = 0;     // chunks of the team consumed by this warp (the team's chunk counter)
  uint32_t n_qf = 0;       // q~ copies issued
  bool timed_out = false;  // a bounded wait of this thread gave up
  bool dead = false;       // CTA-uniform: stop streaming, write empty partials

  while (more) {
    const long long W = segW[b];
    const long long P = seg_start(b, g);
    const long long lo = max(lo_g, P) - P, hi = min(hi_g, P + W) - P;
    const long long bl = (long long)b * s.L + layer;
    const long long seg = (long long)b * s.G + g;
    if (tid == 0 && !dead) {   // the previous segment's readers of qfs are past its last barrier
      fence_proxy_async_smem();
      mbar_arrive_expect_tx(&bar_q, RG * kQfBytes);
      bulk_g2s(smem_addr(qfs), qf + seg * RG * kQfWords, RG * kQfBytes, &bar_q);
    }
    for (int r = tid; r <= kMaxR + 1; r += blockDim.x) {
      if (r <= kMaxR) sm.cnt[r] = bucket_count[bl * (kMaxR + 1) + r];
      sm.base[r] = bucket_base[bl * (kMaxR + 2) + r];
    }
    __syncthreads();
    for (int r = tid; r <= kMaxR; r += blockDim.x) {
      long long i0 = 0, i1 = 0;
      if (r >= s.r_min && r <= s.r_max) bucket_range(sm, r, lo, hi, i0, i1);
      sm.it_lo[r] = (int)i0;
      sm.it_pref[r + 1] = (int)(i1 - i0);
    }
    __syncthreads();
    if (warp == 0) {   // inclusive scan of it_pref[1 .. 129], 5 entries per lane
      constexpr int kPer = (kMaxR + 1 + 31) / 32;
      int v[kPer], acc = 0;
#pragma unroll
      for (int e = 0; e < kPer; ++e) {
        const int r = lane * kPer + e;
        acc += r <= kMaxR ? sm.it_pref[r + 1] : 0;
        v[e] = acc;
      }
      int excl = acc;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, excl, o);
        if (lane >= o) excl += y;
      }
      excl -= acc;
#pragma unroll
      for (int e = 0; e < kPer; ++e) {
        const int r = lane * kPer + e;
        if (r <= kMaxR) sm.it_pref[r + 1] = excl + v[e];
      }
      if (lane == 0) sm.it_pref[0] = 0;
    }
    __syncthreads();

    const __nv_bfloat16* cK = coef + ((bl * s.G + g) * 2) * s.cap;
    const __nv_bfloat16* cV = cK + s.cap;
    const int total = dead ? 0 : sm.it_pref[kMaxR + 1];
    WProd pr;
    pr.k = team; pr.phase = 0; pr.jc = 0;
    if (pr.k < total) pr.item = item_at(sm, pr.k);
    int cons_k = pr.k;
    Item cons = pr.item;

    // chunk n of the team sits in stage n % SPT, completing phase (n / SPT) & 1 of its barrier
    auto produce = [&](bool do_issue, uint32_t n) {
      long long off;
      uint32_t bytes;
      int kv;
      if (!take_chunk<NTEAM>(pr, sm, total, off, bytes, kv)) return;
      if (do_issue && lane == 0) {
        const uint32_t st = n % SPT;
        issc[st] += 1u;   // before the arrive: whoever refills the stage next sees it
        mbar_arrive_expect_tx(&bars[st], bytes);
        fence_proxy_async_smem();
        bulk_g2s_hint(ring_t + st * STAGE, (kv ? cV : cK) + off, bytes, &bars[st], policy);
      }
      __syncwarp();
    };
    auto wait_chunk = [&]() -> bool {
      if (!mbar_wait_bounded(&bars[n_cons % SPT], (n_cons / SPT) & 1u, kWaitTries)) {
        timed_out = true;
        return false;
      }
      return true;
    };
    // this warp has read the stage of chunk n_cons; the last of the team's RG warps refills it
    auto release = [&]() {
      __syncwarp();
      const uint32_t n = n_cons++;
      bool last = true;
      if constexpr (RG > 1) {
        uint32_t old = 0;
        if (lane == 0) old = atom_add_acq_rel_cta_smem(&rel[n % SPT], 1u);
        old = __shfl_sync(0xffffffffu, old, 0);
        last = (old + 1u) % (uint32_t)RG == 0u;
      }
      produce(last, n + SPT);
    };

    for (int i = 0; i < SPT; ++i) produce(rg == 0, n_cons + i);   // the team's ring fills up
    int c0, c1;
    seg_cta_range([&](int i) { return cuts[i]; }, T, C, P, W, c0, c1);
    if (!dead) {
      if (!mbar_wait_bounded(&bar_q, n_qf & 1u, kWaitTries)) timed_out = true;
      ++n_qf;
    }
    __syncwarp();

    float Mx[2][2] = {{-INFINITY, -INFINITY}, {-INFINITY, -INFINITY}};
    float Ls[2][2] = {{0.f, 0.f}, {0.f, 0.f}};
    float oacc[kHeadDim / 16][2][4];
#pragma unroll
    for (int t = 0; t < kHeadDim / 16; ++t)
#pragma unroll
      for (int u = 0; u < 2; ++u) oacc[t][u][0] = oacc[t][u][1] = oacc[t][u][2] = oacc[t][u][3] = 0.f;
    const uint4* qf_w = qfs + rg * (kHeadDim / 16) * 2 * 32 + lane;   // this warp's row group

    while (cons_k < total && !timed_out) {
      const int r = cons.r;
      const long long n_real = sm.cnt[r] - (long long)cons.it * ISL;
      const int tl = (int)min((long long)ISL, pad8(sm.cnt[r]) - (long long)cons.it * ISL);
      const int ng = tl >> 3;
      const bool full_tile = ng == 16;
      const uint32_t row_bytes = (uint32_t)tl * 2u;
      const int lgc = chunk_lg(tl);
      const int nj = (r + (1 << lgc) - 1) >> lgc;
      const int m = lane >> 3, r8 = lane & 7;
      float sc[ISL / 16][2][4];
#pragma unroll
      for (int t = 0; t < ISL / 16; ++t)
#pragma unroll
        for (int u = 0; u < 2; ++u) sc[t][u][0] = sc[t][u][1] = sc[t][u][2] = sc[t][u][3] = 0.f;

      // ---- K chunks: scores for both n-tiles of the warp
      for (int jc = 0; jc < nj; ++jc) {
        if (!wait_chunk()) break;
        const uint32_t st_addr = ring_t + (n_cons % SPT) * STAGE;
        const int j0 = jc << lgc, j1 = min(r, j0 + (1 << lgc));
        for (int j16 = j0; j16 < j1; j16 += 16) {
          const uint4 qa = qf_w[((j16 >> 4) * 2 + 0) * 32];
          const uint4 qb = has_b ? qf_w[((j16 >> 4) * 2 + 1) * 32] : make_uint4(0u, 0u, 0u, 0u);
          const int jrow = (j16 - j0) + (m >> 1) * 8 + r8;
          const int j = j0 + jrow;
          const uint32_t row_addr = st_addr + jrow * row_bytes;
          uint32_t off[ISL / 16];
          if (full_tile) {
            const uint32_t o0 = (uint32_t)(((m & 1) + j) & 15) << 4;
#pragma unroll
            for (int mt = 0; mt < ISL / 16; ++mt) off[mt] = (o0 + 32u * mt) & 255u;
          } else {
            int pg = ((m & 1) + j) % ng;
#pragma unroll
            for (int mt = 0; mt < ISL / 16; ++mt) { off[mt] = 16u * pg; pg = wrap2(pg, ng); }
          }
          const bool tail_rows = j16 + 16 > r;   // warp-uniform
          const int jb = j16 + 2 * c;
          const uint32_t m0 = keep_rows(0xFFFFFFFFu, jb, r), m1 = keep_rows(0xFFFFFFFFu, jb + 8, r);
#pragma unroll
          for (int h = 0; h < 2; ++h) {   // slot tiles 4h .. 4h + 3
            uint32_t a[4][4];
#pragma unroll
            for (int t = 0; t < 4; ++t) {
              ldsm_x4_trans(row_addr + off[4 * h + t], a[t]);
              if (tail_rows) { a[t][0] &= m0; a[t][1] &= m0; a[t][2] &= m1; a[t][3] &= m1; }
            }
#pragma unroll
            for (int t = 0; t < 4; ++t) mma_bf16_16816(sc[4 * h + t][0], a[t], qa.x, qa.y);
#pragma unroll
            for (int t = 0; t < 4; ++t) mma_bf16_16816(sc[4 * h + t][0], a[t], qa.z, qa.w);
            if (has_b) {
#pragma unroll
              for (int t = 0; t < 4; ++t) mma_bf16_16816(sc[4 * h + t][1], a[t], qb.x, qb.y);
#pragma unroll
              for (int t = 0; t < 4; ++t) mma_bf16_16816(sc[4 * h + t][1], a[t], qb.z, qb.w);
            }
          }
        }
        release();
      }
      if (timed_out) break;

      // ---- online softmax, rows 8 nt + 2c + e of n-tile u
      const bool full_item = n_real >= ISL;
      float mloc[2][2] = {{-INFINITY, -INFINITY}, {-INFINITY, -INFINITY}};
#pragma unroll
      for (int mt = 0; mt < ISL / 16; ++mt) {
        if (!full_item) {
          const int s0 = mt * 16 + g8;
          if (s0 >= n_real) { sc[mt][0][0] = sc[mt][0][1] = sc[mt][1][0] = sc[mt][1][1] = -INFINITY; }
          if (s0 + 8 >= n_real) { sc[mt][0][2] = sc[mt][0][3] = sc[mt][1][2] = sc[mt][1][3] = -INFINITY; }
        }
#pragma unroll
        for (int u = 0; u < 2; ++u) {
          if (u == 1 && !has_b) break;
          mloc[u][0] = fmaxf(mloc[u][0], fmaxf(sc[mt][u][0], sc[mt][u][2]));
          mloc[u][1] = fmaxf(mloc[u][1], fmaxf(sc[mt][u][1], sc[mt][u][3]));
        }
      }
      bool fine = true;
#pragma unroll
      for (int u = 0; u < 2; ++u)
        fine = fine && mloc[u][0] <= Mx[u][0] + kSlack && mloc[u][1] <= Mx[u][1] + kSlack;
      if (!__all_sync(0xffffffffu, fine)) {
#pragma unroll
        for (int u = 0; u < 2; ++u)
#pragma unroll
          for (int e = 0; e < 2; ++e) {
            if (u == 1 && !has_b) break;
            float x = mloc[u][e];
#pragma unroll
            for (int o = 4; o < 32; o <<= 1) x = fmaxf(x, __shfl_xor_sync(0xffffffffu, x, o));
            const float nm = fmaxf(Mx[u][e], x);
            const float corr = fast_exp2(Mx[u][e] - nm);
            Mx[u][e] = nm;
            Ls[u][e] *= corr;
#pragma unroll
            for (int t = 0; t < kHeadDim / 16; ++t) { oacc[t][u][e] *= corr; oacc[t][u][e + 2] *= corr; }
          }
      }
      uint32_t pb[ISL / 16][2][2];
#pragma unroll
      for (int mt = 0; mt < ISL / 16; ++mt)
#pragma unroll
        for (int u = 0; u < 2; ++u) {
          if (u == 1 && !has_b) break;
          const float p0 = fast_exp2(sc[mt][u][0] - Mx[u][0]), p1 = fast_exp2(sc[mt][u][1] - Mx[u][1]);
          const float p2 = fast_exp2(sc[mt][u][2] - Mx[u][0]), p3 = fast_exp2(sc[mt][u][3] - Mx[u][1]);
          Ls[u][0] += p0 + p2;
          Ls[u][1] += p1 + p3;
          pb[mt][u][0] = movmatrix_trans(pack_bf16(p0, p1));
          pb[mt][u][1] = movmatrix_trans(pack_bf16(p2, p3));
        }

      // ---- V chunks: weighted coefficient rows for both n-tiles
      {
        int left = 0, j0 = 0;
        uint32_t st_addr = 0;
        bool ok = true;
#pragma unroll
        for (int jt = 0; jt < kHeadDim / 16; ++jt) {
          if (jt * 16 >= r) break;   // warp-uniform
          if (left == 0) {
            if (jt > 0) release();
            if (!wait_chunk()) { ok = false; break; }
            st_addr = ring_t + (n_cons % SPT) * STAGE;
            j0 = jt * 16;
            left = 1 << lgc;
          }
          left -= 16;
          const int jrow = (jt * 16 - j0) + (m & 1) * 8 + r8;
          const int j = j0 + jrow;
          const uint32_t row_addr = st_addr + jrow * row_bytes;
          const bool keep0 = jt * 16 + g8 < r, keep1 = jt * 16 + g8 + 8 < r;
          uint32_t off[ISL / 16];
          if (full_tile) {
            const uint32_t o0 = (uint32_t)(((m >> 1) + j) & 15) << 4;
#pragma unroll
            for (int kt = 0; kt < ISL / 16; ++kt) off[kt] = (o0 + 32u * kt) & 255u;
          } else {
            int pg = ((m >> 1) + j) % ng;
#pragma unroll
            for (int kt = 0; kt < ISL / 16; ++kt) { off[kt] = 16u * pg; pg = wrap2(pg, ng); }
          }
          float t1[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
#pragma unroll
          for (int kt = 0; kt < ISL / 16; kt += 2) {
            uint32_t a[4], a2[4];
            ldsm_x4(row_addr + off[kt], a);
            ldsm_x4(row_addr + off[kt + 1], a2);
            if (jt * 16 + 16 > r) {
              if (!keep0) { a[0] = a[2] = 0u; a2[0] = a2[2] = 0u; }
              if (!keep1) { a[1] = a[3] = 0u; a2[1] = a2[3] = 0u; }
            }
            mma_bf16_16816(oacc[jt][0], a, pb[kt][0][0], pb[kt][0][1]);
            mma_bf16_16816(t1[0], a2, pb[kt + 1][0][0], pb[kt + 1][0][1]);
            if (has_b) {
              mma_bf16_16816(oacc[jt][1], a, pb[kt][1][0], pb[kt][1][1]);
              mma_bf16_16816(t1[1], a2, pb[kt + 1][1][0], pb[kt + 1][1][1]);
            }
          }
#pragma unroll
          for (int u = 0; u < 2; ++u)
#pragma unroll
            for (int e = 0; e < 4; ++e) oacc[jt][u][e] += t1[u][e];
        }
        if (ok) release();
      }
      cons_k += NTEAM;
      if (cons_k < total) cons = next_rr<NTEAM>(sm, cons, cons_k);
    }

    // ---- merge the teams of this CTA for this segment
    __syncwarp();
#pragma unroll
    for (int u = 0; u < 2; ++u)
#pragma unroll
      for (int e = 0; e < 2; ++e)
#pragma unroll
        for (int o = 4; o < 32; o <<= 1) Ls[u][e] += __shfl_xor_sync(0xffffffffu, Ls[u][e], o);
    dead = __syncthreads_or(dead || timed_out);   // every warp has finished the segment
    if (!dead) {
#pragma unroll
      for (int u = 0; u < 2; ++u) {
        if (u == 1 && !has_b) break;
        const int nt = rg + u * RG;
        if (g8 == 0) {
#pragma unroll
          for (int e = 0; e < 2; ++e) {
            mg.M[team][8 * nt + 2 * c + e] = Mx[u][e];
            mg.L[team][8 * nt + 2 * c + e] = Ls[u][e];
          }
        }
#pragma unroll
        for (int t = 0; t < kHeadDim / 16; ++t)
#pragma unroll
          for (int e = 0; e < 4; ++e)
            mg.acc[team][8 * nt + 2 * c + (e & 1)][t * 16 + g8 + (e >> 1) * 8] = oacc[t][u][e];
      }
    }
    __syncthreads();
    const int rows = 8 * ntt;
    if (!dead)
      for (int rho = tid; rho < rows; rho += blockDim.x) {
        float mx = -INFINITY, l = 0.f;
#pragma unroll
        for (int t = 0; t < NTEAM; ++t) mx = fmaxf(mx, mg.M[t][rho]);
#pragma unroll
        for (int t = 0; t < NTEAM; ++t) {
          const float f = mx == -INFINITY ? 0.f : fast_exp2(mg.M[t][rho] - mx);
          mg.F[t][rho] = f;
          l = fmaf(mg.L[t][rho], f, l);
        }
        mg.mx[rho] = mx;
        mg.l[rho] = l;
      }
    __syncthreads();
    // partial of (segment, CTA) in slot cta + seg (unique: a later CTA only meets later segments)
    float* pout = part + (cta + seg) * (long long)rows * kPartStride;
    for (int i = tid; i < rows * kHeadDim; i += blockDim.x) {
      const int rho = i / kHeadDim, j = i % kHeadDim;
      float o = 0.f;
      if (!dead) {
#pragma unroll
        for (int t = 0; t < NTEAM; ++t) o = fmaf(mg.acc[t][rho][j], mg.F[t][rho], o);
      }
      pout[rho * kPartStride + j] = o;
      if (j == 0) {
        pout[rho * kPartStride + kHeadDim] = dead ? -INFINITY : mg.mx[rho];
        pout[rho * kPartStride + kHeadDim + 1] = dead ? 0.f : mg.l[rho];
      }
    }
    __syncthreads();
    if (++g == s.G) { ++b; g = 0; }
    while (b < s.B && segW[b] == 0) ++b;
    more = b < s.B && seg_start(b, g) < hi_g;
    if (more && !dead) {
      fence_proxy_async_smem();   // the merge wrote the ring: before the next copies
      __syncthreads();
    }
  }
  if (dead) {   // last bounded waits for copies that may still be landing in shared memory
    if (tid < Cf::NBAR && iss[tid] > 0u) mbar_wait_bounded(&bar[tid], (iss[tid] - 1u) & 1u, kWaitTries);
    if (tid == Cf::NBAR && n_qf > 0u) mbar_wait_bounded(&bar_q, (n_qf - 1u) & 1u, kWaitTries);
  }
  if (timed_out && lane == 0) raise_status(dev_status, VARRATE_ERR_TIMEOUT);
}

// ------------------------------------------------------------------ 3. combine

constexpr int kTT = 64;                   // tail tokens per step
constexpr int kKsStride = kHeadDim + 2;   // staged tail keys (odd word stride: no bank conflicts)
constexpr int kCombRows = 8;              // query rows per combine CTA: one warp each

struct CombineSmem {
  __nv_bfloat16 us[kHeadDim * kHeadDim];   // U_V[j][col]
  __nv_bfloat16 ks[kTT * kKsStride];        // tail keys of the step
  __nv_bfloat16 vs[kTT * kHeadDim];         // tail values of the step
  float qs[kCombRows][kHeadDim];            // raw query rows (fp32)
  float os[kCombRows][kHeadDim + 4];        // merged o~ per row
  float ws[kCombRows][kTT];                 // tail weights of the step
};

// grid (B G, ceil(R / 8)), 256 threads: warp w owns row rho = 8 blockIdx.y + w, lane l its columns
// l + 32 k (k < 4) and, per step of 64 tail tokens, tokens l and l + 32. part slots as written
// above; out is [B][n_q][H][d].
__global__ void __launch_bounds__(256)
window_combine_kernel(const float* __restrict__ part, const int64_t* __restrict__ bucket_base,
                      const __nv_bfloat16* __restrict__ basis_v, const __nv_bfloat16* __restrict__ q,
                      const __nv_bfloat16* __restrict__ tail_k, const __nv_bfloat16* __restrict__ tail_v,
                      int n_tail, int n_q, __nv_bfloat16* __restrict__ out, Shape s, int layer, int C,
                      int ntt) {
  extern __shared__ __align__(16) unsigned char smem_c[];
  CombineSmem& cs = *reinterpret_cast<CombineSmem*>(smem_c);
  __shared__ long long segW[64];
  __shared__ long long segP[65];
  const int tid = threadIdx.x, lr = tid >> 5, lane = tid & 31;
  const long long seg = blockIdx.x;
  const int b = (int)(seg / s.G), g = (int)(seg % s.G);
  const int R = n_q * s.grp, rows = 8 * ntt;
  const int rho = kCombRows * blockIdx.y + lr;
  const bool valid = rho < R;
  const int iq = valid ? rho / s.grp : 0, h = valid ? rho % s.grp : 0;
  pdl_trigger();
  pdl_wait();
  // U_V of the head (eight 16-byte loads per thread, all in flight) and the query rows
  {
    const uint4* src = reinterpret_cast<const uint4*>(basis_v + ((long long)layer * s.G + g) * kHeadDim * kHeadDim);
    uint4* dst = reinterpret_cast<uint4*>(cs.us);
    uint4 v[kHeadDim * kHeadDim / 8 / 256];
#pragma unroll
    for (int k = 0; k < kHeadDim * kHeadDim / 8 / 256; ++k) v[k] = __ldg(src + tid + 256 * k);
#pragma unroll
    for (int k = 0; k < kHeadDim * kHeadDim / 8 / 256; ++k) dst[tid + 256 * k] = v[k];
    const __nv_bfloat16* qr = q + (((long long)b * n_q + iq) * s.H + (long long)g * s.grp + h) * kHeadDim;
#pragma unroll
    for (int k = 0; k < 4; ++k) cs.qs[lr][lane + 32 * k] = valid ? __bfloat162float(qr[lane + 32 * k]) : 0.f;
  }
  seg_lengths(bucket_base, s, layer, segW, segP, tid);
  // merge the partials of the CTAs that shared the segment: the common maximum first, then the
  // weighted sums (independent loads, four partials at a time)
  float M = -INFINITY, L = 0.f, o[4], ov[4];
#pragma unroll
  for (int k = 0; k < 4; ++k) { o[k] = 0.f; ov[k] = 0.f; }
  const long long W = segW[b];
  if (W > 0 && valid) {
    const long long T = segP[64];
    const long long P = segP[b] + g * (W + kSegCost + kSegEnd) + kSegCost;
    int c0, c1;
    seg_cta_range([&](int i) { return cut_at(T, i, C); }, T, C, P, W, c0, c1);
    const float* pr = part + ((c0 + seg) * (long long)rows + rho) * kPartStride;
    const long long pstride = (long long)rows * kPartStride;
    const int np = c1 - c0 + 1;
#pragma unroll 4
    for (int p = 0; p < np; ++p) M = fmaxf(M, __ldcg(pr + p * pstride + kHeadDim));
    if (M != -INFINITY) {
#pragma unroll 4
      for (int p = 0; p < np; ++p) {
        const float* pp = pr + p * pstride;
        const float mp = __ldcg(pp + kHeadDim);
        const float w = mp == -INFINITY ? 0.f : exp2f(mp - M);
        L = fmaf(w, __ldcg(pp + kHeadDim + 1), L);
#pragma unroll
        for (int k = 0; k < 4; ++k) o[k] = fmaf(w, __ldcg(pp + lane + 32 * k), o[k]);
      }
    }
  }
  // exact tail, causal: row rho (query iq) sees tail tokens t < n_tail - n_q + iq + 1
  const int vis = n_tail - n_q + iq + 1;
  const int last_row = min(R, kCombRows * (int)blockIdx.y + kCombRows) - 1;
  const int vis_max = n_tail - n_q + last_row / s.grp + 1;   // block-uniform
  const float scale = kLog2e * rsqrtf((float)kHeadDim);
  const __nv_bfloat16* tk = tail_k + ((long long)b * s.G + g) * n_tail * kHeadDim;
  const __nv_bfloat16* tv = tail_v + ((long long)b * s.G + g) * n_tail * kHeadDim;
  for (int t0 = 0; t0 < vis_max; t0 += kTT) {
    __syncthreads();   // previous step's readers of ks / vs (and the loads above) are done
    for (int e = tid; e < kTT * kHeadDim / 2; e += blockDim.x) {
      const int t = e / (kHeadDim / 2), i2 = e % (kHeadDim / 2);
      uint32_t kx = 0u, vx = 0u;
      if (t0 + t < n_tail) {
        kx = reinterpret_cast<const uint32_t*>(tk + (long long)(t0 + t) * kHeadDim)[i2];
        vx = reinterpret_cast<const uint32_t*>(tv + (long long)(t0 + t) * kHeadDim)[i2];
      }
      reinterpret_cast<uint32_t*>(cs.ks + t * kKsStride)[i2] = kx;
      reinterpret_cast<uint32_t*>(cs.vs + t * kHeadDim)[i2] = vx;
    }
    __syncthreads();
    float sc[2] = {0.f, 0.f};
    for (int i = 0; i < kHeadDim; i += 2) {
      const float2 qv = *reinterpret_cast<const float2*>(&cs.qs[lr][i]);
#pragma unroll
      for (int k = 0; k < 2; ++k) {
        const __nv_bfloat162 kk = *reinterpret_cast<const __nv_bfloat162*>(cs.ks + (lane + 32 * k) * kKsStride + i);
        sc[k] = fmaf(qv.x, __low2float(kk), fmaf(qv.y, __high2float(kk), sc[k]));
      }
    }
    float tm = -INFINITY;
#pragma unroll
    for (int k = 0; k < 2; ++k) {
      const int t = t0 + lane + 32 * k;
      sc[k] = (valid && t < vis) ? sc[k] * scale : -INFINITY;
      tm = fmaxf(tm, sc[k]);
    }
#pragma unroll
    for (int x = 1; x < 32; x <<= 1) tm = fmaxf(tm, __shfl_xor_sync(0xffffffffu, tm, x));
    const float nm = fmaxf(M, tm);
    float lt = 0.f;
    if (nm != -INFINITY) {
      const float f = M == -INFINITY ? 0.f : exp2f(M - nm);
#pragma unroll
      for (int k = 0; k < 4; ++k) { o[k] *= f; ov[k] *= f; }
      L *= f;
      M = nm;
#pragma unroll
      for (int k = 0; k < 2; ++k) {
        const float w = sc[k] == -INFINITY ? 0.f : exp2f(sc[k] - nm);
        cs.ws[lr][lane + 32 * k] = w;
        lt += w;
      }
    } else {
#pragma unroll
      for (int k = 0; k < 2; ++k) cs.ws[lr][lane + 32 * k] = 0.f;
    }
#pragma unroll
    for (int x = 1; x < 32; x <<= 1) lt += __shfl_xor_sync(0xffffffffu, lt, x);
    L += lt;
    __syncwarp();   // the row's weights were written by this warp
#pragma unroll 4
    for (int t = 0; t < kTT; ++t) {
      const float w = cs.ws[lr][t];
#pragma unroll
      for (int k = 0; k < 4; ++k) ov[k] = fmaf(w, __bfloat162float(cs.vs[t * kHeadDim + lane + 32 * k]), ov[k]);
    }
  }
  // rotate the coded part back: out[col] = sum_j U_V[j][col] o~[j] + tail values, over l
#pragma unroll
  for (int k = 0; k < 4; ++k) cs.os[lr][lane + 32 * k] = o[k];
  __syncthreads();
  float y[4];
#pragma unroll
  for (int k = 0; k < 4; ++k) y[k] = ov[k];
#pragma unroll 4
  for (int j = 0; j < kHeadDim; ++j) {
    const float oj = cs.os[lr][j];
#pragma unroll
    for (int k = 0; k < 4; ++k) y[k] = fmaf(__bfloat162float(cs.us[j * kHeadDim + lane + 32 * k]), oj, y[k]);
  }
  if (valid) {
    __nv_bfloat16* dst = out + (((long long)b * n_q + iq) * s.H + (long long)g * s.grp + h) * kHeadDim;
    const float inv = 1.f / L;
#pragma unroll
    for (int k = 0; k < 4; ++k) dst[lane + 32 * k] = __float2bfloat16_rn(y[k] * inv);
  }
}

template <int RG>
int launch_window_main(const Shape& s, const varrate_packed& c, const uint4* qf, float* part,
                       int32_t* dev_status, int layer, int ntt, int num_sms, cudaStream_t st) {
  const size_t smem = win_smem_bytes<RG>();
  static std::atomic<int> smem_set[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64 ||
      smem_set[dev].load(std::memory_order_acquire) == 0) {
    if (cudaFuncSetAttribute(decode_window_kernel<RG>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem) != cudaSuccess)
      return -1;
    if (dev >= 0 && dev < 64) smem_set[dev].store(1, std::memory_order_release);
  }
  cudaLaunchAttribute pdl[1];
  pdl[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  pdl[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t lc = {};
  lc.gridDim = dim3(num_sms);
  lc.blockDim = dim3(NW * 32);
  lc.dynamicSmemBytes = smem;
  lc.stream = st;
  lc.attrs = pdl;
  lc.numAttrs = 1;
  if (cudaLaunchKernelEx(&lc, decode_window_kernel<RG>, (const __nv_bfloat16*)c.coef,
                         (const int32_t*)c.bucket_count, (const int64_t*)c.bucket_base, qf, part,
                         dev_status, s, layer, ntt) != cudaSuccess)
    return -1;
  return 1;
}

// the shared-memory opt-in of the two helper kernels, once per device
bool helper_smem(int which, const void* fn, size_t bytes) {
  static std::atomic<int> set[2][64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return false;
  if (set[which][dev].load(std::memory_order_acquire)) return true;
  if (cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes) != cudaSuccess)
    return false;
  set[which][dev].store(1, std::memory_order_release);
  return true;
}

int window_rg(int ntt) { return ntt <= 2 ? 1 : (ntt <= 4 ? 2 : (ntt <= 8 ? 4 : 8)); }

}  // namespace

size_t decode_window_ws_bytes(const Shape& s, int num_sms) {
  const size_t segs = (size_t)s.B * s.G;
  const size_t qf = (segs * 8 * kQfBytes + 255) & ~size_t(255);   // RG <= 8 row groups
  const size_t part = ((size_t)(num_sms + segs) * kWindowMaxRows * kPartStride * sizeof(float) + 255) & ~size_t(255);
  return qf + part;
}

bool decode_window_supported(const Shape& s, int n_q, int n_tail, int num_sms) {
  const unsigned long long line = (unsigned long long)s.B * s.G * ((unsigned long long)s.cap + kSegCost + kSegEnd);
  return s.dtype == VARRATE_BF16 && s.B <= 64 && n_q >= 1 && n_q <= n_tail &&
         (long long)n_q * s.grp <= kWindowMaxRows && (long long)s.B * s.G < (1LL << 31) &&
         num_sms >= 1 && num_sms <= kMaxCtas && line <= (1ull << 62) / (unsigned long long)num_sms;
}

int launch_decode_window(const Shape& s, const varrate_packed& c, const void* basis_k, const void* basis_v,
                         const void* q, int n_q, int layer, const void* tail_k, const void* tail_v,
                         int n_tail, void* out, int32_t* dev_status, void* ws, int num_sms,
                         cudaStream_t st) {
  const int R = n_q * s.grp, ntt = (R + 7) / 8, RG = window_rg(ntt);
  const size_t segs = (size_t)s.B * s.G;
  uint4* qf = reinterpret_cast<uint4*>(ws);
  float* part = reinterpret_cast<float*>(static_cast<unsigned char*>(ws) +
                                         ((segs * 8 * kQfBytes + 255) & ~size_t(255)));
  cudaLaunchAttribute pdl[1];
  pdl[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  pdl[0].val.programmaticStreamSerializationAllowed = 1;

  cudaLaunchConfig_t lq = {};
  lq.gridDim = dim3((unsigned)segs, RG, kHeadDim / kQfJ);
  lq.blockDim = dim3(256);
  lq.dynamicSmemBytes = 0;
  lq.stream = st;
  lq.attrs = pdl;
  lq.numAttrs = 1;
  if (cudaLaunchKernelEx(&lq, window_qfrag_kernel, (const __nv_bfloat16*)basis_k, (const __nv_bfloat16*)q,
                         qf, s, layer, n_q, RG, ntt) != cudaSuccess)
    return -1;

  int rc = -1;
  switch (RG) {
    case 1: rc = launch_window_main<1>(s, c, qf, part, dev_status, layer, ntt, num_sms, st); break;
    case 2: rc = launch_window_main<2>(s, c, qf, part, dev_status, layer, ntt, num_sms, st); break;
    case 4: rc = launch_window_main<4>(s, c, qf, part, dev_status, layer, ntt, num_sms, st); break;
    default: rc = launch_window_main<8>(s, c, qf, part, dev_status, layer, ntt, num_sms, st); break;
  }
  if (rc < 0) return -1;

  const size_t csm = sizeof(CombineSmem);
  if (!helper_smem(1, (const void*)window_combine_kernel, csm)) return -1;
  cudaLaunchConfig_t lc = {};
  lc.gridDim = dim3((unsigned)segs, (unsigned)((R + kCombRows - 1) / kCombRows));
  lc.blockDim = dim3(256);
  lc.dynamicSmemBytes = csm;
  lc.stream = st;
  lc.attrs = pdl;
  lc.numAttrs = 1;
  if (cudaLaunchKernelEx(&lc, window_combine_kernel, (const float*)part, (const int64_t*)c.bucket_base,
                         (const __nv_bfloat16*)basis_v, (const __nv_bfloat16*)q, (const __nv_bfloat16*)tail_k,
                         (const __nv_bfloat16*)tail_v, n_tail, n_q, (__nv_bfloat16*)out, s, layer, num_sms,
                         ntt) != cudaSuccess)
    return -1;
  return 3;
}

}  // namespace vr
