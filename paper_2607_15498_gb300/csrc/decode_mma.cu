// Step 4, bf16 — decode attention on the packed coefficients with tensor-core tiles.
//
// Same mathematics as decode.cu (attention of Sec. 3.1 over the cache of Eq. 5, never rebuilding K
// or V): per query head h of KV head g, q~ = U_K q * log2(e)/sqrt(d); score_t = q~[:r_t].c^K_t;
// o = U_V^T (sum_t 2^(score_t - m) c^V_t) / sum_t 2^(score_t - m).
//
// Work split. The coefficient streams of all (sequence, KV head) pairs of the layer form one cost
// line (element offsets, K stream); the persistent grid (one CTA per SM) cuts it into equal
// ranges, so every SM moves the same number of bytes. A CTA walks the (sequence, head) segments its
// range touches; per segment it rotates the query with mma.sync (U_K tile x q), then its warps take
// 128-slot items (one tile of the packed layout) of one rank bucket round-robin. An item of rank r
// is read as K chunks then V chunks of up to 8 KB each (32 rows of a full tile, 64 or 128 rows of a
// short one), each one contiguous block.
//
// Memory path. Each of the 12 warps owns a 2-stage shared-memory ring filled by one 1-D TMA bulk
// copy per chunk that completes on a per-stage mbarrier; while the warp computes on one stage the
// other is in flight (the stage it finishes is refilled with the chunk two ahead), across item
// boundaries, so loads never wait on arithmetic. The per-row rotation of
// the 8-slot groups keeps the unpadded staged rows free of shared-memory bank conflicts. Rows >= r
// of a chunk are never loaded: they are masked out of the K and V fragments (not multiplied by
// zero), so whatever the ring held before never reaches the arithmetic and it is never cleared.
//
// Arithmetic (per warp, fp32 accumulate, all operands exact or split hi+lo in bf16):
//   scores   S^T[slot][head] += K^T[slot][j] * Q~^T[j][head]   (mma m16n8k16; K via ldmatrix.trans,
//            q~ split hi+lo so the product is accurate to ~2^-16)
//   softmax  online, per head, 8 heads per tile (grp <= 8; unused heads are computed and ignored)
//   values   O~^T[j][head] += V[j][slot] * P^T[slot][head]      (P in bf16, <= 2^-9 relative per
//            weight, transposed from the score fragments with movmatrix)
// Partials (max, sum, o~[128]) per (segment, CTA) go to the workspace. The last CTA to finish a
// segment (counted in per-segment arrival counters in the workspace header, DecodeHeader below)
// merges its partials, adds the exact tail, rotates back with U_V^T (staged in the idle ring) and
// normalises, so one launch does the whole step.
//
// Warps reconverge explicitly (__syncwarp) after lane-dependent code and before warp-wide
// shuffles, votes and tensor-core fragments: left to itself a diverged warp reaching those
// instructions was measured to lose thousands of cycles.
#include <stddef.h>

#include <atomic>

#include "common.cuh"
#include "decode_common.cuh"
#include "decode_parts.cuh"
#include "kernels.h"

namespace vr {

namespace {

// Issue the next chunk of this warp's stream into `stage`: consecutive rows of one tile are
// contiguous in the packed layout, so one bulk copy moves the whole chunk.
// Returns false (and issues nothing) when the stream is exhausted.
__device__ __forceinline__ bool issue_chunk(Prod& p, const SegSmem& sm, const __nv_bfloat16* cK,
                                            const __nv_bfloat16* cV, uint32_t stage_addr,
                                            uint64_t* bar, int total, int lane, uint64_t policy) {
  if (p.k >= total) return false;
  const int r = p.item.r;
  const long long n8 = pad8(sm.cnt[r]);
  const long long t0 = (long long)p.item.it * ISL;            // first slot of the tile
  const long long tl = min((long long)ISL, n8 - t0);            // slots in the tile (multiple of 8)
  const int lgc = chunk_lg((int)tl);
  const int j0 = p.jc << lgc;
  const int rows = min(1 << lgc, r - j0);
  // callers have __syncwarp()ed: every lane's ldmatrix reads of this stage are done
  if (lane == 0) {
    const uint32_t bytes = (uint32_t)(rows * tl * 2);           // rows j0.. of the tile: contiguous
    mbar_arrive_expect_tx(bar, bytes);
    fence_proxy_async_smem();  // the generic reads above precede the async write
    bulk_g2s_hint(stage_addr, (p.phase ? cV : cK) + sm.base[r] + t0 * r + (long long)j0 * tl, bytes, bar,
                  policy);
  }
  __syncwarp();   // lane 0 branched off: reconverge before the next warp-wide instruction
  const int nj = (r + (1 << lgc) - 1) >> lgc;
  if (++p.jc == nj) {
    p.jc = 0;
    if (++p.phase == 2) {
      p.phase = 0;
      p.k += NW;
      if (p.k < total) p.item = next_rr<NW>(sm, p.item, p.k);
    }
  }
  return true;
}

__global__ void __launch_bounds__(NW * 32, 1)
decode_mma_kernel(const __nv_bfloat16* __restrict__ coef, const int32_t* __restrict__ bucket_count,
                  const int64_t* __restrict__ bucket_base, const __nv_bfloat16* __restrict__ basis_k,
                  const __nv_bfloat16* __restrict__ basis_v, const __nv_bfloat16* __restrict__ qin,
                  const __nv_bfloat16* __restrict__ tail_k, const __nv_bfloat16* __restrict__ tail_v,
                  int n_tail, __nv_bfloat16* __restrict__ out, float* __restrict__ part,
                  DecodeHeader* __restrict__ hdr, int32_t* __restrict__ dev_status, Shape s,
                  int layer) {
  extern __shared__ __align__(128) unsigned char smem[];
  unsigned char* ring = smem;                                     // NW * ST * STAGE
  static_assert((NW * ST * STAGE) % 16 == 0, "SegSmem must start 16-byte aligned");
  SegSmem& sm = *reinterpret_cast<SegSmem*>(smem + NW * ST * STAGE);
  // the merge and combine buffers alias the ring (idle while a segment is merged)
  static_assert(sizeof(Merge) <= (size_t)NW * ST * STAGE, "merge buffers fit in the ring");
  Merge& mg = *reinterpret_cast<Merge*>(smem);
  __shared__ long long segW[64];                                  // per-sequence stream length
  __shared__ long long segP[65];                                  // start of sequence b on the cost line
  __shared__ long long cuts[kMaxCtas + 1];                        // start of CTA c's range
  __shared__ int n_empty;                                         // sequences with no coded tokens
  __shared__ int last_cta;                                        // this CTA closes the segment
  __shared__ uint32_t parity;                                     // counter set of this call
  __shared__ uint64_t bar_all[NW * ST];                           // one full-barrier per ring stage
  __shared__ uint64_t bar_comb;                                   // U_V copy of a combine

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int g8 = lane >> 2, c = lane & 3;
  const int C = gridDim.x, cta = blockIdx.x;
  const uint64_t policy = l2_evict_first_policy();   // coefficient chunks are read once

  // the next grid in the stream may be scheduled now: it only starts on SMs this grid has left,
  // and waits (griddepcontrol.wait) for this grid to finish before it reads anything
  pdl_trigger();
  // self-contained setup first (it may overlap the tail of the preceding grid)
  if (tid < NW * ST) mbar_init(&bar_all[tid], 1);
  if (tid == NW * ST) mbar_init(&bar_comb, 1);
  fence_mbar_init();
  fence_proxy_async_smem();
  pdl_wait();   // everything below reads data written by earlier grids
  if (tid == 0) parity = (uint32_t)(*reinterpret_cast<volatile unsigned long long*>(&hdr->calls) & 1ull);
  // stream length of every sequence of this layer (same for every head); poisoned tables -> 0
  for (int b = tid; b < s.B; b += blockDim.x) {
    const long long w = bucket_base[((long long)b * s.L + layer) * (kMaxR + 2) + kMaxR + 1];
    segW[b] = (w >= 0 && w <= s.cap) ? w : 0;
  }
  __syncthreads();
  {   // the other set: used by the previous call (finished), counted on by the next one
    uint32_t* other = hdr->arrived[parity ^ 1u];
    for (int i = cta * (int)blockDim.x + tid; i < kDecodeMaxSegs; i += C * (int)blockDim.x) other[i] = 0u;
    if (cta == 0 && tid == 0) hdr->exits[parity ^ 1u] = 0u;
  }
  uint32_t* arrived = hdr->arrived[parity];
  uint32_t n_issued = 0;   // chunks this warp has consumed (== index of its next chunk)
  int n_pending = 0;       // chunks issued but not yet consumed
  bool timed_out = false;  // this thread saw a bounded wait give up
  // CTA-uniform: some wait of this CTA gave up, so bulk copies may still be landing in the ring.
  // From then on nothing writes the ring (merge and combine buffers alias it) and nothing streams;
  // the CTA still writes an empty partial and arrives on every segment it covers, so the counts of
  // the other CTAs stay consistent.
  bool dead = false;
  uint32_t n_comb = 0;     // combines done by this CTA (phase of bar_comb)
  // Cost line: sequence b holds G segments of kSegCost + W_b + kSegEnd elements each (W_b > 0): the
  // set-up allowance, the coefficients, the end allowance. segP = exclusive prefix over sequences (B <= 64: two per lane).
  if (warp == 0) {
    __syncwarp();   // lanes left the loads above apart: reconverge before the shuffles
    const int e0 = 2 * lane, e1 = 2 * lane + 1;
    const long long v0 = (e0 < s.B && segW[e0]) ? (segW[e0] + kSegCost + kSegEnd) * s.G : 0;
    const long long v1 = (e1 < s.B && segW[e1]) ? (segW[e1] + kSegCost + kSegEnd) * s.G : 0;
    long long inc = v0 + v1;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const long long y = __shfl_up_sync(0xffffffffu, inc, o);
      if (lane >= o) inc += y;
    }
    segP[e0] = inc - v0 - v1;
    segP[e1] = inc - v1;
    if (lane == 31) segP[64] = inc;
    const unsigned m0 = __ballot_sync(0xffffffffu, e0 < s.B && segW[e0] == 0);
    const unsigned m1 = __ballot_sync(0xffffffffu, e1 < s.B && segW[e1] == 0);
    if (lane == 0) n_empty = __popc(m0) + __popc(m1);
  }
  __syncthreads();
  const long long T = segP[64];
  for (int c2 = tid; c2 <= C; c2 += blockDim.x) cuts[c2] = cut_at(T, c2, C);
  __syncthreads();
  const long long lo_g = cuts[cta], hi_g = cuts[cta + 1];

  // first segment of this CTA: the sequence whose span holds lo_g, then the head within it
  int b = 0, g = 0;
  {
    int lo_b = 0, hi_b = s.B;
    while (lo_b < hi_b) {
      const int mid = (lo_b + hi_b) >> 1;
      if (segP[mid + 1] > lo_g) hi_b = mid; else lo_b = mid + 1;
    }
    b = lo_b;
    if (b < s.B) {   // g = floor(x / w), estimated in fp32 and corrected
      const long long x = lo_g - segP[b], w = segW[b] + kSegCost + kSegEnd;
      g = (int)((float)x / (float)w);
      while (g > 0 && (long long)g * w > x) --g;
      while ((long long)(g + 1) * w <= x) ++g;
    }
  }
  auto seg_start = [&](int bb, int gg) { return segP[bb] + gg * (segW[bb] + kSegCost + kSegEnd) + kSegCost; };
  if (b < s.B && seg_start(b, g) + segW[b] <= lo_g) {   // the range starts in a segment's end allowance
    if (++g == s.G) { ++b; g = 0; }
    while (b < s.B && segW[b] == 0) ++b;
  }
  bool more = b < s.B && seg_start(b, g) < hi_g;
  while (more) {
    {
      const long long W = segW[b];
      const long long P = seg_start(b, g);   // first coefficient of segment (b, g) on the cost line
      const long long lo = max(lo_g, P) - P, hi = min(hi_g, P + W) - P;
      const long long bl = (long long)b * s.L + layer;
      RotRegs rr;   // this segment's U_K tile and queries, in flight with the table loads below
      rot_load(rr, basis_k + ((long long)layer * s.G + g) * kHeadDim * kHeadDim,
               qin + ((long long)b * s.H + (long long)g * s.grp) * kHeadDim, s.grp, warp, lane);
      // U_V of this head, for whichever CTA merges the segment: into L2 while it streams
      if (tid == 0) bulk_prefetch_l2(basis_v + ((long long)layer * s.G + g) * kHeadDim * kHeadDim, kHeadDim * kHeadDim * 2);
      __syncthreads();
      for (int r = tid; r <= kMaxR + 1; r += blockDim.x) {
        if (r <= kMaxR) sm.cnt[r] = bucket_count[bl * (kMaxR + 1) + r];
        sm.base[r] = bucket_base[bl * (kMaxR + 2) + r];
      }
      __syncthreads();
      for (int r = tid; r <= kMaxR; r += blockDim.x) {
        long long i0 = 0, i1 = 0;
        if (r >= s.r_min && r <= s.r_max) bucket_range(sm, r, lo, hi, i0, i1);
        sm.it_lo[r] = (int)i0;
        sm.it_pref[r + 1] = (int)(i1 - i0);   // counts first, prefixed below
      }
      __syncthreads();
      if (warp == 0) {   // inclusive scan of it_pref[1 .. 129], 5 entries per lane
        __syncwarp();
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
      // start this warp's loads first: they do not depend on the rotated queries
      const __nv_bfloat16* cK = coef + ((bl * s.G + g) * 2) * s.cap;
      const __nv_bfloat16* cV = cK + s.cap;
      const uint32_t ring_w = smem_addr(ring) + warp * ST * STAGE;
      uint64_t* bars = &bar_all[warp * ST];

      float Mx[2] = {-INFINITY, -INFINITY}, Ls[2] = {0.f, 0.f};
      float oacc[kHeadDim / 16][4];
#pragma unroll
      for (int t = 0; t < kHeadDim / 16; ++t) oacc[t][0] = oacc[t][1] = oacc[t][2] = oacc[t][3] = 0.f;

      const int total = dead ? 0 : sm.it_pref[kMaxR + 1];
      Prod pr;
      pr.k = warp; pr.phase = 0; pr.jc = 0;
      if (pr.k < total) pr.item = item_at(sm, pr.k);
      int cons_k = pr.k;
      Item cons = pr.item;
#pragma unroll
      for (int i = 0; i < ST; ++i)   // every stage of the ring in flight
        if (issue_chunk(pr, sm, cK, cV, ring_w + ((n_issued + i) % ST) * STAGE,
                        &bars[(n_issued + i) % ST], total, lane, policy)) ++n_pending;
      int c0, c1;   // the CTAs that share this segment (their partials are merged by the last one)
      seg_cta_range([&](int i) { return cuts[i]; }, T, C, P, W, c0, c1);
      __syncwarp();
      if (warp < kHeadDim / 16) rot_compute(sm, rr, s.grp, warp, lane);
      __syncthreads();
      build_qfrag(sm, tid);
      __syncthreads();

      // chunk k of this warp (counted over the whole kernel) lives in stage k % ST, phase (k/ST)&1

      auto wait_chunk = [&]() -> bool {
        const uint32_t k = n_issued;
        if (!mbar_wait_bounded(&bars[k % ST], (k / ST) & 1u, kWaitTries)) { timed_out = true; return false; }
        return true;
      };
      auto next_chunk = [&]() {
        // the consumed stage is free again: refill it with the chunk ST ahead, so that all the
        // other stages stay in flight while the warp computes
        ++n_issued;
        --n_pending;
        if (issue_chunk(pr, sm, cK, cV, ring_w + ((n_issued + ST - 1) % ST) * STAGE,
                        &bars[(n_issued + ST - 1) % ST], total, lane, policy)) ++n_pending;
      };

      while (cons_k < total && !timed_out) {
        const int r = cons.r;
        const long long n_real = sm.cnt[r] - (long long)cons.it * ISL;   // real slots of this item
        // tile geometry (packed layout, coef_offset): rows of tl slots, 8-slot group g of row j
        // stored at position (g + j) mod (tl / 8)
        const int tl = (int)min((long long)ISL, pad8(sm.cnt[r]) - (long long)cons.it * ISL);
        const int ng = tl >> 3;
        const bool full_tile = ng == 16;
        const uint32_t row_bytes = (uint32_t)tl * 2u;
        const int lgc = chunk_lg(tl);                   // same chunking as the producer
        const int nj = (r + (1 << lgc) - 1) >> lgc;
        float sc[ISL / 16][4];
#pragma unroll
        for (int t = 0; t < ISL / 16; ++t) sc[t][0] = sc[t][1] = sc[t][2] = sc[t][3] = 0.f;

        // ---- K chunks: scores (rows >= r masked in the q~ fragment)
        for (int jc = 0; jc < nj; ++jc) {
          if (!wait_chunk()) break;
          const uint32_t st_addr = ring_w + (n_issued % ST) * STAGE;
          const int m = lane >> 3, r8 = lane & 7;
          const int j0 = jc << lgc, j1 = min(r, j0 + (1 << lgc));
          for (int j16 = j0; j16 < j1; j16 += 16) {
            const uint4 qf = *reinterpret_cast<const uint4*>(&sm.qfrag[j16 >> 4][lane][0]);
            // this lane's row of the 8x8 matrices: coefficient j, staged at row (j - chunk start)
            const int jrow = (j16 - j0) + (m >> 1) * 8 + r8;
            const int j = j0 + jrow;
            const uint32_t row_addr = st_addr + jrow * row_bytes;
            uint32_t a[ISL / 16][4];
            // stored position of slot group 2 mt + (m & 1) in row j: (group + j) mod ng; for a full
            // tile every offset is computed on its own (no chain through the previous one)
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
#pragma unroll
            for (int mt = 0; mt < ISL / 16; ++mt) ldsm_x4_trans(row_addr + off[mt], a[mt]);
            if (j16 + 16 > r) {   // warp-uniform: rows >= r of this k-step are not coefficients
              // A fragment registers 0, 1 hold rows j16 + 2c (+1), registers 2, 3 rows 8 later
              const int jb = j16 + 2 * c;
              const uint32_t m0 = keep_rows(0xFFFFFFFFu, jb, r), m1 = keep_rows(0xFFFFFFFFu, jb + 8, r);
#pragma unroll
              for (int mt = 0; mt < ISL / 16; ++mt) {
                a[mt][0] &= m0; a[mt][1] &= m0; a[mt][2] &= m1; a[mt][3] &= m1;
              }
            }
#pragma unroll
            for (int mt = 0; mt < ISL / 16; ++mt) mma_bf16_16816(sc[mt], a[mt], qf.x, qf.y);
#pragma unroll
            for (int mt = 0; mt < ISL / 16; ++mt) mma_bf16_16816(sc[mt], a[mt], qf.z, qf.w);
          }
          __syncwarp();
          next_chunk();
        }
        if (timed_out) break;

        // ---- online softmax over the item's slots (heads 2c, 2c+1 per lane)
        float mloc[2] = {-INFINITY, -INFINITY};
        const bool full_item = n_real >= ISL;           // warp-uniform: no slot to mask
#pragma unroll
        for (int mt = 0; mt < ISL / 16; ++mt) {
          if (!full_item) {
            const int s0 = mt * 16 + g8;
            if (s0 >= n_real) { sc[mt][0] = sc[mt][1] = -INFINITY; }
            if (s0 + 8 >= n_real) { sc[mt][2] = sc[mt][3] = -INFINITY; }
          }
          mloc[0] = fmaxf(mloc[0], fmaxf(sc[mt][0], sc[mt][2]));
          mloc[1] = fmaxf(mloc[1], fmaxf(sc[mt][1], sc[mt][3]));
        }
        // The reference max only moves when some score exceeds it by more than kSlack (log2
        // units): weights stay <= 2^kSlack, exact after the final normalisation, and the common
        // case costs one warp vote instead of a shuffle reduction and a rescale.
        float corr[2] = {1.f, 1.f};
        if (!__all_sync(0xffffffffu, mloc[0] <= Mx[0] + kSlack && mloc[1] <= Mx[1] + kSlack)) {
#pragma unroll
          for (int o = 4; o < 32; o <<= 1) {
            mloc[0] = fmaxf(mloc[0], __shfl_xor_sync(0xffffffffu, mloc[0], o));
            mloc[1] = fmaxf(mloc[1], __shfl_xor_sync(0xffffffffu, mloc[1], o));
          }
#pragma unroll
          for (int e = 0; e < 2; ++e) {
            const float nm = fmaxf(Mx[e], mloc[e]);
            corr[e] = fast_exp2(Mx[e] - nm);
            Mx[e] = nm;
          }
#pragma unroll
          for (int t = 0; t < kHeadDim / 16; ++t) {
            oacc[t][0] *= corr[0]; oacc[t][1] *= corr[1];
            oacc[t][2] *= corr[0]; oacc[t][3] *= corr[1];
          }
        }
        float lsum[2] = {0.f, 0.f};
        uint32_t pb[ISL / 16][2];   // per slot tile: b0, b1 of P^T (bf16)
#pragma unroll
        for (int mt = 0; mt < ISL / 16; ++mt) {
          const float p0 = fast_exp2(sc[mt][0] - Mx[0]), p1 = fast_exp2(sc[mt][1] - Mx[1]);
          const float p2 = fast_exp2(sc[mt][2] - Mx[0]), p3 = fast_exp2(sc[mt][3] - Mx[1]);
          lsum[0] += p0 + p2;
          lsum[1] += p1 + p3;
          pb[mt][0] = movmatrix_trans(pack_bf16(p0, p1));
          pb[mt][1] = movmatrix_trans(pack_bf16(p2, p3));
        }
        Ls[0] = Ls[0] * corr[0] + lsum[0];
        Ls[1] = Ls[1] * corr[1] + lsum[1];

        // ---- V chunks: weighted coefficient rows (rows >= r masked in the A fragment)
        {
          int left = 0;             // rows of the current chunk not used yet
          int j0 = 0;               // first row of the current chunk
          uint32_t st_addr = 0;
          bool ok = true;
          const int m = lane >> 3, r8 = lane & 7;
#pragma unroll
          for (int jt = 0; jt < kHeadDim / 16; ++jt) {   // 16-row tile of o~
            if (jt * 16 >= r) break;                     // warp-uniform
            if (left == 0) {                             // the tile starts a chunk
              if (jt > 0) { __syncwarp(); next_chunk(); }
              if (!wait_chunk()) { ok = false; break; }
              st_addr = ring_w + (n_issued % ST) * STAGE;
              j0 = jt * 16;
              left = 1 << lgc;
            }
            left -= 16;
            const int jrow = (jt * 16 - j0) + (m & 1) * 8 + r8;
            const int j = j0 + jrow;
            const uint32_t row_addr = st_addr + jrow * row_bytes;
            const bool keep0 = jt * 16 + g8 < r, keep1 = jt * 16 + g8 + 8 < r;
            float t1[4] = {0.f, 0.f, 0.f, 0.f};
            // stored position of slot group 2 kt + (m >> 1) (kt = 0..7) in row j, as in the K loop
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
#pragma unroll
            for (int kt = 0; kt < ISL / 16; kt += 2) {
              uint32_t a[4], b[4];
              ldsm_x4(row_addr + off[kt], a);
              ldsm_x4(row_addr + off[kt + 1], b);
              if (jt * 16 + 16 > r) {                    // warp-uniform: rows >= r in this tile
                if (!keep0) { a[0] = a[2] = 0u; b[0] = b[2] = 0u; }
                if (!keep1) { a[1] = a[3] = 0u; b[1] = b[3] = 0u; }
              }
              mma_bf16_16816(oacc[jt], a, pb[kt][0], pb[kt][1]);
              mma_bf16_16816(t1, b, pb[kt + 1][0], pb[kt + 1][1]);
            }
#pragma unroll
            for (int e = 0; e < 4; ++e) oacc[jt][e] += t1[e];
          }
          if (ok) { __syncwarp(); next_chunk(); }         // the last chunk of the item
        }
        cons_k += NW;
        if (cons_k < total) cons = next_rr<NW>(sm, cons, cons_k);
      }
      // drain: never leave bulk copies in flight into this ring (a copy whose wait gave up stays
      // counted in n_pending and is waited for once more before the CTA exits)
      while (n_pending > 0 && !timed_out) {
        if (!mbar_wait_bounded(&bars[n_issued % ST], (n_issued / ST) & 1u, kWaitTries)) {
          timed_out = true;
          break;
        }
        ++n_issued;
        --n_pending;
      }

      // ---- merge the warps of this CTA for this segment
      __syncwarp();
#pragma unroll
      for (int e = 0; e < 2; ++e)
#pragma unroll
        for (int o = 4; o < 32; o <<= 1) Ls[e] += __shfl_xor_sync(0xffffffffu, Ls[e], o);
      dead = __syncthreads_or(dead || timed_out);   // every warp has finished this segment
      if (!dead && g8 == 0) {
        mg.M[warp][2 * c] = Mx[0]; mg.M[warp][2 * c + 1] = Mx[1];
        mg.L[warp][2 * c] = Ls[0]; mg.L[warp][2 * c + 1] = Ls[1];
      }
      if (!dead) {
#pragma unroll
        for (int t = 0; t < kHeadDim / 16; ++t) {
          mg.acc[warp][2 * c][t * 16 + g8] = oacc[t][0];
          mg.acc[warp][2 * c + 1][t * 16 + g8] = oacc[t][1];
          mg.acc[warp][2 * c][t * 16 + g8 + 8] = oacc[t][2];
          mg.acc[warp][2 * c + 1][t * 16 + g8 + 8] = oacc[t][3];
        }
      }
      if (!dead && tid < kHeadsPad) {
        const int h = tid;
        float mx = -INFINITY, l = 0.f;
#pragma unroll
        for (int w = 0; w < NW; ++w) mx = fmaxf(mx, mg.M[w][h]);
#pragma unroll
        for (int w = 0; w < NW; ++w) {
          const float f = mx == -INFINITY ? 0.f : fast_exp2(mg.M[w][h] - mx);
          mg.F[w][h] = f;
          l = fmaf(mg.L[w][h], f, l);
        }
        mg.mx[h] = mx;
        mg.l[h] = l;
      }
      __syncthreads();
      // partial slot of this (segment, CTA): index cta + segment number (unique: a CTA after this
      // one only meets segments after this one)
      const long long seg = (long long)b * s.G + g;
      float* pout = part + (cta + seg) * (long long)kHeadsPad * kPartStride;
      for (int i = tid; i < kHeadsPad * kHeadDim; i += blockDim.x) {
        const int h = i / kHeadDim, j = i % kHeadDim;
        float o = 0.f;
        if (!dead) {
#pragma unroll
          for (int w = 0; w < NW; ++w) o = fmaf(mg.acc[w][h][j], mg.F[w][h], o);
        }
        pout[h * kPartStride + j] = o;
        if (j == 0) {   // an abandoned CTA contributes an empty partial
          pout[h * kPartStride + kHeadDim] = dead ? -INFINITY : mg.mx[h];
          pout[h * kPartStride + kHeadDim + 1] = dead ? 0.f : mg.l[h];
        }
      }
      // the last CTA to finish this segment merges every partial of it
      __syncthreads();
      if (tid == 0) {
        // release: this CTA's partial (ordered before by the barrier) is visible to whoever sees
        // the count; acquire: the last arrival then sees every other CTA's partial
        const uint32_t n = (uint32_t)(c1 - c0 + 1);   // CTAs that share this segment
        const uint32_t done = atom_add_acq_rel_gpu(&arrived[seg], 1u);
        last_cta = done == n - 1u;
        if (done >= n) raise_status(dev_status, VARRATE_ERR_CORRUPT);   // counts left by an earlier call
      }
      __syncthreads();
      if (last_cta && !dead) {
        if (!combine_segment(*reinterpret_cast<CombSmem*>(ring), &bar_comb, n_comb & 1u, part, c0, c1, seg,
                             qin + ((long long)b * s.H + (long long)g * s.grp) * kHeadDim,
                             basis_v + ((long long)layer * s.G + g) * kHeadDim * kHeadDim,
                             n_tail ? tail_k + ((long long)b * s.G + g) * n_tail * kHeadDim : nullptr,
                             n_tail ? tail_v + ((long long)b * s.G + g) * n_tail * kHeadDim : nullptr, n_tail,
                             out + ((long long)b * s.H + (long long)g * s.grp) * kHeadDim, s.grp, tid)) {
          timed_out = true;
          dead = true;   // CTA-uniform: the U_V copy of the combine may still be landing
        }
        ++n_comb;
      }
      __syncthreads();
    }
    if (++g == s.G) { ++b; g = 0; }
    while (b < s.B && segW[b] == 0) ++b;
    more = b < s.B && seg_start(b, g) < hi_g;
    if (more && !dead) {
      fence_proxy_async_smem();   // the merge and combine wrote the ring: before the next copies
      __syncthreads();
    }
  }
  // segments with an empty coded stream (tail only): one CTA each, no partials
  if (n_empty && !dead)
  for (int b = 0; b < s.B; ++b)
    for (int g = 0; g < s.G; ++g) {
      const long long seg = (long long)b * s.G + g;
      if (segW[b] != 0 || seg % C != cta || dead) continue;   // CTA-uniform
      __syncthreads();
      if (!combine_segment(*reinterpret_cast<CombSmem*>(ring), &bar_comb, n_comb & 1u, part, 0, -1, seg,
                           qin + ((long long)b * s.H + (long long)g * s.grp) * kHeadDim,
                           basis_v + ((long long)layer * s.G + g) * kHeadDim * kHeadDim,
                           n_tail ? tail_k + ((long long)b * s.G + g) * n_tail * kHeadDim : nullptr,
                           n_tail ? tail_v + ((long long)b * s.G + g) * n_tail * kHeadDim : nullptr, n_tail,
                           out + ((long long)b * s.H + (long long)g * s.grp) * kHeadDim, s.grp, tid)) {
        timed_out = true;
        dead = true;
      }
      ++n_comb;
    }
  if (dead) {
    // last bounded waits for copies that may still be landing in this CTA's shared memory
    for (; n_pending > 0; --n_pending, ++n_issued)
      if (!mbar_wait_bounded(&bar_all[warp * ST + n_issued % ST], (n_issued / ST) & 1u, kWaitTries)) break;
    if (n_comb > 0 && tid == 0) mbar_wait_bounded(&bar_comb, (n_comb - 1) & 1u, kWaitTries);
  }
  if (timed_out && lane == 0) raise_status(dev_status, VARRATE_ERR_TIMEOUT);
  // the CTA that completes a multiple of the grid size of exits advances the call count (a
  // multiple rather than exactly C - 1: the count then stays consistent whatever the set held)
  __syncthreads();
  if (tid == 0 && (atomicAdd(&hdr->exits[parity], 1u) + 1u) % (uint32_t)C == 0u)
    atomicAdd(&hdr->calls, 1ull);
}

}  // namespace

size_t decode_mma_smem_bytes() { return (size_t)NW * ST * STAGE + sizeof(SegSmem); }

// partials: one slot per (segment, CTA) pair a CTA can meet (the counters live apart, see kernels.h)
size_t decode_mma_part_bytes(const Shape& s, int num_sms) {
  const size_t p = (size_t)(num_sms + (size_t)s.B * s.G) * kHeadsPad * kPartStride * sizeof(float);
  return (p + 255) & ~size_t(255);
}

bool decode_mma_supported(const Shape& s, int n_tail, int num_sms) {
  // the cost line (at most B G cap elements) times the grid size must stay below 2^62
  const unsigned long long line = (unsigned long long)s.B * s.G * ((unsigned long long)s.cap + kSegCost + kSegEnd);
  return s.dtype == VARRATE_BF16 && s.B <= 64 && (long long)s.B * s.G <= kDecodeMaxSegs &&
         n_tail <= kMaxTailFused && num_sms >= 1 && num_sms <= kMaxCtas &&
         line <= (1ull << 62) / (unsigned long long)num_sms;
}

int launch_decode_mma(const Shape& s, const varrate_packed& c, const void* basis_k,
                      const void* basis_v, const void* q, int layer, const void* tail_k,
                      const void* tail_v, int n_tail, void* out, int32_t* dev_status,
                      void* header, float* part, int num_sms, cudaStream_t st) {
  const size_t smem = decode_mma_smem_bytes();
  // the shared-memory opt-in is a per-device property of the function: set once per device
  static std::atomic<int> smem_set[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64 ||
      smem_set[dev].load(std::memory_order_acquire) == 0) {
    if (cudaFuncSetAttribute(decode_mma_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) !=
        cudaSuccess)
      return -1;
    if (dev >= 0 && dev < 64) smem_set[dev].store(1, std::memory_order_release);
  }
  // the grid may be scheduled while its predecessor drains (programmatic dependent launch); it
  // waits on griddepcontrol.wait before touching anything an earlier operation wrote
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
  cudaLaunchKernelEx(&lc, decode_mma_kernel, (const __nv_bfloat16*)c.coef, (const int32_t*)c.bucket_count,
                     (const int64_t*)c.bucket_base, (const __nv_bfloat16*)basis_k,
                     (const __nv_bfloat16*)basis_v, (const __nv_bfloat16*)q,
                     (const __nv_bfloat16*)tail_k, (const __nv_bfloat16*)tail_v, n_tail,
                     (__nv_bfloat16*)out, part, reinterpret_cast<DecodeHeader*>(header), dev_status, s, layer);
  return 1;
}

}  // namespace vr
