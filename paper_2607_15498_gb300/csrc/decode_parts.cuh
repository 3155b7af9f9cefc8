// Parts shared by the fused tensor-core decode kernels (bf16 coefficients: decode_mma.cu;
// group-quantized coefficients dequantized in the ring: decode_q.cu): the warp layout, the
// per-segment shared-memory tables, the query rotation, the completion-counting header and the
// cross-CTA combine.
#pragma once

#include "common.cuh"
#include "decode_common.cuh"
#include "kernels.h"

namespace vr {

namespace {

// 12 warps of at most 168 registers fill the register file, three per scheduler: more warps hide
// more of the instruction latency of the item loop than deeper rings do (measured: 8 warps with 3
// stages each 54.7 us per llama32 layer call, 12 warps with 2 stages 52.2 us, same 192 KB ring).
constexpr int NW = 12;                // warps per CTA
constexpr int ST = 2;                 // ring stages per warp
constexpr int kPartStride = kHeadDim + 4;   // o~[128], max, sum, pad: rows 16-byte aligned
constexpr int kHeadsPad = 8;

struct SegSmem {
  alignas(16) uint32_t qfrag[kHeadDim / 16][32][4];   // per j-chunk, per lane: b0 hi, b1 hi, b0 lo, b1 lo (read as uint4)
  alignas(16) float qt[kHeadsPad][kHeadDim];          // rotated, scaled queries (fp32)
  long long base[kMaxR + 2];
  int cnt[kMaxR + 1];
  int it_lo[kMaxR + 1];     // first item of bucket r inside this CTA's cost range
  int it_pref[kMaxR + 2];   // exclusive prefix of the per-bucket item counts
};
static_assert(offsetof(SegSmem, qfrag) % 16 == 0, "qfrag is read with 16-byte loads");

struct Merge {
  float M[NW][kHeadsPad], L[NW][kHeadsPad];
  float F[NW][kHeadsPad];             // 2^(M - max): each warp's weight in the CTA's partial
  float mx[kHeadsPad], l[kHeadsPad];
  float acc[NW][kHeadsPad][kHeadDim];
};

// Producer cursor: which chunk of which item comes next in this warp's stream.
struct Prod {
  int k;       // item index (CTA-local)
  Item item;
  int phase;   // 0 = K rows, 1 = V rows
  int jc;      // 16-row chunk index
};

// Rotate the queries of (b, g) into the basis: qt[head][j] = scale * sum_i U_K[j][i] q[head][i],
// warp w computing rows j in [16w, 16w + 16) with one m16n8k16 tile per 16 columns of U_K. The
// loads (rot_load) are issued at the start of a segment, ahead of its table loads, so both take
// one memory round trip together; rot_compute runs once the tables are in.
static_assert(NW * 16 >= kHeadDim, "one 16-row tile of U_K per warp (warps past d / 16 idle)");
struct RotRegs {
  uint32_t a[kHeadDim / 16][4];    // U_K rows 16w .. 16w + 15 (A fragments)
  uint32_t bq[kHeadDim / 16][2];   // q (B fragments; zero for padded heads)
};

// The MMA sums over k, so any one-to-one assignment of U_K's columns to the k slots of the
// fragments gives the same product as long as q uses the same assignment. Lane (g8, c) holds the
// 32 columns {32 i + 8 c + t : i < 4, t < 8} of its rows: four 16-byte loads per row, and the four
// lanes of a row read 64 contiguous bytes. Column 32 i + 8 c + t feeds k-step kc = 2 i + t / 4, as
// fragment register a0 (t % 4 < 2) or a2 (t % 4 >= 2).
__device__ __forceinline__ void rot_load(RotRegs& rr, const __nv_bfloat16* __restrict__ U,
                                         const __nv_bfloat16* __restrict__ q, int grp, int warp, int lane) {
  // warps past d / 16 load (and never use) the tile of warp w mod 8: every address stays in U
  const int g8 = lane >> 2, c = lane & 3, j0 = (warp % (kHeadDim / 16)) * 16;
  const uint4* u0 = reinterpret_cast<const uint4*>(U + (long long)(j0 + g8) * kHeadDim) + c;
  const uint4* u1 = reinterpret_cast<const uint4*>(U + (long long)(j0 + g8 + 8) * kHeadDim) + c;
  const uint4* qr = reinterpret_cast<const uint4*>(q + (long long)(g8 < grp ? g8 : 0) * kHeadDim) + c;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const uint4 x = ld_nc_early_v4(u0 + 4 * i), y = ld_nc_early_v4(u1 + 4 * i), z = ld_nc_early_v4(qr + 4 * i);
    rr.a[2 * i][0] = x.x; rr.a[2 * i][2] = x.y; rr.a[2 * i + 1][0] = x.z; rr.a[2 * i + 1][2] = x.w;
    rr.a[2 * i][1] = y.x; rr.a[2 * i][3] = y.y; rr.a[2 * i + 1][1] = y.z; rr.a[2 * i + 1][3] = y.w;
    rr.bq[2 * i][0] = z.x; rr.bq[2 * i][1] = z.y; rr.bq[2 * i + 1][0] = z.z; rr.bq[2 * i + 1][1] = z.w;
  }
}

__device__ __forceinline__ void rot_compute(SegSmem& sm, const RotRegs& rr, int grp, int warp, int lane) {
  const int g8 = lane >> 2, c = lane & 3, j0 = warp * 16;
  const float scale = kLog2e * rsqrtf((float)kHeadDim);
  float e[2][4] = {};   // even and odd k-steps: two independent MMA chains
#pragma unroll
  for (int kc = 0; kc < kHeadDim / 16; ++kc) {
    const uint32_t b0 = g8 < grp ? rr.bq[kc][0] : 0u, b1 = g8 < grp ? rr.bq[kc][1] : 0u;
    mma_bf16_16816(e[kc & 1], rr.a[kc], b0, b1);
  }
  float d[4];
#pragma unroll
  for (int t = 0; t < 4; ++t) d[t] = e[0][t] + e[1][t];
  // d: rows j0+g8 (+8), heads 2c, 2c+1
  sm.qt[2 * c][j0 + g8] = d[0] * scale;
  sm.qt[2 * c + 1][j0 + g8] = d[1] * scale;
  sm.qt[2 * c][j0 + g8 + 8] = d[2] * scale;
  sm.qt[2 * c + 1][j0 + g8 + 8] = d[3] * scale;
}

// Score-MMA B fragments of q~ (split hi + lo) for every 16-row chunk, one uint4 per lane.
__device__ __noinline__ void build_qfrag(SegSmem& sm, int tid) {
  for (int i = tid; i < (kHeadDim / 16) * 32; i += NW * 32) {
    const int jc = i / 32, lane = i % 32, g8 = lane >> 2, c = lane & 3;
    const int j = jc * 16 + 2 * c;
    uint32_t h0, l0, h1, l1;
    split_bf16(sm.qt[g8][j], sm.qt[g8][j + 1], h0, l0);
    split_bf16(sm.qt[g8][j + 8], sm.qt[g8][j + 9], h1, l1);
    sm.qfrag[jc][lane][0] = h0;
    sm.qfrag[jc][lane][1] = h1;
    sm.qfrag[jc][lane][2] = l0;
    sm.qfrag[jc][lane][3] = l1;
  }
}


// Completion counting (the first kDecodeCounterBytes of the workspace, DecodeHeader): a count of
// the fused calls made on the workspace, and two sets of per-(sequence, KV head) arrival counters
// with a grid-exit counter each. A call reads the call count once (after griddepcontrol.wait, so
// the previous call has finished) and counts on the set of its parity with plain atomicAdd; it
// never resets that set, and instead zeroes the other set, which the previous call used and the
// next call will use. So every call starts from zero counters; counts left by an earlier call that
// overlapped this one or gave up show as an arrival past the expected number (exactly detected:
// VARRATE_ERR_CORRUPT), and are gone one call later without any action by the caller. The CTA that
// brings the grid-exit counter to a multiple of the grid size advances the call count; replaying
// a captured launch advances it the same way.
struct DecodeHeader {
  unsigned long long calls;         // fused calls completed on this workspace
  uint32_t exits[2];                // CTAs that left the kernel, per parity
  uint32_t pad[60];
  uint32_t arrived[2][kDecodeMaxSegs];   // CTAs that finished segment seg, per parity
};
static_assert(sizeof(DecodeHeader) == kDecodeCounterBytes, "decode header layout");
static_assert(offsetof(DecodeHeader, arrived) == 256, "counter sets start 256 bytes in");

constexpr int kMaxTailFused = 256;   // exact tail tokens the fused kernel stages in the ring

struct CombSmem {   // aliases the ring while the last CTA of a segment combines it
  alignas(128) __nv_bfloat16 us[kHeadDim * kHeadDim];       // U_V[g], row j (one bulk copy)
  alignas(128) __nv_bfloat16 tk[kMaxTailFused * kHeadDim];  // exact tail keys, row t (one bulk copy)
  alignas(128) __nv_bfloat16 tv[kMaxTailFused * kHeadDim];  // exact tail values, row t (one bulk copy)
  float ot[kHeadsPad][kHeadDim + 8];                        // merged o~ per head
  float tsc[kHeadsPad][kMaxTailFused + 8];                  // tail scores, then tail weights
  float hl[kHeadsPad];                                      // softmax normaliser per head
};
static_assert(sizeof(CombSmem) <= (size_t)NW * ST * STAGE, "combine buffers fit in the ring");
static_assert(NW >= kHeadsPad, "one warp per head in the combine");

// Merge the partials of segment (b, g) written by CTAs c0..c1 (slot cc + seg; none if c1 < c0),
// add the exact tail, rotate back with U_V^T and normalise. Called by all threads; the ring
// is idle. U_V and the tail's keys and values are staged in the ring by bulk copies while the
// partials are merged (warp h merges head h, lane l columns 4l .. 4l + 3, with the partials of up
// to 8 CTAs in flight at once). Tail scores are m16n8k16 tiles (16 tail tokens x 8 heads, exact
// bf16 products of key and query); the tail's values join the rotation as further k-steps:
//   out^T[col][head] = sum_j U_V[j][col] o~[head][j] + sum_t v_t[col] w[head][t]
// with o~ and the tail weights w split hi + lo in bf16. Returns false if a staging copy timed out.
// Kept out of line (as is build_qfrag): the item loop's code stays compact (measured -0.2 us per
// llama32 layer call).
__device__ __noinline__ bool combine_segment(CombSmem& cs, uint64_t* bar, uint32_t parity, const float* __restrict__ part,
                                int c0, int c1, long long seg, const __nv_bfloat16* __restrict__ q,
                                const __nv_bfloat16* __restrict__ Uv, const __nv_bfloat16* __restrict__ tail_k,
                                const __nv_bfloat16* __restrict__ tail_v, int n_tail,
                                __nv_bfloat16* __restrict__ out, int grp, int tid) {
  const int lane = tid & 31, warp = tid >> 5;
  const int g8 = lane >> 2, c = lane & 3;
  const int n_tt = (n_tail + 15) >> 4;   // 16-token tiles of the tail
  fence_proxy_async_smem();   // earlier generic accesses of the ring precede the async writes
  __syncthreads();
  if (tid == 0) {
    const uint32_t tail_bytes = (uint32_t)n_tail * kHeadDim * 2;
    mbar_arrive_expect_tx(bar, kHeadDim * kHeadDim * 2 + 2 * tail_bytes);
    bulk_g2s(smem_addr(cs.us), Uv, kHeadDim * kHeadDim * 2, bar);
    if (n_tail) {
      bulk_g2s(smem_addr(cs.tk), tail_k, tail_bytes, bar);
      bulk_g2s(smem_addr(cs.tv), tail_v, tail_bytes, bar);
    }
  }
  __syncwarp();
  // rows of the last tail tile past n_tail read as zeros (disjoint from the copies' bytes)
  for (int i = n_tail * kHeadDim + tid; i < n_tt * 16 * kHeadDim; i += blockDim.x) {
    cs.tk[i] = __float2bfloat16_rn(0.f);
    cs.tv[i] = __float2bfloat16_rn(0.f);
  }
  // query B fragments of the tail scores: B[k][n] = q[head n][k], pairs of k per register
  uint32_t qb[kHeadDim / 16][2];
#pragma unroll
  for (int ks = 0; ks < kHeadDim / 16; ++ks) {
    const __nv_bfloat16* qr = q + (long long)(g8 < grp ? g8 : 0) * kHeadDim + ks * 16 + 2 * c;
    qb[ks][0] = g8 < grp && n_tail ? *reinterpret_cast<const uint32_t*>(qr) : 0u;
    qb[ks][1] = g8 < grp && n_tail ? *reinterpret_cast<const uint32_t*>(qr + 8) : 0u;
  }
  // merge the partials of the coded stream
  const int h = warp;
  float M = -INFINITY, L = 0.f;
  float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
  if (h < grp) {
    const int np = c1 - c0 + 1;
    for (int cb = 0; cb < np; cb += 8) {
      float m[8], l[8];
      float4 o[8];
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        if (cb + k < np) {
          const float* pp = part + ((c0 + cb + k + seg) * kHeadsPad + h) * kPartStride;
          m[k] = __ldcg(pp + kHeadDim);
          l[k] = __ldcg(pp + kHeadDim + 1);
          o[k] = __ldcg(reinterpret_cast<const float4*>(pp) + lane);
        } else {
          m[k] = -INFINITY; l[k] = 0.f; o[k] = make_float4(0.f, 0.f, 0.f, 0.f);
        }
      }
      float mx = M;
#pragma unroll
      for (int k = 0; k < 8; ++k) mx = fmaxf(mx, m[k]);
      if (mx != -INFINITY) {
        const float f = M == -INFINITY ? 0.f : exp2f(M - mx);
        acc.x *= f; acc.y *= f; acc.z *= f; acc.w *= f;
        L *= f;
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          const float w = m[k] == -INFINITY ? 0.f : exp2f(m[k] - mx);
          L = fmaf(w, l[k], L);
          acc.x = fmaf(w, o[k].x, acc.x); acc.y = fmaf(w, o[k].y, acc.y);
          acc.z = fmaf(w, o[k].z, acc.z); acc.w = fmaf(w, o[k].w, acc.w);
        }
        M = mx;
      }
    }
  }
  if (!__syncthreads_and(mbar_wait_bounded(bar, parity, kWaitTries))) return false;
  __syncwarp();
  // exact tail scores (log2 units): warp w takes tail tiles w, w + NW, ...
  const float scale = kLog2e * rsqrtf((float)kHeadDim);
  for (int tt = warp; tt < n_tt; tt += NW) {
    float sc[4] = {0.f, 0.f, 0.f, 0.f};
    const int row = tt * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
#pragma unroll
    for (int ks = 0; ks < kHeadDim / 16; ++ks) {
      uint32_t a[4];
      ldsm_x4(smem_addr(&cs.tk[row * kHeadDim + ks * 16 + (lane >> 4) * 8]), a);
      mma_bf16_16816(sc, a, qb[ks][0], qb[ks][1]);
    }
#pragma unroll
    for (int e = 0; e < 4; ++e) {   // rows tt*16 + g8 (+8), heads 2c, 2c+1
      const int t = tt * 16 + g8 + (e >> 1) * 8;
      cs.tsc[2 * c + (e & 1)][t] = t < n_tail ? sc[e] * scale : -INFINITY;
    }
  }
  __syncthreads();
  // per head: fold the tail into the softmax, tail weights in place of the scores
  {
    float tm = -INFINITY;
    if (h < grp)
      for (int t = lane; t < n_tail; t += 32) tm = fmaxf(tm, cs.tsc[h][t]);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) tm = fmaxf(tm, __shfl_xor_sync(0xffffffffu, tm, o));
    const float mx = fmaxf(M, tm);
    const float f = (M == -INFINITY || mx == -INFINITY) ? 0.f : exp2f(M - mx);
    acc.x *= f; acc.y *= f; acc.z *= f; acc.w *= f;
    float lt = 0.f;
    for (int t = lane; t < n_tt * 16; t += 32) {
      const float w = (h < grp && t < n_tail) ? exp2f(cs.tsc[h][t] - mx) : 0.f;
      if (h < kHeadsPad) cs.tsc[h][t] = w;   // zero for padded heads and rows past the tail
      lt += w;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) lt += __shfl_xor_sync(0xffffffffu, lt, o);
    if (lane == 0 && h < kHeadsPad) cs.hl[h] = L * f + lt;
    if (h >= grp) acc = make_float4(0.f, 0.f, 0.f, 0.f);
    if (h < kHeadsPad) *reinterpret_cast<float4*>(&cs.ot[h][4 * lane]) = acc;   // zero for padded heads
  }
  __syncthreads();
  // out^T[col][head]: warp w < 8 owns columns 16w .. 16w + 15
  if (warp < kHeadDim / 16) {
    // four independent accumulators (hi / lo part of the B operand, even / odd k-step) keep the
    // chain of dependent MMAs short
    float d[4][4] = {};
    const int col0 = warp * 16;
    const int col = col0 + ((lane >> 3) & 1) * 8;
    const int jr = (lane & 7) + ((lane >> 4) & 1) * 8;
#pragma unroll
    for (int ks = 0; ks < kHeadDim / 16; ++ks) {
      uint32_t a[4];
      ldsm_x4_trans(smem_addr(&cs.us[(ks * 16 + jr) * kHeadDim + col]), a);
      const int jb = ks * 16 + 2 * c;
      uint32_t h0, l0, h1, l1;
      split_bf16(cs.ot[g8][jb], cs.ot[g8][jb + 1], h0, l0);
      split_bf16(cs.ot[g8][jb + 8], cs.ot[g8][jb + 9], h1, l1);
      mma_bf16_16816(d[ks & 1], a, h0, h1);
      mma_bf16_16816(d[2 + (ks & 1)], a, l0, l1);
    }
    for (int ts = 0; ts < n_tt; ts += 2) {   // the tail's values, 16 tokens per k-step
#pragma unroll
      for (int u = 0; u < 2; ++u) {
        if (ts + u < n_tt) {
          uint32_t a[4];
          ldsm_x4_trans(smem_addr(&cs.tv[((ts + u) * 16 + jr) * kHeadDim + col]), a);
          const int tb = (ts + u) * 16 + 2 * c;
          uint32_t h0, l0, h1, l1;
          split_bf16(cs.tsc[g8][tb], cs.tsc[g8][tb + 1], h0, l0);
          split_bf16(cs.tsc[g8][tb + 8], cs.tsc[g8][tb + 9], h1, l1);
          mma_bf16_16816(d[u], a, h0, h1);
          mma_bf16_16816(d[2 + u], a, l0, l1);
        }
      }
    }
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int oc = col0 + g8 + (e >> 1) * 8, hh = 2 * c + (e & 1);
      if (hh < grp) {
        const float y = (d[0][e] + d[1][e]) + (d[2][e] + d[3][e]);
        out[(long long)hh * kHeadDim + oc] = __float2bfloat16_rn(y / cs.hl[hh]);
      }
    }
  }
  return true;
}

}  // namespace

}  // namespace vr
