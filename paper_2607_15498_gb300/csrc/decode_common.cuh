// Work split shared by the bf16 tensor-core decode kernels (single query: decode_mma.cu; window of
// queries: decode_window.cu).
//
// Cost line. The K coefficient streams of all (sequence, KV head) pairs of a layer are laid end to
// end, each preceded by a fixed set-up allowance (kSegCost elements); the persistent grid cuts the
// line into equal ranges, so every SM moves about the same number of bytes. A CTA walks the
// (sequence, head) segments its range touches; inside one segment its share is a run of 128-slot
// items (one tile of the packed layout, Eq. 5 storage), enumerated bucket by bucket.
#pragma once

#include "common.cuh"

namespace vr {

constexpr int kMaxR = kHeadDim;
constexpr int ISL = 128;              // slots per item (one tile of the packed layout)
constexpr int CH = 32;                // coefficient rows per chunk of a full 128-slot tile
constexpr int STAGE = CH * ISL * 2;   // one chunk: up to 32 rows of a 128-slot tile (8 KB)
constexpr uint32_t kWaitTries = 1u << 22;   // bounded mbarrier polls (well over a second)
constexpr float kSlack = 8.f;                // headroom of the running max, log2 units
// Cost-line allowance per (sequence, KV head) segment, in K-stream elements: a CTA that enters a
// segment pays its set-up (tables, query rotation, pipeline ramp, partial write, and for one CTA
// the combine), about as long as streaming this many coefficients at a CTA's share of HBM
// bandwidth, so ranges that straddle segments are shortened by that much.
constexpr long long kSegCost = 90112;
// Cost-line allowance after each segment's coefficients: the CTA that takes a segment's last
// stretch also pays its arrival, often the segment's combine, and the uneven finish of its warps on
// the last items, so its range is shortened by this much. Both allowances were swept on the GPU
// for the 32-layer, 8-sequence llama shape (64 segments over 152 CTAs); shapes with few segments
// per grid barely feel them.
constexpr long long kSegEnd = 163840;
constexpr int kMaxCtas = 1024;   // grid size bound (64-bit cost-line arithmetic)

// A 64-bit integer division is a long instruction sequence (measured ~600 cycles here), so the
// cost-line arithmetic avoids it. n / d for d < 2^16 by long division in 16-bit digits: four
// 32-bit divisions.
__device__ __forceinline__ unsigned long long udiv_small(unsigned long long n, uint32_t d) {
  unsigned long long q = 0;
  uint32_t r = 0;
#pragma unroll
  for (int sh = 48; sh >= 0; sh -= 16) {
    const uint32_t cur = (r << 16) | (uint32_t)((n >> sh) & 0xFFFFu);   // r < d < 2^16
    const uint32_t qd = cur / d;
    r = cur - qd * d;
    q = (q << 16) | qd;
  }
  return q;
}
static_assert(kMaxCtas < (1 << 16), "udiv_small divides by the grid size");

// Start of CTA c's range on a cost line of T elements cut into C equal ranges: floor(T c / C).
// The launcher guarantees T * C < 2^63 and C <= kMaxCtas < 2^16.
__device__ __forceinline__ long long cut_at(long long T, long long c, int C) {
  return (long long)udiv_small((unsigned long long)T * (unsigned long long)c, (uint32_t)C);
}

// CTAs whose cost range [cuts[c], cuts[c + 1]) meets [P, P + W): c0..c1 (W > 0, P + W <= T,
// cuts[c] = floor(T c / C)). c0 is the first c with cuts[c + 1] > P, i.e. ceil((P + 1) C / T) - 1,
// and c1 + 1 the first c with cuts[c] > P + W - 1, i.e. ceil((P + W) C / T) (at most C). Both are
// estimated in fp32 and then corrected against the cuts, which makes them exact. `cut(c)` returns
// cuts[c] (a shared-memory table, or cut_at itself).
template <class Cut>
__device__ __forceinline__ void seg_cta_range(Cut cut, long long T, int C, long long P, long long W,
                                              int& c0, int& c1) {
  int c = (int)ceilf((float)(P + 1) * (float)C / (float)T) - 1;
  c = max(0, min(C - 1, c));
  while (c > 0 && cut(c) > P) --c;
  while (c < C - 1 && cut(c + 1) <= P) ++c;
  c0 = c;
  const long long X = P + W - 1;
  c = min((int)ceilf((float)(P + W) * (float)C / (float)T), C) - 1;
  c = max(0, min(C - 1, c));
  while (c < C - 1 && cut(c + 1) <= X) ++c;
  while (c > 0 && cut(c) > X) --c;
  c1 = c;
}

// Per-segment tables in shared memory (any struct with these members): bucket counts and element
// bases of the (sequence, layer), and the CTA's items in (rank, slot) order: item k lies in bucket
// r with it_pref[r] <= k < it_pref[r + 1] and is item it_lo[r] + (k - it_pref[r]) of that bucket.

// Items of bucket r inside the cost range [lo, hi) of a stream: [i0, i1).
template <class Tb>
__device__ __forceinline__ void bucket_range(const Tb& sm, int r, long long lo, long long hi,
                                             long long& i0, long long& i1) {
  const int n = sm.cnt[r];
  if (n == 0) { i0 = i1 = 0; return; }
  const long long n8 = pad8(n), b0 = sm.base[r];
  const long long nit = (n8 + ISL - 1) / ISL;
  // ceil(x / (128 r)) = ceil(ceil(x / 128) / r)
  auto items_before = [&](long long x) -> long long {
    if (x <= 0) return 0;
    const unsigned long long a = ((unsigned long long)x + ISL - 1) / ISL;
    if (a < (1ull << 31)) return (long long)(((uint32_t)a + (uint32_t)r - 1u) / (uint32_t)r);
    return (long long)udiv_small(a + r - 1, (uint32_t)r);
  };
  i0 = items_before(lo - b0);
  i1 = items_before(hi - b0);
  if (i1 > nit) i1 = nit;
  if (i0 > i1) i0 = i1;
}

struct Item {
  int r;    // bucket (rank)
  int it;   // item index inside the bucket
};

template <class Tb>
__device__ __forceinline__ Item item_at(const Tb& sm, int k) {
  int lo = 0, hi = kMaxR + 1;   // it_pref[lo] <= k < it_pref[hi]
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (sm.it_pref[mid] <= k) lo = mid; else hi = mid;
  }
  Item x;
  x.r = lo;
  x.it = sm.it_lo[lo] + (k - sm.it_pref[lo]);
  return x;
}

// Item k after item x = item k - STRIDE (round-robin): STRIDE further in the same bucket, else a
// search.
template <int STRIDE, class Tb>
__device__ __forceinline__ Item next_rr(const Tb& sm, Item x, int k) {
  if (k < sm.it_pref[x.r + 1]) { x.it += STRIDE; return x; }
  return item_at(sm, k);
}

// Rows per chunk of a tile of tl slots, as log2: as many rows as fill one 8 KB stage (32 rows of a
// full 128-slot tile, 64 of a tile of at most 64 slots, all 128 of a tile of at most 32). The
// sparse high-rank buckets end in short tiles; reading them in few chunks keeps their items from
// being a chain of small, latency-bound copies.
__device__ __forceinline__ int chunk_lg(int tl) { return tl > 64 ? 5 : (tl > 32 ? 6 : 7); }
static_assert((ISL * 2) << 5 == STAGE, "a full tile's chunk fills a stage");

// (x + 2) mod n for 0 <= x < n, n >= 1
__device__ __forceinline__ int wrap2(int x, int n) {
  x += 2;
  x -= (x >= n) ? n : 0;
  x -= (x >= n) ? n : 0;
  return x;
}

// Keep the bf16 halves of `w` whose row index (lo half: j, hi half: j + 1) is below r.
__device__ __forceinline__ uint32_t keep_rows(uint32_t w, int j, int r) {
  const uint32_t m = (j < r ? 0x0000FFFFu : 0u) | (j + 1 < r ? 0xFFFF0000u : 0u);
  return w & m;
}

// Per-sequence stream length segW[b] (equal for every head of the sequence; a table outside
// [0, cap] counts as empty) and cost-line start segP[b] of sequence b, whose G segments take
// kSegCost + segW[b] + kSegEnd elements each (an empty sequence takes none); segP[64] = T, the
// line's length. Segment (b, g)'s coefficients start at segP[b] + g (W_b + kSegCost + kSegEnd) +
// kSegCost.
// Called by every thread of the block (B <= 64, two sequences per lane of warp 0 in the scan);
// ends with __syncthreads().
__device__ __forceinline__ void seg_lengths(const int64_t* __restrict__ bucket_base, const Shape& s,
                                            int layer, long long* segW, long long* segP, int tid) {
  for (int b = tid; b < s.B; b += blockDim.x) {
    const long long w = bucket_base[((long long)b * s.L + layer) * (kMaxR + 2) + kMaxR + 1];
    segW[b] = (w >= 0 && w <= s.cap) ? w : 0;
  }
  __syncthreads();
  if (tid < 32) {
    const int lane = tid;
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
  }
  __syncthreads();
}

// The first segment (b, g) whose coefficients end after cost-line position x: the segment whose
// span [segP[b] + g (W_b + kSegCost + kSegEnd), ...) holds x, or the next one when x lies in that
// span's end allowance (b = B when there is none).
__device__ __forceinline__ void segment_at(const long long* segP, const long long* segW, int B, int G,
                                           long long x, int& b, int& g) {
  int lo_b = 0, hi_b = B;
  while (lo_b < hi_b) {
    const int mid = (lo_b + hi_b) >> 1;
    if (segP[mid + 1] > x) hi_b = mid; else lo_b = mid + 1;
  }
  b = lo_b;
  g = 0;
  if (b < B) {   // g = floor(y / w), estimated in fp32 and corrected
    const long long y = x - segP[b], w = segW[b] + kSegCost + kSegEnd;
    g = (int)((float)y / (float)w);
    while (g > 0 && (long long)g * w > y) --g;
    while ((long long)(g + 1) * w <= y) ++g;
    if (y - (long long)g * w >= kSegCost + segW[b]) {   // in the end allowance: the next segment
      if (++g == G) {
        g = 0;
        ++b;
        while (b < B && segW[b] == 0) ++b;
      }
    }
  }
}

// Shared-memory atomic add with acquire-release ordering at CTA scope: the releases of a ring stage
// by several warps (their reads of the stage precede the add) and the refill by the last of them.
__device__ __forceinline__ uint32_t atom_add_acq_rel_cta_smem(uint32_t* p, uint32_t v) {
  uint32_t old;
  asm volatile("atom.acq_rel.cta.shared::cta.add.u32 %0, [%1], %2;\n"
               : "=r"(old) : "r"(smem_addr(p)), "r"(v) : "memory");
  return old;
}

}  // namespace vr
