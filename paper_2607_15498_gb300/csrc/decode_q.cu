// Step 4 on a group-quantized cache (Sec. 3.3, "Composability": the stored coefficients are
// quantized without changing the allocation) — the fused tensor-core decode of decode_mma.cu with
// the coefficients dequantized inside each warp's ring, so a layer call reads the b-bit codes from
// HBM (31.5 % of the bf16 footprint at 4 bits, 56.5 % at 8) and nothing else of the cache.
//
// Same work split, cost line, online softmax, merge and combine as the bf16 kernel (the shared
// parts are in decode_parts.cuh). What differs:
//  - The cost line is measured in bytes of the quantized K stream (qbase), its allowances scaled
//    from the bf16 ones by the bytes of a 128-slot row (qrow(128) per 128 elements), and an item of
//    rank r spans r * qrow(128) bytes.
//  - A chunk is a run of quantized rows of one tile (qrow(tl) bytes each: the codes, then (fp16 lo,
//    fp16 step) per 32-slot group), one 1-D bulk copy into a 4 KB ring stage. Once it lands, the
//    warp expands it, one row per lane, into its own 8 KB staging buffer as fp16 rows laid out like
//    the bf16 packed layout (8-slot group g of row j at position (g + j) mod (tl / 8); at 4 bits the
//    slots inside a group in the order 0 4 1 5 2 6 3 7, see expand8), refills the stage at once and
//    computes from the staging rows with the bf16 kernel's fragment code.
//  - Expansion in fp16 half2 arithmetic: a code becomes the fp16 value 1024 + code by a byte
//    permute and a mask (the exponent of 1024 put above it), 1024 is subtracted exactly, and
//    code * step + lo is one fused multiply-add rounded once to fp16 (the format's lo and step are
//    fp16 already); x^ = lo + code * step of the format is therefore held to within an fp16
//    rounding, finer than the bf16 rounding of the bf16 path.
//  - The tensor-core tiles are fp16 (mma m16n8k16 f16): q~ split hi + lo in fp16, the softmax
//    weights P in fp16 scaled by 2^kPShift (weights down to 2^-31 of the running max stay normal
//    numbers; the partials carry max - kPShift as their reference, so nothing downstream changes).
#include <atomic>

#include "common.cuh"
#include "decode_common.cuh"
#include "decode_parts.cuh"
#include "kernels.h"

namespace vr {

namespace {

constexpr int kPShift = 7;     // P in fp16 as 2^(score - max + kPShift) <= 2^(kSlack + kPShift)
static_assert(kSlack + kPShift <= 15, "scaled weights stay below the fp16 range");

// Bytes of a full 128-slot quantized row, and the cost-line allowances in bytes of the quantized
// K stream (the bf16 allowances, in elements, times the bytes per element of a full row).
template <int BITS> struct QLine {
  static constexpr long long row = ((128 * BITS / 8 + 4 * 4) + 15) & ~15;   // qrow(128)
  // ring stage: the largest chunk (4 bits: 32 rows x 80, 64 x 48 or 128 x 32 bytes; 8 bits:
  // 32 rows x 144 or x 80, 64 x 48)
  static constexpr int stage = BITS == 4 ? 4096 : 4608;
  static constexpr long long seg_cost = kSegCost * row / ISL;
  static constexpr long long seg_end = kSegEnd * row / ISL;
};
static_assert(QLine<4>::row == 80 && QLine<8>::row == 144, "quantized row sizes");

// Rows per chunk (log2): the bf16 kernel's chunking at 4 bits (32 rows of a full tile, 64 of one of
// at most 64 slots, 128 of one of at most 32); at 8 bits 32 rows of any tile over 32 slots and 64
// below, so that a chunk fits a stage and its expansion the 8 KB staging buffer.
__device__ __forceinline__ int chunk_lg_q(int tl, int bits) {
  return bits == 4 ? chunk_lg(tl) : (tl > 32 ? 5 : 6);
}

// Items of bucket r inside the byte range [lo, hi) of a quantized stream: [i0, i1). Item i starts
// at qbase[r] + i * r * qrow(128), so the items starting before x are ceil(x / (r * qrow(128))).
template <int BITS>
__device__ __forceinline__ void bucket_range_q(const SegSmem& sm, int r, long long lo, long long hi,
                                               long long& i0, long long& i1) {
  const int n = sm.cnt[r];
  if (n == 0) { i0 = i1 = 0; return; }
  const long long nit = (pad8(n) + ISL - 1) / ISL, b0 = sm.base[r];
  auto items_before = [&](long long x) -> long long {
    if (x <= 0) return 0;
    const unsigned long long a = ((unsigned long long)x + QLine<BITS>::row - 1) / QLine<BITS>::row;
    if (a < (1ull << 31)) return (long long)(((uint32_t)a + (uint32_t)r - 1u) / (uint32_t)r);
    return (long long)udiv_small(a + r - 1, (uint32_t)r);
  };
  i0 = items_before(lo - b0);
  i1 = items_before(hi - b0);
  if (i1 > nit) i1 = nit;
  if (i0 > i1) i0 = i1;
}

// D(16x8, fp32) += A(16x16, fp16, row) * B(16x8, fp16, col)
__device__ __forceinline__ void mma_f16_16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm("mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
      "{%8,%9}, {%0,%1,%2,%3};\n"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
__device__ __forceinline__ uint32_t pack_f16(float lo, float hi) {
  __half2 v = __floats2half2_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}
// Two floats as fp16 hi parts and fp16 residuals: x ~ hi + lo to ~2^-22 relative.
__device__ __forceinline__ void split_f16(float x0, float x1, uint32_t& hi, uint32_t& lo) {
  __half2 h = __floats2half2_rn(x0, x1);
  const float2 hf = __half22float2(h);
  __half2 l = __floats2half2_rn(x0 - hf.x, x1 - hf.y);
  hi = *reinterpret_cast<uint32_t*>(&h);
  lo = *reinterpret_cast<uint32_t*>(&l);
}

// Score-MMA B fragments of q~ in fp16 (hi + lo) for every 16-row chunk, one uint4 per lane.
__device__ __noinline__ void build_qfrag_f16(SegSmem& sm, int tid) {
  for (int i = tid; i < (kHeadDim / 16) * 32; i += NW * 32) {
    const int jc = i / 32, lane = i % 32, g8 = lane >> 2, c = lane & 3;
    const int j = jc * 16 + 2 * c;
    uint32_t h0, l0, h1, l1;
    split_f16(sm.qt[g8][j], sm.qt[g8][j + 1], h0, l0);
    split_f16(sm.qt[g8][j + 8], sm.qt[g8][j + 9], h1, l1);
    sm.qfrag[jc][lane][0] = h0;
    sm.qfrag[jc][lane][1] = h1;
    sm.qfrag[jc][lane][2] = l0;
    sm.qfrag[jc][lane][3] = l1;
  }
}

// Issue the next chunk of this warp's stream into `stage`: consecutive quantized rows of one tile
// are contiguous, so one bulk copy moves the chunk (qrow is a multiple of 16 bytes, and so is every
// tile and bucket start). Returns false (and issues nothing) when the stream is exhausted.
template <int BITS>
__device__ __forceinline__ bool issue_chunk_q(Prod& p, const SegSmem& sm, const uint8_t* cK, const uint8_t* cV,
                                              uint32_t stage_addr, uint64_t* bar, int total, int lane,
                                              uint64_t policy) {
  if (p.k >= total) return false;
  const int r = p.item.r;
  const long long n8 = pad8(sm.cnt[r]);
  const long long t0 = (long long)p.item.it * ISL;            // first slot of the tile
  const int tl = (int)min((long long)ISL, n8 - t0);             // slots in the tile (multiple of 8)
  const int lgc = chunk_lg_q(tl, BITS);
  const int j0 = p.jc << lgc;
  const int rows = min(1 << lgc, r - j0);
  const int qrow = qrow_bytes(tl, BITS);
  if (lane == 0) {
    const uint32_t bytes = (uint32_t)(rows * qrow);
    mbar_arrive_expect_tx(bar, bytes);
    fence_proxy_async_smem();  // the generic reads above precede the async write
    bulk_g2s_hint(stage_addr, (p.phase ? cV : cK) + sm.base[r] + (long long)p.item.it * r * QLine<BITS>::row +
                                  (long long)j0 * qrow, bytes, bar, policy);
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

__device__ __forceinline__ uint4 ld_shared_v4(uint32_t a) {
  uint4 v;
  asm volatile("ld.shared.v4.u32 {%0,%1,%2,%3}, [%4];\n" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(a));
  return v;
}
__device__ __forceinline__ uint32_t ld_shared_u32(uint32_t a) {
  uint32_t v;
  asm volatile("ld.shared.u32 %0, [%1];\n" : "=r"(v) : "r"(a));
  return v;
}
__device__ __forceinline__ void st_shared_v4(uint32_t a, uint4 v) {
  asm volatile("st.shared.v4.u32 [%0], {%1,%2,%3,%4};\n" ::"r"(a), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w) : "memory");
}

// Eight codes (one 8-slot group) -> eight fp16 values lo + code * step, as four half2. A code c
// becomes the fp16 number 1024 + c (0x6400 | c, exact for c < 1024). At 8 bits half2 p holds slots
// 2p, 2p + 1; at 4 bits it holds slots p and p + 4 (nibbles p and p + 4 of the word, one mask
// apiece), so within each group the staged order of slots is 0 4 1 5 2 6 3 7. Nothing depends on
// the order of slots inside a tile except the mask of padding slots, which maps it back.
__device__ __forceinline__ uint4 expand8(uint32_t w0, uint32_t w1, __half2 lo2, __half2 st2, int bits) {
  const __half2 k1024 = __halves2half2(__ushort_as_half(0x6400), __ushort_as_half(0x6400));
  uint32_t t[4];
  if (bits == 4) {   // nibble e holds slot e
#pragma unroll
    for (int p = 0; p < 4; ++p) t[p] = ((w0 >> (4 * p)) & 0x000F000Fu) | 0x64006400u;
  } else {           // byte e of (w0, w1) holds slot e
    t[0] = __byte_perm(w0, 0x64646464u, 0x4140);
    t[1] = __byte_perm(w0, 0x64646464u, 0x4342);
    t[2] = __byte_perm(w1, 0x64646464u, 0x4140);
    t[3] = __byte_perm(w1, 0x64646464u, 0x4342);
  }
  uint32_t o[4];
#pragma unroll
  for (int p = 0; p < 4; ++p) {
    const __half2 code = __hsub2(*reinterpret_cast<const __half2*>(&t[p]), k1024);
    const __half2 x = __hfma2(code, st2, lo2);
    o[p] = *reinterpret_cast<const uint32_t*>(&x);
  }
  return make_uint4(o[0], o[1], o[2], o[3]);
}

// Expand `rows` staged quantized rows (tile rows j0 .., tl slots) into fp16 rows at `dst` in the
// packed layout's order (group g of tile row j at position (g + j) mod (tl / 8)). Lane l takes rows
// l, l + 32, ...; a full 4-bit row is five 16-byte loads (codes, then the four (lo, step) pairs)
// and sixteen 16-byte stores, whose banks the row stride (80 bytes) and the rotation spread.
template <int BITS>
__device__ __forceinline__ void dequant_chunk(uint32_t src, uint32_t dst, int rows, int j0, int tl, int lane) {
  const int ng = tl >> 3, qrow = qrow_bytes(tl, BITS), pbase = tl * BITS / 8;
  if (tl == ISL) {   // warp-uniform: full tile, 16-byte loads of four groups' codes at a time
    for (int jr = lane; jr < rows; jr += 32) {
      const uint32_t row = src + jr * qrow, orow = dst + jr * (ISL * 2);
      const int j = j0 + jr;
      const uint4 pr = ld_shared_v4(row + pbase);   // (lo, step) of slot groups 0..3 of 32
#pragma unroll
      for (int q = 0; q < 4; ++q) {   // 32 slots: four 8-slot groups
        const uint32_t pq = q == 0 ? pr.x : q == 1 ? pr.y : q == 2 ? pr.z : pr.w;
        const __half2 ph = *reinterpret_cast<const __half2*>(&pq);
        const __half2 lo2 = __low2half2(ph), st2 = __high2half2(ph);
        uint32_t w[8];
        if (BITS == 4) {
          const uint4 c4 = ld_shared_v4(row + 16 * q);
          w[0] = c4.x; w[1] = c4.y; w[2] = c4.z; w[3] = c4.w;
        } else {
          const uint4 a = ld_shared_v4(row + 32 * q), b = ld_shared_v4(row + 32 * q + 16);
          w[0] = a.x; w[1] = a.y; w[2] = a.z; w[3] = a.w; w[4] = b.x; w[5] = b.y; w[6] = b.z; w[7] = b.w;
        }
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int gi = 4 * q + e;
          const uint4 v = BITS == 4 ? expand8(w[e], 0u, lo2, st2, 4) : expand8(w[2 * e], w[2 * e + 1], lo2, st2, 8);
          st_shared_v4(orow + 16 * ((gi + j) & 15), v);
        }
      }
    }
  } else {           // a short tile: group by group
    for (int jr = lane; jr < rows; jr += 32) {
      const uint32_t row = src + jr * qrow, orow = dst + jr * (tl * 2);
      const int j = j0 + jr;
      for (int gi = 0; gi < ng; ++gi) {
        const uint32_t pq = ld_shared_u32(row + pbase + 4 * (gi >> 2));
        const __half2 ph = *reinterpret_cast<const __half2*>(&pq);
        const __half2 lo2 = __low2half2(ph), st2 = __high2half2(ph);
        const uint32_t w0 = ld_shared_u32(row + (BITS == 4 ? 4 : 8) * gi);
        const uint32_t w1 = BITS == 8 ? ld_shared_u32(row + 8 * gi + 4) : 0u;
        const uint4 v = expand8(w0, w1, lo2, st2, BITS);
        st_shared_v4(orow + 16 * ((gi + j) % ng), v);
      }
    }
  }
}

template <int BITS>
__global__ void __launch_bounds__(NW * 32, 1)
decode_q_kernel(const uint8_t* __restrict__ qdata, const int32_t* __restrict__ bucket_count,
                  const int64_t* __restrict__ bucket_base, const __nv_bfloat16* __restrict__ basis_k,
                  const __nv_bfloat16* __restrict__ basis_v, const __nv_bfloat16* __restrict__ qin,
                  const __nv_bfloat16* __restrict__ tail_k, const __nv_bfloat16* __restrict__ tail_v,
                  int n_tail, __nv_bfloat16* __restrict__ out, float* __restrict__ part,
                  DecodeHeader* __restrict__ hdr, int32_t* __restrict__ dev_status, Shape s,
                  int layer, int64_t qcap) {
  constexpr long long kSegCostQ = QLine<BITS>::seg_cost, kSegEndQ = QLine<BITS>::seg_end;
  extern __shared__ __align__(128) unsigned char smem[];
  constexpr int STQ = QLine<BITS>::stage;
  unsigned char* ring = smem;   // NW * ST * STQ of quantized chunks, then NW * STAGE of fp16 rows
  constexpr int kRing = NW * (ST * STQ + STAGE);
  static_assert(kRing % 16 == 0 && kRing >= NW * ST * STAGE, "SegSmem 16-byte aligned; merge and combine fit");
  SegSmem& sm = *reinterpret_cast<SegSmem*>(smem + kRing);
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
    segW[b] = (w >= 0 && w <= qcap) ? w : 0;
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
    const long long v0 = (e0 < s.B && segW[e0]) ? (segW[e0] + kSegCostQ + kSegEndQ) * s.G : 0;
    const long long v1 = (e1 < s.B && segW[e1]) ? (segW[e1] + kSegCostQ + kSegEndQ) * s.G : 0;
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
      const long long x = lo_g - segP[b], w = segW[b] + kSegCostQ + kSegEndQ;
      g = (int)((float)x / (float)w);
      while (g > 0 && (long long)g * w > x) --g;
      while ((long long)(g + 1) * w <= x) ++g;
    }
  }
  auto seg_start = [&](int bb, int gg) { return segP[bb] + gg * (segW[bb] + kSegCostQ + kSegEndQ) + kSegCostQ; };
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
        if (r >= s.r_min && r <= s.r_max) bucket_range_q<BITS>(sm, r, lo, hi, i0, i1);
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
      const uint8_t* cK = qdata + ((bl * s.G + g) * 2) * qcap;
      const uint8_t* cV = cK + qcap;
      const uint32_t ring_w = smem_addr(ring) + warp * ST * STQ;
      const uint32_t stg_w = smem_addr(ring) + NW * ST * STQ + warp * STAGE;   // this warp's fp16 rows
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
        if (issue_chunk_q<BITS>(pr, sm, cK, cV, ring_w + ((n_issued + i) % ST) * STQ,
                        &bars[(n_issued + i) % ST], total, lane, policy)) ++n_pending;
      int c0, c1;   // the CTAs that share this segment (their partials are merged by the last one)
      seg_cta_range([&](int i) { return cuts[i]; }, T, C, P, W, c0, c1);
      __syncwarp();
      if (warp < kHeadDim / 16) rot_compute(sm, rr, s.grp, warp, lane);
      __syncthreads();
      build_qfrag_f16(sm, tid);
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
        if (issue_chunk_q<BITS>(pr, sm, cK, cV, ring_w + ((n_issued + ST - 1) % ST) * STQ,
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
        const int lgc = chunk_lg_q(tl, BITS);           // same chunking as the producer
        const int nj = (r + (1 << lgc) - 1) >> lgc;
        float sc[ISL / 16][4];
#pragma unroll
        for (int t = 0; t < ISL / 16; ++t) sc[t][0] = sc[t][1] = sc[t][2] = sc[t][3] = 0.f;

        // ---- K chunks: scores (rows >= r masked in the q~ fragment)
        for (int jc = 0; jc < nj; ++jc) {
          if (!wait_chunk()) break;
          const int j0 = jc << lgc, j1 = min(r, j0 + (1 << lgc));
          dequant_chunk<BITS>(ring_w + (n_issued % ST) * STQ, stg_w, j1 - j0, j0, tl, lane);
          __syncwarp();
          next_chunk();   // the stage is free once its rows are dequantized: refill it now
          const uint32_t st_addr = stg_w;
          const int m = lane >> 3, r8 = lane & 7;
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
            for (int mt = 0; mt < ISL / 16; ++mt) mma_f16_16816(sc[mt], a[mt], qf.x, qf.y);
#pragma unroll
            for (int mt = 0; mt < ISL / 16; ++mt) mma_f16_16816(sc[mt], a[mt], qf.z, qf.w);
          }
          __syncwarp();   // every lane has read the staged rows before the next chunk replaces them
        }
        if (timed_out) break;

        // ---- online softmax over the item's slots (heads 2c, 2c+1 per lane)
        float mloc[2] = {-INFINITY, -INFINITY};
        const bool full_item = n_real >= ISL;           // warp-uniform: no slot to mask
#pragma unroll
        for (int mt = 0; mt < ISL / 16; ++mt) {
          if (!full_item) {
            // stored position g8 of an 8-slot group holds slot g8 (8 bits) or g8 / 2 + 4 (g8 % 2) (4 bits)
            const int s0 = mt * 16 + (BITS == 4 ? (g8 >> 1) + 4 * (g8 & 1) : g8);
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
        const float Mr[2] = {Mx[0] - kPShift, Mx[1] - kPShift};   // weights scaled by 2^kPShift
        uint32_t pb[ISL / 16][2];   // per slot tile: b0, b1 of P^T (bf16)
#pragma unroll
        for (int mt = 0; mt < ISL / 16; ++mt) {
          const float p0 = fast_exp2(sc[mt][0] - Mr[0]), p1 = fast_exp2(sc[mt][1] - Mr[1]);
          const float p2 = fast_exp2(sc[mt][2] - Mr[0]), p3 = fast_exp2(sc[mt][3] - Mr[1]);
          lsum[0] += p0 + p2;
          lsum[1] += p1 + p3;
          pb[mt][0] = movmatrix_trans(pack_f16(p0, p1));
          pb[mt][1] = movmatrix_trans(pack_f16(p2, p3));
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
              __syncwarp();   // (jt > 0) the previous chunk's staged rows have been read
              if (!wait_chunk()) { ok = false; break; }
              j0 = jt * 16;
              dequant_chunk<BITS>(ring_w + (n_issued % ST) * STQ, stg_w, min(r - j0, 1 << lgc), j0, tl, lane);
              __syncwarp();
              next_chunk();
              st_addr = stg_w;
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
              mma_f16_16816(oacc[jt], a, pb[kt][0], pb[kt][1]);
              mma_f16_16816(t1, b, pb[kt + 1][0], pb[kt + 1][1]);
            }
#pragma unroll
            for (int e = 0; e < 4; ++e) oacc[jt][e] += t1[e];
          }
          (void)ok;
          __syncwarp();   // the staged rows are read before the next item's first chunk
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
        mg.M[warp][2 * c] = Mx[0] - kPShift; mg.M[warp][2 * c + 1] = Mx[1] - kPShift;
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

size_t decode_q_smem_bytes(int bits) {
  const int stq = bits == 4 ? QLine<4>::stage : QLine<8>::stage;
  return (size_t)NW * (ST * stq + STAGE) + sizeof(SegSmem);
}

bool decode_q_supported(const Shape& s, int bits, int64_t qcap, int n_tail, int num_sms) {
  const long long cost = bits == 4 ? QLine<4>::seg_cost + QLine<4>::seg_end : QLine<8>::seg_cost + QLine<8>::seg_end;
  const unsigned long long line = (unsigned long long)s.B * s.G * ((unsigned long long)qcap + (unsigned long long)cost);
  return s.dtype == VARRATE_BF16 && (bits == 4 || bits == 8) && qcap > 0 && qcap % 16 == 0 && s.B <= 64 &&
         (long long)s.B * s.G <= kDecodeMaxSegs && n_tail <= kMaxTailFused && num_sms >= 1 &&
         num_sms <= kMaxCtas && line <= (1ull << 62) / (unsigned long long)num_sms;
}

int launch_decode_q_fused(const Shape& s, const varrate_qpacked& c, const void* basis_k, const void* basis_v,
                          const void* q, int layer, const void* tail_k, const void* tail_v, int n_tail, void* out,
                          int32_t* dev_status, void* header, float* part, int num_sms, cudaStream_t st) {
  const size_t smem = decode_q_smem_bytes(c.bits);
  auto kern = c.bits == 4 ? decode_q_kernel<4> : decode_q_kernel<8>;
  static std::atomic<int> smem_set[2][64];   // the opt-in is per device and per instantiation
  const int bi = c.bits == 4 ? 0 : 1;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64 ||
      smem_set[bi][dev].load(std::memory_order_acquire) == 0) {
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess)
      return -1;
    if (dev >= 0 && dev < 64) smem_set[bi][dev].store(1, std::memory_order_release);
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
  cudaLaunchKernelEx(&lc, kern, (const uint8_t*)c.data, (const int32_t*)c.bucket_count, (const int64_t*)c.qbase,
                     (const __nv_bfloat16*)basis_k, (const __nv_bfloat16*)basis_v, (const __nv_bfloat16*)q,
                     (const __nv_bfloat16*)tail_k, (const __nv_bfloat16*)tail_v, n_tail, (__nv_bfloat16*)out, part,
                     reinterpret_cast<DecodeHeader*>(header), dev_status, s, layer, (int64_t)c.qcap_bytes);
  return 1;
}

}  // namespace vr
