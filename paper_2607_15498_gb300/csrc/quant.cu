// Group-wise b-bit quantization of the packed coefficients (Sec. 3.3, "Composability": the stored
// coefficients can be quantized without changing the allocation).
//
// Groups: 32 consecutive slots (tokens of one rank, in bucket order) of one coefficient row j of a
// 128-slot tile. Asymmetric min-max with fp16 offset and step:
//   lo = fp16(min), step = fp16(fl32(max - lo) / (2^b - 1)),
//   code = clip(rint(fl32(fl32(x - lo) / step)), 0, 2^b - 1)   (step = 0: code 0),
// every operation an explicitly rounded IEEE fp32 operation, so the codes are a function of the
// stored bf16 coefficients. Quantized stream layout: bucket r at byte qbase[r], its tiles back to
// back, each r rows of qrow(tl) bytes: the tl codes (b = 4: two per byte, the even slot in the low
// nibble; b = 8: one per byte), then (fp16 lo, fp16 step) for each group of 32 slots, then zero
// padding to a multiple of 16 bytes.
#include "common.cuh"
#include "kernels.h"

namespace vr {

namespace {

constexpr int kMaxR = kHeadDim;
constexpr int kGroup = 32;

// qbase per (b, l): one thread per (sequence, layer) (129 buckets, a serial prefix).
__global__ void qtables_kernel(const int32_t* __restrict__ bucket_count, int64_t* __restrict__ qbase,
                               Shape s, int bits) {
  const int64_t bl = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (bl >= (int64_t)s.B * s.L) return;
  const int32_t* cnt = bucket_count + bl * (kMaxR + 1);
  int64_t* qb = qbase + bl * (kMaxR + 2);
  const int64_t full = qrow_bytes(128, bits);
  int64_t acc = 0;
  for (int r = 0; r <= kMaxR; ++r) {
    qb[r] = acc;
    if (r >= s.r_min && r <= s.r_max) {
      const int64_t n8 = pad8(cnt[r]);
      const int64_t last = n8 % 128;
      acc += (int64_t)r * ((n8 / 128) * full + (last ? qrow_bytes((int)last, bits) : 0));
    }
  }
  qb[kMaxR + 1] = acc;
}

// grid (2 G, B L, kQuantSplit), 256 threads: CTA (stream, bl, z) quantizes the z-th share of the
// tiles of stream (b, l, g, kv). A warp takes one tile at a time, two rows per step: lane (lr, gp)
// reads the 8 bf16 coefficients of slot group gp of row 2 jj + lr (stored at position (gp + j) mod
// (tl / 8)), the four lanes of a 32-slot group agree on its min and max by shuffles, and each lane
// writes its 8 codes (one 32-bit word at 4 bits, two at 8 bits); the group's first lane writes
// (lo, step) and the row's padding bytes are zeroed.
constexpr int kQuantSplit = 8;
constexpr int kDeqRows = 8;   // rows per lane whose loads are in flight together

template <int BITS>
__global__ void __launch_bounds__(256)
quantize_kernel(const __nv_bfloat16* __restrict__ coef, const int32_t* __restrict__ bucket_count,
                const int64_t* __restrict__ bucket_base, const int64_t* __restrict__ qbase,
                uint8_t* __restrict__ qdata, int32_t* __restrict__ dev_status, Shape s, int64_t qcap) {
  __shared__ int cnt[kMaxR + 1];
  __shared__ long long base[kMaxR + 2];
  __shared__ long long qb[kMaxR + 2];
  __shared__ int tiles_pre[kMaxR + 2];   // tiles of the buckets before r
  const int kv = blockIdx.x & 1, g = blockIdx.x >> 1, z = blockIdx.z;
  const int64_t bl = blockIdx.y;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  for (int r = tid; r <= kMaxR + 1; r += blockDim.x) {
    if (r <= kMaxR) cnt[r] = bucket_count[bl * (kMaxR + 1) + r];
    base[r] = bucket_base[bl * (kMaxR + 2) + r];
    qb[r] = qbase[bl * (kMaxR + 2) + r];
  }
  __syncthreads();
  if (tid == 0) {
    int tiles = 0;
    for (int r = 0; r <= kMaxR; ++r) {
      tiles_pre[r] = tiles;
      if (r >= s.r_min && r <= s.r_max && cnt[r] > 0) tiles += (int)((pad8(cnt[r]) + 127) / 128);
    }
    tiles_pre[kMaxR + 1] = tiles;
  }
  __syncthreads();
  // a table that does not fit the buffers (corrupt ranks upstream) is skipped
  if (base[kMaxR + 1] > s.cap || qb[kMaxR + 1] > qcap) {
    if (tid == 0 && blockIdx.x == 0 && z == 0) raise_status(dev_status, VARRATE_ERR_CORRUPT);
    return;
  }
  const int64_t stream = (bl * s.G + g) * 2 + kv;
  const __nv_bfloat16* src = coef + stream * s.cap;
  uint8_t* dst = qdata + stream * qcap;
  constexpr float kQmax = (float)((1 << BITS) - 1);
  const int total = tiles_pre[kMaxR + 1];
  const int T0 = (int)((long long)total * z / kQuantSplit), T1 = (int)((long long)total * (z + 1) / kQuantSplit);
  const int lr = lane >> 4, gp = lane & 15;
  for (int T = T0 + warp; T < T1; T += blockDim.x / 32) {
    int lo_r = 0, hi_r = kMaxR + 1;   // tiles_pre[lo_r] <= T < tiles_pre[hi_r]
    while (hi_r - lo_r > 1) {
      const int mid = (lo_r + hi_r) >> 1;
      if (tiles_pre[mid] <= T) lo_r = mid; else hi_r = mid;
    }
    const int r = lo_r;
    const long long i = T - tiles_pre[r];
    const int tl = (int)min(128ll, pad8(cnt[r]) - 128 * i);
    const int ng = tl >> 3;
    const int qrow = qrow_bytes(tl, BITS);
    const int raw = tl * BITS / 8 + 4 * ((tl + kGroup - 1) / kGroup);
    const __nv_bfloat16* stile = src + base[r] + 128 * i * r;
    uint8_t* qtile = dst + qb[r] + i * (long long)r * qrow_bytes(128, BITS);
    const bool on = gp < ng;
    for (int j0 = 0; j0 < r; j0 += 2 * kDeqRows) {
      uint4 x[kDeqRows];
#pragma unroll
      for (int u = 0; u < kDeqRows; ++u) {   // every row's load in flight before the first use
        const int j = j0 + 2 * u + lr;
        if (on && j < r) x[u] = *reinterpret_cast<const uint4*>(stile + (long long)j * tl + 8 * ((gp + j) % ng));
      }
#pragma unroll
      for (int u = 0; u < kDeqRows; ++u) {
        if (j0 + 2 * u >= r) break;   // warp-uniform: no row of this step in either half
        const int j = j0 + 2 * u + lr;
        const bool valid = on && j < r;   // the other half-warp may still have a row: no early exit
        float v[8];
        v[0] = __uint_as_float(x[u].x << 16); v[1] = __uint_as_float(x[u].x & 0xffff0000u);
        v[2] = __uint_as_float(x[u].y << 16); v[3] = __uint_as_float(x[u].y & 0xffff0000u);
        v[4] = __uint_as_float(x[u].z << 16); v[5] = __uint_as_float(x[u].z & 0xffff0000u);
        v[6] = __uint_as_float(x[u].w << 16); v[7] = __uint_as_float(x[u].w & 0xffff0000u);
        float mn = INFINITY, mx = -INFINITY;
        if (valid) {
#pragma unroll
          for (int e = 0; e < 8; ++e) { mn = fminf(mn, v[e]); mx = fmaxf(mx, v[e]); }
        }
        // the four lanes of a 32-slot group (gp = 4 q .. 4 q + 3 of the same half)
        mn = fminf(mn, __shfl_xor_sync(0xffffffffu, mn, 1));
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
        mn = fminf(mn, __shfl_xor_sync(0xffffffffu, mn, 2));
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
        const __half lo = __float2half_rn(mn);
        const float lo32 = __half2float(lo);
        // a range beyond the fp16 range saturates the step at the largest finite fp16
        const __half st = __float2half_rn(fminf(__fdiv_rn(__fsub_rn(mx, lo32), kQmax), 65504.f));
        const float s32 = __half2float(st);
        uint32_t q[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          int cq = 0;
          if (s32 != 0.f) cq = __float2int_rn(__fdiv_rn(__fsub_rn(v[e], lo32), s32));
          q[e] = (uint32_t)min(max(cq, 0), (int)kQmax);
        }
        if (j >= r) continue;
        uint8_t* row = qtile + (long long)j * qrow;
        if (on) {
          if (BITS == 4) {
            uint32_t w = 0;
#pragma unroll
            for (int e = 0; e < 8; ++e) w |= q[e] << (4 * e);
            *reinterpret_cast<uint32_t*>(row + 4 * gp) = w;
          } else {
            *reinterpret_cast<uint2*>(row + 8 * gp) =
                make_uint2(q[0] | (q[1] << 8) | (q[2] << 16) | (q[3] << 24), q[4] | (q[5] << 8) | (q[6] << 16) | (q[7] << 24));
          }
          if ((gp & 3) == 0) *reinterpret_cast<__half2*>(row + tl * BITS / 8 + 4 * (gp >> 2)) = __halves2half2(lo, st);
        }
        if (gp < qrow - raw) row[raw + gp] = 0;   // zero padding of the row to its 16-byte size
      }
    }
  }
}

}  // namespace

int launch_quantize(const Shape& s, const varrate_packed& in, const varrate_qpacked& out,
                    int32_t* dev_status, cudaStream_t st) {
  const int64_t pairs = (int64_t)s.B * s.L;
  qtables_kernel<<<(unsigned)((pairs + 127) / 128), 128, 0, st>>>(in.bucket_count, out.qbase, s, out.bits);
  const dim3 grid(2 * s.G, (unsigned)pairs, kQuantSplit);
  if (out.bits == 4)
    quantize_kernel<4><<<grid, 256, 0, st>>>((const __nv_bfloat16*)in.coef, in.bucket_count,
                                             in.bucket_base, out.qbase, out.data, dev_status, s,
                                             out.qcap_bytes);
  else
    quantize_kernel<8><<<grid, 256, 0, st>>>((const __nv_bfloat16*)in.coef, in.bucket_count,
                                             in.bucket_base, out.qbase, out.data, dev_status, s,
                                             out.qcap_bytes);
  return 2;
}

}  // namespace vr
