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

// grid (2 G, B L), 256 threads: one CTA per stream (b, l, g, kv); warp w quantizes coefficient rows
// w, w + 8, ... of the stream, the rows enumerated bucket by bucket, tile by tile.
template <int BITS>
__global__ void __launch_bounds__(256)
quantize_kernel(const __nv_bfloat16* __restrict__ coef, const int32_t* __restrict__ bucket_count,
                const int64_t* __restrict__ bucket_base, const int64_t* __restrict__ qbase,
                uint8_t* __restrict__ qdata, int32_t* __restrict__ dev_status, Shape s, int64_t qcap) {
  __shared__ int cnt[kMaxR + 1];
  __shared__ long long base[kMaxR + 2];
  __shared__ long long qb[kMaxR + 2];
  __shared__ long long rows_pre[kMaxR + 2];   // rows of the buckets before r (r rows per tile)
  const int kv = blockIdx.x & 1, g = blockIdx.x >> 1;
  const int64_t bl = blockIdx.y;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  for (int r = tid; r <= kMaxR + 1; r += blockDim.x) {
    if (r <= kMaxR) cnt[r] = bucket_count[bl * (kMaxR + 1) + r];
    base[r] = bucket_base[bl * (kMaxR + 2) + r];
    qb[r] = qbase[bl * (kMaxR + 2) + r];
  }
  __syncthreads();
  if (tid == 0) {
    long long acc = 0;
    for (int r = 0; r <= kMaxR; ++r) {
      rows_pre[r] = acc;
      if (r >= s.r_min && r <= s.r_max) acc += (long long)r * ((pad8(cnt[r]) + 127) / 128);
    }
    rows_pre[kMaxR + 1] = acc;
  }
  __syncthreads();
  // a table that does not fit the buffers (corrupt ranks upstream) is skipped
  if (base[kMaxR + 1] > s.cap || qb[kMaxR + 1] > qcap) {
    if (tid == 0) raise_status(dev_status, VARRATE_ERR_CORRUPT);
    return;
  }
  const int64_t stream = (bl * s.G + g) * 2 + kv;
  const __nv_bfloat16* src = coef + stream * s.cap;
  uint8_t* dst = qdata + stream * qcap;
  constexpr float kQmax = (float)((1 << BITS) - 1);
  const long long total = rows_pre[kMaxR + 1];
  for (long long R = warp; R < total; R += blockDim.x / 32) {
    int lo_r = 0, hi_r = kMaxR + 1;   // rows_pre[lo_r] <= R < rows_pre[hi_r]
    while (hi_r - lo_r > 1) {
      const int mid = (lo_r + hi_r) >> 1;
      if (rows_pre[mid] <= R) lo_r = mid; else hi_r = mid;
    }
    const int r = lo_r;
    const long long k = R - rows_pre[r];
    const long long i = k / r;
    const int j = (int)(k - i * r);
    const long long n8 = pad8(cnt[r]);
    const int tl = (int)min(128ll, n8 - 128 * i);
    const int ng = tl >> 3;
    // bf16 row j of tile i: 8-slot group gp at position (gp + j) mod ng
    const __nv_bfloat16* row = src + base[r] + 128 * i * r + (long long)j * tl;
    const int p0 = lane * 4;                  // this lane's 4 slots (one half of an 8-slot group)
    const bool on = p0 < tl;
    float x[4] = {0.f, 0.f, 0.f, 0.f};
    if (on) {
      const int gp = p0 >> 3;
      const uint2 u = *reinterpret_cast<const uint2*>(row + 8 * ((gp + j) % ng) + (p0 & 7));
      x[0] = __uint_as_float(u.x << 16); x[1] = __uint_as_float(u.x & 0xffff0000u);
      x[2] = __uint_as_float(u.y << 16); x[3] = __uint_as_float(u.y & 0xffff0000u);
    }
    float mn = on ? fminf(fminf(x[0], x[1]), fminf(x[2], x[3])) : INFINITY;
    float mx = on ? fmaxf(fmaxf(x[0], x[1]), fmaxf(x[2], x[3])) : -INFINITY;
#pragma unroll
    for (int o = 1; o < 8; o <<= 1) {   // the 8 lanes of a 32-slot group
      mn = fminf(mn, __shfl_xor_sync(0xffffffffu, mn, o));
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    }
    const __half lo = __float2half_rn(mn);
    const float lo32 = __half2float(lo);
    // a range beyond the fp16 range saturates the step at the largest finite fp16
    const __half st = __float2half_rn(fminf(__fdiv_rn(__fsub_rn(mx, lo32), kQmax), 65504.f));
    const float s32 = __half2float(st);
    uint32_t q[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      int c = 0;
      if (s32 != 0.f) c = __float2int_rn(__fdiv_rn(__fsub_rn(x[e], lo32), s32));
      q[e] = (uint32_t)min(max(c, 0), (int)kQmax);
    }
    uint8_t* qrow = dst + qb[r] + i * (long long)r * qrow_bytes(128, BITS) + (long long)j * qrow_bytes(tl, BITS);
    if (on) {
      if (BITS == 4) {
        const uint16_t w = (uint16_t)(q[0] | (q[1] << 4) | (q[2] << 8) | (q[3] << 12));
        *reinterpret_cast<uint16_t*>(qrow + (p0 >> 1)) = w;
      } else {
        *reinterpret_cast<uint32_t*>(qrow + p0) = q[0] | (q[1] << 8) | (q[2] << 16) | (q[3] << 24);
      }
      if ((lane & 7) == 0) {
        __half2 par = __halves2half2(lo, st);
        *reinterpret_cast<__half2*>(qrow + tl * BITS / 8 + 4 * (p0 / kGroup)) = par;
      }
    }
    // zero padding of the row to its 16-byte size
    const int raw = tl * BITS / 8 + 4 * ((tl + kGroup - 1) / kGroup);
    if (lane < qrow_bytes(tl, BITS) - raw) qrow[raw + lane] = 0;
    __syncwarp();
  }
}

}  // namespace

int launch_quantize(const Shape& s, const varrate_packed& in, const varrate_qpacked& out,
                    int32_t* dev_status, cudaStream_t st) {
  const int64_t pairs = (int64_t)s.B * s.L;
  qtables_kernel<<<(unsigned)((pairs + 127) / 128), 128, 0, st>>>(in.bucket_count, out.qbase, s, out.bits);
  const dim3 grid(2 * s.G, (unsigned)pairs);
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
