// Step 4 — decode attention on the packed coefficients of one layer (attention of Sec. 3.1 on the
// cache of Eq. 5, never rebuilding K or V).
//
// For query head h of KV head g:  q~ = U_K q * log2(e)/sqrt(d);  score_t = q~[:r_t] . c^K_t[:r_t];
// o = U_V^T (sum_t 2^(score_t - m) c^V_t[:r_t]) / sum_t 2^(score_t - m)   (+ exact tail tokens).
//
// decode_rotate  q~ for every head (fp32 workspace).
// decode_split   grid (S, G, B), 8 warps. The coded elements of the (b, l, g) stream are split
//                into S contiguous cost ranges; a warp item is one 128-slot tile of a rank bucket
//                (8 slots per lane on 16 lanes, one 16-byte load per coefficient row, addressed
//                through the packed layout's coef_offset). Scores: 8 slots x GP heads per lane, no cross-lane work. Value rows: every
//                lane forms GP x RG partial sums (GP heads x RG rows, GP * RG = 32) and one
//                31-shuffle transpose-reduction leaves lane i with the full sum of pair i, so each
//                lane owns 128 / RG output coordinates. Online softmax per warp; warps then merge
//                in shared memory and write one (max, sum, o~[128]) partial per head.
// decode_combine merges the S partials (and the exact tail), rotates back with U_V^T, writes out.
#include "common.cuh"
#include "kernels.h"

namespace vr {

namespace {

constexpr int kMaxR = kHeadDim;
constexpr int kWarps = 8;
constexpr int kItem = 128;        // slots per warp item: one tile of the packed layout
constexpr int kMaxTail = 4096;

// Raw 8-element row fragment: bf16 -> one uint4, fp32 -> two float4.
template <typename T> struct Frag;
template <> struct Frag<__nv_bfloat16> {
  uint4 u;
  __device__ __forceinline__ void load(const __nv_bfloat16* p) { u = __ldcs(reinterpret_cast<const uint4*>(p)); }
  __device__ __forceinline__ void zero() { u = make_uint4(0, 0, 0, 0); }
  __device__ __forceinline__ float get(int i) const {
    const uint32_t w = (i < 2) ? u.x : (i < 4) ? u.y : (i < 6) ? u.z : u.w;
    return (i & 1) ? __uint_as_float(w & 0xffff0000u) : __uint_as_float(w << 16);
  }
};
template <> struct Frag<float> {
  float4 a, b;
  __device__ __forceinline__ void load(const float* p) {
    a = __ldcs(reinterpret_cast<const float4*>(p));
    b = __ldcs(reinterpret_cast<const float4*>(p) + 1);
  }
  __device__ __forceinline__ void zero() { a = b = make_float4(0.f, 0.f, 0.f, 0.f); }
  __device__ __forceinline__ float get(int i) const {
    switch (i) { case 0: return a.x; case 1: return a.y; case 2: return a.z; case 3: return a.w;
                 case 4: return b.x; case 5: return b.y; case 6: return b.z; default: return b.w; }
  }
};

// Quantized 8-slot row fragment (group-wise b-bit codes, varrate_qpacked layout): the raw codes of
// slots p0 .. p0 + 7 of one coefficient row (one 32-slot group) and the group's (offset, step);
// get(i) dequantizes slot p0 + i as fl32(lo + fl32(code * step)).
template <int BITS> struct QFrag {
  uint32_t w0, w1;
  float lo, st;
  __device__ __forceinline__ void zero() { w0 = w1 = 0u; lo = 0.f; st = 0.f; }
  __device__ __forceinline__ void load(const uint8_t* row, int p0, int tl) {
    if (BITS == 4) {
      w0 = __ldcs(reinterpret_cast<const unsigned int*>(row + (p0 >> 1)));
      w1 = 0u;
    } else {
      const uint2 u = __ldcs(reinterpret_cast<const uint2*>(row + p0));
      w0 = u.x; w1 = u.y;
    }
    const __half2 par = *reinterpret_cast<const __half2*>(row + tl * BITS / 8 + 4 * (p0 >> 5));
    lo = __low2float(par);
    st = __high2float(par);
  }
  __device__ __forceinline__ float get(int i) const {
    const uint32_t c = BITS == 4 ? (w0 >> (4 * i)) & 15u : ((i < 4 ? w0 : w1) >> (8 * (i & 3))) & 255u;
    return __fadd_rn(lo, __fmul_rn((float)c, st));
  }
};

// Where the split kernel reads coefficient rows from. DenseSrc: the packed cache of `T` elements
// (bucket offsets from its table). QuantSrc: the quantized cache (bucket element offsets rebuilt
// from the counts, byte offsets from qbase).
template <typename T> struct DenseSrc {
  using F = Frag<T>;
  static constexpr bool kTableBase = true;
  const T* coef;
  const int64_t* bucket_base;
  int64_t stride;   // elements per stream
  const T* cK;
  const T* cV;
  __device__ __forceinline__ void bind(int64_t stream0) { cK = coef + stream0 * stride; cV = cK + stride; }
  __device__ __forceinline__ void load(F& f, int kv, int r, long long b0, long long qb0, long long n8,
                                       long long s0, int j) const {
    (void)qb0;
    f.load((kv ? cV : cK) + b0 + coef_offset(r, n8, s0, j));
  }
};
template <int BITS> struct QuantSrc {
  using F = QFrag<BITS>;
  static constexpr bool kTableBase = false;
  const uint8_t* data;
  const int64_t* qbase;
  int64_t stride;   // bytes per stream
  const uint8_t* qK;
  const uint8_t* qV;
  __device__ __forceinline__ void bind(int64_t stream0) { qK = data + stream0 * stride; qV = qK + stride; }
  __device__ __forceinline__ void load(F& f, int kv, int r, long long b0, long long qb0, long long n8,
                                       long long s0, int j) const {
    (void)b0;
    const long long it = s0 >> 7;
    const int p0 = (int)(s0 & 127);
    const int tl = (int)min(128ll, n8 - (it << 7));
    f.load((kv ? qV : qK) + qb0 + it * r * qrow_bytes(128, BITS) + (long long)j * qrow_bytes(tl, BITS), p0, tl);
  }
};

// v[32] holds partials of 32 (head, row) pairs; afterwards v[0] of lane i is the warp-wide sum of
// pair i (each halving step keeps the half selected by the lane's bit and trades the other).
__device__ __forceinline__ float transpose_reduce32(float (&v)[32]) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int n = 16; n >= 1; n >>= 1) {
    const bool upper = lane & n;
#pragma unroll
    for (int i = 0; i < n; ++i) {
      const float send = upper ? v[i] : v[i + n];
      const float keep = upper ? v[i + n] : v[i];
      v[i] = keep + __shfl_xor_sync(0xffffffffu, send, n);
    }
  }
  return v[0];
}

// grid (G, B), 256 threads: qt[b][h][j] = scale * sum_i U_K[j][i] q[b][h][i].
template <typename T>
__global__ void __launch_bounds__(256)
decode_rotate_kernel(const T* __restrict__ q, const T* __restrict__ basis_k, float* __restrict__ qt,
                     Shape s, int layer) {
  __shared__ float qs[8][kHeadDim];
  const int g = blockIdx.x, b = blockIdx.y;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  for (int i = tid; i < s.grp * kHeadDim; i += blockDim.x)
    qs[i / kHeadDim][i % kHeadDim] = to_f(q[((int64_t)b * s.H + g * s.grp) * kHeadDim + i]);
  __syncthreads();
  const T* U = basis_k + ((int64_t)layer * s.G + g) * kHeadDim * kHeadDim;
  const float scale = kLog2e * rsqrtf((float)kHeadDim);
  for (int j = warp; j < kHeadDim; j += kWarps) {
    float u[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) u[i] = to_f(U[j * kHeadDim + lane * 4 + i]);
    for (int hh = 0; hh < s.grp; ++hh) {
      float acc = 0.f;
#pragma unroll
      for (int i = 0; i < 4; ++i) acc = fmaf(u[i], qs[hh][lane * 4 + i], acc);
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
      if (lane == 0) qt[((int64_t)b * s.H + g * s.grp + hh) * kHeadDim + j] = acc * scale;
    }
  }
}

template <class Src, int GP>
__global__ void __launch_bounds__(256, (GP == 4 || GP == 2) ? 2 : 1)
decode_split_kernel(Src src, const int32_t* __restrict__ bucket_count, const float* __restrict__ qt,
                    float* __restrict__ part, Shape s, int layer, int S, long long table_cap) {
  constexpr int RG = 32 / GP;             // value rows per transpose-reduction
  constexpr int NACC = kHeadDim / RG;     // output coordinates owned per lane
  __shared__ __align__(16) float q_s[kHeadDim][GP];
  __shared__ int cnt[kMaxR + 1];
  __shared__ long long base[kMaxR + 2];
  __shared__ long long qb[kMaxR + 2];   // quantized source: byte offset of each bucket
  __shared__ float wM[kWarps][GP], wL[kWarps][GP];
  __shared__ float wacc[kWarps][GP][kHeadDim];

  const int split = blockIdx.x, g = blockIdx.y, b = blockIdx.z;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int64_t bl = (int64_t)b * s.L + layer;
  for (int r = tid; r <= kMaxR + 1; r += blockDim.x) {
    if (r <= kMaxR) cnt[r] = bucket_count[bl * (kMaxR + 1) + r];
    if constexpr (Src::kTableBase) base[r] = src.bucket_base[bl * (kMaxR + 2) + r];
    else qb[r] = src.qbase[bl * (kMaxR + 2) + r];
  }
  if constexpr (!Src::kTableBase) {   // element offsets of the buckets, as the packed table has them
    __syncthreads();
    if (tid == 0) {
      long long acc = 0;
      for (int r = 0; r <= kMaxR; ++r) {
        base[r] = acc;
        if (r >= s.r_min && r <= s.r_max) acc += (long long)r * pad8(cnt[r]);
      }
      base[kMaxR + 1] = acc;
    }
  }
  for (int i = tid; i < kHeadDim * GP; i += blockDim.x) {
    const int j = i / GP, hh = i % GP;
    q_s[j][hh] = hh < s.grp ? qt[((int64_t)b * s.H + g * s.grp + hh) * kHeadDim + j] : 0.f;
  }
  __syncthreads();

  float M[GP], Ls[GP], acc[NACC];
#pragma unroll
  for (int h = 0; h < GP; ++h) { M[h] = -INFINITY; Ls[h] = 0.f; }
#pragma unroll
  for (int a = 0; a < NACC; ++a) acc[a] = 0.f;

  const long long W = base[kMaxR + 1];
  const bool table_ok = W <= s.cap && (Src::kTableBase || qb[kMaxR + 1] <= table_cap);
  const long long lo = table_ok ? W * split / S : 0, hi = table_ok ? W * (split + 1) / S : 0;
  src.bind((bl * s.G + g) * 2);
  int counter = 0;
  for (int r = s.r_min; r <= s.r_max && table_ok; ++r) {
    const int n = cnt[r];
    if (n == 0) continue;
    const long long n8 = pad8(n), b0 = base[r], unit = (long long)kItem * r;
    const long long nit = (n8 + kItem - 1) / kItem;
    long long i_lo = lo > b0 ? (lo - b0 + unit - 1) / unit : 0;
    long long i_hi = hi > b0 ? (hi - b0 + unit - 1) / unit : 0;
    if (i_hi > nit) i_hi = nit;
    for (long long it = i_lo; it < i_hi; ++it, ++counter) {
      if ((counter % kWarps) != warp) continue;
      const long long s0 = it * kItem + lane * 8;
      const bool lane_ok = lane < kItem / 8 && s0 < n8;   // lanes 16..31 idle: 8 slots per lane
      const long long qb0 = Src::kTableBase ? 0 : qb[r];

      // scores for 8 slots x GP heads
      float sc[GP][8];
#pragma unroll
      for (int h = 0; h < GP; ++h)
#pragma unroll
        for (int i = 0; i < 8; ++i) sc[h][i] = 0.f;
      for (int j0 = 0; j0 < r; j0 += 8) {
        typename Src::F f[8];
#pragma unroll
        for (int jj = 0; jj < 8; ++jj) {
          if (lane_ok && j0 + jj < r) src.load(f[jj], 0, r, b0, qb0, n8, s0, j0 + jj);
          else f[jj].zero();
        }
#pragma unroll
        for (int jj = 0; jj < 8; ++jj) {
          if (j0 + jj < r) {
            float qv[GP];
#pragma unroll
            for (int h = 0; h < GP; ++h) qv[h] = q_s[j0 + jj][h];
#pragma unroll
            for (int i = 0; i < 8; ++i) {
              const float kx = f[jj].get(i);
#pragma unroll
              for (int h = 0; h < GP; ++h) sc[h][i] = fmaf(qv[h], kx, sc[h][i]);
            }
          }
        }
      }
      // online softmax over this item
      float corr[GP];
#pragma unroll
      for (int h = 0; h < GP; ++h) {
        float mloc = -INFINITY;
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          if (!(lane_ok && s0 + i < n)) sc[h][i] = -INFINITY;
          mloc = fmaxf(mloc, sc[h][i]);
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) mloc = fmaxf(mloc, __shfl_xor_sync(0xffffffffu, mloc, o));
        const float nm = fmaxf(M[h], mloc);
        corr[h] = exp2f(M[h] - nm);
        float sum = 0.f;
#pragma unroll
        for (int i = 0; i < 8; ++i) { sc[h][i] = exp2f(sc[h][i] - nm); sum += sc[h][i]; }
        Ls[h] = Ls[h] * corr[h] + sum;
        M[h] = nm;
      }
      float my_corr = corr[0];
#pragma unroll
      for (int h = 1; h < GP; ++h) if (lane / RG == h) my_corr = corr[h];
#pragma unroll
      for (int a = 0; a < NACC; ++a) acc[a] *= my_corr;

      // weighted value rows, RG rows at a time
#pragma unroll
      for (int gi = 0; gi < NACC; ++gi) {
        if (gi * RG >= r) break;
        typename Src::F f[RG];
#pragma unroll
        for (int jj = 0; jj < RG; ++jj) {
          if (lane_ok && gi * RG + jj < r) src.load(f[jj], 1, r, b0, qb0, n8, s0, gi * RG + jj);
          else f[jj].zero();
        }
        float pv[32];
#pragma unroll
        for (int jj = 0; jj < RG; ++jj) {
#pragma unroll
          for (int h = 0; h < GP; ++h) {
            float a2 = 0.f;
#pragma unroll
            for (int i = 0; i < 8; ++i) a2 = fmaf(sc[h][i], f[jj].get(i), a2);
            pv[h * RG + jj] = a2;
          }
        }
        acc[gi] += transpose_reduce32(pv);
      }
    }
  }

  // merge the warps of this CTA
#pragma unroll
  for (int h = 0; h < GP; ++h) {
    float l = Ls[h];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) l += __shfl_xor_sync(0xffffffffu, l, o);
    if (lane == 0) { wM[warp][h] = M[h]; wL[warp][h] = l; }
  }
#pragma unroll
  for (int a = 0; a < NACC; ++a) wacc[warp][lane / RG][a * RG + (lane % RG)] = acc[a];
  __syncthreads();
  float* out = part + (((int64_t)b * s.G + g) * S + split) * GP * (kHeadDim + 2);
  for (int i = tid; i < GP * kHeadDim; i += blockDim.x) {
    const int h = i / kHeadDim, j = i % kHeadDim;
    float mx = -INFINITY;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) mx = fmaxf(mx, wM[w][h]);
    float o = 0.f, l = 0.f;
    if (mx != -INFINITY) {
#pragma unroll
      for (int w = 0; w < kWarps; ++w) {
        const float f = exp2f(wM[w][h] - mx);
        o = fmaf(wacc[w][h][j], f, o);
        l = fmaf(wL[w][h], f, l);
      }
    }
    out[h * (kHeadDim + 2) + j] = o;
    if (j == 0) { out[h * (kHeadDim + 2) + kHeadDim] = mx; out[h * (kHeadDim + 2) + kHeadDim + 1] = l; }
  }
}

// grid (G, B), 128 threads: merge partials and the exact tail, rotate back, normalise.
template <typename T, int GP>
__global__ void __launch_bounds__(128)
decode_combine_kernel(const float* __restrict__ part, const T* __restrict__ q,
                      const T* __restrict__ basis_v, const T* __restrict__ tail_k,
                      const T* __restrict__ tail_v, int n_tail, T* __restrict__ out, Shape s,
                      int layer, int S) {
  __shared__ float ot[kHeadDim];
  __shared__ float tsc[kMaxTail];
  __shared__ float qrow[kHeadDim];
  const int g = blockIdx.x, b = blockIdx.y;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const T* U = basis_v + ((int64_t)layer * s.G + g) * kHeadDim * kHeadDim;
  const float scale = kLog2e * rsqrtf((float)kHeadDim);
  const float* pb = part + ((int64_t)b * s.G + g) * S * GP * (kHeadDim + 2);
  for (int hh = 0; hh < s.grp; ++hh) {
    const int h = g * s.grp + hh;
    __syncthreads();
    qrow[tid] = to_f(q[((int64_t)b * s.H + h) * kHeadDim + tid]);
    __syncthreads();
    // exact tail scores (log2 units)
    float tmax = -INFINITY;
    if (n_tail > 0) {
      const T* tk = tail_k + ((int64_t)b * s.G + g) * n_tail * kHeadDim;
      for (int t = warp; t < n_tail; t += 4) {
        float a = 0.f;
#pragma unroll
        for (int i = 0; i < 4; ++i) a = fmaf(qrow[lane * 4 + i], to_f(tk[(int64_t)t * kHeadDim + lane * 4 + i]), a);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) a += __shfl_xor_sync(0xffffffffu, a, o);
        if (lane == 0) tsc[t] = a * scale;
      }
      __syncthreads();
      for (int t = 0; t < n_tail; ++t) tmax = fmaxf(tmax, tsc[t]);
    }
    float mx = tmax;
    for (int sp = 0; sp < S; ++sp) mx = fmaxf(mx, pb[(sp * GP + hh) * (kHeadDim + 2) + kHeadDim]);
    float l = 0.f, o = 0.f;
    for (int sp = 0; sp < S; ++sp) {
      const float* pp = pb + (sp * GP + hh) * (kHeadDim + 2);
      const float m = pp[kHeadDim];
      if (m == -INFINITY) continue;
      const float f = exp2f(m - mx);
      l = fmaf(pp[kHeadDim + 1], f, l);
      o = fmaf(pp[tid], f, o);
    }
    ot[tid] = o;
    __syncthreads();
    float y = 0.f;
    for (int j = 0; j < kHeadDim; ++j) y = fmaf(to_f(U[j * kHeadDim + tid]), ot[j], y);
    if (n_tail > 0) {
      const T* tv = tail_v + ((int64_t)b * s.G + g) * n_tail * kHeadDim;
      for (int t = 0; t < n_tail; ++t) {
        const float p = exp2f(tsc[t] - mx);
        l += p;
        y = fmaf(p, to_f(tv[(int64_t)t * kHeadDim + tid]), y);
      }
    }
    out[((int64_t)b * s.H + h) * kHeadDim + tid] = from_f<T>(y / l);
  }
}

template <typename T, int GP>
void launch_decode_t(const Shape& s, const varrate_packed& c, const void* basis_k, const void* basis_v,
                     const void* q, int layer, const void* tail_k, const void* tail_v, int n_tail,
                     void* out, float* qt, float* part, int S, cudaStream_t st) {
  decode_rotate_kernel<T><<<dim3(s.G, s.B), 256, 0, st>>>((const T*)q, (const T*)basis_k, qt, s, layer);
  DenseSrc<T> src{(const T*)c.coef, c.bucket_base, s.cap, nullptr, nullptr};
  decode_split_kernel<DenseSrc<T>, GP><<<dim3(S, s.G, s.B), 256, 0, st>>>(src, c.bucket_count, qt, part,
                                                                           s, layer, S, 0);
  decode_combine_kernel<T, GP><<<dim3(s.G, s.B), 128, 0, st>>>(part, (const T*)q, (const T*)basis_v,
                                                               (const T*)tail_k, (const T*)tail_v,
                                                               n_tail, (T*)out, s, layer, S);
}

template <typename T>
void dispatch_gp(int gp, const Shape& s, const varrate_packed& c, const void* bk, const void* bv,
                 const void* q, int layer, const void* tk, const void* tv, int nt, void* out,
                 float* qt, float* part, int S, cudaStream_t st) {
  switch (gp) {
    case 1: launch_decode_t<T, 1>(s, c, bk, bv, q, layer, tk, tv, nt, out, qt, part, S, st); break;
    case 2: launch_decode_t<T, 2>(s, c, bk, bv, q, layer, tk, tv, nt, out, qt, part, S, st); break;
    case 4: launch_decode_t<T, 4>(s, c, bk, bv, q, layer, tk, tv, nt, out, qt, part, S, st); break;
    default: launch_decode_t<T, 8>(s, c, bk, bv, q, layer, tk, tv, nt, out, qt, part, S, st); break;
  }
}

int group_pad(int grp) { return grp <= 1 ? 1 : grp <= 2 ? 2 : grp <= 4 ? 4 : 8; }

template <int GP>
void launch_decode_qt(const Shape& s, const varrate_qpacked& c, const void* basis_k, const void* basis_v,
                      const void* q, int layer, const void* tail_k, const void* tail_v, int n_tail,
                      void* out, float* qt, float* part, int S, cudaStream_t st) {
  using bf = __nv_bfloat16;
  decode_rotate_kernel<bf><<<dim3(s.G, s.B), 256, 0, st>>>((const bf*)q, (const bf*)basis_k, qt, s, layer);
  if (c.bits == 4) {
    QuantSrc<4> src{c.data, c.qbase, c.qcap_bytes, nullptr, nullptr};
    decode_split_kernel<QuantSrc<4>, GP><<<dim3(S, s.G, s.B), 256, 0, st>>>(src, c.bucket_count, qt, part,
                                                                           s, layer, S, c.qcap_bytes);
  } else {
    QuantSrc<8> src{c.data, c.qbase, c.qcap_bytes, nullptr, nullptr};
    decode_split_kernel<QuantSrc<8>, GP><<<dim3(S, s.G, s.B), 256, 0, st>>>(src, c.bucket_count, qt, part,
                                                                           s, layer, S, c.qcap_bytes);
  }
  decode_combine_kernel<bf, GP><<<dim3(s.G, s.B), 128, 0, st>>>(part, (const bf*)q, (const bf*)basis_v,
                                                               (const bf*)tail_k, (const bf*)tail_v,
                                                               n_tail, (bf*)out, s, layer, S);
}

}  // namespace

int decode_splits(const Shape& s, int num_sms) {
  const int64_t units = (int64_t)s.B * s.G;
  int64_t S = (4LL * num_sms + units - 1) / units;
  if (S < 1) S = 1;
  if (S > 128) S = 128;
  return (int)S;
}

size_t decode_ws_bytes(const Shape& s, int num_sms) {
  const int S = decode_splits(s, num_sms);
  size_t a = (size_t)s.B * s.H * kHeadDim * sizeof(float);
  a = (a + 255) & ~size_t(255);
  a += (size_t)s.B * s.G * S * group_pad(s.grp) * (kHeadDim + 2) * sizeof(float);
  const size_t m = decode_mma_part_bytes(s, num_sms);
  if (m > a) a = m;
  return kDecodeCounterBytes + ((a + 255) & ~size_t(255));
}

int launch_decode(const Shape& s, const varrate_packed& cache, const void* basis_k,
                  const void* basis_v, const void* q, int layer, const void* tail_k,
                  const void* tail_v, int n_tail, void* out, int32_t* dev_status, void* ws,
                  int num_sms, cudaStream_t st) {
  void* header = ws;   // completion counting: the first kDecodeCounterBytes of the workspace
  ws = static_cast<char*>(ws) + kDecodeCounterBytes;
  if (decode_mma_supported(s, n_tail, num_sms))
    return launch_decode_mma(s, cache, basis_k, basis_v, q, layer, tail_k, tail_v, n_tail, out,
                             dev_status, header, reinterpret_cast<float*>(ws), num_sms, st);
  const int S = decode_splits(s, num_sms);
  float* qt = reinterpret_cast<float*>(ws);
  size_t a = (size_t)s.B * s.H * kHeadDim * sizeof(float);
  a = (a + 255) & ~size_t(255);
  float* part = reinterpret_cast<float*>(static_cast<char*>(ws) + a);
  const int gp = group_pad(s.grp);
  if (s.dtype == VARRATE_BF16)
    dispatch_gp<__nv_bfloat16>(gp, s, cache, basis_k, basis_v, q, layer, tail_k, tail_v, n_tail, out, qt, part, S, st);
  else
    dispatch_gp<float>(gp, s, cache, basis_k, basis_v, q, layer, tail_k, tail_v, n_tail, out, qt, part, S, st);
  return 3;
}

int launch_decode_q(const Shape& s, const varrate_qpacked& cache, const void* basis_k,
                    const void* basis_v, const void* q, int layer, const void* tail_k,
                    const void* tail_v, int n_tail, void* out, void* ws, int num_sms, cudaStream_t st) {
  ws = static_cast<char*>(ws) + kDecodeCounterBytes;   // same scratch layout as the general path
  const int S = decode_splits(s, num_sms);
  float* qt = reinterpret_cast<float*>(ws);
  size_t a = (size_t)s.B * s.H * kHeadDim * sizeof(float);
  a = (a + 255) & ~size_t(255);
  float* part = reinterpret_cast<float*>(static_cast<char*>(ws) + a);
  switch (group_pad(s.grp)) {
    case 1: launch_decode_qt<1>(s, cache, basis_k, basis_v, q, layer, tail_k, tail_v, n_tail, out, qt, part, S, st); break;
    case 2: launch_decode_qt<2>(s, cache, basis_k, basis_v, q, layer, tail_k, tail_v, n_tail, out, qt, part, S, st); break;
    case 4: launch_decode_qt<4>(s, cache, basis_k, basis_v, q, layer, tail_k, tail_v, n_tail, out, qt, part, S, st); break;
    default: launch_decode_qt<8>(s, cache, basis_k, basis_v, q, layer, tail_k, tail_v, n_tail, out, qt, part, S, st); break;
  }
  return 3;
}

}  // namespace vr
