// C ABI of the VarRate hot path (declared in include/varrate.h): argument validation, workspace
// carving and kernel launches. No device memory is allocated here.
#include <algorithm>
#include <atomic>
#include <initializer_list>
#include <math.h>
#include <stdint.h>

#include "common.cuh"
#include "kernels.h"

using vr::Shape;

namespace {

constexpr int32_t kVersion = 1 * 10000 + 0 * 100 + 0;

bool valid_dtype(int32_t d) { return d == VARRATE_F32 || d == VARRATE_BF16; }

varrate_status check(const varrate_config* c) {
  if (c == nullptr) return VARRATE_ERR_ARG;
  if (c->n_layers < 1 || c->n_kv_heads < 1 || c->group < 1 || c->batch < 1 || c->window < 1 ||
      c->n_ctx < 1 || c->r_min < 1 || !valid_dtype(c->dtype) ||
      (c->mode != VARRATE_SALIENCE && c->mode != VARRATE_UNIFORM))
    return VARRATE_ERR_ARG;
  if (!(c->budget_frac > 0.0) || !(c->budget_frac <= 1.0)) return VARRATE_ERR_ARG;
  if (c->window > c->n_ctx || c->n_ctx >= (int64_t(1) << 31)) return VARRATE_ERR_ARG;
  if (c->pool_len < 1 || c->pool_len > 31 || (c->pool_len % 2) == 0) return VARRATE_ERR_ARG;
  if (c->head_dim != vr::kHeadDim) return VARRATE_ERR_UNSUPPORTED;
  if (c->r_min > c->head_dim) return VARRATE_ERR_ARG;
  if (c->group > 8 || (int64_t)c->group * c->window > 256) return VARRATE_ERR_UNSUPPORTED;
  if (c->dtype == VARRATE_BF16 &&
      (int64_t)c->batch * c->n_layers * c->n_kv_heads * c->n_ctx > (int64_t)INT32_MAX)
    return VARRATE_ERR_UNSUPPORTED;
  return VARRATE_OK;
}

int64_t coded_budget(const varrate_config* c) {
  return (int64_t)floor(c->budget_frac * (double)(c->n_ctx * (int64_t)c->head_dim)) -
         (int64_t)c->window * c->head_dim;
}

int64_t cap_elems(const varrate_config* c) {
  const int64_t n_coded = c->n_ctx - c->window;
  int64_t coded = coded_budget(c);
  if ((int64_t)c->r_min * n_coded > coded) coded = (int64_t)c->r_min * n_coded;
  if (coded < 0) coded = 0;
  int64_t pads = 0;
  for (int r = c->r_min; r <= c->head_dim; ++r) pads += 7 * r;
  const int64_t cap = coded + (int64_t)c->window * c->head_dim + pads;
  return (cap + 7) & ~int64_t(7);
}

Shape make_shape(const varrate_config* c, int64_t cap) {
  Shape s;
  s.B = c->batch; s.L = c->n_layers; s.G = c->n_kv_heads; s.grp = c->group;
  s.H = c->n_kv_heads * c->group; s.d = c->head_dim; s.w = c->window; s.pool = c->pool_len;
  s.r_min = c->r_min; s.r_max = c->head_dim; s.dtype = c->dtype; s.mode = c->mode;
  s.N = c->n_ctx; s.n_coded = c->n_ctx - c->window; s.Bc = coded_budget(c); s.cap = cap;
  return s;
}

// SM count of each device, cached per process (a property of the device: every thread that fills
// an entry writes the same value).
int num_sms() {
  static std::atomic<int> cached[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 148;
  int n = cached[dev].load(std::memory_order_relaxed);
  if (n == 0) {
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) n = 148;
    cached[dev].store(n, std::memory_order_relaxed);
  }
  return n;
}


size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

size_t ws_bytes(const varrate_config* c, int32_t which) {
  const Shape s = make_shape(c, cap_elems(c));
  const int sms = num_sms();
  switch (which) {
    case VARRATE_CALL_SALIENCE: return vr::salience_ws_bytes(s, sms);
    case VARRATE_CALL_PACK: return 0;
    case VARRATE_CALL_ENCODE:
      return vr::salience_ws_bytes(s, sms) + align256((size_t)s.B * s.L * s.n_coded * sizeof(float)) +
             align256((size_t)s.B * s.L * sizeof(int64_t));
    case VARRATE_CALL_DECODE: return vr::decode_ws_bytes(s, sms);
    case VARRATE_CALL_DECODE_WINDOW: return vr::decode_window_ws_bytes(s, sms);
    case VARRATE_CALL_DECODE_Q: return vr::decode_ws_bytes(s, sms);
    default: return 0;
  }
}

varrate_status launched() {
  return cudaGetLastError() == cudaSuccess ? VARRATE_OK : VARRATE_ERR_CUDA;
}

// Every device pointer must be 16-byte aligned: the kernels move data with 16-byte vector loads,
// 1-D bulk copies and TMA tiles, which fault on misaligned addresses. NULL passes.
bool aligned16(std::initializer_list<const void*> ps) {
  for (const void* p : ps)
    if ((reinterpret_cast<uintptr_t>(p) & 15u) != 0) return false;
  return true;
}

int64_t qcap_bytes(const varrate_config* c, int bits) {
  const int64_t n_coded = c->n_ctx - c->window;
  int64_t sum = coded_budget(c);
  if ((int64_t)c->r_min * n_coded > sum) sum = (int64_t)c->r_min * n_coded;
  if (sum < 0) sum = 0;
  sum += (int64_t)c->window * c->head_dim;
  int64_t rsum = 0;
  for (int r = c->r_min; r <= c->head_dim; ++r) rsum += r;
  const int64_t full = vr::qrow_bytes(128, bits);
  const int64_t cap = (full * (sum + 7 * rsum) + 127) / 128 + 19 * rsum;
  return (cap + 15) & ~int64_t(15);
}

bool qpacked_ok(const varrate_config* c, const varrate_qpacked* p) {
  return p && p->data && p->qbase && p->bucket_count && (p->bits == 4 || p->bits == 8) &&
         p->qcap_bytes >= qcap_bytes(c, p->bits) && (p->qcap_bytes % 16) == 0 &&
         aligned16({p->data, p->qbase, p->bucket_count});
}

bool packed_ok(const varrate_config* c, const varrate_packed* p) {
  return p && p->coef && p->bucket_count && p->bucket_base && p->perm && p->pos && p->ranks &&
         p->cap_elems >= cap_elems(c) && (p->cap_elems % 8) == 0 &&
         aligned16({p->coef, p->bucket_count, p->bucket_base, p->perm, p->pos, p->ranks});
}

}  // namespace

extern "C" {

int32_t varrate_version(void) { return kVersion; }

const char* varrate_status_string(int32_t st) {
  switch (st) {
    case VARRATE_OK: return "ok";
    case VARRATE_FLOOR_BINDS: return "budget below the rank floor: every coded token at r_min";
    case VARRATE_ERR_ARG: return "invalid argument";
    case VARRATE_ERR_WORKSPACE: return "workspace too small";
    case VARRATE_ERR_CUDA: return "CUDA launch or runtime error";
    case VARRATE_ERR_TIMEOUT: return "bounded device wait timed out";
    case VARRATE_ERR_UNSUPPORTED: return "unsupported shape";
    case VARRATE_ERR_CORRUPT: return "rank or layout table out of range, or decode workspace left inconsistent";
    default: return "unknown status";
  }
}

varrate_status varrate_check_config(const varrate_config* cfg) { return check(cfg); }

int64_t varrate_coded_budget(const varrate_config* cfg) {
  return check(cfg) == VARRATE_OK ? coded_budget(cfg) : INT64_MIN;
}

int64_t varrate_packed_cap_elems(const varrate_config* cfg) {
  return check(cfg) == VARRATE_OK ? cap_elems(cfg) : -1;
}

size_t varrate_workspace_bytes(const varrate_config* cfg, int32_t which_call) {
  return check(cfg) == VARRATE_OK ? ws_bytes(cfg, which_call) : 0;
}

varrate_status varrate_salience(const varrate_config* cfg, const void* q_win, const void* k,
                                float* sal_out, void* ws, size_t ws_bytes_, void* stream) {
  varrate_status st = check(cfg);
  if (st != VARRATE_OK) return st;
  const bool empty = cfg->n_ctx == cfg->window;   // no coded token: nothing to score
  if (!empty && (!q_win || !k || !sal_out)) return VARRATE_ERR_ARG;
  if (cfg->mode == VARRATE_UNIFORM) return VARRATE_ERR_ARG;
  if (!aligned16({q_win, k, sal_out, ws})) return VARRATE_ERR_ARG;
  const size_t need = ws_bytes(cfg, VARRATE_CALL_SALIENCE);
  if (ws_bytes_ < need || (need > 0 && ws == nullptr)) return VARRATE_ERR_WORKSPACE;
  const Shape s = make_shape(cfg, cap_elems(cfg));
  if (vr::launch_salience(s, q_win, k, sal_out, ws, nullptr, num_sms(), (cudaStream_t)stream) < 0)
    return VARRATE_ERR_CUDA;
  return launched();
}

varrate_status varrate_allocate(const varrate_config* cfg, const float* sal, uint8_t* ranks,
                                int64_t* realized_sum, int32_t* dev_status, void* stream) {
  varrate_status st = check(cfg);
  if (st != VARRATE_OK) return st;
  if (!ranks || (cfg->mode == VARRATE_SALIENCE && !sal && cfg->n_ctx > cfg->window))
    return VARRATE_ERR_ARG;
  if (!aligned16({sal, ranks, realized_sum, dev_status})) return VARRATE_ERR_ARG;
  const Shape s = make_shape(cfg, cap_elems(cfg));
  vr::launch_allocate(s, sal, ranks, realized_sum, dev_status, (cudaStream_t)stream);
  return launched();
}

varrate_status varrate_pack(const varrate_config* cfg, const void* k, const void* v,
                            const void* basis_k, const void* basis_v, varrate_packed* out,
                            int32_t* dev_status, void* ws, size_t ws_bytes_, void* stream) {
  (void)ws; (void)ws_bytes_;
  varrate_status st = check(cfg);
  if (st != VARRATE_OK) return st;
  if (!k || !v || !basis_k || !basis_v || !packed_ok(cfg, out)) return VARRATE_ERR_ARG;
  if (!aligned16({k, v, basis_k, basis_v, dev_status})) return VARRATE_ERR_ARG;
  const Shape s = make_shape(cfg, out->cap_elems);
  if (!vr::pack_ready(s, k, v)) return VARRATE_ERR_CUDA;   // before anything is enqueued
  if (vr::launch_pack(s, k, v, basis_k, basis_v, *out, dev_status, num_sms(), (cudaStream_t)stream) < 0)
    return VARRATE_ERR_CUDA;
  return launched();
}

varrate_status varrate_encode(const varrate_config* cfg, const void* q_win, const void* k,
                              const void* v, const void* basis_k, const void* basis_v,
                              float* sal_out, varrate_packed* out, int64_t* realized_sum,
                              int32_t* dev_status, void* ws, size_t ws_bytes_, void* stream) {
  varrate_status st = check(cfg);
  if (st != VARRATE_OK) return st;
  if (!k || !v || !basis_k || !basis_v || !packed_ok(cfg, out)) return VARRATE_ERR_ARG;
  if (cfg->mode == VARRATE_SALIENCE && !q_win && cfg->n_ctx > cfg->window) return VARRATE_ERR_ARG;
  if (!aligned16({q_win, k, v, basis_k, basis_v, sal_out, realized_sum, dev_status, ws}))
    return VARRATE_ERR_ARG;
  const size_t need = ws_bytes(cfg, VARRATE_CALL_ENCODE);
  if (ws_bytes_ < need || ws == nullptr) return VARRATE_ERR_WORKSPACE;
  const Shape s = make_shape(cfg, out->cap_elems);
  if (!vr::pack_ready(s, k, v)) return VARRATE_ERR_CUDA;   // before anything is enqueued
  const int sms = num_sms();
  cudaStream_t cs = (cudaStream_t)stream;
  char* w = static_cast<char*>(ws);
  const size_t sal_ws = vr::salience_ws_bytes(s, sms);
  float* sal = sal_out ? sal_out : reinterpret_cast<float*>(w + sal_ws);
  int64_t* realized = realized_sum
      ? realized_sum
      : reinterpret_cast<int64_t*>(w + sal_ws + align256((size_t)s.B * s.L * s.n_coded * sizeof(float)));
  if (cfg->mode == VARRATE_SALIENCE && vr::launch_salience(s, q_win, k, sal, w, dev_status, sms, cs) < 0)
    return VARRATE_ERR_CUDA;
  vr::launch_allocate(s, sal, out->ranks, realized, dev_status, cs);
  if (vr::launch_pack(s, k, v, basis_k, basis_v, *out, dev_status, sms, cs) < 0) return VARRATE_ERR_CUDA;
  return launched();
}

varrate_status varrate_decode_attn(const varrate_config* cfg, const varrate_packed* cache,
                                   const void* basis_k, const void* basis_v, const void* q,
                                   int32_t layer, const void* tail_k, const void* tail_v,
                                   int32_t n_tail, void* out, int32_t* dev_status, void* ws,
                                   size_t ws_bytes_, void* stream) {
  varrate_status st = check(cfg);
  if (st != VARRATE_OK) return st;
  if (!packed_ok(cfg, cache) || !basis_k || !basis_v || !q || !out) return VARRATE_ERR_ARG;
  if (layer < 0 || layer >= cfg->n_layers || n_tail < 0) return VARRATE_ERR_ARG;
  if (n_tail > 4096) return VARRATE_ERR_UNSUPPORTED;
  if (n_tail > 0 && (!tail_k || !tail_v)) return VARRATE_ERR_ARG;
  if (!aligned16({basis_k, basis_v, q, tail_k, tail_v, out, dev_status, ws})) return VARRATE_ERR_ARG;
  const size_t need = ws_bytes(cfg, VARRATE_CALL_DECODE);
  if (ws_bytes_ < need || ws == nullptr) return VARRATE_ERR_WORKSPACE;
  const Shape s = make_shape(cfg, cache->cap_elems);
  if (vr::launch_decode(s, *cache, basis_k, basis_v, q, layer, tail_k, tail_v, n_tail, out, dev_status,
                        ws, num_sms(), (cudaStream_t)stream) < 0)
    return VARRATE_ERR_CUDA;
  return launched();
}

varrate_status varrate_decode_window(const varrate_config* cfg, const varrate_packed* cache,
                                     const void* basis_k, const void* basis_v, const void* q,
                                     int32_t n_q, int32_t layer, const void* tail_k,
                                     const void* tail_v, int32_t n_tail, void* out,
                                     int32_t* dev_status, void* ws, size_t ws_bytes_, void* stream) {
  varrate_status st = check(cfg);
  if (st != VARRATE_OK) return st;
  if (cfg->dtype != VARRATE_BF16) return VARRATE_ERR_UNSUPPORTED;
  if (!packed_ok(cfg, cache) || !basis_k || !basis_v || !q || !out || !tail_k || !tail_v)
    return VARRATE_ERR_ARG;
  if (layer < 0 || layer >= cfg->n_layers || n_q < 1 || n_tail < n_q) return VARRATE_ERR_ARG;
  if (n_tail > 4096) return VARRATE_ERR_UNSUPPORTED;
  if (!aligned16({basis_k, basis_v, q, tail_k, tail_v, out, dev_status, ws})) return VARRATE_ERR_ARG;
  const Shape s = make_shape(cfg, cache->cap_elems);
  if (!vr::decode_window_supported(s, n_q, n_tail, num_sms())) return VARRATE_ERR_UNSUPPORTED;
  const size_t need = ws_bytes(cfg, VARRATE_CALL_DECODE_WINDOW);
  if (ws_bytes_ < need || ws == nullptr) return VARRATE_ERR_WORKSPACE;
  if (vr::launch_decode_window(s, *cache, basis_k, basis_v, q, n_q, layer, tail_k, tail_v, n_tail, out,
                               dev_status, ws, num_sms(), (cudaStream_t)stream) < 0)
    return VARRATE_ERR_CUDA;
  return launched();
}

int64_t varrate_qpacked_cap_bytes(const varrate_config* cfg, int32_t bits) {
  if (check(cfg) != VARRATE_OK || (bits != 4 && bits != 8)) return -1;
  return qcap_bytes(cfg, bits);
}

varrate_status varrate_quantize(const varrate_config* cfg, const varrate_packed* in,
                                varrate_qpacked* out, int32_t* dev_status, void* stream) {
  varrate_status st = check(cfg);
  if (st != VARRATE_OK) return st;
  if (cfg->dtype != VARRATE_BF16) return VARRATE_ERR_UNSUPPORTED;
  if (!packed_ok(cfg, in) || !qpacked_ok(cfg, out) || out->bucket_count != in->bucket_count)
    return VARRATE_ERR_ARG;
  if (!aligned16({dev_status})) return VARRATE_ERR_ARG;
  const Shape s = make_shape(cfg, in->cap_elems);
  if ((int64_t)s.B * s.L > 65535) return VARRATE_ERR_UNSUPPORTED;   // grid.y of the quantize kernel
  vr::launch_quantize(s, *in, *out, dev_status, (cudaStream_t)stream);
  return launched();
}

varrate_status varrate_decode_attn_q(const varrate_config* cfg, const varrate_qpacked* cache,
                                     const void* basis_k, const void* basis_v, const void* q,
                                     int32_t layer, const void* tail_k, const void* tail_v,
                                     int32_t n_tail, void* out, int32_t* dev_status, void* ws,
                                     size_t ws_bytes_, void* stream) {
  varrate_status st = check(cfg);
  if (st != VARRATE_OK) return st;
  if (cfg->dtype != VARRATE_BF16) return VARRATE_ERR_UNSUPPORTED;
  if (!qpacked_ok(cfg, cache) || !basis_k || !basis_v || !q || !out) return VARRATE_ERR_ARG;
  if (layer < 0 || layer >= cfg->n_layers || n_tail < 0) return VARRATE_ERR_ARG;
  if (n_tail > 4096) return VARRATE_ERR_UNSUPPORTED;
  if (n_tail > 0 && (!tail_k || !tail_v)) return VARRATE_ERR_ARG;
  if (!aligned16({basis_k, basis_v, q, tail_k, tail_v, out, dev_status, ws})) return VARRATE_ERR_ARG;
  const size_t need = ws_bytes(cfg, VARRATE_CALL_DECODE);
  if (ws_bytes_ < need || ws == nullptr) return VARRATE_ERR_WORKSPACE;
  const Shape s = make_shape(cfg, cap_elems(cfg));
  const int sms = num_sms();
  if (vr::decode_q_supported(s, cache->bits, cache->qcap_bytes, n_tail, sms) && aligned16({cache->data})) {
    char* w = static_cast<char*>(ws);
    if (vr::launch_decode_q_fused(s, *cache, basis_k, basis_v, q, layer, tail_k, tail_v, n_tail, out, dev_status,
                                  w, reinterpret_cast<float*>(w + vr::kDecodeCounterBytes), sms,
                                  (cudaStream_t)stream) < 0)
      return VARRATE_ERR_CUDA;
    return launched();
  }
  vr::launch_decode_q(s, *cache, basis_k, basis_v, q, layer, tail_k, tail_v, n_tail, out, ws, sms,
                      (cudaStream_t)stream);
  return launched();
}

size_t varrate_anchor_search_ws_bytes(const varrate_config* cfg, int32_t stride) {
  if (check(cfg) != VARRATE_OK || stride < 1 || stride > cfg->n_ctx) return 0;
  return vr::anchor_search_ws_bytes(make_shape(cfg, cap_elems(cfg)), stride);
}

varrate_status varrate_anchor_search(const varrate_config* cfg, const void* k, const void* v,
                                     int32_t stride, int32_t c, int32_t* idx_out, float* dist_out,
                                     int32_t* dev_status, void* ws, size_t ws_bytes_, void* stream) {
  varrate_status st = check(cfg);
  if (st != VARRATE_OK) return st;
  if (cfg->dtype != VARRATE_BF16) return VARRATE_ERR_UNSUPPORTED;
  if (!k || !v || !idx_out || stride < 1 || stride > cfg->n_ctx || c < 1) return VARRATE_ERR_ARG;
  if (!aligned16({k, v, idx_out, dist_out, dev_status, ws})) return VARRATE_ERR_ARG;
  const Shape s = make_shape(cfg, cap_elems(cfg));
  if (!vr::anchor_search_supported(s, stride, c)) return VARRATE_ERR_UNSUPPORTED;
  const size_t need = vr::anchor_search_ws_bytes(s, stride);
  if (ws_bytes_ < need || ws == nullptr) return VARRATE_ERR_WORKSPACE;
  if (vr::launch_anchor_search(s, k, v, stride, c, idx_out, dist_out, dev_status, ws,
                               (cudaStream_t)stream) < 0)
    return VARRATE_ERR_CUDA;
  return launched();
}

varrate_status varrate_anchor_residual(const varrate_config* cfg, const void* k, const void* v,
                                       int32_t stride, int32_t c, const int32_t* idx, void* e_out,
                                       int32_t* dev_status, void* stream) {
  varrate_status st = check(cfg);
  if (st != VARRATE_OK) return st;
  if (cfg->dtype != VARRATE_BF16) return VARRATE_ERR_UNSUPPORTED;
  if (!k || !v || !idx || !e_out || stride < 1 || stride > cfg->n_ctx || c < 1) return VARRATE_ERR_ARG;
  if (!aligned16({k, v, idx, e_out, dev_status})) return VARRATE_ERR_ARG;
  const Shape s = make_shape(cfg, cap_elems(cfg));
  if (!vr::anchor_residual_supported(s, stride, c)) return VARRATE_ERR_UNSUPPORTED;
  vr::launch_anchor_residual(s, k, v, stride, c, idx, e_out, dev_status, (cudaStream_t)stream);
  return launched();
}

}  // extern "C"
