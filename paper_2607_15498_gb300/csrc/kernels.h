// Host-side launchers of the VarRate kernels (internal; the public ABI is include/varrate.h).
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "common.cuh"

namespace vr {

// ---- step 1: salience
struct SalPlan {
  int n_rb;          // row blocks of 128 window rows per KV head
  int n_chunks;      // token chunks of pass 1
  int64_t chunk;
  int n_chunks2;     // token chunks of pass 2
  int64_t chunk2;
};
SalPlan salience_plan(const Shape& s, int num_sms);
size_t salience_ws_bytes(const Shape& s, int num_sms);
// Returns the number of kernels launched.
int launch_salience(const Shape& s, const void* q_win, const void* k, float* sal_out, void* ws,
                    int32_t* dev_status, int num_sms, cudaStream_t st);
// bf16 tensor-core salience (salience_tc.cu); returns -1 if a TMA descriptor cannot be built
bool salience_tc_supported(const Shape& s);
SalPlan salience_tc_plan(const Shape& s, int num_sms);
size_t salience_tc_ws_bytes(const Shape& s, int num_sms);
int launch_salience_tc(const Shape& s, const void* q_win, const void* k, float* sal_out, void* ws,
                       int32_t* dev_status, int num_sms, cudaStream_t st);

// ---- step 2: allocation
int launch_allocate(const Shape& s, const float* sal, uint8_t* ranks, int64_t* realized,
                    int32_t* dev_status, cudaStream_t st);

// ---- step 3: tables + projection
// Host-side checks of what launch_pack builds before its first launch (bf16: the TMA tensor maps
// of k and v); false means launch_pack would fail.
bool pack_ready(const Shape& s, const void* k, const void* v);
int launch_pack(const Shape& s, const void* k, const void* v, const void* basis_k,
                const void* basis_v, const varrate_packed& out, int32_t* dev_status,
                int num_sms, cudaStream_t st);

// bf16 tensor-core projection (project_tc.cu)
size_t project_tc_smem_bytes();
int launch_project_tc(const Shape& s, const void* k, const void* v, const void* basis_k,
                      const void* basis_v, const varrate_packed& out, int32_t* dev_status,
                      int num_sms, cudaStream_t st);

// ---- step 4: decode attention
// The decode workspace starts with a fixed header used by the bf16 tensor-core kernel: a count of
// its calls and two alternating sets of per-(sequence, KV head) arrival counters (decode_mma.cu);
// the rest of the workspace is scratch that every call writes before it reads.
constexpr int kDecodeMaxSegs = 4096;
constexpr size_t kDecodeCounterBytes = 256 + 2 * (size_t)kDecodeMaxSegs * sizeof(uint32_t);
int decode_splits(const Shape& s, int num_sms);
size_t decode_ws_bytes(const Shape& s, int num_sms);
// bf16 tensor-core decode (decode_mma.cu)
size_t decode_mma_smem_bytes();
size_t decode_mma_part_bytes(const Shape& s, int num_sms);
bool decode_mma_supported(const Shape& s, int n_tail, int num_sms);
int launch_decode_mma(const Shape& s, const varrate_packed& c, const void* basis_k,
                      const void* basis_v, const void* q, int layer, const void* tail_k,
                      const void* tail_v, int n_tail, void* out, int32_t* dev_status,
                      void* header, float* part, int num_sms, cudaStream_t st);
int launch_decode(const Shape& s, const varrate_packed& cache, const void* basis_k,
                  const void* basis_v, const void* q, int layer, const void* tail_k,
                  const void* tail_v, int n_tail, void* out, int32_t* dev_status, void* ws,
                  int num_sms, cudaStream_t st);

// ---- decode of a window of n_q new tokens, bf16 (decode_window.cu): q~ fragments, the coded part
// on the cost line, then merge + causal exact tail + U_V^T per (sequence, KV head). The workspace
// holds the q~ fragments and the per-(segment, CTA) partials, sized for kWindowMaxRows query rows.
constexpr int kWindowMaxRows = 128;   // n_q * group
size_t decode_window_ws_bytes(const Shape& s, int num_sms);
bool decode_window_supported(const Shape& s, int n_q, int n_tail, int num_sms);
int launch_decode_window(const Shape& s, const varrate_packed& c, const void* basis_k, const void* basis_v,
                         const void* q, int n_q, int layer, const void* tail_k, const void* tail_v,
                         int n_tail, void* out, int32_t* dev_status, void* ws, int num_sms,
                         cudaStream_t st);

// ---- quantized coefficients (quant.cu)
int launch_quantize(const Shape& s, const varrate_packed& in, const varrate_qpacked& out,
                    int32_t* dev_status, cudaStream_t st);
// Fused decode on a group-quantized cache (decode_q.cu): the bf16 kernel's work split with the
// codes dequantized in each warp's ring. Workspace: that of the bf16 fused decode (header, then
// the partials). Shapes it does not take run the general kernels on x^ (launch_decode_q,
// decode.cu).
bool decode_q_supported(const Shape& s, int bits, int64_t qcap, int n_tail, int num_sms);
int launch_decode_q_fused(const Shape& s, const varrate_qpacked& cache, const void* basis_k,
                          const void* basis_v, const void* q, int layer, const void* tail_k,
                          const void* tail_v, int n_tail, void* out, int32_t* dev_status, void* header,
                          float* part, int num_sms, cudaStream_t st);
int launch_decode_q(const Shape& s, const varrate_qpacked& cache, const void* basis_k,
                    const void* basis_v, const void* q, int layer, const void* tail_k,
                    const void* tail_v, int n_tail, void* out, void* ws, int num_sms, cudaStream_t st);

// ---- joint codec: nearest-anchor search (anchor_search.cu)
int anchor_count(int64_t N, int stride);
int anchor_count_padded(int64_t N, int stride);   // rounded up to the 256-anchor MMA tile
size_t anchor_search_ws_bytes(const Shape& s, int stride);
bool anchor_search_supported(const Shape& s, int stride, int c);
int launch_anchor_search(const Shape& s, const void* k, const void* v, int stride, int c, int32_t* idx_out,
                         float* dist_out, int32_t* dev_status, void* ws, cudaStream_t st);
bool anchor_residual_supported(const Shape& s, int stride, int c);
int launch_anchor_residual(const Shape& s, const void* k, const void* v, int stride, int c,
                           const int32_t* idx, void* e_out, int32_t* dev_status, cudaStream_t st);

}  // namespace vr
