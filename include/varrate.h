/*
 * varrate.h — C ABI of the GB300 (sm_103a) VarRate hot path.
 *
 * VarRate (arXiv 2607.15498) compresses a KV cache by giving every cached token its own rank in
 * a fixed orthonormal basis: salience from an observation window decides how many basis
 * coefficients each token keeps (Sec. 3.2), the coefficients are the projection onto the basis
 * truncated to that rank (Sec. 3.3, Eq. 5), and decode attention runs directly on the stored
 * coefficients with the query rotated into the basis.
 *
 * Conventions shared by every entry point
 *  - Every tensor argument is a caller-owned DEVICE pointer (CUDA global memory), row-major and
 *    densely packed in the layout stated next to it, and 16-byte aligned (as cudaMalloc and
 *    PyTorch allocations are); a misaligned pointer is VARRATE_ERR_ARG. The library never
 *    allocates or frees device memory. Calls are reentrant and thread-safe. Across calls the
 *    library keeps only per-process values that do not change results: each device's SM count,
 *    the driver entry point that encodes TMA descriptors, whether a kernel's shared-memory opt-in
 *    was made on a device, and the device address of the allocation-free entry point's scratch
 *    array. All are held in atomics.
 *  - `stream` is a cudaStream_t passed as void* (NULL = the legacy default stream). Every call
 *    only enqueues work on `stream` and returns without synchronising.
 *  - The return value reports what the host can see: bad arguments (VARRATE_ERR_ARG), a workspace
 *    that is too small (VARRATE_ERR_WORKSPACE), an unsupported shape (VARRATE_ERR_UNSUPPORTED) or
 *    a failed launch (VARRATE_ERR_CUDA). Nothing is enqueued when the return value is negative.
 *  - Outcomes that depend on the data are written by the kernels to `*dev_status` (one int32 in
 *    device memory). Kernels only raise it: a warning (VARRATE_FLOOR_BINDS) replaces 0, an error
 *    (negative) replaces anything larger. The caller zeroes it before a sequence of calls and
 *    reads it after synchronising.
 *  - dtype VARRATE_BF16: keys, values, queries, bases and packed coefficients are bfloat16 and all
 *    arithmetic accumulates in fp32. dtype VARRATE_F32: all of them are fp32. Salience is fp32 in
 *    both cases.
 *  - Limits: head_dim == 128, 1 <= group <= 8, 1 <= window and group * window <= 256,
 *    window <= n_ctx < 2^31, 1 <= r_min <= head_dim, pool_len odd in [1, 31],
 *    0 < budget_frac <= 1; in bf16, batch * n_layers * n_kv_heads * n_ctx < 2^31 (the K and V
 *    tensors are read through TMA tensor maps with 32-bit row coordinates).
 *
 * Notation: B = batch (sequences), L = n_layers, G = n_kv_heads, H = G * group query heads,
 * d = head_dim, N = n_ctx, w = window. The exact set is the last w tokens [N - w, N) (kept at
 * full rank d); the coded set is [0, N - w).
 */
#ifndef VARRATE_H
#define VARRATE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  VARRATE_OK = 0,
  VARRATE_FLOOR_BINDS = 1,       /* warning: budget below r_min * |C|; every coded token at r_min */
  VARRATE_ERR_ARG = -1,          /* invalid argument (null pointer, size out of range) */
  VARRATE_ERR_WORKSPACE = -2,    /* ws_bytes smaller than varrate_workspace_bytes() */
  VARRATE_ERR_CUDA = -3,         /* a CUDA launch or runtime call failed */
  VARRATE_ERR_TIMEOUT = -4,      /* a bounded device-side wait gave up */
  VARRATE_ERR_UNSUPPORTED = -5,  /* a shape outside the limits above */
  VARRATE_ERR_CORRUPT = -6       /* rank or layout table outside its valid range, or decode
                                    completion words left inconsistent by an earlier call */
} varrate_status;

typedef enum { VARRATE_F32 = 0, VARRATE_BF16 = 1 } varrate_dtype;

/* Allocation mode: salience-driven water-filling (Sec. 3.2, Eq. 4) or the uniform-rank "flat"
 * ablation (every coded token at the same rank; the constant-salience limit of Eq. 4). */
typedef enum { VARRATE_SALIENCE = 0, VARRATE_UNIFORM = 1 } varrate_mode;

/* Problem statement (Sec. 3.1 "Attention and the KV cache", "Budget"; Sec. 4.1). r_max is head_dim. */
typedef struct {
  int32_t n_layers;     /* L */
  int32_t n_kv_heads;   /* G */
  int32_t group;        /* query heads per KV head (GQA) */
  int32_t head_dim;     /* d (must be 128) */
  int64_t n_ctx;        /* N, cached tokens per sequence */
  int32_t batch;        /* B, independent sequences */
  int32_t r_min;        /* rank floor (Eq. 4) */
  double budget_frac;   /* kappa: fraction of the full cache kept (Eq. 3) */
  int32_t window;       /* w = observation window = exact recent window */
  int32_t pool_len;     /* moving-average length of the salience (5 in SnapKV) */
  int32_t dtype;        /* varrate_dtype */
  int32_t mode;         /* varrate_mode */
} varrate_config;

/* Packed variable-rank cache (all device pointers, caller-owned).
 *
 * For each (sequence b, layer l) one bucket table, shared by every KV head and by K and V, groups
 * the tokens by rank. With n_r tokens of rank r and n8_r = n_r rounded up to a multiple of 8:
 *   bucket_base[r_min] = 0, bucket_base[r + 1] = bucket_base[r] + r * n8_r.
 * Bucket r's slots p in [0, n8_r) (token perm-order; p = pos[t]) are cut into tiles of 128 slots,
 * the last one holding tl = n8_r - 128 i slots. Tile i stores r rows of tl elements back to back,
 * one row per coefficient, from element bucket_base[r] + 128 i r; in row j the group of 8 slots
 * g = (p mod 128) / 8 sits at position (g + j) mod (tl / 8). So coefficient j (< r_t) of token t of
 * stream (b, l, g, kv) is at element
 *   coef[(((b * L + l) * G + g) * 2 + kv) * cap_elems + bucket_base[r] + 128 i r + j * tl
 *        + 8 * ((g + j) mod (tl / 8)) + p mod 8],   i = p / 128, r = r_t, p = pos[t].
 * Every tile, and every run of its rows, is one contiguous block (one bulk copy); the rotation keeps
 * a block copied verbatim to shared memory free of bank conflicts. Padding slots p in [n_r, n8_r)
 * hold zeros. kv = 0 is K, 1 is V. */
typedef struct {
  void* coef;             /* [B][L][G][2][cap_elems] dtype */
  int32_t* bucket_count;  /* [B][L][d + 1]  n_r (0 for r < r_min) */
  int64_t* bucket_base;   /* [B][L][d + 2]  element offset of bucket r (0 for r <= r_min) */
  int32_t* perm;          /* [B][L][N] bucketed slot -> token (buckets in increasing rank, stable) */
  int32_t* pos;           /* [B][L][N] token -> position inside its bucket */
  uint8_t* ranks;         /* [B][L][N] rank of every token (exact set at d) */
  int64_t cap_elems;      /* elements per stream, >= varrate_packed_cap_elems() */
} varrate_packed;

/* Quantized packed cache: the coefficients of a varrate_packed cache in group-wise b-bit form
 * (Sec. 3.3, "Composability"; the allocation and bucket tables are unchanged). A group is 32
 * consecutive slots of one coefficient row of a 128-slot tile (one coefficient of up to 32 tokens of
 * equal rank, in bucket order, bucket padding slots included as zeros); its values x map to codes
 *   lo = fp16(min x), step = fp16(min(fl32(max x - lo) / (2^b - 1), 65504)),
 *   code = clip(rint(fl32(fl32(x - lo) / step)), 0, 2^b - 1)   (step == 0: code 0),
 * and back to x^ = fl32(lo + fl32(code * step)). Stream (b, l, g, kv) occupies qcap_bytes bytes from
 * data + (((b * L + l) * G + g) * 2 + kv) * qcap_bytes; bucket r starts at byte qbase[b][l][r]; its
 * tiles follow back to back (the last one pad8(n_r) mod 128 slots), each r rows of
 * qrow(tl) = roundup16(tl * b / 8 + 4 * ceil(tl / 32)) bytes: row j of tile i at
 * qbase[r] + i * r * qrow(128) + j * qrow(tl) holds the codes of slots 0 .. tl - 1 (b = 4: two per
 * byte, the even slot in the low nibble; b = 8: one per byte), then (fp16 lo, fp16 step) of each
 * group of 32 slots, then zeros. Slot p of the tile is bucket position 128 i + p. */
typedef struct {
  uint8_t* data;                /* [B][L][G][2][qcap_bytes] */
  int64_t* qbase;               /* [B][L][d + 2] byte offset of bucket r in a stream */
  const int32_t* bucket_count;  /* [B][L][d + 1] the source cache's bucket counts */
  int32_t bits;                 /* 4 or 8 */
  int64_t qcap_bytes;           /* bytes per stream, >= varrate_qpacked_cap_bytes(cfg, bits) */
} varrate_qpacked;

/* Which call a workspace is sized for. */
typedef enum {
  VARRATE_CALL_SALIENCE = 0,
  VARRATE_CALL_PACK = 1,
  VARRATE_CALL_ENCODE = 2,
  VARRATE_CALL_DECODE = 3,
  VARRATE_CALL_DECODE_WINDOW = 4,
  VARRATE_CALL_DECODE_Q = 5
} varrate_call;

/* Library version (major * 10000 + minor * 100 + patch). */
int32_t varrate_version(void);

/* Readable name of a status code; never NULL. */
const char* varrate_status_string(int32_t status);

/* Validates a configuration against the limits above; VARRATE_OK or the error it would cause. */
varrate_status varrate_check_config(const varrate_config* cfg);

/* Coded budget B_c of one (sequence, layer) in per-head rank units: Eq. 3 (Sec. 3.1) with
 * D -> d and n_ref = w, i.e. floor(budget_frac * (N * d)) - w * d, the product in double.
 * Returns INT64_MIN if cfg is invalid. */
int64_t varrate_coded_budget(const varrate_config* cfg);

/* Upper bound on the packed length of one stream, independent of the data:
 * max(B_c, r_min * (N - w)) + w * d + 7 * sum_{r = r_min..d} r. Returns -1 if cfg is invalid. */
int64_t varrate_packed_cap_elems(const varrate_config* cfg);

/* Bytes of device workspace a call needs (0 is a valid answer). Returns 0 if cfg is invalid. */
size_t varrate_workspace_bytes(const varrate_config* cfg, int32_t which_call);

/* Step 1 — salience (Sec. 3.2, Eq. salience, and SnapKV's length-pool_len moving average).
 *   q_win   [B][L][w][H][d]  queries of the last w tokens (window query q is at position N - w + q)
 *   k       [B][L][G][N][d]  keys; query head h reads KV head h / group
 *   sal_out [B][L][N - w]    fp32: s'_t = pooled mean over the w queries and H heads of the
 *                            causal softmax weight alpha_{q,t} = softmax_{u <= p}(<q,k_u>/sqrt(d))
 *   ws      workspace of at least varrate_workspace_bytes(cfg, VARRATE_CALL_SALIENCE) bytes. */
varrate_status varrate_salience(const varrate_config* cfg, const void* q_win, const void* k,
                                float* sal_out, void* ws, size_t ws_bytes, void* stream);

/* Step 2 — rank allocation (Sec. 3.2, Eq. 4 and Algorithm 1's water level), per (b, l):
 * min-max normalise sal over the coded set in IEEE fp32 (s_hat = (s - min) / (max - min); 1 if
 * max == min or mode is UNIFORM), then rank_t = r_max if x_t >= r_max else max(r_min, floor(x_t))
 * with x_t = fl(fl(lambda * s_hat_t) + r_min), lambda the largest fp32 value whose ranks sum to at
 * most B_c. If r_min * |C| > B_c every coded token gets r_min and *dev_status is raised to
 * VARRATE_FLOOR_BINDS; if B_c >= d * |C| every token gets d. The exact set gets d.
 *   sal          [B][L][N - w] fp32 (e.g. from varrate_salience; ignored in UNIFORM mode, may be NULL)
 *   ranks        [B][L][N] uint8 out
 *   realized_sum [B][L] int64 out: sum of the coded ranks (<= B_c unless FLOOR_BINDS); may be NULL
 * The result is a deterministic function of the fp32 input bits. */
varrate_status varrate_allocate(const varrate_config* cfg, const float* sal, uint8_t* ranks,
                                int64_t* realized_sum, int32_t* dev_status, void* stream);

/* Step 3 — projection and packing (Algorithm 1's projection; Eq. 5 with the anchor mean at 0):
 * builds the bucket tables of `out` from `out->ranks` (which the caller fills, e.g. with
 * varrate_allocate), then writes c_t = U_{g} x_t truncated to r_t for every stream.
 *   k, v        [B][L][G][N][d]
 *   basis_k/_v  [L][G][d][d]  row j = basis vector j (ordered by decreasing singular value)
 * A rank outside [r_min, d] in out->ranks raises VARRATE_ERR_CORRUPT and leaves coef undefined. */
varrate_status varrate_pack(const varrate_config* cfg, const void* k, const void* v,
                            const void* basis_k, const void* basis_v, varrate_packed* out,
                            int32_t* dev_status, void* ws, size_t ws_bytes, void* stream);

/* Steps 1-3 for every (b, l): varrate_salience, varrate_allocate and varrate_pack in one call.
 * sal_out and realized_sum may be NULL (then kept in the workspace). */
varrate_status varrate_encode(const varrate_config* cfg, const void* q_win, const void* k,
                              const void* v, const void* basis_k, const void* basis_v,
                              float* sal_out, varrate_packed* out, int64_t* realized_sum,
                              int32_t* dev_status, void* ws, size_t ws_bytes, void* stream);

/* Step 4 — decode attention on the packed coefficients of one layer (attention of Sec. 3.1 over
 * the cache of Eq. 5, without rebuilding K or V): per query head h of KV head g,
 *   q~ = U_K q;  score_t = q~[:r_t] . c^K_t[:r_t] / sqrt(d);  alpha = softmax over all N tokens
 *   (and the n_tail exact tail tokens);  o = U_V^T sum_t alpha_t c^V_t[:r_t] + sum_tail alpha v.
 *   q       [B][H][d]  one query per head per sequence
 *   tail_k/_v [B][G][n_tail][d] uncompressed tokens appended after the cache (may be NULL if
 *           n_tail == 0); 0 <= n_tail <= 4096 (more is VARRATE_ERR_UNSUPPORTED)
 *   out     [B][H][d]  dtype
 *   ws      at least varrate_workspace_bytes(cfg, VARRATE_CALL_DECODE) bytes, zero-filled before
 *           the first decode call that uses it. Its first 33024 bytes are a header kept by the
 *           fused kernel (below): a count of its calls on this workspace and two alternating sets
 *           of per-(sequence, KV head) arrival counters (at most 4096 pairs). A call counts on the
 *           set of its call count's parity and clears the other set for the next call; the rest of
 *           the workspace is scratch that a call writes before it reads. So one workspace serves
 *           any number of later decode calls (any shape), provided they are ordered on one stream,
 *           and captured launches can be replayed. Calls that overlap on one workspace (different
 *           streams, host threads) race and give wrong results. A call that finds counts left by
 *           an earlier call (an overlapping call, a call that gave up with VARRATE_ERR_TIMEOUT, or
 *           garbage) raises VARRATE_ERR_CORRUPT in *dev_status; its results are not to be trusted,
 *           and the next call on the workspace is clean again without any action by the caller.
 * Kernels: in bf16 with n_tail <= 256, batch <= 64 and batch * n_kv_heads <= 4096 one fused kernel
 * runs. It is launched with programmatic stream serialization and allows the next kernel on
 * `stream` to be scheduled while it runs: a following kernel launched with that attribute must wait
 * for it (griddepcontrol.wait / cudaGridDependencySynchronize) before it reads `out` or
 * `*dev_status`. Kernels launched without the attribute, and every other stream operation, still
 * start only after it has finished. Other shapes (and fp32) run three ordinary kernels (query
 * rotation, split over tokens, combine), launched without that attribute. */
varrate_status varrate_decode_attn(const varrate_config* cfg, const varrate_packed* cache,
                                   const void* basis_k, const void* basis_v, const void* q,
                                   int32_t layer, const void* tail_k, const void* tail_v,
                                   int32_t n_tail, void* out, int32_t* dev_status, void* ws,
                                   size_t ws_bytes, void* stream);

/* Step 4 for a window of new tokens — decode attention of n_q consecutive queries per sequence in
 * one call (the multi-token form of varrate_decode_attn: speculative or chunked decoding). The last
 * n_q tokens of the exact tail are the window; query i (0 <= i < n_q) sits at tail position
 * n_tail - n_q + i and, as in causal attention (Sec. 3.1), attends to every coded token and to the
 * tail tokens 0 .. n_tail - n_q + i. Per query head h of KV head g the result is that of
 * varrate_decode_attn for query i with the tail cut after its own position.
 *   q         [B][n_q][H][d] bf16
 *   tail_k/_v [B][G][n_tail][d] bf16, n_q <= n_tail <= 4096
 *   out       [B][n_q][H][d] bf16
 *   ws        at least varrate_workspace_bytes(cfg, VARRATE_CALL_DECODE_WINDOW) bytes: scratch that
 *             a call writes before it reads (no state is kept between calls; no zero-fill needed).
 *             Calls that overlap on one workspace race.
 * Limits: dtype VARRATE_BF16, batch <= 64, 1 <= n_q and n_q * group <= 128 (VARRATE_ERR_UNSUPPORTED
 * otherwise; n_q > n_tail is VARRATE_ERR_ARG). Three kernels run (query rotation into MMA fragments,
 * the coded part over the persistent grid, merge + causal tail + back-rotation), each launched
 * with programmatic stream serialization; the same rule as for varrate_decode_attn applies to a
 * following kernel launched with that attribute. */
varrate_status varrate_decode_window(const varrate_config* cfg, const varrate_packed* cache,
                                     const void* basis_k, const void* basis_v, const void* q,
                                     int32_t n_q, int32_t layer, const void* tail_k,
                                     const void* tail_v, int32_t n_tail, void* out,
                                     int32_t* dev_status, void* ws, size_t ws_bytes, void* stream);

/* Upper bound on the bytes of one quantized stream for any allocation within the budget:
 * with S = max(B_c, r_min * (N - w)) + w * d, R = sum_{r = r_min..d} r and F = qrow(128):
 * roundup16(ceil(F * (S + 7 R) / 128) + 19 R). Returns -1 if cfg or bits is invalid. */
int64_t varrate_qpacked_cap_bytes(const varrate_config* cfg, int32_t bits);

/* Quantize a bf16 packed cache (every stream of every (sequence, layer)) into `out` (layout above):
 * fills out->qbase from in->bucket_count and writes the codes and group parameters. out->bits is 4
 * or 8 and out->bucket_count must be in->bucket_count. A table that does not fit in->cap_elems or
 * out->qcap_bytes raises VARRATE_ERR_CORRUPT in *dev_status and leaves that (b, l) unwritten.
 * dtype must be VARRATE_BF16 (VARRATE_ERR_UNSUPPORTED otherwise). No workspace. */
varrate_status varrate_quantize(const varrate_config* cfg, const varrate_packed* in,
                                varrate_qpacked* out, int32_t* dev_status, void* stream);

/* Decode attention of one layer on a quantized cache: the same mathematics and arguments as
 * varrate_decode_attn with each stored coefficient c replaced by its dequantized value x^
 * = fl32(lo + fl32(code * step)); 0 <= n_tail <= 4096; dtype VARRATE_BF16 only (queries, bases,
 * tail and output bf16). ws holds at least varrate_workspace_bytes(cfg, VARRATE_CALL_DECODE) bytes
 * (VARRATE_CALL_DECODE_Q asks for the same size), zero-filled before first use like the decode
 * workspace (its header is the same).
 *  - With n_tail <= 256, batch <= 64, batch * n_kv_heads <= 4096 and qcap_bytes a multiple of 16,
 *    one fused kernel runs, with the shape limits and the programmatic stream serialization of the
 *    fused kernel of varrate_decode_attn: it reads the codes and their group parameters (nothing
 *    else of the cache) into shared memory, turns them into x^ rounded to fp16 (one fused
 *    multiply-add from the exact code and the fp16 lo and step) and runs the tensor-core
 *    attention on those fp16 values.
 *  - Otherwise the general kernels (query rotation, split over tokens, combine) decode on x^ in
 *    fp32 directly. */
varrate_status varrate_decode_attn_q(const varrate_config* cfg, const varrate_qpacked* cache,
                                     const void* basis_k, const void* basis_v, const void* q,
                                     int32_t layer, const void* tail_k, const void* tail_v,
                                     int32_t n_tail, void* out, int32_t* dev_status, void* ws,
                                     size_t ws_bytes, void* stream);

/* Decode attention without caller workspace (the paper has no counterpart: this is an interface
 * for callers that cannot allocate device memory, such as a plugin that a host framework hands only
 * input and output pointers, or a serving loop that must not allocate after start-up).
 * Same arguments and results as varrate_decode_attn, minus ws/ws_bytes: the scratch lives in a
 * fixed 4 MiB array in device memory defined by the library (held by every GPU that loads the
 * library until the process exits). Nothing is allocated, by this call or by the library.
 *  - Returns VARRATE_ERR_WORKSPACE when the shape needs more than 4 MiB of decode scratch
 *    (varrate_workspace_bytes(cfg, VARRATE_CALL_DECODE) > 4 MiB).
 *  - The first call on a device looks up the array's device address (once per device, for the
 *    current device) and caches it; make that first call before any stream capture. After
 *    cudaDeviceReset of a device the cached address is stale: do not call this entry point on
 *    that device again in the process.
 *  - All calls share the one array: calls that overlap on the GPU (other streams, other host
 *    threads) race on it and must be serialised by the caller. The array starts zero-filled and
 *    keeps the last call's contents: its header works as described for varrate_decode_attn (after
 *    an overlap or a timed-out call one call reports VARRATE_ERR_CORRUPT and the next is clean
 *    again, which matters here because the caller cannot clear this array), and the rest is
 *    written before it is read. */
varrate_status varrate_decode_attn_noalloc(const varrate_config* cfg, const varrate_packed* cache,
                                           const void* basis_k, const void* basis_v, const void* q,
                                           int32_t layer, const void* tail_k, const void* tail_v,
                                           int32_t n_tail, void* out, int32_t* dev_status,
                                           void* stream);

/* Self-test of the device-side failure path (no counterpart in the paper). Every TMA, tcgen05 and
 * bulk-copy wait in the library is a bounded loop of mbarrier polls; one that gives up raises
 * VARRATE_ERR_TIMEOUT in *dev_status and the kernel returns, leaving the context usable. This call
 * runs one block that waits on an mbarrier phase nothing completes, for 1 <= polls <= 2^24 polls, so
 * it always raises VARRATE_ERR_TIMEOUT in *dev_status (an int32 in device memory, 4-byte aligned);
 * no copy is in flight, so nothing can fault. VARRATE_ERR_ARG for a NULL or misaligned status word
 * or polls out of range. */
varrate_status varrate_selftest_wait_timeout(int32_t* dev_status, uint32_t polls, void* stream);

/* Joint codec, nearest anchors (Sec. 3.1, Eq. 1-2) — the search step of the paper's residual codec.
 * For one (sequence, layer) the joint per-token vector stacks every KV head's key and value,
 *   z_t = [k_t of heads 0..G-1 ; v_t of heads 0..G-1]  (D = 2 G d),
 * the anchors are the tokens a * stride (a = 0 .. n_a - 1, n_a = ceil(N / stride)), and for every
 * token t this call lists the c anchors nearest z_t in squared Euclidean distance,
 *   dist(t, a) = max(0, |z_t|^2 + |z_a|^2 - 2 z_t . z_a),
 * with the bf16 products exact and the sums in fp32 (tensor cores for the dot products), ordered by
 * (distance, a). Tokens that are anchors are listed too (their own anchor comes first).
 *   k, v      [B][L][G][N][d] bf16 (the encode inputs)
 *   stride    1 <= stride <= N;  c: 1 <= c <= 8
 *   idx_out   [B][L][N][c] int32 anchor numbers (the anchor token is a * stride); -1 past n_a
 *   dist_out  [B][L][N][c] fp32 squared distances, +inf past n_a; may be NULL
 *   ws        at least varrate_anchor_search_ws_bytes(cfg, stride) bytes of scratch (the anchors
 *             copied densely, their norms and the token norms), written before it is read.
 * Limits: dtype VARRATE_BF16, batch * n_layers <= 65535, n_kv_heads <= 64 (VARRATE_ERR_UNSUPPORTED
 * otherwise). Only n_layers, n_kv_heads, head_dim, n_ctx, batch and dtype of cfg are used (the
 * rest must still pass varrate_check_config). Two kernels run: one pass over K and V for the
 * norms and the anchor copy, then the tensor-core search. A wait that gives up raises
 * VARRATE_ERR_TIMEOUT in *dev_status and leaves the outputs of that tile unwritten. */
size_t varrate_anchor_search_ws_bytes(const varrate_config* cfg, int32_t stride);
varrate_status varrate_anchor_search(const varrate_config* cfg, const void* k, const void* v,
                                     int32_t stride, int32_t c, int32_t* idx_out, float* dist_out,
                                     int32_t* dev_status, void* ws, size_t ws_bytes, void* stream);

/* Joint codec, residuals (Sec. 3.1, Eq. 2; the third step of Algorithm 1): for every token t,
 *   e_t = z_t - mean of the anchors z_{a * stride} listed for t,
 * with z_t the joint vector of varrate_anchor_search. Arithmetic: the listed anchors' bf16 values
 * summed in list order in fp32, divided (IEEE) by their count, subtracted from z_t in fp32,
 * rounded to bf16.
 *   k, v    [B][L][G][N][d] bf16
 *   idx     [B][L][N][c] int32 anchor lists (e.g. from varrate_anchor_search); entries -1 are skipped
 *   e_out   [B][L][N][2 G d] bf16, in the joint order (head g's key at g d, its value at G d + g d)
 * A list with an entry outside [-1, n_a) or no valid entry raises VARRATE_ERR_CORRUPT in *dev_status
 * and leaves that token's row unwritten. Limits: dtype VARRATE_BF16, 1 <= stride <= N,
 * 1 <= c <= 8, batch * n_layers <= 65535. One kernel, no workspace. */
varrate_status varrate_anchor_residual(const varrate_config* cfg, const void* k, const void* v,
                                       int32_t stride, int32_t c, const int32_t* idx, void* e_out,
                                       int32_t* dev_status, void* stream);

#ifdef __cplusplus
}
#endif
#endif /* VARRATE_H */
