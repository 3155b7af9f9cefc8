"""VarRate CPU oracle: TEST INFRASTRUCTURE, not part of the library.

A plain, slow, obviously-correct restatement of the VarRate hot path (arXiv 2607.15498,
"VarRate: Training-Free Variable-Rate KV Cache Compression for Long-Context LLMs") in numpy.
Floating point is fp64 except the normalisation and the rank allocation, which are specified in
IEEE fp32 (separately rounded multiply and add, no FMA) so that an implementation fed the same
salience can reproduce the ranks bit for bit.

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline / reference leg may
import this module. It shares no code with the CUDA library and imports nothing from it.

Readings of the paper taken here (each one is also listed in the design notes):
  * per-head bases: every (layer, KV head, K-or-V) stream has its own d x d orthonormal basis
    (rows ordered by decreasing singular value), and a token has ONE rank r_t per layer shared by
    all KV heads and by K and V (Sec. 3.1 "Joint per-token vector" restricted to head blocks);
  * the residual/anchor codec of Eq. 2 is off (anchor mean 0, e_t = z_t); the exact set is the
    last ``window`` tokens, coded at full rank d;
  * no RoPE: keys are coded in the frame they are given;
  * budget in per-head rank units: B_c = floor(kappa * N * d) - w * d (Eq. 3);
  * integer ranks come from the largest fp32 water level lambda whose allocation does not exceed
    B_c (the paper's rounding overshoots B by < 0.4%; this reading never exceeds it);
  * salience softmax is causal over all tokens up to the query's position; salience is kept for
    the coded set only; the length-5 moving average is zero-padded with divisor 5;
  * decode attention runs on the stored coefficients (Eq. 5 with the query rotated into the basis).
"""
from __future__ import annotations

import math

import numpy as np

# status codes (match the library's public enum values)
OK = 0
FLOOR_BINDS = 1

SALIENCE = 0
UNIFORM = 1

F32_MAX_BITS = 0x7F7FFFFF


# ----------------------------------------------------------------------------- budget (Eq. 3)

def coded_budget(n_ctx: int, head_dim: int, window: int, budget_frac: float) -> int:
    """Coded budget B_c in per-head rank units (Sec. 3.1 "Budget", Eq. 3).

    The paper's B = D (kappa L - n_ref) with D -> d (one head stream) and n_ref = window:
    B_c = floor(kappa * (N d)) - w d, the product taken once in double precision."""
    return int(math.floor(budget_frac * float(n_ctx * head_dim))) - window * head_dim


def packed_cap_elems(n_ctx: int, head_dim: int, window: int, budget_frac: float,
                     r_min: int) -> int:
    """Static upper bound on the packed length of one (sequence, layer, head, K-or-V) stream:
    sum of ranks (at most max(B_c, r_min |C|) + w d) plus up to 7 padding slots per bucket."""
    n_coded = n_ctx - window
    bc = coded_budget(n_ctx, head_dim, window, budget_frac)
    return max(bc, r_min * n_coded, 0) + window * head_dim + 7 * sum(range(r_min, head_dim + 1))


# ----------------------------------------------------------------------- salience (Sec. 3.2)

def salience_raw(q_win: np.ndarray, k: np.ndarray, group: int) -> np.ndarray:
    """SnapKV salience of Sec. 3.2, Eq. (salience), before pooling.

    q_win: [w][H][d] queries of the last w tokens (window query q sits at position N - w + q).
    k:     [G][N][d] keys; query head h reads KV head h // group.
    For every window query and head, alpha = softmax over t <= p of <q, k_t> / sqrt(d) (every
    token up to the query's own position, Sec. 3.1 "Attention and the KV cache"); s_t is the mean of alpha over the
    w queries and H heads. Returns s for the coded set t in [0, N - w), fp64."""
    q_win = np.asarray(q_win, dtype=np.float64)
    k = np.asarray(k, dtype=np.float64)
    w, H, d = q_win.shape
    G, N, _ = k.shape
    assert H == G * group
    pos = N - w + np.arange(w)
    future = np.arange(N)[None, :] > pos[:, None]          # [w][N]
    s = np.zeros(N)
    for h in range(H):
        scores = (q_win[:, h, :] @ k[h // group].T) / math.sqrt(d)   # [w][N]
        scores[future] = -np.inf
        m = scores.max(axis=1, keepdims=True)
        e = np.exp(scores - m)
        alpha = e / e.sum(axis=1, keepdims=True)
        s += alpha.sum(axis=0)
    s /= (w * H)
    return s[: N - w]


def pool(s: np.ndarray, pool_len: int = 5) -> np.ndarray:
    """SnapKV's moving average over adjacent tokens (Sec. 3.2): the mean of the pool_len values
    centred on t, indices outside the coded set counting as 0 (divisor is always pool_len)."""
    s = np.asarray(s, dtype=np.float64)
    half = pool_len // 2
    padded = np.concatenate([np.zeros(half), s, np.zeros(half)])
    out = np.zeros_like(s)
    for i in range(pool_len):
        out += padded[i: i + s.size]
    return out / pool_len


def salience(q_win, k, group, pool_len=5) -> np.ndarray:
    """Pooled salience s'_t (fp64) for the coded set."""
    return pool(salience_raw(q_win, k, group), pool_len)


# ------------------------------------------------------------- normalisation (Sec. 3.2), fp32

def normalize(sal32: np.ndarray, mode: int = SALIENCE) -> np.ndarray:
    """Min-max normalisation over the coded set to s_hat in [0, 1] (Sec. 3.2), in IEEE fp32:
    s_hat = fl(fl(s - min) / fl(max - min)). A constant signal (max == min) and the uniform-rank
    ablation both give s_hat = 1 for every token, the limit in which Eq. 4 collapses to the
    uniform-rank codec."""
    sal32 = np.asarray(sal32, dtype=np.float32)
    if mode == UNIFORM or sal32.size == 0:
        return np.ones(sal32.size, dtype=np.float32)
    mn = sal32.min()
    mx = sal32.max()
    if mx == mn:
        return np.ones(sal32.size, dtype=np.float32)
    num = (sal32 - mn).astype(np.float32)
    den = np.float32(mx - mn)
    return (num / den).astype(np.float32)


# ---------------------------------------------------------- water-filling (Sec. 3.2, Eq. 4)

def bits_to_f32(bits: int) -> np.float32:
    return np.array([bits], dtype=np.uint32).view(np.float32)[0]


def f32_to_bits(x) -> int:
    return int(np.array([x], dtype=np.float32).view(np.uint32)[0])


def rank_at(lam, shat: np.ndarray, r_min: int, r_max: int) -> np.ndarray:
    """Integer rank of every coded token at water level lambda (Eq. 4 with integer ranks):
    x_t = fl(fl(lambda * s_hat_t) + r_min); rank = r_max if x_t >= r_max (or x_t = inf),
    else max(r_min, floor(x_t))."""
    lam = np.float32(lam)
    with np.errstate(over="ignore"):
        prod = (lam * shat).astype(np.float32)
        x = (prod + np.float32(r_min)).astype(np.float32)
    r = np.maximum(np.floor(x), np.float32(r_min))
    r = np.where(x >= np.float32(r_max), np.float32(r_max), r)
    return r.astype(np.int64)


def allocate(shat: np.ndarray, budget: int, r_min: int, r_max: int):
    """Rank allocation of Sec. 3.2 (Eq. 4, Algorithm 1's water level) for the coded set.

    Returns (ranks int64 [|C|], lambda_bits, status, realised_sum).
      * infeasible (r_min |C| > B_c): every token at r_min, status FLOOR_BINDS;
      * full (B_c >= r_max |C|): every token at r_max (kappa = 1 reconstructs exactly);
      * otherwise lambda* = the largest finite fp32 lambda >= 0 with sum_t rank_t(lambda) <= B_c,
        found by bisection over the fp32 bit patterns (the sum is non-decreasing in lambda);
        if even lambda = FLT_MAX fits, lambda* = FLT_MAX and the slack stays unspent.
    """
    shat = np.asarray(shat, dtype=np.float32)
    n = shat.size
    if n == 0:
        return np.zeros(0, dtype=np.int64), 0, OK, 0
    if r_min * n > budget:
        r = np.full(n, r_min, dtype=np.int64)
        return r, 0, FLOOR_BINDS, int(r.sum())
    if budget >= r_max * n:
        r = np.full(n, r_max, dtype=np.int64)
        return r, F32_MAX_BITS, OK, int(r.sum())

    def total(bits):
        return int(rank_at(bits_to_f32(bits), shat, r_min, r_max).sum())

    if total(F32_MAX_BITS) <= budget:
        lo = F32_MAX_BITS
    else:
        lo, hi = 0, F32_MAX_BITS          # total(lo) <= budget < total(hi)
        while hi - lo > 1:
            mid = (lo + hi) // 2
            if total(mid) <= budget:
                lo = mid
            else:
                hi = mid
    r = rank_at(bits_to_f32(lo), shat, r_min, r_max)
    return r, lo, OK, int(r.sum())


def waterfill_continuous(shat: np.ndarray, budget: float, r_min: float, r_max: float,
                         max_iter: int = 10_000) -> np.ndarray:
    """Algorithm 1's clip-and-redistribute recursion in fp64 (continuous ranks), for reference:
    start every coded token at r_min, spread the remaining budget over the unclipped tokens in
    proportion to s_hat, clip those that pass r_max and repeat until none do."""
    shat = np.asarray(shat, dtype=np.float64)
    r = np.full(shat.size, float(r_min))
    active = np.ones(shat.size, dtype=bool)
    for _ in range(max_iter):
        delta = budget - r.sum()
        w = shat[active].sum()
        if w <= 0:
            break
        r[active] += delta * shat[active] / w
        over = active & (r > r_max)
        r[over] = r_max
        active &= ~over
        if not over.any():
            break
    return r


def allocate_layer(sal32: np.ndarray, n_ctx: int, head_dim: int, window: int,
                   budget_frac: float, r_min: int, mode: int = SALIENCE):
    """Ranks of all N tokens of one (sequence, layer): coded tokens from the allocation, the last
    ``window`` tokens (the exact set) at full rank d. Returns (ranks uint8-valued int64 [N],
    status, realised coded sum)."""
    n_coded = n_ctx - window
    bc = coded_budget(n_ctx, head_dim, window, budget_frac)
    shat = normalize(np.asarray(sal32, dtype=np.float32)[:n_coded], mode)
    rc, _, status, total = allocate(shat, bc, r_min, head_dim)
    ranks = np.concatenate([rc, np.full(window, head_dim, dtype=np.int64)])
    return ranks, status, total


# ---------------------------------------------------------------------- packed layout tables

def pack_tables(ranks: np.ndarray, r_min: int, r_max: int):
    """Rank-bucketed layout of one (sequence, layer) (shared by every head and by K and V).

    count[r]  = number of tokens of rank r                               (int32 [r_max + 1])
    base[r]   = element offset of bucket r: base[r_min] = 0,
                base[r + 1] = base[r] + r * pad8(count[r])                (int64 [r_max + 2])
    pos[t]    = number of earlier tokens with the same rank (stable)      (int32 [N])
    perm[s]   = token in bucketed slot s, buckets in rank order           (int32 [N])
    Coefficient j of token t sits at base[r_t] + j * pad8(count[r_t]) + pos[t]."""
    ranks = np.asarray(ranks, dtype=np.int64)
    count = np.zeros(r_max + 1, dtype=np.int64)
    for r in ranks:
        count[r] += 1
    base = np.zeros(r_max + 2, dtype=np.int64)
    for r in range(r_min, r_max + 1):
        base[r + 1] = base[r] + r * ((count[r] + 7) // 8 * 8)
    slot_start = np.zeros(r_max + 2, dtype=np.int64)
    for r in range(r_max + 1):
        slot_start[r + 1] = slot_start[r] + count[r]
    seen = np.zeros(r_max + 1, dtype=np.int64)
    pos = np.zeros(ranks.size, dtype=np.int64)
    perm = np.zeros(ranks.size, dtype=np.int64)
    for t, r in enumerate(ranks):
        pos[t] = seen[r]
        perm[slot_start[r] + seen[r]] = t
        seen[r] += 1
    return count.astype(np.int32), base, pos.astype(np.int32), perm.astype(np.int32)


# ------------------------------------------------------------- projection (Eq. 5, Alg. 1)

def project(x: np.ndarray, basis: np.ndarray) -> np.ndarray:
    """Coefficients c_t = U x_t at full rank (Algorithm 1's projection onto the basis, Eq. 5 with
    the anchor mean at 0). x: [N][d], basis U: [d][d] (row j = basis vector j). fp64 [N][d]."""
    return np.asarray(x, dtype=np.float64) @ np.asarray(basis, dtype=np.float64).T


def truncate(coef: np.ndarray, ranks: np.ndarray) -> np.ndarray:
    """Nested mask m_{t,j} = 1[j < r_t] applied to full coefficients (Eq. 5)."""
    d = coef.shape[-1]
    mask = np.arange(d)[None, :] < np.asarray(ranks)[:, None]
    return np.where(mask, coef, 0.0)


def reconstruct(coef: np.ndarray, ranks: np.ndarray, basis: np.ndarray) -> np.ndarray:
    """z_hat_t = U^T (m_t * c_t) (Eq. 5 with the anchor mean at 0)."""
    return truncate(coef, ranks) @ np.asarray(basis, dtype=np.float64)


def pack_stream(coef: np.ndarray, ranks: np.ndarray, count, base, pos) -> np.ndarray:
    """Lay the truncated coefficients of one stream out in the bucketed layout (pads zero)."""
    r_max = len(count) - 1
    out = np.zeros(int(base[r_max + 1]))
    for t, r in enumerate(np.asarray(ranks)):
        n8 = (int(count[r]) + 7) // 8 * 8
        for j in range(int(r)):
            out[int(base[r]) + j * n8 + int(pos[t])] = coef[t, j]
    return out


def unpack_stream(buf: np.ndarray, ranks: np.ndarray, count, base, pos) -> np.ndarray:
    """Inverse of pack_stream: [N][d] truncated coefficients (zero beyond each rank)."""
    ranks = np.asarray(ranks)
    d = len(count) - 1
    out = np.zeros((ranks.size, d))
    for t, r in enumerate(ranks):
        n8 = (int(count[r]) + 7) // 8 * 8
        for j in range(int(r)):
            out[t, j] = buf[int(base[r]) + j * n8 + int(pos[t])]
    return out


# ---------------------------------------------------------------- decode attention (Eq. 5)

def attention(q: np.ndarray, k: np.ndarray, v: np.ndarray) -> np.ndarray:
    """Plain softmax attention of one query per head (Sec. 3.1): q [H][d], k, v [G][N][d]
    (query head h reads KV head h // (H / G)). fp64 [H][d]."""
    q = np.asarray(q, dtype=np.float64)
    H, d = q.shape
    G = k.shape[0]
    grp = H // G
    out = np.zeros((H, d))
    for h in range(H):
        g = h // grp
        sc = np.asarray(k[g], dtype=np.float64) @ q[h] / math.sqrt(d)
        a = np.exp(sc - sc.max())
        a /= a.sum()
        out[h] = a @ np.asarray(v[g], dtype=np.float64)
    return out


def decode_coef(q, coef_k, coef_v, ranks, basis_k, basis_v, tail_k=None, tail_v=None):
    """Decode attention computed on the coefficients (route i).

    q [H][d]; coef_k, coef_v [G][N][d] full coefficients (truncated here by ranks);
    basis_k, basis_v [G][d][d]; optional tail_k, tail_v [G][n_tail][d] exact tokens appended after
    the cache (the recent window kept exact, Sec. 3.1 "Residual codec"). Per head:
    q~ = U_K q; score_t = q~[:r_t] . c^K_t[:r_t] / sqrt(d) (tail: q . k / sqrt(d)); alpha = softmax
    over all N (+ n_tail) tokens; o = U_V^T sum_t alpha_t (m_t * c^V_t) + sum_tail alpha v.
    Equal to attention over the reconstructed cache because U_K^T is the inverse rotation."""
    q = np.asarray(q, dtype=np.float64)
    H, d = q.shape
    G = coef_k.shape[0]
    grp = H // G
    out = np.zeros((H, d))
    for h in range(H):
        g = h // grp
        uk = np.asarray(basis_k[g], dtype=np.float64)
        uv = np.asarray(basis_v[g], dtype=np.float64)
        qt = uk @ q[h]
        ck = truncate(np.asarray(coef_k[g], dtype=np.float64), ranks)
        cv = truncate(np.asarray(coef_v[g], dtype=np.float64), ranks)
        sc = ck @ qt / math.sqrt(d)
        if tail_k is not None and len(tail_k[g]):
            tk = np.asarray(tail_k[g], dtype=np.float64)
            tv = np.asarray(tail_v[g], dtype=np.float64)
            st = tk @ q[h] / math.sqrt(d)
        else:
            tv = np.zeros((0, d))
            st = np.zeros(0)
        m = max(sc.max(), st.max() if st.size else -np.inf)
        a = np.exp(sc - m)
        at = np.exp(st - m)
        z = a.sum() + at.sum()
        out[h] = (uv.T @ (a @ cv) + at @ tv) / z
    return out


def decode_recon(q, coef_k, coef_v, ranks, basis_k, basis_v, tail_k=None, tail_v=None):
    """Decode attention on the reconstructed cache (route ii): rebuild k_hat, v_hat by Eq. 5,
    append the exact tail tokens and run plain attention (the paper's reconstruct-in-place decode)."""
    G = coef_k.shape[0]
    kh = np.stack([reconstruct(coef_k[g], ranks, basis_k[g]) for g in range(G)])
    vh = np.stack([reconstruct(coef_v[g], ranks, basis_v[g]) for g in range(G)])
    if tail_k is not None:
        kh = np.concatenate([kh, np.asarray(tail_k, dtype=np.float64)], axis=1)
        vh = np.concatenate([vh, np.asarray(tail_v, dtype=np.float64)], axis=1)
    return attention(q, kh, vh)


def decode_window(q, coef_k, coef_v, ranks, basis_k, basis_v, tail_k, tail_v):
    """Decode attention for a window of n_q consecutive new tokens in one call (the multi-query
    form of the exact-tail decode: the recent tokens are kept exact, Sec. 3.1 "Residual codec").

    q [n_q][H][d] are the queries of the last n_q tokens of the exact tail tail_k, tail_v
    [G][n_tail][d] (n_tail >= n_q). Query i sits at tail position n_tail - n_q + i and, as in
    causal attention (Sec. 3.1 "Attention and the KV cache"), attends to every cached token and to
    the tail tokens up to and including its own position. Returns [n_q][H][d]."""
    q = np.asarray(q, dtype=np.float64)
    n_q = q.shape[0]
    n_tail = np.asarray(tail_k).shape[1]
    if n_q > n_tail:
        raise ValueError("every window query is one of the tail tokens")
    out = np.zeros(q.shape)
    for i in range(n_q):
        m = n_tail - n_q + i + 1                    # tail tokens visible to query i
        out[i] = decode_coef(q[i], coef_k, coef_v, ranks, basis_k, basis_v,
                             np.asarray(tail_k)[:, :m], np.asarray(tail_v)[:, :m])
    return out


# --------------------------------------------------------------------------- whole layer

def encode_layer(q_win, k, v, basis_k, basis_v, group, budget_frac, r_min, pool_len=5,
                 mode=SALIENCE):
    """Steps 1-3 for one (sequence, layer): salience -> ranks -> coefficients and tables.
    k, v: [G][N][d]; basis_*: [G][d][d]. Returns a dict with fp32 salience, ranks, status,
    realised coded sum, tables and full fp64 coefficients [G][N][d] for K and V."""
    G, N, d = k.shape
    w = q_win.shape[0]
    sal32 = salience(q_win, k, group, pool_len).astype(np.float32) if mode == SALIENCE \
        else np.zeros(N - w, dtype=np.float32)
    ranks, status, total = allocate_layer(sal32, N, d, w, budget_frac, r_min, mode)
    count, base, pos, perm = pack_tables(ranks, r_min, d)
    ck = np.stack([project(k[g], basis_k[g]) for g in range(G)])
    cv = np.stack([project(v[g], basis_v[g]) for g in range(G)])
    return dict(sal=sal32, ranks=ranks, status=status, total=total, count=count, base=base,
                pos=pos, perm=perm, coef_k=ck, coef_v=cv)


# ------------------------------------------- coefficient quantization (Sec. 3.3, "Composability")

# The paper states that the coefficients c_t can be quantized with standard group-wise b-bit
# quantization without touching the allocation. Reading taken here: a group is 32 consecutive slots
# (tokens of one rank, in bucket order) of one coefficient row j inside a 128-slot tile of the
# packed layout, so a group holds one coefficient of up to 32 tokens of equal rank; quantization is
# asymmetric min-max with the group's offset and step stored in fp16:
#     lo = fp16(min), step = fp16(fl32(max - lo) / (2^b - 1)),
#     code = clip(rint(fl32(fl32(x - lo) / step)), 0, 2^b - 1)   (step = 0: code 0),
#     x^ = fl32(lo + fl32(code * step)).
# Padding slots of a bucket (zeros) belong to the group of their tile like the others.

QGROUP = 32


def qrow_bytes(tl: int, bits: int) -> int:
    """Bytes of one quantized coefficient row of a tile of tl slots: the codes (tl * bits / 8),
    then (fp16 offset, fp16 step) per group of 32 slots, rounded up to 16 bytes."""
    raw = tl * bits // 8 + 4 * ((tl + QGROUP - 1) // QGROUP)
    return (raw + 15) // 16 * 16


def quantize_group(x, bits: int):
    """One group: float32 values -> (uint8 codes, fp16 offset, fp16 step)."""
    x = np.asarray(x, dtype=np.float32)
    qmax = np.float32(2 ** bits - 1)
    lo = np.float16(x.min())
    lo32 = np.float32(lo)
    # a range beyond the fp16 range saturates the step at the largest finite fp16
    step = np.float16(min(np.float32(np.float32(x.max()) - lo32) / qmax, np.float32(65504.0)))
    s32 = np.float32(step)
    if s32 == 0:
        return np.zeros(x.size, dtype=np.uint8), lo, step
    with np.errstate(over="ignore", invalid="ignore"):
        q = np.rint(((x - lo32).astype(np.float32) / s32).astype(np.float32))
    q = np.clip(q, 0, qmax)
    return q.astype(np.uint8), lo, step


def dequantize_group(codes, lo, step):
    """x^ = fl32(lo + fl32(code * step)) (separately rounded multiply and add)."""
    prod = (np.asarray(codes, dtype=np.float32) * np.float32(step)).astype(np.float32)
    return (np.float32(lo) + prod).astype(np.float32)


def qpack_tables(count, r_min: int, r_max: int, bits: int) -> np.ndarray:
    """Byte offset of each rank bucket in a quantized stream (int64 [r_max + 2]): bucket r holds
    its tiles (128 slots; the last one pad8(n_r) mod 128 slots) back to back, r rows each."""
    qbase = np.zeros(r_max + 2, dtype=np.int64)
    full = qrow_bytes(128, bits)
    for r in range(r_min, r_max + 1):
        n8 = (int(count[r]) + 7) // 8 * 8
        last = n8 % 128
        qbase[r + 1] = qbase[r] + r * ((n8 // 128) * full + (qrow_bytes(last, bits) if last else 0))
    return qbase


def qpacked_cap_bytes(n_ctx: int, head_dim: int, window: int, budget_frac: float, r_min: int,
                      bits: int) -> int:
    """Static upper bound on the bytes of one quantized stream for any allocation: with
    S = max(B_c, r_min |C|) + w d rank units (+ 7 padding slots per bucket and row), a full-tile
    row costs qrow_bytes(128) / 128 per unit and a short last tile at most 19 bytes per row more
    than its share (group parameters of a partial group, 16-byte rounding)."""
    n_coded = n_ctx - window
    s = max(coded_budget(n_ctx, head_dim, window, budget_frac), r_min * n_coded, 0) \
        + window * head_dim
    rsum = sum(range(r_min, head_dim + 1))
    full = qrow_bytes(128, bits)
    cap = (full * (s + 7 * rsum) + 127) // 128 + 19 * rsum
    return (cap + 15) // 16 * 16


def quantize_coefficients(coef, ranks, count, pos, bits: int):
    """Quantize one stream given its per-token coefficients coef [N][d] (float32: the stored values)
    and the bucket tables. Returns (codes [N][d] uint8 (0 beyond each rank), lo [N][d] fp16 and
    step [N][d] fp16 of the group each coefficient belongs to, dequantized [N][d] float32)."""
    coef = np.asarray(coef, dtype=np.float32)
    ranks = np.asarray(ranks, dtype=np.int64)
    N, d = coef.shape
    codes = np.zeros((N, d), dtype=np.uint8)
    lo = np.zeros((N, d), dtype=np.float16)
    step = np.zeros((N, d), dtype=np.float16)
    deq = np.zeros((N, d), dtype=np.float32)
    for r in np.unique(ranks):
        toks = np.nonzero(ranks == r)[0]
        order = toks[np.argsort(np.asarray(pos)[toks], kind="stable")]   # bucket order
        n = order.size
        n8 = (n + 7) // 8 * 8
        for g0 in range(0, n8, QGROUP):                 # groups never cross a 128-slot tile
            g1 = min(g0 + QGROUP, n8, (g0 // 128 + 1) * 128)
            members = order[g0:min(g1, n)]
            n_pad = (g1 - g0) - members.size            # padding slots of the bucket: zeros
            for j in range(int(r)):
                x = np.concatenate([coef[members, j], np.zeros(n_pad, dtype=np.float32)])
                q, a, s = quantize_group(x, bits)
                codes[members, j] = q[: members.size]
                lo[members, j] = a
                step[members, j] = s
                deq[members, j] = dequantize_group(q[: members.size], a, s)
    return codes, lo, step, deq
