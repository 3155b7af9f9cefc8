"""VarRate joint-codec CPU oracle: TEST INFRASTRUCTURE, not part of the library.

The paper-faithful form of the codec (Sec. 3.1): one basis per layer over the joint per-token
vector of all KV heads' keys and values (Eq. 1), strided anchor tokens kept exact, every other
token coded as its residual to the mean of its c nearest anchors (Eq. 2), ranks capped at the
basis size R (Eq. 4), reconstruction by Eq. 5 with the anchor mean added back. Plain numpy,
fp64, in the order of Algorithm 1; the salience, normalisation and integer water level are the
ones of ``varrate_oracle`` (pinned there), applied to the joint coded set.

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline / reference leg may
import this module. It shares no code with the CUDA library and imports nothing from it.

Readings of the paper taken here (each one is also listed in the design notes):
  * z_t = [k_t of heads 0..G-1 ; v_t of heads 0..G-1] (Eq. 1), so element i of head g's key is
    z[g d + i] and of its value z[G d + g d + i]; keys are taken in the frame they are given
    (no RoPE in the synthetic workloads);
  * anchors are the tokens at positions 0, stride, 2 stride, ... (0-based form of the paper's
    z_1, z_{1+Delta}, ...); the exact set is the anchors plus the last ``window`` tokens
    (Algorithm 1, line 2); the coded set is every other token;
  * the nearest anchors of a token are searched among all anchors of the sequence by squared
    Euclidean distance over the whole joint vector (Eq. 2); equal distances are ordered by the
    lower anchor index; with fewer than c anchors every anchor is used (the indices past the
    anchor count are -1 and their distances +inf);
  * the coded budget is B = floor(kappa N D) - |E| D (Eq. 3 with the product taken once in double
    precision, as in the per-head codec) and ranks lie in [r_min, R];
  * salience is computed for the tokens before the recent window and pooled there (as in the
    per-head codec); the allocation sees the salience of the coded tokens only, in position order.
"""
from __future__ import annotations

import math

import numpy as np

from . import varrate_oracle as vo


# ------------------------------------------------------------ joint vector (Sec. 3.1, Eq. 1)

def joint_vector(k: np.ndarray, v: np.ndarray) -> np.ndarray:
    """z_t = [k_t of every KV head ; v_t of every KV head] for one (sequence, layer).
    k, v: [G][N][d]. Returns fp64 [N][2 G d]."""
    k = np.asarray(k, dtype=np.float64)
    v = np.asarray(v, dtype=np.float64)
    G, N, d = k.shape
    z = np.zeros((N, 2 * G * d))
    for g in range(G):
        z[:, g * d:(g + 1) * d] = k[g]
        z[:, G * d + g * d:G * d + (g + 1) * d] = v[g]
    return z


def split_joint(z: np.ndarray, G: int, d: int):
    """Inverse of joint_vector: [N][2 G d] -> (k [G][N][d], v [G][N][d])."""
    z = np.asarray(z, dtype=np.float64)
    k = np.stack([z[:, g * d:(g + 1) * d] for g in range(G)])
    v = np.stack([z[:, G * d + g * d:G * d + (g + 1) * d] for g in range(G)])
    return k, v


# ------------------------------------------------- anchors and exact set (Algorithm 1, line 2)

def anchor_positions(n_ctx: int, stride: int) -> np.ndarray:
    """Positions of the anchor tokens: 0, stride, 2 stride, ... < n_ctx."""
    return np.arange(0, n_ctx, stride, dtype=np.int64)


def exact_mask(n_ctx: int, stride: int, window: int) -> np.ndarray:
    """Exact set E = anchors plus the last ``window`` tokens, as a boolean mask over [0, n_ctx)."""
    m = np.zeros(n_ctx, dtype=bool)
    m[anchor_positions(n_ctx, stride)] = True
    m[max(0, n_ctx - window):] = True
    return m


# ------------------------------------------------------- nearest anchors (Sec. 3.1, Eq. 2)

def nearest_anchors(z: np.ndarray, stride: int, c: int, rows=None):
    """The c anchors nearest every token in squared Euclidean distance over the joint vector.

    Returns (idx int64 [N][c]: anchor numbers a, the anchor token being z[a * stride],
    dist fp64 [N][c]: the squared distances), each row ordered by (distance, anchor number).
    Rows of tokens that are themselves anchors are included (their nearest anchor is themselves).
    With ``rows`` (token indices) only those tokens are searched and the results have one row per
    listed token, in the given order."""
    z = np.asarray(z, dtype=np.float64)
    N = z.shape[0]
    pos = anchor_positions(N, stride)
    anchors = z[pos]
    n_a = pos.size
    tokens = np.arange(N) if rows is None else np.asarray(rows, dtype=np.int64)
    idx = np.full((tokens.size, c), -1, dtype=np.int64)
    dist = np.full((tokens.size, c), np.inf)
    for i, t in enumerate(tokens):
        diff = anchors - z[t]
        d2 = np.einsum("ad,ad->a", diff, diff)
        order = np.lexsort((np.arange(n_a), d2))       # by distance, then anchor number
        take = order[:min(c, n_a)]
        idx[i, :take.size] = take
        dist[i, :take.size] = d2[take]
    return idx, dist


def anchor_mean(z: np.ndarray, idx: np.ndarray, stride: int) -> np.ndarray:
    """z_bar_t = mean of the anchors listed in idx[t] (Eq. 2); entries -1 are not anchors."""
    z = np.asarray(z, dtype=np.float64)
    out = np.zeros_like(z)
    for t in range(z.shape[0]):
        sel = [a for a in idx[t] if a >= 0]
        out[t] = z[np.asarray(sel, dtype=np.int64) * stride].mean(axis=0)
    return out


def residual(z: np.ndarray, idx: np.ndarray, stride: int) -> np.ndarray:
    """e_t = z_t - z_bar_t (Eq. 2)."""
    return np.asarray(z, dtype=np.float64) - anchor_mean(z, idx, stride)


# --------------------------------------------------------------- budget and ranks (Eq. 3, 4)

def joint_budget(n_ctx: int, dim: int, n_exact: int, budget_frac: float) -> int:
    """Coded budget in joint-coefficient units: B = floor(kappa * N * D) - |E| D (Eq. 3)."""
    return int(math.floor(budget_frac * float(n_ctx * dim))) - n_exact * dim


def joint_ranks(sal32: np.ndarray, n_ctx: int, dim: int, rank_cap: int, stride: int,
                window: int, budget_frac: float, r_min: int, mode: int = vo.SALIENCE):
    """Ranks of all N tokens of one (sequence, layer) under the joint codec.

    sal32: fp32 pooled salience of the tokens before the window ([N - window]). Coded tokens get
    the integer water level of Eq. 4 over their own min-max normalised salience, in [r_min, R];
    exact tokens get rank 0 (they are stored whole). Returns (ranks int64 [N], status, realised
    coded sum, coded budget)."""
    exact = exact_mask(n_ctx, stride, window)
    coded = np.flatnonzero(~exact)
    bc = joint_budget(n_ctx, dim, int(exact.sum()), budget_frac)
    shat = vo.normalize(np.asarray(sal32, dtype=np.float32)[coded], mode)
    rc, _, status, total = vo.allocate(shat, bc, r_min, rank_cap)
    ranks = np.zeros(n_ctx, dtype=np.int64)
    ranks[coded] = rc
    return ranks, status, total, bc


def joint_footprint(n_ctx: int, dim: int, stride: int, window: int, budget_frac: float, c: int,
                    coef_bits: float = 16.0, group: int = 32, param_bits: int = 32,
                    index_bytes: int = 2, elem_bytes: int = 2) -> float:
    """Stored bytes of one (sequence, layer) under the joint codec as a fraction of the full cache
    (N D values of elem_bytes): the exact set whole (|E| D values), the coded budget B of Eq. 3 in
    coefficients of coef_bits bits (quantized: plus param_bits of group parameters per group of
    ``group`` coefficients; coef_bits = 16 means unquantized), and c anchor indices of index_bytes
    per coded token (Sec. 3.1, Budget: the indices are counted in the reported footprint)."""
    exact = int(exact_mask(n_ctx, stride, window).sum())
    coded = n_ctx - exact
    b = joint_budget(n_ctx, dim, exact, budget_frac)
    per_coef = coef_bits / 8.0 if coef_bits >= 16 else (coef_bits + param_bits / group) / 8.0
    total = exact * dim * elem_bytes + max(b, 0) * per_coef + coded * c * index_bytes
    return total / (n_ctx * dim * elem_bytes)


# ------------------------------------------------ projection and reconstruction (Eq. 5)

def joint_project(e: np.ndarray, basis: np.ndarray) -> np.ndarray:
    """c_t = V e_t at full rank R. e: [N][D], basis V: [R][D] (row j = basis vector j)."""
    return np.asarray(e, dtype=np.float64) @ np.asarray(basis, dtype=np.float64).T


def joint_reconstruct(z: np.ndarray, idx: np.ndarray, coef: np.ndarray, ranks: np.ndarray,
                      basis: np.ndarray, stride: int) -> np.ndarray:
    """z_hat_t = z_bar_t + V^T (m_t * c_t) for coded tokens (rank > 0), z_hat_t = z_t for exact
    tokens (rank 0) (Eq. 5)."""
    z = np.asarray(z, dtype=np.float64)
    basis = np.asarray(basis, dtype=np.float64)
    zbar = anchor_mean(z, idx, stride)
    out = z.copy()
    R = basis.shape[0]
    for t in range(z.shape[0]):
        r = int(ranks[t])
        if r > 0:
            m = (np.arange(R) < r).astype(np.float64)
            out[t] = zbar[t] + basis.T @ (m * coef[t])
    return out


def encode_joint(q_win, k, v, basis, group, budget_frac, r_min, stride, c, window,
                 pool_len=5, mode=vo.SALIENCE):
    """Algorithm 1 for one (sequence, layer) under the joint codec: joint vectors, anchors and
    exact set, nearest anchors and residuals, salience and ranks, full-rank coefficients.
    k, v: [G][N][d]; basis: [R][2 G d]. Returns a dict."""
    k = np.asarray(k, dtype=np.float64)
    G, N, d = k.shape
    z = joint_vector(k, v)
    idx, dist = nearest_anchors(z, stride, c)
    e = residual(z, idx, stride)
    sal32 = vo.salience(q_win, k, group, pool_len).astype(np.float32) if mode == vo.SALIENCE \
        else np.zeros(N - window, dtype=np.float32)
    ranks, status, total, bc = joint_ranks(sal32, N, 2 * G * d, basis.shape[0], stride, window,
                                           budget_frac, r_min, mode)
    coef = joint_project(e, basis)
    return dict(z=z, idx=idx, dist=dist, ranks=ranks, status=status, total=total, budget=bc,
                coef=coef, sal=sal32)


# ----------------------------------------------------------- decode attention on the joint code

def joint_decode_coef(q, z, idx, coef, ranks, basis, stride, G):
    """Decode attention of one new token computed on the joint code (route i).

    q [H][d]; z [N][D] supplies the exact tokens (rank 0) and the anchors; coef [N][R] full
    coefficients (truncated here by ranks). Per query head h on KV head g, with V_Kg = the key
    columns of head g of the basis (V[:, g d:(g+1) d]) and V_Vg its value columns:
      exact t:  score = q . k_t / sqrt(d)
      coded t:  score = (mean over the anchors a of t of q . k_a + (V_Kg q)[:r_t] . c_t[:r_t]) / sqrt(d)
    and, with alpha the softmax over all N tokens,
      o = sum_{t exact} alpha_t v_t + sum_a w_a v_a + V_Vg^T sum_{t coded} alpha_t (m_t * c_t),
    where w_a collects alpha_t / (number of anchors of t) from every coded t that lists anchor a.
    Equal to attention over the reconstructed cache (Eq. 5)."""
    q = np.asarray(q, dtype=np.float64)
    z = np.asarray(z, dtype=np.float64)
    coef = np.asarray(coef, dtype=np.float64)
    basis = np.asarray(basis, dtype=np.float64)
    H, d = q.shape
    N = z.shape[0]
    R = basis.shape[0]
    grp = H // G
    coded = np.asarray(ranks) > 0
    mask = (np.arange(R)[None, :] < np.asarray(ranks)[:, None]).astype(np.float64)
    ct = coef * mask
    out = np.zeros((H, d))
    for h in range(H):
        g = h // grp
        kz = z[:, g * d:(g + 1) * d]
        vz = z[:, G * d + g * d:G * d + (g + 1) * d]
        vk = basis[:, g * d:(g + 1) * d]
        vv = basis[:, G * d + g * d:G * d + (g + 1) * d]
        exact_sc = kz @ q[h]                          # q . k_t of every token (used for exact ones)
        qt = vk @ q[h]
        sc = np.zeros(N)
        for t in range(N):
            if coded[t]:
                sel = np.asarray([a for a in idx[t] if a >= 0], dtype=np.int64)
                sc[t] = exact_sc[sel * stride].mean() + ct[t] @ qt
            else:
                sc[t] = exact_sc[t]
        sc /= math.sqrt(d)
        a = np.exp(sc - sc.max())
        a /= a.sum()
        wz = np.where(coded, 0.0, a)                  # weights on the stored tokens themselves
        for t in np.flatnonzero(coded):
            sel = np.asarray([x for x in idx[t] if x >= 0], dtype=np.int64)
            wz[sel * stride] += a[t] / sel.size
        out[h] = wz @ vz + vv.T @ (a @ ct)
    return out


def joint_decode_recon(q, z, idx, coef, ranks, basis, stride, G):
    """Decode attention on the reconstructed joint cache (route ii): z_hat by Eq. 5, split into
    keys and values, plain attention."""
    zh = joint_reconstruct(z, idx, coef, ranks, basis, stride)
    d = np.asarray(q).shape[1]
    kh, vh = split_joint(zh, G, d)
    return vo.attention(q, kh, vh)
