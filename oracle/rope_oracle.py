"""VarRate pre-RoPE coding, CPU oracle: TEST INFRASTRUCTURE, not part of the library.

The paper codes keys before the rotary position embedding (Sec. 3.1, "Joint per-token vector";
Algorithm 1, first and last steps): every post-RoPE key is un-rotated to its pre-RoPE form, coded,
reconstructed, and re-rotated to post-RoPE; values carry no rotation. RoPE's per-position rotation
raises the numerical rank of the key cache, which is why the coding happens before it. Plain numpy,
fp64, on top of the per-head codec of ``varrate_oracle``.

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline / reference leg may
import this module. It shares no code with the CUDA library and imports nothing from it.

Readings of the paper taken here (each one is also listed in the design notes):
  * the paper names RoPE without restating it; this oracle uses the rotary embedding of the models
    it evaluates, in the half-split pairing: coordinate i is paired with i + d/2 (i < d/2) and the
    pair at position p is turned by the angle p * f_i, f_i = base^(-2 i / d);
  * the frequencies are an explicit input (``inv_freq``, d/2 values), so a model's own frequency
    table (a different base, or a long-context rescaling of the low frequencies) plugs in unchanged;
    ``rope_inv_freq`` gives the plain table;
  * positions are the cache positions 0 .. N-1 of the tokens; a decode query at position p is
    rotated by p like any key (the model hands it over post-RoPE).
"""
from __future__ import annotations

import math

import numpy as np

from . import varrate_oracle as vo


def rope_inv_freq(head_dim: int, base: float) -> np.ndarray:
    """Plain RoPE frequencies f_i = base^(-2 i / d), i < d / 2 (fp64)."""
    i = np.arange(head_dim // 2, dtype=np.float64)
    return base ** (-2.0 * i / head_dim)


def rope_rotate(x: np.ndarray, pos, inv_freq: np.ndarray) -> np.ndarray:
    """Post-RoPE form of x [..., N, d] at positions pos [N]: the pair (x_i, x_{i + d/2}) turned by
    the angle pos * f_i, i.e. (x_i cos - x_{i+d/2} sin, x_{i+d/2} cos + x_i sin)."""
    x = np.asarray(x, dtype=np.float64)
    h = x.shape[-1] // 2
    ang = np.asarray(pos, dtype=np.float64)[:, None] * np.asarray(inv_freq, dtype=np.float64)[None, :]
    c, s = np.cos(ang), np.sin(ang)
    a, b = x[..., :h], x[..., h:]
    return np.concatenate([a * c - b * s, b * c + a * s], axis=-1)


def rope_unrotate(x: np.ndarray, pos, inv_freq: np.ndarray) -> np.ndarray:
    """Pre-RoPE form of a post-RoPE x: the inverse turn (angle -pos * f_i)."""
    return rope_rotate(x, -np.asarray(pos, dtype=np.float64), inv_freq)


def rotation_matrix(p: float, inv_freq: np.ndarray) -> np.ndarray:
    """The d x d matrix R_p with rope_rotate(x, [p]) = R_p x (for the per-token query turn of the
    coefficient route)."""
    h = len(inv_freq)
    R = np.zeros((2 * h, 2 * h))
    for i in range(h):
        c, s = math.cos(p * inv_freq[i]), math.sin(p * inv_freq[i])
        R[i, i], R[i, i + h] = c, -s
        R[i + h, i], R[i + h, i + h] = s, c
    return R


def encode_prerope(k_post: np.ndarray, pos, inv_freq: np.ndarray, basis_k: np.ndarray) -> np.ndarray:
    """Algorithm 1's first step for the keys of one head, then the projection: un-rotate the
    post-RoPE keys k_post [N][d] and project them on the (pre-RoPE) key basis. Returns the full
    coefficients [N][d]."""
    return vo.project(rope_unrotate(k_post, pos, inv_freq), basis_k)


def reconstruct_post(coef: np.ndarray, ranks: np.ndarray, basis_k: np.ndarray, pos,
                     inv_freq: np.ndarray) -> np.ndarray:
    """Algorithm 1's last steps for the keys of one head: rebuild the pre-RoPE keys from the
    truncated coefficients (Eq. 5) and re-rotate them to post-RoPE."""
    return rope_rotate(vo.reconstruct(coef, ranks, basis_k), pos, inv_freq)


def decode_prerope_recon(q_post, coef_k, coef_v, ranks, basis_k, basis_v, pos, inv_freq):
    """Decode attention of one post-RoPE query per head over a pre-RoPE-coded cache, by the paper's
    route: rebuild every key (re-rotated to post-RoPE) and value, then plain attention.
    q_post [H][d]; coef_k, coef_v [G][N][d]; basis_k, basis_v [G][d][d]; pos [N]."""
    G = coef_k.shape[0]
    kh = np.stack([reconstruct_post(coef_k[g], ranks, basis_k[g], pos, inv_freq) for g in range(G)])
    vh = np.stack([vo.reconstruct(coef_v[g], ranks, basis_v[g]) for g in range(G)])
    return vo.attention(q_post, kh, vh)


def decode_prerope_coef(q_post, coef_k, coef_v, ranks, basis_k, basis_v, pos, inv_freq):
    """The same attention computed on the coefficients: the score of token t needs the query turned
    back by the token's own position, q~_t = U_K R_t^T q (the query cannot absorb the rotation once
    for all tokens), then score_t = q~_t[:r_t] . c^K_t[:r_t] / sqrt(d); the values are not rotated,
    so o = U_V^T sum_t alpha_t c^V_t[:r_t] as without RoPE."""
    q = np.asarray(q_post, dtype=np.float64)
    H, d = q.shape
    G = coef_k.shape[0]
    grp = H // G
    out = np.zeros((H, d))
    for h in range(H):
        g = h // grp
        uk = np.asarray(basis_k[g], dtype=np.float64)
        uv = np.asarray(basis_v[g], dtype=np.float64)
        ck = vo.truncate(np.asarray(coef_k[g], dtype=np.float64), ranks)
        cv = vo.truncate(np.asarray(coef_v[g], dtype=np.float64), ranks)
        sc = np.zeros(ck.shape[0])
        for t, p in enumerate(pos):
            qt = uk @ (rotation_matrix(float(p), inv_freq).T @ q[h])
            sc[t] = ck[t] @ qt / math.sqrt(d)
        a = np.exp(sc - sc.max())
        a /= a.sum()
        out[h] = uv.T @ (a @ cv)
    return out
