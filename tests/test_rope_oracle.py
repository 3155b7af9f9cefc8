"""Pins of the pre-RoPE coding oracle (Sec. 3.1 "Joint per-token vector"; Algorithm 1, first and
last steps) against facts that do not come from the oracle itself: rotations worked out by hand,
the complex-number form of the rotary embedding, its relative-position property, torch SDPA, and
the paper's remark that RoPE raises the numerical rank of the keys."""
import math

import numpy as np
import torch

import oracle as O
from oracle import rope_oracle as R


def _orthonormal(rng, d):
    q, _ = np.linalg.qr(rng.standard_normal((d, d)))
    return q.T


def test_rotation_by_hand():
    f = R.rope_inv_freq(4, 100.0)
    np.testing.assert_allclose(f, [1.0, 0.1], rtol=0, atol=1e-15)
    # pair (0, 2) turned by 1 rad at position 1
    np.testing.assert_allclose(R.rope_rotate(np.array([[1.0, 0, 0, 0]]), [1], f),
                               [[math.cos(1), 0, math.sin(1), 0]], atol=1e-15)
    # pair (1, 3) turned by 3 * 0.1 rad at position 3
    np.testing.assert_allclose(R.rope_rotate(np.array([[0, 2.0, 0, 0]]), [3], f),
                               [[0, 2 * math.cos(0.3), 0, 2 * math.sin(0.3)]], atol=1e-15)


def test_rotation_is_complex_multiplication():
    rng = np.random.default_rng(0)
    d, n = 16, 40
    f = R.rope_inv_freq(d, 10000.0)
    x = rng.standard_normal((n, d))
    pos = rng.integers(0, 5000, n)
    zc = (x[:, :d // 2] + 1j * x[:, d // 2:]) * np.exp(1j * pos[:, None] * f[None, :])
    np.testing.assert_allclose(R.rope_rotate(x, pos, f), np.concatenate([zc.real, zc.imag], axis=1),
                               atol=1e-12)


def test_rotation_is_orthogonal_and_inverted():
    rng = np.random.default_rng(1)
    d, n = 32, 25
    f = R.rope_inv_freq(d, 500000.0)
    x = rng.standard_normal((n, d))
    pos = np.arange(n) * 997
    y = R.rope_rotate(x, pos, f)
    np.testing.assert_allclose(np.linalg.norm(y, axis=1), np.linalg.norm(x, axis=1), rtol=1e-13)
    np.testing.assert_allclose(R.rope_unrotate(y, pos, f), x, atol=1e-12)
    for t in (0, 7, 24):
        np.testing.assert_allclose(R.rotation_matrix(float(pos[t]), f) @ x[t], y[t], atol=1e-12)


def test_scores_depend_only_on_the_offset():
    rng = np.random.default_rng(2)
    d = 16
    f = R.rope_inv_freq(d, 10000.0)
    q, k = rng.standard_normal((1, d)), rng.standard_normal((1, d))
    base = float((R.rope_rotate(q, [50], f) @ R.rope_rotate(k, [20], f).T)[0, 0])
    for s in (1, 333, 4096):
        shifted = float((R.rope_rotate(q, [50 + s], f) @ R.rope_rotate(k, [20 + s], f).T)[0, 0])
        assert abs(shifted - base) < 1e-10


def test_rope_raises_the_numerical_rank_of_keys():
    # Sec. 3.1: keys of low rank before RoPE are of much higher rank after it
    rng = np.random.default_rng(3)
    d, n, r = 64, 512, 8
    f = R.rope_inv_freq(d, 10000.0)
    pre = rng.standard_normal((n, r)) @ rng.standard_normal((r, d))
    post = R.rope_rotate(pre, np.arange(n), f)

    def num_rank(m):
        s = np.linalg.svd(m, compute_uv=False)
        return int((s > 1e-8 * s[0]).sum())
    assert num_rank(pre) == r
    assert num_rank(post) >= 4 * r


def _case(seed, G=2, grp=2, n=60, d=8, full=False):
    rng = np.random.default_rng(seed)
    f = R.rope_inv_freq(d, 10000.0)
    pos = np.arange(n) * 3 + 5
    k_post = rng.standard_normal((G, n, d))
    v = rng.standard_normal((G, n, d))
    q = rng.standard_normal((G * grp, d))
    bk = np.stack([_orthonormal(rng, d) for _ in range(G)])
    bv = np.stack([_orthonormal(rng, d) for _ in range(G)])
    ck = np.stack([R.encode_prerope(k_post[g], pos, f, bk[g]) for g in range(G)])
    cv = np.stack([O.project(v[g], bv[g]) for g in range(G)])
    ranks = np.full(n, d) if full else rng.integers(1, d + 1, n)
    return q, k_post, v, ck, cv, ranks, bk, bv, pos, f


def test_full_rank_round_trip_gives_the_post_rope_keys():
    q, k_post, v, ck, cv, ranks, bk, bv, pos, f = _case(4, full=True)
    for g in range(k_post.shape[0]):
        np.testing.assert_allclose(R.reconstruct_post(ck[g], ranks, bk[g], pos, f), k_post[g], atol=1e-12)


def test_decode_routes_agree():
    for seed in range(3):
        q, k_post, v, ck, cv, ranks, bk, bv, pos, f = _case(10 + seed)
        a = R.decode_prerope_coef(q, ck, cv, ranks, bk, bv, pos, f)
        b = R.decode_prerope_recon(q, ck, cv, ranks, bk, bv, pos, f)
        np.testing.assert_allclose(a, b, rtol=0, atol=1e-10)


def test_decode_at_full_rank_is_sdpa_on_the_post_rope_cache():
    q, k_post, v, ck, cv, ranks, bk, bv, pos, f = _case(20, full=True)
    out = R.decode_prerope_coef(q, ck, cv, ranks, bk, bv, pos, f)
    H, d = q.shape
    grp = H // k_post.shape[0]
    for h in range(H):
        g = h // grp
        want = torch.nn.functional.scaled_dot_product_attention(
            torch.as_tensor(q[h])[None, None, None], torch.as_tensor(k_post[g])[None, None],
            torch.as_tensor(v[g])[None, None])[0, 0, 0].numpy()
        np.testing.assert_allclose(out[h], want, atol=1e-10)


def test_position_zero_everywhere_is_the_plain_codec():
    q, k_post, v, ck, cv, ranks, bk, bv, pos, f = _case(30)
    zero = np.zeros_like(pos)
    ck0 = np.stack([R.encode_prerope(k_post[g], zero, f, bk[g]) for g in range(k_post.shape[0])])
    np.testing.assert_allclose(R.decode_prerope_coef(q, ck0, cv, ranks, bk, bv, zero, f),
                               O.decode_coef(q, ck0, cv, ranks, bk, bv), atol=1e-12)
