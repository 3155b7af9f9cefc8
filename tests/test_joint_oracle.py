"""Pins of the joint-codec oracle (Sec. 3.1, Eq. 1-3 and 5; Algorithm 1) against facts that do not
come from the oracle itself: hand-derived values (tests/golden/joint_budgets.json), brute force
in plain Python on tiny inputs, scipy's cdist, torch SDPA, orthonormal-basis identities and the
exact-set share the paper states for stride 16 (appendix "The Stride Ablation")."""
import json
import math
import os

import numpy as np
import pytest
import torch
from scipy.spatial.distance import cdist

import oracle as O
from oracle import joint_oracle as J

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _orthonormal_rows(rng, r, dim):
    q, _ = np.linalg.qr(rng.standard_normal((dim, dim)))
    return q.T[:r]


def _sdpa(q, k, v):
    """One query per head through torch's scaled_dot_product_attention (fp64)."""
    H, d = q.shape
    G = k.shape[0]
    grp = H // G
    out = np.zeros((H, d))
    for h in range(H):
        g = h // grp
        o = torch.nn.functional.scaled_dot_product_attention(
            torch.as_tensor(q[h], dtype=torch.float64)[None, None, None],
            torch.as_tensor(k[g], dtype=torch.float64)[None, None],
            torch.as_tensor(v[g], dtype=torch.float64)[None, None])
        out[h] = o[0, 0, 0].numpy()
    return out


# ------------------------------------------------------------------------- Eq. 1 layout

def test_joint_vector_layout_by_hand():
    # G = 2 heads, d = 2: token t of head g has key (10 g + t, 10 g + t + 0.5) and value minus that
    G, N, d = 2, 3, 2
    k = np.zeros((G, N, d))
    for g in range(G):
        for t in range(N):
            k[g, t] = [10 * g + t, 10 * g + t + 0.5]
    v = -k
    z = J.joint_vector(k, v)
    assert z.shape == (3, 8)
    np.testing.assert_array_equal(z[1], [1, 1.5, 11, 11.5, -1, -1.5, -11, -11.5])
    kk, vv = J.split_joint(z, G, d)
    np.testing.assert_array_equal(kk, k)
    np.testing.assert_array_equal(vv, v)


# ------------------------------------------------------------------ exact set (Algorithm 1)

def test_exact_set_by_hand():
    np.testing.assert_array_equal(np.flatnonzero(J.exact_mask(10, 4, 3)), [0, 4, 7, 8, 9])
    np.testing.assert_array_equal(np.flatnonzero(J.exact_mask(5, 8, 0)), [0])
    assert J.exact_mask(7, 1, 0).all()
    np.testing.assert_array_equal(J.anchor_positions(33, 16), [0, 16, 32])


def test_joint_budget_golden():
    with open(os.path.join(GOLDEN, "joint_budgets.json")) as f:
        cases = json.load(f)["cases"]
    for c in cases:
        n_exact = int(J.exact_mask(c["n_ctx"], c["stride"], c["window"]).sum())
        assert n_exact == c["n_exact"], c["name"]
        dim = 2 * c["G"] * c["head_dim"]
        assert J.joint_budget(c["n_ctx"], dim, n_exact, c["budget_frac"]) == c["budget"], c["name"]


def test_exact_share_at_stride_16_matches_the_paper():
    # appendix "The Stride Ablation": at stride 16 the anchors are 6.25 % of the cache, so at a
    # 10 % budget they alone take ~66 % of it (62.5 % anchors, the recent window the rest)
    n, D, w = 16384, 2048, 64
    anchors = J.anchor_positions(n, 16).size
    assert anchors / n == 0.0625
    exact = int(J.exact_mask(n, 16, w).sum())
    share = exact * D / (0.1 * n * D)
    assert 0.62 <= share <= 0.67


# ------------------------------------------------------------------ nearest anchors (Eq. 2)

def _brute_nearest(z, stride, c):
    n = len(z)
    out_i, out_d = [], []
    for t in range(n):
        cand = []
        for a, p in enumerate(range(0, n, stride)):
            s = 0.0
            for x, y in zip(z[t], z[p]):
                s += (float(x) - float(y)) ** 2
            cand.append((s, a))
        cand.sort()
        take = cand[:c]
        out_i.append([a for _, a in take] + [-1] * (c - len(take)))
        out_d.append([s for s, _ in take] + [math.inf] * (c - len(take)))
    return np.array(out_i), np.array(out_d)


@pytest.mark.parametrize("n,dim,stride,c", [(13, 3, 4, 2), (20, 5, 3, 4), (9, 2, 2, 1), (6, 4, 4, 4)])
def test_nearest_anchors_brute_force(n, dim, stride, c):
    rng = np.random.default_rng(n * 7 + c)
    z = np.round(rng.standard_normal((n, dim)) * 4) / 4       # repeated values -> some ties
    idx, dist = J.nearest_anchors(z, stride, c)
    bi, bd = _brute_nearest(z.tolist(), stride, c)
    np.testing.assert_array_equal(idx, bi)
    np.testing.assert_allclose(dist, bd, rtol=0, atol=1e-12)


def test_nearest_anchors_scipy_cdist():
    rng = np.random.default_rng(5)
    z = rng.standard_normal((300, 24))
    stride, c = 16, 4
    idx, dist = J.nearest_anchors(z, stride, c)
    d2 = cdist(z, z[::stride], "sqeuclidean")
    ref = np.argsort(d2, axis=1, kind="stable")[:, :c]
    np.testing.assert_array_equal(idx, ref)
    np.testing.assert_allclose(dist, np.take_along_axis(d2, ref, axis=1), rtol=1e-12, atol=1e-12)
    rows = np.array([299, 0, 17, 150])
    ri, rd = J.nearest_anchors(z, stride, c, rows=rows)
    np.testing.assert_array_equal(ri, ref[rows])
    np.testing.assert_array_equal(rd, dist[rows])


def test_anchor_tokens_pick_themselves_and_ties_take_the_lower_index():
    rng = np.random.default_rng(9)
    z = rng.standard_normal((40, 6))
    idx, dist = J.nearest_anchors(z, 8, 3)
    for a in range(5):
        assert idx[a * 8, 0] == a and dist[a * 8, 0] == 0.0
    z[16] = z[8]                                   # anchors 1 and 2 identical
    idx, _ = J.nearest_anchors(z, 8, 2)
    assert list(idx[8]) == [1, 2] and list(idx[16]) == [1, 2]


def test_fewer_anchors_than_c():
    z = np.arange(10, dtype=np.float64).reshape(5, 2)
    idx, dist = J.nearest_anchors(z, 4, 4)          # anchors at 0 and 4 only
    assert (idx[:, 2:] == -1).all() and np.isinf(dist[:, 2:]).all()
    np.testing.assert_array_equal(J.anchor_mean(z, idx, 4)[2], (z[0] + z[4]) / 2)


def test_residual_by_hand():
    # one dimension, stride 2: anchors z0 = 0, z2 = 5, z4 = 10; c = 2
    z = np.array([[0.0], [1.0], [5.0], [2.0], [10.0]])
    idx, dist = J.nearest_anchors(z, 2, 2)
    np.testing.assert_array_equal(idx[1], [0, 1])      # |1-0|^2 = 1, |1-5|^2 = 16
    np.testing.assert_array_equal(dist[1], [1.0, 16.0])
    np.testing.assert_array_equal(idx[3], [0, 1])      # |2-0|^2 = 4, |2-5|^2 = 9
    e = J.residual(z, idx, 2)
    assert e[1, 0] == -1.5 and e[3, 0] == -0.5
    assert e[2, 0] == 2.5                              # anchor z2 = 5: nearest {5, 0 or 10 -> 0}


# ------------------------------------------------------------------------- ranks (Eq. 4)

def test_joint_ranks_invariants():
    rng = np.random.default_rng(3)
    n, D, R, stride, w = 400, 64, 48, 16, 8
    sal = rng.random(n - w).astype(np.float32) ** 3
    ranks, status, total, bc = J.joint_ranks(sal, n, D, R, stride, w, 0.4, 4)
    exact = J.exact_mask(n, stride, w)
    assert status == O.OK
    assert (ranks[exact] == 0).all()
    assert ranks[~exact].min() >= 4 and ranks[~exact].max() <= R
    assert total == ranks.sum() <= bc
    assert bc == math.floor(0.4 * n * D) - int(exact.sum()) * D
    # uniform salience: one rank for every coded token (Eq. 4 collapses to the flat codec)
    ru, _, _, _ = J.joint_ranks(np.full(n - w, 0.5, np.float32), n, D, R, stride, w, 0.4, 4)
    assert np.unique(ru[~exact]).size == 1
    # a negative budget binds the floor
    rf, st, _, _ = J.joint_ranks(sal, n, D, R, stride, w, 0.05, 4)
    assert st == O.FLOOR_BINDS and (rf[~exact] == 4).all()


# ---------------------------------------------------------- projection, reconstruction (Eq. 5)

def test_full_rank_reconstruction_is_exact():
    rng = np.random.default_rng(4)
    n, D, stride, c = 50, 12, 4, 3
    z = rng.standard_normal((n, D))
    V = _orthonormal_rows(rng, D, D)
    idx, _ = J.nearest_anchors(z, stride, c)
    coef = J.joint_project(J.residual(z, idx, stride), V)
    ranks = np.where(J.exact_mask(n, stride, 5), 0, D)
    np.testing.assert_allclose(J.joint_reconstruct(z, idx, coef, ranks, V, stride), z, atol=1e-12)


def test_truncation_error_is_the_dropped_energy():
    rng = np.random.default_rng(6)
    n, D, stride, c = 60, 10, 5, 2
    z = rng.standard_normal((n, D))
    V = _orthonormal_rows(rng, D, D)
    idx, _ = J.nearest_anchors(z, stride, c)
    coef = J.joint_project(J.residual(z, idx, stride), V)
    exact = J.exact_mask(n, stride, 4)
    ranks = np.where(exact, 0, rng.integers(1, D + 1, n))
    zh = J.joint_reconstruct(z, idx, coef, ranks, V, stride)
    for t in np.flatnonzero(~exact):
        dropped = (coef[t, ranks[t]:] ** 2).sum()
        assert abs(((zh[t] - z[t]) ** 2).sum() - dropped) < 1e-10
    np.testing.assert_array_equal(zh[exact], z[exact])


# ------------------------------------------------------------------------------- decode

def _case(seed, G=2, grp=2, n=70, d=4, R=None, stride=8, c=3, w=6):
    rng = np.random.default_rng(seed)
    D = 2 * G * d
    k = rng.standard_normal((G, n, d))
    v = rng.standard_normal((G, n, d))
    q = rng.standard_normal((G * grp, d))
    V = _orthonormal_rows(rng, R or D, D)
    z = J.joint_vector(k, v)
    idx, _ = J.nearest_anchors(z, stride, c)
    coef = J.joint_project(J.residual(z, idx, stride), V)
    exact = J.exact_mask(n, stride, w)
    ranks = np.where(exact, 0, rng.integers(1, (R or D) + 1, n))
    return q, k, v, z, idx, coef, ranks, V, stride, G


def test_decode_routes_agree():
    for seed in range(3):
        q, k, v, z, idx, coef, ranks, V, stride, G = _case(seed, R=9)
        a = J.joint_decode_coef(q, z, idx, coef, ranks, V, stride, G)
        b = J.joint_decode_recon(q, z, idx, coef, ranks, V, stride, G)
        np.testing.assert_allclose(a, b, rtol=0, atol=1e-10)


def test_decode_at_full_rank_is_sdpa():
    q, k, v, z, idx, coef, ranks, V, stride, G = _case(11)
    D = V.shape[1]
    ranks = np.where(ranks > 0, D, 0)
    out = J.joint_decode_coef(q, z, idx, coef, ranks, V, stride, G)
    np.testing.assert_allclose(out, _sdpa(q, k, v), atol=1e-10)


def test_decode_every_token_an_anchor_is_sdpa():
    # stride 1: every token is exact, whatever the basis and the ranks
    q, k, v, z, idx, coef, ranks, V, stride, G = _case(12, stride=1, R=3)
    assert (ranks == 0).all()
    np.testing.assert_allclose(J.joint_decode_coef(q, z, idx, coef, ranks, V, 1, G), _sdpa(q, k, v),
                               atol=1e-10)


def test_decode_tokens_on_their_anchor_mean_are_exact_at_rank_one():
    # coded tokens placed on the midpoint of two neighbouring anchors (anchors spread along a line,
    # so those two are the nearest) have a zero residual: the anchor term alone must reproduce them
    # (a dropped or mis-weighted anchor term fails here)
    rng = np.random.default_rng(13)
    G, grp, n, d, stride, c, w = 2, 2, 48, 4, 6, 2, 4
    D = 2 * G * d
    u = rng.standard_normal(D)
    u /= np.linalg.norm(u)
    pos = J.anchor_positions(n, stride)
    z = np.zeros((n, D))
    for j, p in enumerate(pos):
        z[p] = 10.0 * j * u + 0.1 * rng.standard_normal(D)
    exact = J.exact_mask(n, stride, w)
    for t in np.flatnonzero(~exact):
        j = min(t // stride, pos.size - 2)
        z[t] = (z[pos[j]] + z[pos[j + 1]]) / 2
    for t in np.flatnonzero(exact):
        if t not in pos:
            z[t] = rng.standard_normal(D)
    idx, _ = J.nearest_anchors(z, stride, c)
    np.testing.assert_allclose(J.residual(z, idx, stride)[~exact], 0, atol=1e-12)
    V = _orthonormal_rows(rng, 5, D)
    coef = J.joint_project(J.residual(z, idx, stride), V)
    ranks = np.where(exact, 0, 1)
    q = rng.standard_normal((G * grp, d)) * 0.3
    k, v = J.split_joint(z, G, d)
    np.testing.assert_allclose(J.joint_decode_coef(q, z, idx, coef, ranks, V, stride, G),
                               _sdpa(q, k, v), atol=1e-10)


def test_encode_joint_at_kappa_one_reconstructs_exactly():
    rng = np.random.default_rng(14)
    G, grp, n, d, w = 1, 2, 64, 4, 4
    D = 2 * G * d
    k = rng.standard_normal((G, n, d))
    v = rng.standard_normal((G, n, d))
    q_win = rng.standard_normal((w, G * grp, d))
    V = _orthonormal_rows(rng, D, D)
    enc = J.encode_joint(q_win, k, v, V, grp, 1.0, 1, 8, 4, w)
    exact = J.exact_mask(n, 8, w)
    assert (enc["ranks"][~exact] == D).all() and (enc["ranks"][exact] == 0).all()
    zh = J.joint_reconstruct(enc["z"], enc["idx"], enc["coef"], enc["ranks"], V, 8)
    np.testing.assert_allclose(zh, J.joint_vector(k, v), atol=1e-12)


def test_footprint_matches_the_papers_measured_memory():
    # Table "Coefficient quantization sweep" (Llama, keep 20 %): memory ~20 % in fp16, ~14 % with
    # 8-bit, ~10 % with 4-bit and ~9 % with 3-bit coefficients; Sec. 3.1 "Budget": the anchor
    # indices add 0.2 % of the cache. Paper setting: D = 2 x 8 x 128, stride 16, c = 4, w = 64; a
    # 16K context; group parameters of two fp16 values per 32 coefficients.
    n, D, stride, w, kappa, c = 16384, 2048, 16, 64, 0.2, 4
    for bits, paper in ((16, 20.0), (8, 14.0), (4, 10.0), (3, 9.0)):
        got = 100 * J.joint_footprint(n, D, stride, w, kappa, c, coef_bits=bits)
        assert abs(got - paper) <= 1.5, (bits, got)
    idx = 100 * (J.joint_footprint(n, D, stride, w, kappa, c) - J.joint_footprint(n, D, stride, w, kappa, 0))
    assert 0.15 <= idx <= 0.25
    # the budget is matched: without quantization or indices the footprint is kappa up to the floor
    assert abs(J.joint_footprint(n, D, stride, w, kappa, 0) - kappa) < 1e-6
