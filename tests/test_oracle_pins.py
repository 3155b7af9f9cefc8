"""Pins of the CPU oracle against facts that do not come from the oracle itself: library routines
(torch SDPA for softmax attention weights, numpy QR), closed forms, brute force on tiny inputs,
hand-derived values (tests/golden/) and invariants the paper states by construction."""
import json
import math
import os

import numpy as np
import pytest
import torch

import oracle as O
import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _sdpa_weights(q, k, causal_pos):
    """Attention weights from torch's scaled_dot_product_attention (fp64), obtained by attending
    to an identity value matrix: row q of the output is alpha_{q, .}."""
    w, d = q.shape
    n = k.shape[0]
    mask = torch.arange(n)[None, :] <= torch.as_tensor(causal_pos)[:, None]
    out = torch.nn.functional.scaled_dot_product_attention(
        torch.as_tensor(q, dtype=torch.float64)[None, None],
        torch.as_tensor(k, dtype=torch.float64)[None, None],
        torch.eye(n, dtype=torch.float64)[None, None], attn_mask=mask[None, None])
    return out[0, 0].numpy()


# ------------------------------------------------------------------------------ salience

@pytest.mark.parametrize("G,grp,w,N,d", [(1, 1, 1, 9, 4), (2, 3, 4, 23, 8), (1, 4, 5, 40, 16)])
def test_salience_matches_sdpa_weights(G, grp, w, N, d):
    rng = np.random.default_rng(G * 100 + N)
    q = rng.standard_normal((w, G * grp, d))
    k = rng.standard_normal((G, N, d)) * 1.5
    pos = N - w + np.arange(w)
    acc = np.zeros(N)
    for h in range(G * grp):
        acc += _sdpa_weights(q[:, h], k[h // grp], pos).sum(axis=0)
    want = acc[: N - w] / (w * G * grp)
    got = O.salience_raw(q, k, grp)
    np.testing.assert_allclose(got, want, rtol=1e-12, atol=1e-15)


def test_salience_equal_keys_closed_form():
    # every key equal => each window query spreads weight 1/(p+1) over tokens 0..p
    w, G, grp, N, d = 6, 2, 2, 30, 8
    rng = np.random.default_rng(3)
    q = rng.standard_normal((w, G * grp, d))
    k = np.tile(rng.standard_normal(d), (G, N, 1))
    got = O.salience_raw(q, k, grp)
    want = np.mean([1.0 / (N - w + i + 1) for i in range(w)])
    np.testing.assert_allclose(got, np.full(N - w, want), rtol=1e-13)


def test_salience_rows_sum_to_one():
    # with w = 1 the single query sees every token: coded weight + own weight = 1 per head
    rng = np.random.default_rng(5)
    G, grp, N, d = 2, 2, 17, 8
    q = rng.standard_normal((1, G * grp, d))
    k = rng.standard_normal((G, N, d))
    s = O.salience_raw(q, k, grp)
    last = np.mean([_sdpa_weights(q[:, h], k[h // grp], [N - 1])[0, N - 1]
                    for h in range(G * grp)])
    assert abs(s.sum() + last - 1.0) < 1e-13


def test_salience_picks_gqa_group():
    # a key that matches only head 3's query raises salience only through KV head 3 // grp
    G, grp, N, d = 2, 2, 12, 4
    q = np.zeros((1, 4, d))
    q[0, 3] = [10.0, 0, 0, 0]
    k = np.zeros((G, N, d))
    k[1, 5] = [10.0, 0, 0, 0]
    s = O.salience_raw(q, k, grp)
    assert np.argmax(s) == 5
    k2 = np.zeros((G, N, d))
    k2[0, 5] = [10.0, 0, 0, 0]
    assert np.ptp(O.salience_raw(q, k2, grp)) < 1e-15


def test_pool_delta_and_edges():
    s = np.zeros(11)
    s[5] = 1.0
    p = O.pool(s, 5)
    np.testing.assert_allclose(p, [0, 0, 0, .2, .2, .2, .2, .2, 0, 0, 0])
    c = O.pool(np.ones(6), 5)
    np.testing.assert_allclose(c, [3 / 5, 4 / 5, 1, 1, 4 / 5, 3 / 5])
    np.testing.assert_allclose(O.pool(np.arange(4.0), 1), np.arange(4.0))


# ----------------------------------------------------------------------- normalisation

def test_normalize_fp32_values():
    s = np.array([0.5, 0.25, 1.0, 0.75, 0.25], dtype=np.float32)
    np.testing.assert_array_equal(O.normalize(s), np.array([1 / 3, 0, 1, 2 / 3, 0], np.float32))
    assert O.normalize(s).dtype == np.float32
    np.testing.assert_array_equal(O.normalize(np.full(4, 7.0, np.float32)), np.ones(4, np.float32))
    np.testing.assert_array_equal(O.normalize(s, O.UNIFORM), np.ones(5, np.float32))


# ------------------------------------------------------------------- budget and ranks

def test_budget_golden():
    with open(os.path.join(GOLDEN, "budgets.json")) as f:
        cases = json.load(f)["cases"]
    for c in cases:
        assert O.coded_budget(c["n_ctx"], c["head_dim"], c["window"], c["budget_frac"]) == c["B_c"], c


def test_rank_at_golden():
    with open(os.path.join(GOLDEN, "rank_at.json")) as f:
        cases = json.load(f)["cases"]
    for c in cases:
        got = O.rank_at(np.float32(c["lambda"]), np.array(c["s_hat"], np.float32), c["r_min"],
                        c["r_max"])
        assert got.tolist() == c["ranks"], c


def _check_invariants(shat, B, rmin, rmax, r, status):
    n = shat.size
    if status == O.FLOOR_BINDS:
        assert rmin * n > B and np.all(r == rmin)
        return
    assert r.sum() <= B
    assert r.min() >= rmin and r.max() <= rmax
    order = np.argsort(shat, kind="stable")
    assert np.all(np.diff(r[order]) >= 0), "rank must be non-decreasing in salience"


@pytest.mark.parametrize("seed", range(8))
def test_allocate_invariants_and_maximality(seed):
    rng = np.random.default_rng(seed)
    n = int(rng.integers(5, 400))
    rmin, rmax = 16, 128
    shat = O.normalize(rng.exponential(size=n).astype(np.float32))
    B = int(rng.integers(rmin * n, rmax * n))
    r, bits, status, total = O.allocate(shat, B, rmin, rmax)
    _check_invariants(shat, B, rmin, rmax, r, status)
    assert total == r.sum()
    if bits < O.F32_MAX_BITS:   # the next fp32 level would overspend
        assert O.rank_at(O.bits_to_f32(bits + 1), shat, rmin, rmax).sum() > B


def test_allocate_two_token_closed_form():
    # s_hat = [0, 1]: the salient token takes every unit above the floor, up to r_max
    for extra in [0, 1, 7, 50, 112]:
        r, _, st, _ = O.allocate(np.array([0, 1], np.float32), 32 + extra, 16, 128)
        assert st == O.OK and r.tolist() == [16, 16 + extra]


@pytest.mark.parametrize("n,B", [(4, 70), (10, 255), (7, 16 * 7), (3, 3 * 128 - 1)])
def test_allocate_uniform_is_flat(n, B):
    r, _, st, _ = O.allocate(np.ones(n, np.float32), B, 16, 128)
    assert st == O.OK and np.all(r == min(128, B // n))


def test_allocate_full_and_infeasible():
    shat = np.linspace(0, 1, 9).astype(np.float32)
    r, _, st, _ = O.allocate(shat, 128 * 9, 16, 128)
    assert st == O.OK and np.all(r == 128)
    r, _, st, _ = O.allocate(shat, 16 * 9 - 1, 16, 128)
    assert st == O.FLOOR_BINDS and np.all(r == 16)


def _fp32_threshold(sh, k, rmin, rmax):
    """Smallest fp32 lambda >= 0 with rank_t(lambda) >= k, found by an ulp walk around the real
    threshold (k - r_min) / s_hat."""
    def rank(lam):
        return int(O.rank_at(np.float32(lam), np.array([sh], np.float32), rmin, rmax)[0])
    lam = np.float32((k - rmin) / float(sh))
    while rank(lam) >= k and lam > 0:
        lam = np.nextafter(lam, np.float32(0))
    while rank(lam) < k:
        lam = np.nextafter(lam, np.float32(np.inf))
    return lam


@pytest.mark.parametrize("seed", range(12))
def test_allocate_brute_force_tiny(seed):
    rng = np.random.default_rng(1000 + seed)
    n = int(rng.integers(1, 7))
    rmin, rmax = 2, 9
    shat = O.normalize(rng.random(n).astype(np.float32))
    if seed % 3 == 0:
        shat[: n // 2] = shat[-1]   # ties
    B = int(rng.integers(rmin * n, rmax * n + 1))
    r, bits, st, _ = O.allocate(shat, B, rmin, rmax)
    # every place the allocation can change, by brute force
    cands = {np.float32(0.0), np.float32(np.finfo(np.float32).max)}
    for sh in shat:
        if sh <= 0:
            continue
        for k in range(rmin + 1, rmax + 1):
            th = _fp32_threshold(sh, k, rmin, rmax)
            if np.isfinite(th) and th > 0:
                cands.add(np.nextafter(th, np.float32(0)))
    feas = [c for c in cands if O.rank_at(c, shat, rmin, rmax).sum() <= B]
    best = max(feas) if B < rmax * n else np.float32(np.finfo(np.float32).max)
    np.testing.assert_array_equal(r, O.rank_at(best, shat, rmin, rmax))


@pytest.mark.parametrize("seed", range(4))
def test_allocate_tracks_algorithm1_continuous(seed):
    rng = np.random.default_rng(77 + seed)
    n, rmin, rmax = 300, 16, 128
    shat = O.normalize(rng.lognormal(sigma=1.5, size=n).astype(np.float32))
    B = int(25.5 * n)
    r, _, st, _ = O.allocate(shat, B, rmin, rmax)
    rc = O.waterfill_continuous(shat, B, rmin, rmax)
    assert abs(rc.sum() - B) < 1e-6 * B
    assert np.all(rc >= rmin - 1e-9) and np.all(rc <= rmax + 1e-9)
    assert np.all(r >= np.floor(rc) - 1)          # integer level is at or above the continuous one
    assert B - n <= r.sum() <= B


# ------------------------------------------------------------------------- pack tables

@pytest.mark.parametrize("seed", range(5))
def test_pack_tables_brute_force(seed):
    rng = np.random.default_rng(seed)
    rmin, rmax = 3, 12
    ranks = rng.integers(rmin, rmax + 1, size=int(rng.integers(1, 300)))
    count, base, pos, perm = O.pack_tables(ranks, rmin, rmax)
    order = sorted(range(ranks.size), key=lambda t: (ranks[t], t))
    assert perm.tolist() == order
    assert count.sum() == ranks.size
    for t in range(ranks.size):
        assert pos[t] == sum(1 for u in range(t) if ranks[u] == ranks[t])
    off = 0
    for r in range(rmin, rmax + 1):
        assert base[r] == off
        off += r * (-(-int(count[r]) // 8) * 8)
    assert base[rmax + 1] == off
    assert np.all(base[: rmin + 1] == 0)


def test_pack_roundtrip():
    rng = np.random.default_rng(9)
    rmin, rmax, n = 2, 8, 61
    ranks = rng.integers(rmin, rmax + 1, size=n)
    coef = rng.standard_normal((n, rmax))
    count, base, pos, _ = O.pack_tables(ranks, rmin, rmax)
    buf = O.pack_stream(coef, ranks, count, base, pos)
    assert buf.size == base[rmax + 1]
    np.testing.assert_array_equal(O.unpack_stream(buf, ranks, count, base, pos),
                                  O.truncate(coef, ranks))
    assert np.count_nonzero(buf) == int(ranks.sum())   # pads are zero


# -------------------------------------------------------------------------- projection

def test_basis_is_orthonormal_and_projection_is_parseval():
    wl = synth.workload("tiny")
    uk, _ = synth.bases(wl, 0)
    u = uk[0]
    np.testing.assert_allclose(u @ u.T, np.eye(wl.head_dim), atol=1e-12)
    x = np.random.default_rng(2).standard_normal((50, wl.head_dim))
    c = O.project(x, u)
    np.testing.assert_allclose((c ** 2).sum(1), (x ** 2).sum(1), rtol=1e-12)
    np.testing.assert_allclose(O.reconstruct(c, np.full(50, wl.head_dim), u), x, atol=1e-12)
    # truncation error is the dropped energy and is non-increasing in the rank
    errs = [((O.reconstruct(c, np.full(50, r), u) - x) ** 2).sum() for r in range(0, 129, 8)]
    dropped = [(c[:, r:] ** 2).sum() for r in range(0, 129, 8)]
    np.testing.assert_allclose(errs, dropped, rtol=1e-9, atol=1e-9)
    assert all(a >= b for a, b in zip(errs, errs[1:]))


def test_projection_energy_matches_spectrum():
    # with the generator's frame as basis, E[c_j^2] = (sigma_j * scale)^2 + noise^2
    wl = synth.workload("llama1", n_kv_heads=1, n_ctx=8192)
    k, _ = synth.layer_kv(wl, 0, 0, out_dtype=torch.float64)
    uk, _ = synth.bases(wl, 0)
    c = O.project(k[0].numpy(), uk[0])
    sig = synth.spectrum(wl) * synth._scale(wl)
    want = sig ** 2 + wl.noise_std ** 2
    got = (c ** 2).mean(0)
    np.testing.assert_allclose(got[:40], want[:40], rtol=0.08)
    np.testing.assert_allclose(got[40:], want[40:], rtol=0.08)


# ------------------------------------------------------------------------------ decode

def _sdpa_attention(q, k, v):
    H = q.shape[0]
    G = k.shape[0]
    kk = torch.as_tensor(k).repeat_interleave(H // G, dim=0)[None]
    vv = torch.as_tensor(v).repeat_interleave(H // G, dim=0)[None]
    out = torch.nn.functional.scaled_dot_product_attention(torch.as_tensor(q)[None, :, None],
                                                           kk, vv)
    return out[0, :, 0].numpy()


def test_attention_matches_sdpa():
    rng = np.random.default_rng(4)
    q = rng.standard_normal((8, 16))
    k = rng.standard_normal((2, 50, 16))
    v = rng.standard_normal((2, 50, 16))
    np.testing.assert_allclose(O.attention(q, k, v), _sdpa_attention(q, k, v), atol=1e-13)


def test_decode_routes_agree_and_full_rank_is_exact():
    wl = synth.workload("tiny", n_ctx=300, window=8, n_kv_heads=2)
    k, v = synth.layer_kv(wl, 0, 0, out_dtype=torch.float64)
    k, v = k.numpy(), v.numpy()
    uk, uv = synth.bases(wl, 0)
    q = np.random.default_rng(1).standard_normal((wl.n_q_heads, wl.head_dim))
    ck = np.stack([O.project(k[g], uk[g]) for g in range(2)])
    cv = np.stack([O.project(v[g], uv[g]) for g in range(2)])
    ranks = np.random.default_rng(2).integers(16, 129, size=300)
    a = O.decode_coef(q, ck, cv, ranks, uk, uv)
    b = O.decode_recon(q, ck, cv, ranks, uk, uv)
    np.testing.assert_allclose(a, b, atol=1e-10)
    full = O.decode_coef(q, ck, cv, np.full(300, 128), uk, uv)
    np.testing.assert_allclose(full, _sdpa_attention(q, k, v), atol=1e-10)


def test_decode_with_exact_tail():
    wl = synth.workload("tiny", n_ctx=200, window=8, n_kv_heads=2)
    k, v = synth.layer_kv(wl, 0, 0, out_dtype=torch.float64)
    k, v = k.numpy(), v.numpy()
    uk, uv = synth.bases(wl, 0)
    rng = np.random.default_rng(11)
    q = rng.standard_normal((wl.n_q_heads, wl.head_dim))
    tk = rng.standard_normal((2, 5, wl.head_dim))
    tv = rng.standard_normal((2, 5, wl.head_dim))
    ck = np.stack([O.project(k[g], uk[g]) for g in range(2)])
    cv = np.stack([O.project(v[g], uv[g]) for g in range(2)])
    ranks = rng.integers(16, 129, size=200)
    a = O.decode_coef(q, ck, cv, ranks, uk, uv, tk, tv)
    np.testing.assert_allclose(a, O.decode_recon(q, ck, cv, ranks, uk, uv, tk, tv), atol=1e-10)
    full = O.decode_coef(q, ck, cv, np.full(200, 128), uk, uv, tk, tv)
    want = _sdpa_attention(q, np.concatenate([k, tk], 1), np.concatenate([v, tv], 1))
    np.testing.assert_allclose(full, want, atol=1e-10)


def _sdpa_window(q, k, v, n_tail):
    """Causal attention of the last n_q of n = N + n_tail tokens, from torch SDPA (fp64):
    query i (token n - n_q + i) sees tokens 0 .. n - n_q + i. q [n_q][H][d]; k, v [G][n][d]."""
    n_q, H, d = q.shape
    G, n, _ = k.shape
    kk = torch.as_tensor(k).repeat_interleave(H // G, dim=0)[None]      # [1][H][n][d]
    vv = torch.as_tensor(v).repeat_interleave(H // G, dim=0)[None]
    qq = torch.as_tensor(q).permute(1, 0, 2)[None]                      # [1][H][n_q][d]
    mask = torch.arange(n)[None, :] <= (n - n_q + torch.arange(n_q))[:, None]
    out = torch.nn.functional.scaled_dot_product_attention(qq, kk, vv, attn_mask=mask[None, None])
    return out[0].permute(1, 0, 2).numpy()


def _window_case(n_ctx=160, n_tail=9, n_q=4, seed=21):
    wl = synth.workload("tiny", n_ctx=n_ctx, window=8, n_kv_heads=2)
    k, v = synth.layer_kv(wl, 0, 0, out_dtype=torch.float64)
    k, v = k.numpy(), v.numpy()
    uk, uv = synth.bases(wl, 0)
    rng = np.random.default_rng(seed)
    q = rng.standard_normal((n_q, wl.n_q_heads, wl.head_dim))
    tk = rng.standard_normal((2, n_tail, wl.head_dim))
    tv = rng.standard_normal((2, n_tail, wl.head_dim))
    ck = np.stack([O.project(k[g], uk[g]) for g in range(2)])
    cv = np.stack([O.project(v[g], uv[g]) for g in range(2)])
    return k, v, uk, uv, q, tk, tv, ck, cv, rng


def test_window_decode_full_rank_is_causal_attention():
    """At full rank the window decode is causal attention over cache + tail (torch SDPA, masked)."""
    k, v, uk, uv, q, tk, tv, ck, cv, _ = _window_case()
    got = O.decode_window(q, ck, cv, np.full(k.shape[1], 128), uk, uv, tk, tv)
    want = _sdpa_window(q, np.concatenate([k, tk], 1), np.concatenate([v, tv], 1), tk.shape[1])
    np.testing.assert_allclose(got, want, atol=1e-10)


def test_window_decode_sees_no_later_token():
    """Query i is unchanged when the tail tokens after its own position change, and changes when
    an earlier one does; with n_q = 1 it is the single-query decode over the whole tail."""
    k, v, uk, uv, q, tk, tv, ck, cv, rng = _window_case()
    ranks = rng.integers(16, 129, size=k.shape[1])
    n_tail, n_q = tk.shape[1], q.shape[0]
    base = O.decode_window(q, ck, cv, ranks, uk, uv, tk, tv)
    tk2, tv2 = tk.copy(), tv.copy()
    tk2[:, -1] += 3.0
    tv2[:, -1] -= 2.0                                   # the last query's own token
    moved = O.decode_window(q, ck, cv, ranks, uk, uv, tk2, tv2)
    np.testing.assert_array_equal(moved[:-1], base[:-1])
    assert np.abs(moved[-1] - base[-1]).max() > 1e-6
    one = O.decode_window(q[-1:], ck, cv, ranks, uk, uv, tk, tv)
    np.testing.assert_allclose(one[0], O.decode_coef(q[-1], ck, cv, ranks, uk, uv, tk, tv), atol=1e-12)
    with pytest.raises(ValueError):
        O.decode_window(np.zeros((n_tail + 1,) + q.shape[1:]), ck, cv, ranks, uk, uv, tk, tv)


def test_decode_single_token_and_flat_scores():
    d = 16
    rng = np.random.default_rng(8)
    u = np.linalg.qr(rng.standard_normal((d, d)))[0].T
    ck = rng.standard_normal((1, 1, d))
    cv = rng.standard_normal((1, 1, d))
    q = rng.standard_normal((2, d))
    o = O.decode_coef(q, ck, cv, np.array([5]), u[None], u[None])
    vhat = O.reconstruct(cv[0], np.array([5]), u)[0]
    np.testing.assert_allclose(o, np.stack([vhat, vhat]), atol=1e-13)
    ck = rng.standard_normal((1, 7, d))
    cv = rng.standard_normal((1, 7, d))
    ranks = rng.integers(1, d + 1, size=7)
    o = O.decode_coef(np.zeros((1, d)), ck, cv, ranks, u[None], u[None])
    np.testing.assert_allclose(o[0], O.reconstruct(cv[0], ranks, u).mean(0), atol=1e-13)


def test_budget_one_matches_uncompressed_attention():
    wl = synth.workload("tiny", n_ctx=512, budget_frac=1.0)
    k, v = synth.layer_kv(wl, 0, 0)
    qw = synth.window_queries(wl, 0, 0)
    uk, uv = synth.bases(wl, 0)
    enc = O.encode_layer(qw.numpy(), k.numpy(), v.numpy(), uk, uv, wl.group, 1.0, wl.r_min)
    assert np.all(enc["ranks"] == wl.head_dim) and enc["status"] == O.OK
    q = synth.decode_queries(wl, 0, 0, 1)[0].numpy()
    o = O.decode_coef(q, enc["coef_k"], enc["coef_v"], enc["ranks"], uk, uv)
    np.testing.assert_allclose(o, O.attention(q, k.numpy(), v.numpy()), atol=1e-5)


def test_uniform_mode_gives_one_rank():
    wl = synth.workload("tiny", n_ctx=700)
    k, v = synth.layer_kv(wl, 0, 0)
    uk, uv = synth.bases(wl, 0)
    enc = O.encode_layer(synth.window_queries(wl, 0, 0).numpy(), k.numpy(), v.numpy(), uk, uv,
                         wl.group, wl.budget_frac, wl.r_min, mode=O.UNIFORM)
    coded = enc["ranks"][: wl.n_ctx - wl.window]
    bc = O.coded_budget(wl.n_ctx, wl.head_dim, wl.window, wl.budget_frac)
    assert np.all(coded == bc // coded.size)


def test_salient_outliers_get_higher_ranks():
    wl = synth.workload("tiny")
    k, v = synth.layer_kv(wl, 0, 0)
    uk, uv = synth.bases(wl, 0)
    enc = O.encode_layer(synth.window_queries(wl, 0, 0).numpy(), k.numpy(), v.numpy(), uk, uv,
                         wl.group, wl.budget_frac, wl.r_min)
    out = synth.outlier_tokens(wl, 0, 0)
    r = enc["ranks"][: wl.n_ctx - wl.window]
    assert r[out].mean() > r.mean()
    assert enc["total"] <= O.coded_budget(wl.n_ctx, wl.head_dim, wl.window, wl.budget_frac)
