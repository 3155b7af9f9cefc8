"""Pins of the oracle's coefficient quantization (group-wise b-bit, Sec. 3.3 "Composability"), on the
CPU: what the definition of asymmetric min-max quantization with fp16 parameters fixes, checked
against closed forms, brute force and invariants rather than against itself."""
import numpy as np
import pytest

import oracle as O


@pytest.mark.parametrize("bits", [4, 8])
def test_round_trip_error_within_half_a_step(bits):
    rng = np.random.default_rng(bits)
    for _ in range(200):
        x = (rng.standard_normal(32) * rng.uniform(0.01, 20)).astype(np.float32)
        q, lo, step = O.quantize_group(x, bits)
        xh = O.dequantize_group(q, lo, step)
        bound = 0.5 * np.float32(step) + 2.0 ** -10 * np.abs(x).max()
        assert np.abs(xh - x).max() <= bound
        assert q.max() <= 2 ** bits - 1


@pytest.mark.parametrize("bits", [4, 8])
def test_grid_values_round_trip_exactly(bits):
    """Values lo + k * step with fp16 lo and step (computed exactly in fp32) are reproduced."""
    lo, step = np.float16(-1.5), np.float16(0.25)
    k = np.array([0, 1, 3, 2 ** bits - 1, 7, 2 ** bits - 1, 0, 5], dtype=np.float32)
    x = (np.float32(lo) + k * np.float32(step)).astype(np.float32)
    q, lo2, step2 = O.quantize_group(x, bits)
    assert lo2 == lo and step2 == step
    np.testing.assert_array_equal(q, k.astype(np.uint8))
    np.testing.assert_array_equal(O.dequantize_group(q, lo2, step2), x)


def test_extremes_and_constant_groups():
    x = np.array([3.0, -2.0, 0.5, 1.25, -2.0, 3.0], dtype=np.float32)
    for bits in (4, 8):
        q, lo, step = O.quantize_group(x, bits)
        assert q[1] == 0 and q[4] == 0                   # the minimum maps to code 0
        assert q[0] == 2 ** bits - 1 and q[5] == 2 ** bits - 1   # the maximum to the top code
    q, lo, step = O.quantize_group(np.full(7, 0.375, dtype=np.float32), 4)
    assert step == 0 and np.all(q == 0)
    np.testing.assert_array_equal(O.dequantize_group(q, lo, step), np.full(7, 0.375, np.float32))


def test_more_bits_is_more_accurate():
    rng = np.random.default_rng(0)
    x = rng.standard_normal((500, 32)).astype(np.float32)
    err = {b: np.mean([np.abs(O.dequantize_group(*O.quantize_group(r, b)) - r).max() for r in x])
           for b in (4, 8)}
    # uniform rounding error: about range / (2^b - 1) / 4 on average
    assert err[8] < err[4] / 10


def test_row_bytes_closed_form():
    assert O.qrow_bytes(128, 4) == 64 + 16 == 80
    assert O.qrow_bytes(128, 8) == 128 + 16 == 144
    assert O.qrow_bytes(8, 4) == 16          # 4 code bytes + one group's 4 parameter bytes -> 16
    assert O.qrow_bytes(40, 8) == 48         # 40 code bytes + 2 groups -> 48
    for tl in range(8, 129, 8):
        for b in (4, 8):
            n = O.qrow_bytes(tl, b)
            assert n % 16 == 0 and tl * b // 8 + 4 * ((tl + 31) // 32) <= n < tl * b // 8 + 4 * ((tl + 31) // 32) + 16


@pytest.mark.parametrize("bits", [4, 8])
def test_stream_bytes_by_brute_force_and_static_cap(bits):
    """qpack_tables equals a tile-by-tile count, and never exceeds the static cap for random
    allocations within the budget (including the floor-binds and all-at-r_max extremes)."""
    n_ctx, d, w, rmin = 3000, 128, 32, 16
    rng = np.random.default_rng(bits)
    for kappa in (0.1, 0.2, 0.5, 1.0):
        cap = O.qpacked_cap_bytes(n_ctx, d, w, kappa, rmin, bits)
        bc = O.coded_budget(n_ctx, d, w, kappa)
        n_coded = n_ctx - w
        for trial in range(20):
            if trial == 0:
                rc = np.full(n_coded, rmin)
            elif trial == 1:
                rc = np.full(n_coded, min(d, max(rmin, bc // n_coded)))
            else:   # random ranks scaled under the budget
                raw = rng.exponential(size=n_coded)
                rc = np.clip(np.floor(rmin + raw / raw.sum() * max(bc - rmin * n_coded, 0)), rmin, d).astype(int)
            ranks = np.concatenate([rc, np.full(w, d)])
            count = np.bincount(ranks, minlength=d + 1)
            qbase = O.qpack_tables(count, rmin, d, bits)
            brute = 0
            for r in range(rmin, d + 1):
                n8 = (int(count[r]) + 7) // 8 * 8
                for t0 in range(0, n8, 128):
                    brute += r * O.qrow_bytes(min(128, n8 - t0), bits)
            assert qbase[-1] == brute
            if rc.sum() <= max(bc, rmin * n_coded):
                assert brute <= cap, (kappa, trial, brute, cap)


def test_quantize_coefficients_groups_follow_the_bucket_layout():
    """Groups are 32 consecutive bucket slots of one coefficient row inside a 128-slot tile:
    tokens of one group share (offset, step); padding slots count as zeros."""
    rng = np.random.default_rng(5)
    n, d = 300, 128
    ranks = rng.choice([16, 20, 128], size=n, p=[0.7, 0.25, 0.05])
    count, base, pos, perm = O.pack_tables(ranks, 16, d)
    coef = rng.standard_normal((n, d)).astype(np.float32)
    codes, lo, step, deq = O.quantize_coefficients(coef, ranks, count, pos, 4)
    for t in range(n):
        r = ranks[t]
        assert np.all(codes[t, r:] == 0) and np.all(deq[t, r:] == 0)
        # members of the same group: same bucket, same tile, same 32-slot block
        same = [u for u in range(n) if ranks[u] == r and pos[u] // 32 == pos[t] // 32]
        for j in range(0, r, 7):
            assert all(lo[u, j] == lo[t, j] and step[u, j] == step[t, j] for u in same)
            members = coef[same, j]
            n8 = (int(count[r]) + 7) // 8 * 8
            blk = pos[t] // 32 * 32
            n_pad = min(blk + 32, n8) - blk - len(same)
            x = np.concatenate([members, np.zeros(n_pad, np.float32)])
            assert lo[t, j] == np.float16(x.min())
    err = np.abs(deq - O.truncate(coef, ranks))
    assert err.max() < 0.5            # 4-bit of unit-variance values: about range/30


def test_decode_on_8_bit_coefficients_close_to_unquantized():
    rng = np.random.default_rng(9)
    G, N, d, grp = 1, 700, 128, 4
    ranks = np.concatenate([rng.integers(16, 40, N - 32), np.full(32, d)])
    count, base, pos, perm = O.pack_tables(ranks, 16, d)
    uk = np.linalg.qr(rng.standard_normal((d, d)))[0].T[None]
    uv = np.linalg.qr(rng.standard_normal((d, d)))[0].T[None]
    ck = (rng.standard_normal((G, N, d))).astype(np.float32)
    cv = (rng.standard_normal((G, N, d))).astype(np.float32)
    q = rng.standard_normal((G * grp, d))
    ref = O.decode_coef(q, ck, cv, ranks, uk, uv)
    for bits, tol in ((8, 0.02), (4, 0.3)):
        dk = O.quantize_coefficients(ck[0], ranks, count, pos, bits)[3][None]
        dv = O.quantize_coefficients(cv[0], ranks, count, pos, bits)[3][None]
        got = O.decode_coef(q, dk, dv, ranks, uk, uv)
        rel = np.abs(got - ref).max(axis=-1) / np.abs(ref).max(axis=-1)
        assert rel.max() < tol, (bits, rel.max())
