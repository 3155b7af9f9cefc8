"""GPU vs oracle parity, through the C ABI, element by element on the same seeded inputs.

Bars: ranks, realised sums and every layout table bit-exact (from identical fp32 salience / ranks);
salience within 1e-4 relative; coefficients within their storage rounding; decode attention within
2e-2 max-abs (bf16) or 1e-4 (fp32) of the fp64 oracle and, per output row, within 2^-6 (bf16) or
1e-4 (fp32) of that row's largest magnitude (the derivation is in gpu_helpers.py)."""
import numpy as np
import pytest
import torch

from gpu_helpers import (O, V, cfg_for, coef_tol, decode_close, decode_errors, f64, gpu_allocate,
                         gpu_decode, gpu_encode, gpu_pack, oracle_layer, salience_close, synth,
                         unpack)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _gpu(vlib):
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")


# workloads small enough for the oracle, spanning several tiles and ragged tails
CASES = {
    "tiny": synth.workload("tiny"),
    "llama_ragged": synth.workload("llama1", n_kv_heads=2, n_ctx=4096 + 37, batch=2, n_layers=2),
    "qwen_g7": synth.workload("qwen", n_kv_heads=2, n_ctx=3000 + 5, n_layers=1),
    "group1": synth.workload("llama1", n_kv_heads=3, group=1, n_ctx=1500 + 3),
    "group2_f32": synth.workload("tiny", n_kv_heads=2, group=2, n_ctx=999, window=7),
}


def _inputs(wl):
    return synth.stack_inputs(wl, device="cpu")


@pytest.fixture(scope="module")
def inputs():
    return {name: _inputs(wl) for name, wl in CASES.items()}


# ----------------------------------------------------------------------------- salience

@pytest.mark.parametrize("name", list(CASES))
def test_salience_matches_oracle(inputs, name):
    wl = CASES[name]
    k, v, qw, bk, bv = inputs[name]
    cfg = cfg_for(wl)
    r = gpu_encode(cfg, k, v, qw, bk, bv)
    for b in range(wl.batch):
        for l in range(wl.n_layers):
            want = O.salience(f64(qw[b, l]), f64(k[b, l]), wl.group)
            ok, nbad, worst = salience_close(r["sal"][b, l].numpy(), want)
            assert ok, (name, b, l, nbad, worst)


# --------------------------------------------------------------------------- allocation

def _alloc_case(sal, wl, budget_frac=None, mode=O.SALIENCE):
    cfg = cfg_for(wl, mode=mode, budget_frac=budget_frac)
    ranks, realized, status = gpu_allocate(cfg, sal)
    bf = wl.budget_frac if budget_frac is None else budget_frac
    sal = np.asarray(sal, dtype=np.float32).reshape(wl.batch * wl.n_layers, -1)
    want_status = O.OK
    for i in range(sal.shape[0]):
        wr, st, tot = O.allocate_layer(sal[i], wl.n_ctx, wl.head_dim, wl.window, bf, wl.r_min, mode)
        np.testing.assert_array_equal(ranks.reshape(sal.shape[0], -1)[i], wr)
        assert realized.reshape(-1)[i] == tot
        want_status = max(want_status, st)
    assert status == want_status


@pytest.mark.parametrize("name", list(CASES))
def test_allocation_bit_exact_from_oracle_salience(inputs, name):
    wl = CASES[name]
    k, v, qw, bk, bv = inputs[name]
    sal = np.stack([np.stack([O.salience(f64(qw[b, l]), f64(k[b, l]), wl.group).astype(np.float32)
                              for l in range(wl.n_layers)]) for b in range(wl.batch)])
    _alloc_case(sal, wl)


@pytest.mark.parametrize("kind", ["exponential", "ties", "constant", "denormal", "spiky",
                                  "zeros_and_one", "huge_range"])
@pytest.mark.parametrize("budget_frac", [0.1, 0.2, 0.37, 1.0])
def test_allocation_bit_exact_edge_salience(kind, budget_frac):
    wl = synth.workload("llama1", n_ctx=5000 + 11, batch=2, n_layers=1)
    rng = np.random.default_rng(hash((kind, budget_frac)) % 2 ** 32)
    n = wl.n_ctx - wl.window
    shape = (wl.batch * wl.n_layers, n)
    if kind == "exponential":
        s = rng.exponential(size=shape)
    elif kind == "ties":
        s = rng.integers(0, 5, size=shape).astype(np.float64)
    elif kind == "constant":
        s = np.full(shape, 0.25)
    elif kind == "denormal":
        s = rng.random(shape) * 1e-39
    elif kind == "spiky":
        s = rng.random(shape) * 1e-6
        s[:, rng.integers(0, n, 20)] = 1.0
    elif kind == "zeros_and_one":
        s = np.zeros(shape)
        s[:, 7] = 1.0
    else:
        s = np.exp(rng.uniform(-80, 80, size=shape))
    _alloc_case(s.astype(np.float32), wl, budget_frac=budget_frac)


def test_allocation_uniform_mode_one_rank():
    wl = synth.workload("llama1", n_ctx=4096, n_layers=2)
    cfg = cfg_for(wl, mode=V.UNIFORM)
    ranks = torch.zeros((1, 2, wl.n_ctx), dtype=torch.uint8, device="cuda")
    realized = torch.zeros((1, 2), dtype=torch.int64, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    V.check(V.varrate_allocate(cfg, None, ranks, realized, status))
    torch.cuda.synchronize()
    coded = ranks[:, :, : wl.n_ctx - wl.window].cpu().numpy()
    bc = O.coded_budget(wl.n_ctx, wl.head_dim, wl.window, wl.budget_frac)
    assert np.all(coded == bc // coded.shape[-1])
    assert np.all(ranks[:, :, wl.n_ctx - wl.window:].cpu().numpy() == 128)


def test_allocation_floor_binds_status():
    wl = synth.workload("qwen", n_ctx=4096, n_kv_heads=4, n_layers=1)
    sal = np.random.default_rng(1).exponential(size=(1, wl.n_ctx - wl.window)).astype(np.float32)
    ranks, realized, status = gpu_allocate(cfg_for(wl, budget_frac=0.10), sal)
    assert status == V.FLOOR_BINDS
    assert np.all(ranks[0, 0, : wl.n_ctx - wl.window] == wl.r_min)


def test_allocation_empty_coded_set():
    wl = synth.workload("llama1", n_ctx=32, window=32)
    ranks, realized, status = gpu_allocate(cfg_for(wl), np.zeros((1, 0), np.float32))
    assert status == V.OK and np.all(ranks == 128) and realized.sum() == 0


# ---------------------------------------------------------------------- pack + project

@pytest.mark.parametrize("name", list(CASES))
def test_pack_tables_bit_exact_and_coefficients(inputs, name):
    wl = CASES[name]
    k, v, qw, bk, bv = inputs[name]
    cfg = cfg_for(wl)
    refs = [[oracle_layer(wl, k, v, qw, bk, bv, b, l) for l in range(wl.n_layers)]
            for b in range(wl.batch)]
    ranks = np.stack([np.stack([refs[b][l]["ranks"] for l in range(wl.n_layers)])
                      for b in range(wl.batch)])
    packed, status = gpu_pack(cfg, ranks, k, v, bk, bv)
    assert status == V.OK
    rtol, atol = coef_tol(cfg)
    for b in range(wl.batch):
        for l in range(wl.n_layers):
            ref = refs[b][l]
            np.testing.assert_array_equal(packed.bucket_count[b, l].cpu().numpy(), ref["count"])
            np.testing.assert_array_equal(packed.bucket_base[b, l].cpu().numpy(), ref["base"])
            np.testing.assert_array_equal(packed.pos[b, l].cpu().numpy(), ref["pos"])
            np.testing.assert_array_equal(packed.perm[b, l].cpu().numpy(), ref["perm"])
            total = int(ref["base"][-1])
            for g in range(wl.n_kv_heads):
                for kv, full in ((0, ref["coef_k"][g]), (1, ref["coef_v"][g])):
                    got = unpack(packed, b, l, g, kv, ref["ranks"], ref["count"], ref["base"], ref["pos"])
                    want = O.truncate(full, ref["ranks"])
                    err = np.abs(got - want) - (rtol * np.abs(want) + atol)
                    assert err.max() <= 0, (name, b, l, g, kv, float(err.max()))
                    # padding slots are zero and nothing lies beyond the last bucket's slots
                    buf = f64(packed.coef[b, l, g, kv])[:total]
                    assert np.count_nonzero(buf) <= int(ref["ranks"].sum())


def test_pack_rejects_corrupt_ranks():
    wl = synth.workload("llama1", n_kv_heads=1, n_ctx=1024)
    k, v, qw, bk, bv = synth.stack_inputs(wl)
    ranks = np.full((1, 1, 1024), 20, dtype=np.int64)
    ranks[0, 0, 100] = 3     # below r_min
    packed, status = gpu_pack(cfg_for(wl), ranks, k, v, bk, bv)
    assert status == V.ERR_CORRUPT
    # the poisoned table makes decode skip the layer instead of reading garbage
    assert packed.bucket_base[0, 0, -1].item() > packed.cap_elems


# ------------------------------------------------------------------------------ decode

def _decode_check(wl, inputs, mode=O.SALIENCE, budget_frac=None, n_steps=3, n_tail=0):
    k, v, qw, bk, bv = inputs
    cfg = cfg_for(wl, mode=mode, budget_frac=budget_frac)
    refs = [[oracle_layer(wl, k, v, qw, bk, bv, b, l, mode=mode, budget_frac=budget_frac)
             for l in range(wl.n_layers)] for b in range(wl.batch)]
    ranks = np.stack([np.stack([refs[b][l]["ranks"] for l in range(wl.n_layers)])
                      for b in range(wl.batch)])
    packed, status = gpu_pack(cfg, ranks, k, v, bk, bv)
    dt = synth.torch_dtype(wl)
    worst = (0.0, 0.0)
    for l in range(wl.n_layers):
        qs = synth.stack_decode_queries(wl, l, n_steps)
        tk = tv = None
        if n_tail:
            g = torch.Generator().manual_seed(77 + l)
            tk = torch.randn((wl.batch, wl.n_kv_heads, n_tail, wl.head_dim), generator=g).to(dt)
            tv = torch.randn((wl.batch, wl.n_kv_heads, n_tail, wl.head_dim), generator=g).to(dt)
        for step in range(n_steps):
            out, st = gpu_decode(cfg, packed, bk, bv, qs[step], l, tk, tv)
            assert st == V.OK
            for b in range(wl.batch):
                ref = refs[b][l]
                want = O.decode_coef(f64(qs[step][b]), ref["coef_k"], ref["coef_v"], ref["ranks"],
                                     f64(bk[l]), f64(bv[l]),
                                     None if tk is None else f64(tk[b]),
                                     None if tv is None else f64(tv[b]))
                assert decode_close(out[b], want, cfg), (l, step, b, decode_errors(out[b], want))
                worst = tuple(max(a, e) for a, e in zip(worst, decode_errors(out[b], want)))
    print(f"decode worst relative / absolute error: {worst[0]:.3e} / {worst[1]:.3e}")
    return worst


@pytest.mark.parametrize("name", list(CASES))
def test_decode_matches_oracle(inputs, name):
    _decode_check(CASES[name], inputs[name])


@pytest.mark.parametrize("n_tail", [1, 37, 160, 256])
def test_decode_with_exact_tail(inputs, n_tail):
    # the fused bf16 kernel stages up to 256 tail tokens (160 = a 32-token window plus 128 decode
    # steps appended after the cache)
    _decode_check(CASES["llama_ragged"], inputs["llama_ragged"], n_tail=n_tail, n_steps=2)


def test_decode_with_long_exact_tail(inputs):
    # more than 256 tail tokens: the bf16 call takes the general split-and-combine kernels
    _decode_check(CASES["llama_ragged"], inputs["llama_ragged"], n_tail=300, n_steps=1)


def test_decode_tail_only(inputs):
    """Empty coded set: the whole context is the exact window, plus an exact tail."""
    wl = synth.workload("llama1", n_kv_heads=2, n_ctx=32, window=32, batch=2)
    _decode_check(wl, synth.stack_inputs(wl), n_tail=45, n_steps=1)


def test_decode_uniform_mode(inputs):
    _decode_check(CASES["llama_ragged"], inputs["llama_ragged"], mode=O.UNIFORM, n_steps=2)


def test_decode_floor_binds(inputs):
    _decode_check(CASES["qwen_g7"], inputs["qwen_g7"], budget_frac=0.10, n_steps=2)


def _decode_with_ws(cfg, packed, bk, bv, q, layer, ws):
    out = torch.empty_like(q, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    V.check(V.varrate_decode_attn(cfg, packed, bk.cuda(), bv.cuda(), q.cuda(), layer, None, None, 0,
                                  out, status, ws), "varrate_decode_attn")
    torch.cuda.synchronize()
    return f64(out), int(status.item())


HEADER_BYTES = 33024   # decode workspace header: call count, exit counters, 2 x 4096 arrival counters


def _header(ws):
    h = ws[:HEADER_BYTES]
    calls = int(h[:8].view(torch.int64).item())
    arrived = h[256:].view(torch.int32).cpu().numpy().reshape(2, 4096)
    return calls, arrived


def test_decode_workspace_reuse_and_counter_check(inputs):
    """One zero-filled workspace serves decode calls of different shapes in any order, with outputs
    equal to those of a call on a fresh workspace; the header counts the calls. Counts left in the
    header by an earlier call (garbage, or a call that stopped after some thread blocks arrived) are
    reported as corrupt by the next call, and the call after that is clean again on the same
    workspace, without the caller clearing anything."""
    runs = []
    for name in ("llama_ragged", "qwen_g7"):
        wl = CASES[name]
        k, v, qw, bk, bv = inputs[name]
        cfg = cfg_for(wl)
        r = gpu_encode(cfg, k, v, qw, bk, bv)
        runs.append((cfg, r["packed"], bk, bv, synth.stack_decode_queries(wl, 0, 1)[0]))
    ref = [gpu_decode(cfg, p, bk, bv, q, 0)[0] for (cfg, p, bk, bv, q) in runs]
    n = max(V.varrate_workspace_bytes(run[0], V.CALL_DECODE) for run in runs)
    ws = torch.zeros(n, dtype=torch.uint8, device="cuda")
    for _ in range(3):
        for i, (cfg, p, bk, bv, q) in enumerate(runs):
            out, st = _decode_with_ws(cfg, p, bk, bv, q, 0, ws)
            assert st == V.OK
            np.testing.assert_array_equal(out, ref[i])
    calls, _ = _header(ws)
    assert calls == 6
    cfg, p, bk, bv, q = runs[0]
    n_segs = cfg.batch * cfg.n_kv_heads
    ws[:HEADER_BYTES].fill_(0x7F)                        # garbage
    _, st = _decode_with_ws(cfg, p, bk, bv, q, 0, ws)
    assert st == V.ERR_CORRUPT
    out, st = _decode_with_ws(cfg, p, bk, bv, q, 0, ws)   # clean again
    assert st == V.OK
    np.testing.assert_array_equal(out, ref[0])
    # an earlier call that stopped after one thread block arrived on every segment
    calls, _ = _header(ws)
    ws[256:HEADER_BYTES].view(torch.int32).view(2, 4096)[calls & 1, :n_segs] = 1
    _, st = _decode_with_ws(cfg, p, bk, bv, q, 0, ws)
    assert st == V.ERR_CORRUPT
    for _ in range(2):
        out, st = _decode_with_ws(cfg, p, bk, bv, q, 0, ws)
        assert st == V.OK
        np.testing.assert_array_equal(out, ref[0])


def test_budget_one_matches_uncompressed_attention():
    wl = synth.workload("tiny", n_ctx=1500, budget_frac=1.0)
    k, v, qw, bk, bv = synth.stack_inputs(wl)
    cfg = cfg_for(wl)
    r = gpu_encode(cfg, k, v, qw, bk, bv)
    assert np.all(r["packed"].ranks.cpu().numpy() == 128)
    q = synth.stack_decode_queries(wl, 0, 1)[0]
    out, _ = gpu_decode(cfg, r["packed"], bk, bv, q, 0)
    want = O.attention(f64(q[0]), f64(k[0, 0]), f64(v[0, 0]))
    assert np.abs(out[0] - want).max() <= 1e-5


def test_empty_coded_set_decodes_exactly():
    wl = synth.workload("tiny", n_ctx=48, window=48)
    k, v, qw, bk, bv = synth.stack_inputs(wl)
    cfg = cfg_for(wl)
    r = gpu_encode(cfg, k, v, qw, bk, bv)
    assert r["status"] == V.OK and np.all(r["packed"].ranks.cpu().numpy() == 128)
    q = synth.stack_decode_queries(wl, 0, 1)[0]
    out, _ = gpu_decode(cfg, r["packed"], bk, bv, q, 0)
    assert np.abs(out[0] - O.attention(f64(q[0]), f64(k[0, 0]), f64(v[0, 0]))).max() <= 1e-5


# ------------------------------------------------------------------- encode end to end

@pytest.mark.parametrize("name", list(CASES))
def test_encode_end_to_end(inputs, name):
    """Full GPU path (salience -> ranks -> pack -> decode) against the full oracle path. Ranks
    come from each side's own salience, so a token at a rounding boundary may differ by one; the
    decode outputs must still agree within the decode bound."""
    wl = CASES[name]
    k, v, qw, bk, bv = inputs[name]
    cfg = cfg_for(wl)
    r = gpu_encode(cfg, k, v, qw, bk, bv)
    bc = O.coded_budget(wl.n_ctx, wl.head_dim, wl.window, wl.budget_frac)
    worst = (0.0, 0.0)
    for b in range(wl.batch):
        for l in range(wl.n_layers):
            ref = oracle_layer(wl, k, v, qw, bk, bv, b, l)
            got = r["packed"].ranks[b, l].cpu().numpy().astype(np.int64)
            agree = np.mean(got == ref["ranks"])
            assert agree >= 0.999 and np.abs(got - ref["ranks"]).max() <= 1, (agree,)
            assert int(r["realized"][b, l]) <= bc
            assert int(r["realized"][b, l]) == int(got[: wl.n_ctx - wl.window].sum())
            q = synth.stack_decode_queries(wl, l, 1)[0]
            out, _ = gpu_decode(cfg, r["packed"], bk, bv, q, l)
            want = O.decode_coef(f64(q[b]), ref["coef_k"], ref["coef_v"], ref["ranks"],
                                 f64(bk[l]), f64(bv[l]))
            assert decode_close(out[b], want, cfg), (b, l, decode_errors(out[b], want))
            worst = tuple(max(a, e) for a, e in zip(worst, decode_errors(out[b], want)))
    print(f"{name}: decode worst relative / absolute error {worst[0]:.3e} / {worst[1]:.3e}")
