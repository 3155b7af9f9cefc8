"""GPU parity at the full workload sizes, in the launch configuration bench.py times.

* llama32 layer call: 8 sequences x 8 KV heads x N = 32768, 32 query heads (GQA 4), head_dim 128,
  bf16, budget 0.2, r_min 16, window 32. Two layers are drawn: one decode launch covers one layer,
  so its grid, cost line and partition are those of the 32-layer stack.
* long-context layer: N = 131072, batch 1 (the reuse workload's layer shape).

The inputs are drawn on the device; the oracle recomputes sampled (sequence, layer) pairs one by
one from host copies of the same tensors."""
import numpy as np
import pytest

from gpu_helpers import (O, V, cfg_for, coef_tol, decode_close, decode_errors, f64, gpu_decode,
                         gpu_encode, gpu_pack, oracle_layer, salience_close, synth, unpack,
                         uniform_weight_output)

pytestmark = pytest.mark.gpu


def _encode_and_sample(wl, samples):
    k, v, qw, bk, bv = synth.stack_inputs(wl, device="cuda")
    cfg = cfg_for(wl)
    r = gpu_encode(cfg, k, v, qw, bk, bv)
    assert r["status"] == V.OK
    refs = {(b, l): oracle_layer(wl, k, v, qw, bk, bv, b, l) for (b, l) in samples}
    return dict(wl=wl, cfg=cfg, inputs=(k, v, qw, bk, bv), gpu=r, refs=refs)


@pytest.fixture(scope="module")
def llama32():
    return _encode_and_sample(synth.workload("llama32", n_layers=2), [(0, 1), (5, 0)])


@pytest.fixture(scope="module")
def long_ctx():
    return _encode_and_sample(synth.workload("reuse", n_layers=1), [(0, 0)])


def _check_encode(run):
    wl, r = run["wl"], run["gpu"]
    bc = O.coded_budget(wl.n_ctx, wl.head_dim, wl.window, wl.budget_frac)
    for (b, l), ref in run["refs"].items():
        ok, nbad, worst = salience_close(r["sal"][b, l].numpy(), ref["sal"])
        assert ok, (b, l, nbad, worst)
        got = r["packed"].ranks[b, l].cpu().numpy().astype(np.int64)
        # ranks come from each side's own salience: a token at a rounding boundary may move by one
        assert np.mean(got == ref["ranks"]) >= 0.999 and np.abs(got - ref["ranks"]).max() <= 1
        assert int(r["realized"][b, l]) <= bc
        assert got.min() >= wl.r_min and got.max() <= wl.head_dim


def _check_decode(run, n_steps=2):
    """Decode of the sampled pairs within the per-row relative bar; at the same size a score-blind
    output (uniform weights) must fail that bar, so the check is able to catch a wrong kernel."""
    wl, cfg, r = run["wl"], run["cfg"], run["gpu"]
    _, _, _, bk, bv = run["inputs"]
    worst = (0.0, 0.0)
    for (b, l), ref in run["refs"].items():
        qs = synth.stack_decode_queries(wl, l, n_steps)
        blind = uniform_weight_output(ref, f64(bv[l]), wl.group)
        for step in range(n_steps):
            out, st = gpu_decode(cfg, r["packed"], bk, bv, qs[step], l)
            assert st == V.OK
            want = O.decode_coef(f64(qs[step][b]), ref["coef_k"], ref["coef_v"], ref["ranks"],
                                 f64(bk[l]), f64(bv[l]))
            assert decode_close(out[b], want, cfg), (b, l, step, decode_errors(out[b], want))
            assert not decode_close(blind, want, cfg), (b, l, step, decode_errors(blind, want))
            worst = tuple(max(a, e) for a, e in zip(worst, decode_errors(out[b], want)))
    print(f"N={wl.n_ctx}: decode worst relative / absolute error {worst[0]:.3e} / {worst[1]:.3e}")


def _check_pack(run, n_tokens=4096):
    """Pack fed the oracle's ranks for the sampled pairs: tables bit-exact, coefficients of a
    random token sample within the coefficient bound."""
    wl, cfg, r = run["wl"], run["cfg"], run["gpu"]
    k, v, _, bk, bv = run["inputs"]
    ranks = r["packed"].ranks.cpu().numpy().astype(np.int64)
    for (b, l), ref in run["refs"].items():
        ranks[b, l] = ref["ranks"]
    packed, st = gpu_pack(cfg, ranks, k, v, bk, bv)
    assert st == V.OK
    rtol, atol = coef_tol(cfg)
    rng = np.random.default_rng(3)
    for (b, l), ref in run["refs"].items():
        np.testing.assert_array_equal(packed.bucket_count[b, l].cpu().numpy(), ref["count"])
        np.testing.assert_array_equal(packed.bucket_base[b, l].cpu().numpy(), ref["base"])
        tok = np.sort(rng.choice(wl.n_ctx, size=min(n_tokens, wl.n_ctx), replace=False))
        for g in (0, wl.n_kv_heads - 1):
            for kv, full in ((0, ref["coef_k"][g]), (1, ref["coef_v"][g])):
                got = unpack(packed, b, l, g, kv, ref["ranks"], ref["count"], ref["base"],
                             ref["pos"])[tok]
                want = O.truncate(full, ref["ranks"])[tok]
                err = np.abs(got - want) - (rtol * np.abs(want) + atol)
                assert err.max() <= 0, (b, l, g, kv, float(err.max()))
        np.testing.assert_array_equal(packed.pos[b, l].cpu().numpy(), ref["pos"])
        np.testing.assert_array_equal(packed.perm[b, l].cpu().numpy(), ref["perm"])


def test_llama32_encode_full_size(llama32):
    _check_encode(llama32)


def test_llama32_decode_full_size(llama32):
    _check_decode(llama32)


def test_llama32_pack_full_size(llama32):
    _check_pack(llama32)


def test_long_context_encode_and_decode(long_ctx):
    _check_encode(long_ctx)
    _check_decode(long_ctx, n_steps=1)


def test_long_context_window_decode(long_ctx):
    """The window call of the reuse workload (N = 131072, 32 window queries x GQA 4 = 128 query rows
    per KV head, exact tail = the window's own 32 tokens), in the launch configuration bench.py
    times. Sampled queries against the oracle with each query's causal cut of the tail, and the
    score-blind control failing the same bar."""
    import torch
    wl, cfg, r = long_ctx["wl"], long_ctx["cfg"], long_ctx["gpu"]
    _, _, _, bk, bv = long_ctx["inputs"]
    ref = long_ctx["refs"][(0, 0)]
    n_q = 32
    q = synth.stack_decode_queries(wl, 0, n_q).permute(1, 0, 2, 3).contiguous()   # [B][n_q][H][d]
    g = torch.Generator().manual_seed(5)
    shape = (wl.batch, wl.n_kv_heads, n_q, wl.head_dim)
    tk = torch.randn(shape, generator=g).to(torch.bfloat16)
    tv = torch.randn(shape, generator=g).to(torch.bfloat16)
    out = torch.empty_like(q, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    ws = V.workspace(cfg, V.CALL_DECODE_WINDOW, "cuda")
    V.check(V.varrate_decode_window(cfg, r["packed"], bk.cuda(), bv.cuda(), q.cuda(), n_q, 0,
                                    tk.cuda(), tv.cuda(), n_q, out, status, ws),
            "varrate_decode_window")
    torch.cuda.synchronize()
    assert int(status.item()) == V.OK
    got = f64(out)
    blind = uniform_weight_output(ref, f64(bv[0]), wl.group)
    worst = (0.0, 0.0)
    for i in (0, 13, n_q - 1):
        m = i + 1                                 # tail tokens visible to query i
        want = O.decode_coef(f64(q[0, i]), ref["coef_k"], ref["coef_v"], ref["ranks"], f64(bk[0]),
                             f64(bv[0]), f64(tk[0, :, :m]), f64(tv[0, :, :m]))
        assert decode_close(got[0, i], want, cfg), (i, decode_errors(got[0, i], want))
        assert not decode_close(blind, want, cfg), (i, decode_errors(blind, want))
        worst = tuple(max(a, e) for a, e in zip(worst, decode_errors(got[0, i], want)))
    print(f"N={wl.n_ctx} window of {n_q}: worst relative / absolute error {worst[0]:.3e} / {worst[1]:.3e}")
