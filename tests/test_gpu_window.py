"""GPU vs oracle parity of the window decode (n_q new tokens per sequence in one call, causal
within the window), through the C ABI.

Bars: the decode bars of gpu_helpers.py per output row (one window query and head). The cases cover
every row-group size of the kernel (n_q * group rows in 1, 2, 4 and 8 groups of 16), a partial
second n-tile (group 7), a window that is the whole tail, tails past 256 tokens, an empty coded set,
and causality: changing tail tokens after query i's position leaves queries 0..i bit-identical."""
import numpy as np
import pytest
import torch

from gpu_helpers import (O, V, cfg_for, decode_close, decode_errors, f64, gpu_pack, oracle_layer,
                         synth)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _gpu(vlib):
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")


WL = {
    "llama": synth.workload("llama1", n_kv_heads=2, n_ctx=4096 + 37, batch=2, n_layers=2),
    "qwen_g7": synth.workload("qwen", n_kv_heads=2, n_ctx=3000 + 5, n_layers=1),
}


@pytest.fixture(scope="module")
def caches():
    out = {}
    for name, wl in WL.items():
        k, v, qw, bk, bv = synth.stack_inputs(wl, device="cpu")
        refs = [[oracle_layer(wl, k, v, qw, bk, bv, b, l) for l in range(wl.n_layers)]
                for b in range(wl.batch)]
        ranks = np.stack([np.stack([refs[b][l]["ranks"] for l in range(wl.n_layers)])
                          for b in range(wl.batch)])
        cfg = cfg_for(wl)
        packed, st = gpu_pack(cfg, ranks, k, v, bk, bv)
        assert st == V.OK
        out[name] = dict(wl=wl, cfg=cfg, refs=refs, packed=packed, bk=bk, bv=bv)
    return out


def _window_inputs(wl, layer, n_q, n_tail, seed):
    """Queries [B][n_q][H][d] and an exact tail [B][G][n_tail][d] (the window's own tokens last)."""
    g = torch.Generator().manual_seed(seed)
    dt = synth.torch_dtype(wl)
    q = synth.stack_decode_queries(wl, layer, n_q).permute(1, 0, 2, 3).contiguous()
    tk = torch.randn((wl.batch, wl.n_kv_heads, n_tail, wl.head_dim), generator=g).to(dt)
    tv = torch.randn((wl.batch, wl.n_kv_heads, n_tail, wl.head_dim), generator=g).to(dt)
    return q, tk, tv


def gpu_window(cfg, packed, bk, bv, q, layer, tk, tv, ws=None):
    out = torch.empty_like(q, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    if ws is None:
        ws = V.workspace(cfg, V.CALL_DECODE_WINDOW, "cuda")
    V.check(V.varrate_decode_window(cfg, packed, bk.cuda(), bv.cuda(), q.cuda(), q.shape[1], layer,
                                    tk.cuda(), tv.cuda(), tk.shape[2], out, status, ws),
            "varrate_decode_window")
    torch.cuda.synchronize()
    return out, int(status.item())


def _check(c, layer, n_q, n_tail, seed=5):
    wl, cfg = c["wl"], c["cfg"]
    q, tk, tv = _window_inputs(wl, layer, n_q, n_tail, seed)
    out, st = gpu_window(cfg, c["packed"], c["bk"], c["bv"], q, layer, tk, tv)
    assert st == V.OK
    got = f64(out)
    worst = (0.0, 0.0)
    for b in range(wl.batch):
        ref = c["refs"][b][layer]
        want = O.decode_window(f64(q[b]), ref["coef_k"], ref["coef_v"], ref["ranks"],
                               f64(c["bk"][layer]), f64(c["bv"][layer]), f64(tk[b]), f64(tv[b]))
        for i in range(n_q):
            assert decode_close(got[b, i], want[i], cfg), (b, i, decode_errors(got[b, i], want[i]))
        worst = tuple(max(a, e) for a, e in zip(worst, decode_errors(got[b], want)))
    print(f"window n_q={n_q} n_tail={n_tail}: worst relative / absolute {worst[0]:.3e} / {worst[1]:.3e}")
    return q, tk, tv, out


# llama group 4: n_q = 1, 4 -> one row group; 8 -> two; 16 -> four; 32 -> eight (128 rows)
@pytest.mark.parametrize("n_q,n_tail", [(1, 1), (4, 37), (8, 8), (16, 160), (32, 32), (32, 300)])
def test_window_matches_oracle_llama(caches, n_q, n_tail):
    _check(caches["llama"], 1, n_q, n_tail)


# group 7: 3 queries = 21 rows (two row groups, the second with one n-tile), 18 queries = 126 rows
@pytest.mark.parametrize("n_q,n_tail", [(3, 40), (18, 18), (5, 257)])
def test_window_matches_oracle_group7(caches, n_q, n_tail):
    _check(caches["qwen_g7"], 0, n_q, n_tail)


def test_window_is_causal(caches):
    """Replacing the tail tokens after query i's own position changes nothing for queries <= i."""
    c = caches["llama"]
    n_q, n_tail, i = 16, 40, 9
    q, tk, tv, out = _check(c, 0, n_q, n_tail)
    pos = n_tail - n_q + i                      # query i's position in the tail
    g = torch.Generator().manual_seed(99)
    tk2, tv2 = tk.clone(), tv.clone()
    tk2[:, :, pos + 1:] = torch.randn(tk2[:, :, pos + 1:].shape, generator=g).to(tk.dtype)
    tv2[:, :, pos + 1:] = torch.randn(tv2[:, :, pos + 1:].shape, generator=g).to(tv.dtype)
    out2, st = gpu_window(c["cfg"], c["packed"], c["bk"], c["bv"], q, 0, tk2, tv2)
    assert st == V.OK
    assert torch.equal(out[:, : i + 1], out2[:, : i + 1])
    assert not torch.equal(out[:, i + 1:], out2[:, i + 1:])


def test_window_deterministic_and_workspace_reuse(caches):
    """Two calls on one workspace (garbage-filled first: it is scratch) give identical outputs."""
    c = caches["llama"]
    q, tk, tv = _window_inputs(c["wl"], 0, 8, 20, 7)
    ws = V.workspace(c["cfg"], V.CALL_DECODE_WINDOW, "cuda")
    ws.fill_(0x5A)
    a, st = gpu_window(c["cfg"], c["packed"], c["bk"], c["bv"], q, 0, tk, tv, ws)
    assert st == V.OK
    b, st = gpu_window(c["cfg"], c["packed"], c["bk"], c["bv"], q, 0, tk, tv, ws)
    assert st == V.OK
    assert torch.equal(a, b)


def test_window_tail_only():
    """Empty coded set: the whole context is the exact window, plus the exact tail."""
    wl = synth.workload("llama1", n_kv_heads=2, n_ctx=32, window=32, batch=2)
    k, v, qw, bk, bv = synth.stack_inputs(wl)
    refs = [[oracle_layer(wl, k, v, qw, bk, bv, b, 0)] for b in range(wl.batch)]
    ranks = np.stack([np.stack([refs[b][0]["ranks"]]) for b in range(wl.batch)])
    cfg = cfg_for(wl)
    packed, st = gpu_pack(cfg, ranks, k, v, bk, bv)
    assert st == V.OK
    c = dict(wl=wl, cfg=cfg, refs=refs, packed=packed, bk=bk, bv=bv)
    _check(c, 0, 6, 45)


def test_window_rejects_bad_shapes(caches):
    c = caches["llama"]
    cfg = c["cfg"]
    q, tk, tv = _window_inputs(c["wl"], 0, 8, 8, 1)
    out = torch.empty_like(q, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    ws = V.workspace(cfg, V.CALL_DECODE_WINDOW, "cuda")
    args = (c["bk"].cuda(), c["bv"].cuda(), q.cuda())
    # more window queries than tail tokens
    assert V.varrate_decode_window(cfg, c["packed"], *args, 8, 0, tk[:, :, :4].contiguous().cuda(),
                                   tv[:, :, :4].contiguous().cuda(), 4, out, status, ws) == V.ERR_ARG
    # 33 queries x group 4 = 132 rows > 128
    assert V.varrate_decode_window(cfg, c["packed"], *args, 33, 0, tk.cuda(), tv.cuda(), 40, out,
                                   status, ws) == V.ERR_UNSUPPORTED
    # workspace too small
    assert V.varrate_decode_window(cfg, c["packed"], *args, 8, 0, tk.cuda(), tv.cuda(), 8, out,
                                   status, ws[:1024]) == V.ERR_WORKSPACE
