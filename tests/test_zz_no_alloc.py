"""The allocation-free decode entry point, through the C ABI.

Some callers cannot allocate device memory: a plugin that a host framework hands only the input and
output pointers, or a serving loop that must not allocate once it has started. For them
varrate_decode_attn_noalloc takes its scratch from a fixed array inside the library. It runs the
same kernels as varrate_decode_attn with the same grid and merge order, so its output must equal,
bit for bit, that of a call with caller workspace, on two calls in a row (the array is reused and
keeps the previous call's contents). Covered: the fused bf16 kernel (no tail), the general bf16
kernels (a 300-token exact tail) and the fp32 kernels, which place their scratch differently.
Collected last, so that a run stopping at the first failure has already run every other test."""
import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu


def _cases():
    import synth
    return {
        "bf16_fused": (synth.workload("llama1", n_kv_heads=4, n_ctx=6000 + 13, batch=2, n_layers=2), 0),
        "bf16_long_tail": (synth.workload("llama1", n_kv_heads=2, n_ctx=3000 + 7, batch=2, n_layers=2), 300),
        "f32": (synth.workload("tiny", n_kv_heads=2, group=2, n_ctx=999, window=7, n_layers=2), 5),
    }


@pytest.mark.parametrize("name", ["bf16_fused", "bf16_long_tail", "f32"])
def test_decode_noalloc_matches_workspace_decode(vlib, name):
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    import synth
    from gpu_helpers import cfg_for, gpu_encode

    V = vlib
    wl, n_tail = _cases()[name]
    k, v, qw, bk, bv = synth.stack_inputs(wl)
    cfg = cfg_for(wl)
    r = gpu_encode(cfg, k, v, qw, bk, bv)
    bk, bv = bk.cuda(), bv.cuda()
    ws = V.workspace(cfg, V.CALL_DECODE)
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    gen = torch.Generator().manual_seed(5)
    dt = synth.torch_dtype(wl)
    for call in range(2):
        layer = call % wl.n_layers
        q = synth.stack_decode_queries(wl, layer, 1)[0].cuda()
        tk = tv = None
        if n_tail:
            shape = (wl.batch, wl.n_kv_heads, n_tail, wl.head_dim)
            tk = torch.randn(shape, generator=gen).to(dt).cuda()
            tv = torch.randn(shape, generator=gen).to(dt).cuda()
        want = torch.empty_like(q)
        got = torch.full_like(q, float("nan"))
        V.check(V.varrate_decode_attn(cfg, r["packed"], bk, bv, q, layer, tk, tv, n_tail, want,
                                      status, ws))
        V.check(V.varrate_decode_attn_noalloc(cfg, r["packed"], bk, bv, q, layer, tk, tv, n_tail,
                                              got, status))
        torch.cuda.synchronize()
        assert int(status.item()) == V.OK, (name, call, V.status_string(int(status.item())))
        assert torch.isfinite(want.float()).all()
        assert torch.equal(got, want), (name, call, (got.double() - want.double()).abs().max().item())


def test_decode_noalloc_rejects_shapes_beyond_its_scratch(vlib):
    import ctypes
    V = vlib
    cfg = V.make_config(1, 8, 8, 32768, batch=512)
    assert V.varrate_workspace_bytes(cfg, V.CALL_DECODE) > (4 << 20)
    p = V.varrate_packed(1, 1, 1, 1, 1, 1, V.varrate_packed_cap_elems(cfg))
    rc = V.lib().varrate_decode_attn_noalloc(ctypes.byref(cfg), ctypes.byref(p), 1, 1, 1, 0, None,
                                             None, 0, 1, None, None)
    assert rc == V.ERR_WORKSPACE
