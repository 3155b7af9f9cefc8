"""The allocation-free decode entry point (for callers that cannot allocate device memory, e.g. a
plugin handed only input/output pointers): through the C ABI it must give the same result as
varrate_decode_attn with caller workspace, on two calls in a row (the fixed scratch array is
reused and keeps the previous call's contents). Kept last in collection order."""
import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu


def test_decode_noalloc_matches_workspace_decode(vlib):
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    import synth
    from gpu_helpers import cfg_for, decode_tol, gpu_encode

    V = vlib
    wl = synth.workload("llama1", n_kv_heads=4, n_ctx=6000 + 13, batch=2, n_layers=2)
    k, v, qw, bk, bv = synth.stack_inputs(wl)
    cfg = cfg_for(wl)
    r = gpu_encode(cfg, k, v, qw, bk, bv)
    bk, bv = bk.cuda(), bv.cuda()
    ws = V.workspace(cfg, V.CALL_DECODE)
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    for call in range(2):
        layer = call % wl.n_layers
        q = synth.stack_decode_queries(wl, layer, 1)[0].cuda()
        want = torch.empty_like(q)
        got = torch.full_like(q, float("nan"))
        V.check(V.varrate_decode_attn(cfg, r["packed"], bk, bv, q, layer, None, None, 0, want,
                                      status, ws))
        V.check(V.varrate_decode_attn_noalloc(cfg, r["packed"], bk, bv, q, layer, None, None, 0,
                                              got, status))
        torch.cuda.synchronize()
        assert int(status.item()) == V.OK
        err = (got.double() - want.double()).abs().max().item()
        assert np.isfinite(err) and err <= decode_tol(cfg), (call, err)


def test_decode_noalloc_rejects_shapes_beyond_its_scratch(vlib):
    import ctypes
    V = vlib
    cfg = V.make_config(1, 8, 8, 32768, batch=512)
    assert V.varrate_workspace_bytes(cfg, V.CALL_DECODE) > (4 << 20)
    p = V.varrate_packed(1, 1, 1, 1, 1, 1, V.varrate_packed_cap_elems(cfg))
    rc = V.lib().varrate_decode_attn_noalloc(ctypes.byref(cfg), ctypes.byref(p), 1, 1, 1, 0, None,
                                             None, 0, 1, None, None)
    assert rc == V.ERR_WORKSPACE
