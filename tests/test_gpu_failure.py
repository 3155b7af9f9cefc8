"""GPU side of failure detection, without faulting, trapping or hanging the GPU.

Every TMA, tcgen05 and bulk-copy wait of the library is a bounded loop of mbarrier polls; one that
gives up raises VARRATE_ERR_TIMEOUT in the device status word and lets the kernel return. The test
hook `varrate_selftest_wait_timeout` waits on an mbarrier phase that nothing completes (no copy in
flight), so its wait always runs out: the status must read TIMEOUT, and the context must stay usable,
i.e. a fused decode launched right after it on the same stream still matches the oracle with a clean
status word."""
import numpy as np
import pytest
import torch

from gpu_helpers import O, V, decode_close, decode_errors, f64, gpu_decode, gpu_pack, cfg_for, oracle_layer, synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _gpu(vlib):
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")


@pytest.mark.parametrize("polls", [1, 64, 4096])
def test_bounded_wait_raises_timeout(polls):
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    assert V.varrate_selftest_wait_timeout(status, polls) == V.OK
    torch.cuda.synchronize()
    assert int(status.item()) == V.ERR_TIMEOUT


def test_context_usable_after_timeout():
    wl = synth.workload("llama1", n_kv_heads=2, n_ctx=2048 + 11, batch=2)
    k, v, qw, bk, bv = synth.stack_inputs(wl)
    refs = [oracle_layer(wl, k, v, qw, bk, bv, b, 0) for b in range(wl.batch)]
    ranks = np.stack([refs[b]["ranks"][None] for b in range(wl.batch)])
    cfg = cfg_for(wl)
    packed, st = gpu_pack(cfg, ranks, k, v, bk, bv)
    assert st == V.OK
    bad = torch.zeros(1, dtype=torch.int32, device="cuda")
    for _ in range(3):   # several timed-out waits in a row, queued ahead of the decode
        assert V.varrate_selftest_wait_timeout(bad, 256) == V.OK
    q = synth.stack_decode_queries(wl, 0, 1)[0]
    out, st = gpu_decode(cfg, packed, bk, bv, q, 0, None, None)
    assert int(bad.item()) == V.ERR_TIMEOUT
    assert st == V.OK
    for b in range(wl.batch):
        want = O.decode_coef(f64(q[b]), refs[b]["coef_k"], refs[b]["coef_v"], refs[b]["ranks"],
                             f64(bk[0]), f64(bv[0]))
        assert decode_close(out[b], want, cfg), (b, decode_errors(out[b], want))
