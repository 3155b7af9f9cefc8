"""GPU parity of the joint codec's nearest-anchor search (Sec. 3.1, Eq. 1-2) through the C ABI,
against the joint oracle on the same bf16 inputs.

The kernel forms |z_t|^2 + |z_a|^2 - 2 z_t . z_a with exact bf16 products and fp32 sums; the
oracle takes exact fp64 distances. Bars, per token row t with TOL = 1e-4 (|z_t|^2 + max_a |z_a|^2)
(fp32 accumulation over D terms stays orders of magnitude below it; a lost head or a wrong sign
moves a distance by a sizeable fraction of |z|^2):
  * every reported distance within TOL of the exact distance of the same (token, anchor) pair;
  * the listed anchors distinct, within [0, n_a), ordered by (reported distance, anchor);
  * the s-th listed anchor's exact distance within 2 TOL of the s-th smallest exact distance (the
    list is a valid top-c: its s-th reported value is at most the s-th smallest reported value);
  * wherever the oracle's c + 1 smallest exact distances are more than 2 TOL apart (one correct
    answer), the list identical to the oracle's;
  * past the anchor count: -1 and +inf, exactly."""
import numpy as np
import pytest
import torch

from gpu_helpers import V, synth
from oracle import joint_oracle as J

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _gpu(vlib):
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")


def _search(wl, k, v, stride, c):
    cfg = V.make_config(wl.n_layers, wl.n_kv_heads, wl.group, wl.n_ctx, batch=wl.batch,
                        window=min(wl.window, wl.n_ctx), dtype=V.BF16)
    B, L, N = wl.batch, wl.n_layers, wl.n_ctx
    ws = torch.zeros(max(V.varrate_anchor_search_ws_bytes(cfg, stride), 256), dtype=torch.uint8,
                     device="cuda")
    idx = torch.full((B, L, N, c), -7, dtype=torch.int32, device="cuda")
    dist = torch.full((B, L, N, c), float("nan"), dtype=torch.float32, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    V.check(V.varrate_anchor_search(cfg, k, v, stride, c, idx, dist, status, ws), "varrate_anchor_search")
    torch.cuda.synchronize()
    assert int(status.item()) == 0, V.status_string(int(status.item()))
    return idx.cpu().numpy(), dist.cpu().numpy()


def _check_rows(z, stride, c, idx, dist, rows):
    """Compare the kernel's lists (idx, dist: [len(rows)][c]) with the oracle on the given rows."""
    n = z.shape[0]
    pos = J.anchor_positions(n, stride)
    n_a = pos.size
    na = np.einsum("ad,ad->a", z[pos], z[pos])
    oi, od = J.nearest_anchors(z, stride, min(c + 1, n_a), rows=rows)
    worst = 0.0
    for i, t in enumerate(rows):
        tol = 1e-4 * (float(z[t] @ z[t]) + float(na.max()))
        m = min(c, n_a)
        ki, kd = idx[i], dist[i]
        assert (ki[m:] == -1).all() and np.isinf(kd[m:]).all(), t
        ki, kd = ki[:m].astype(np.int64), kd[:m].astype(np.float64)
        assert ((ki >= 0) & (ki < n_a)).all() and np.unique(ki).size == m, (t, ki)
        assert all((kd[s], ki[s]) <= (kd[s + 1], ki[s + 1]) for s in range(m - 1)), (t, ki, kd)
        diff = z[pos[ki]] - z[t]
        exact = np.einsum("ad,ad->a", diff, diff)
        err = np.abs(kd - exact).max()
        worst = max(worst, err / tol)
        assert err <= tol, (t, err, tol)
        assert (exact <= od[i, :m] + 2 * tol).all(), (t, exact, od[i])
        gaps = np.diff(od[i][np.isfinite(od[i])])
        if gaps.size == 0 or gaps.min() > 2 * tol:
            np.testing.assert_array_equal(ki, oi[i, :m], err_msg=f"token {t}")
    return worst


CASES = {
    # D = 512, 65 anchors (one partial tile), ragged last token tile, 2 sequences x 2 layers
    "llama_g2": (synth.workload("llama1", n_kv_heads=2, n_ctx=1000 + 37, batch=2, n_layers=2), 16, 4),
    # D = 1024, stride 7: 430 anchors over two anchor tiles (both epilogue groups), c = 8
    "qwen_g4_s7": (synth.workload("qwen", n_kv_heads=4, n_ctx=3000 + 5, n_layers=1), 7, 8),
    # fewer anchors than c: 3 anchors, c = 4
    "few_anchors": (synth.workload("llama1", n_kv_heads=1, n_ctx=40, n_layers=1), 16, 4),
    # every token an anchor: 300 anchors, two tiles; each token finds itself first
    "stride1": (synth.workload("llama1", n_kv_heads=1, n_ctx=300, n_layers=1), 1, 2),
}


@pytest.mark.parametrize("name", list(CASES))
def test_anchor_search_matches_oracle(name):
    wl, stride, c = CASES[name]
    k, v, _, _, _ = synth.stack_inputs(wl, device="cuda")
    idx, dist = _search(wl, k, v, stride, c)
    kc, vc = k.cpu(), v.cpu()
    worst = 0.0
    for b in range(wl.batch):
        for l in range(wl.n_layers):
            z = J.joint_vector(kc[b, l].double().numpy(), vc[b, l].double().numpy())
            rows = np.arange(wl.n_ctx)
            worst = max(worst, _check_rows(z, stride, c, idx[b, l], dist[b, l], rows))
    if stride == 1:
        assert (idx[..., 0] == np.arange(wl.n_ctx)).all()
    print(f"{name}: worst distance error {worst:.3g} of the bar")
    # a second call gives the same bits
    idx2, dist2 = _search(wl, k, v, stride, c)
    np.testing.assert_array_equal(idx2, idx)
    np.testing.assert_array_equal(dist2.view(np.int32), dist.view(np.int32))


def test_anchor_search_full_size_llama_layer():
    """One Llama-shaped layer at N = 32768 (G = 8, D = 2048, stride 16: 2048 anchors, c = 4):
    every output checked for range and order, 384 sampled tokens against the oracle."""
    wl = synth.workload("llama1")
    stride, c = 16, 4
    k, v, _, _, _ = synth.stack_inputs(wl, device="cuda")
    idx, dist = _search(wl, k, v, stride, c)
    n_a = J.anchor_positions(wl.n_ctx, stride).size
    assert ((idx >= 0) & (idx < n_a)).all() and np.isfinite(dist).all() and (dist >= 0).all()
    assert (np.diff(dist, axis=-1) >= 0).all()
    z = J.joint_vector(k[0, 0].cpu().double().numpy(), v[0, 0].cpu().double().numpy())
    rng = np.random.default_rng(1)
    rows = np.unique(np.concatenate([[0, 1, 16, 127, 128, wl.n_ctx - 1, wl.n_ctx - 16],
                                     rng.choice(wl.n_ctx, 377, replace=False)]))
    worst = _check_rows(z, stride, c, idx[0, 0, rows], dist[0, 0, rows], rows)
    anchors = rows[rows % stride == 0]
    assert (idx[0, 0, anchors, 0] == anchors // stride).all()
    print(f"full size: worst distance error {worst:.3g} of the bar")


def _residual(wl, k, v, stride, c, idx_dev):
    cfg = V.make_config(wl.n_layers, wl.n_kv_heads, wl.group, wl.n_ctx, batch=wl.batch,
                        window=min(wl.window, wl.n_ctx), dtype=V.BF16)
    D = 2 * wl.n_kv_heads * wl.head_dim
    e = torch.full((wl.batch, wl.n_layers, wl.n_ctx, D), float("nan"), dtype=torch.bfloat16, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    V.check(V.varrate_anchor_residual(cfg, k, v, stride, c, idx_dev, e, status), "varrate_anchor_residual")
    torch.cuda.synchronize()
    return e, int(status.item())


@pytest.mark.parametrize("name", ["llama_g2", "qwen_g4_s7", "few_anchors"])
def test_anchor_residual_matches_oracle(name):
    """Eq. 2 on the GPU's own anchor lists: e_t = z_t - mean of the listed anchors, against the
    oracle's residual in fp64. Bar per coordinate: twice the bf16 rounding of the result (unit
    roundoff 2^-8, so 2^-7 |want|) plus the fp32 rounding of the sum (2^-20 (|z_t| + the listed
    anchors' magnitudes)). A numpy emulation of the kernel's arithmetic reaches 0.50 of this bar;
    a dropped anchor mean or a wrong divisor exceed it by four orders of magnitude."""
    wl, stride, c = CASES[name]
    k, v, _, _, _ = synth.stack_inputs(wl, device="cuda")
    idx, _ = _search(wl, k, v, stride, c)
    e, st = _residual(wl, k, v, stride, c, torch.as_tensor(idx, device="cuda"))
    assert st == 0, V.status_string(st)
    got = e.to(torch.float64).cpu().numpy()
    kc, vc = k.cpu(), v.cpu()
    for b in range(wl.batch):
        for l in range(wl.n_layers):
            z = J.joint_vector(kc[b, l].double().numpy(), vc[b, l].double().numpy())
            lists = idx[b, l].astype(np.int64)
            want = J.residual(z, lists, stride)
            mag = np.abs(z).copy()
            for s in range(c):
                ok = lists[:, s] >= 0
                mag[ok] += np.abs(z[lists[ok, s] * stride])
            bar = 2.0 ** -7 * np.abs(want) + 2.0 ** -20 * mag
            err = np.abs(got[b, l] - want)
            assert (err <= bar).all(), (name, b, l, float((err / np.maximum(bar, 1e-30)).max()))


def test_anchor_residual_rejects_a_bad_list():
    """An anchor number past the anchor count is caught by the kernel's own check: the call raises
    VARRATE_ERR_CORRUPT, leaves that token's row unwritten and writes the others."""
    wl, stride, c = CASES["llama_g2"]
    k, v, _, _, _ = synth.stack_inputs(wl, device="cuda")
    idx, _ = _search(wl, k, v, stride, c)
    n_a = J.anchor_positions(wl.n_ctx, stride).size
    bad = idx.copy()
    bad[0, 0, 5, 1] = n_a + 3
    e, st = _residual(wl, k, v, stride, c, torch.as_tensor(bad, device="cuda"))
    assert st == V.ERR_CORRUPT
    assert torch.isnan(e[0, 0, 5].float()).all()
    good, st2 = _residual(wl, k, v, stride, c, torch.as_tensor(idx, device="cuda"))
    assert st2 == 0
    np.testing.assert_array_equal(e[0, 0, 6].float().cpu().numpy(), good[0, 0, 6].float().cpu().numpy())
