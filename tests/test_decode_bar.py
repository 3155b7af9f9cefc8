"""The decode parity bar of the GPU tests can fail (CPU only, no GPU).

The outer 2e-2 max-abs bound alone is met even by a decode that ignores the scores once the
context is long (max|o| is then ~0.02). These checks fix the inner per-row relative bound from
both sides on the Llama-shaped layer at N = 4133: plausible kernel mistakes, planted in outputs
computed here from the oracle's own coefficients, must fail it, and the bf16 roundings the kernel
makes (coefficients, softmax weights and output stored in bf16) must pass it."""
import numpy as np
import pytest
import torch

import oracle as O
import synth
from gpu_helpers import V, decode_close, decode_errors, f64, uniform_weight_output


def _bf16(x):
    return torch.tensor(x, dtype=torch.float64).to(torch.bfloat16).to(torch.float64).numpy()


def _decode_variant(q, ref, uk, uv, keep=None, bf16=False):
    """Attention on the coefficients as the oracle states it, optionally over a subset of tokens
    (`keep`, a mask) and with the bf16 roundings of the kernel (stored coefficients, weights P,
    output); the normaliser stays the fp32-or-better sum of unrounded weights."""
    H, d = q.shape
    G = ref["coef_k"].shape[0]
    grp = H // G
    rnd = _bf16 if bf16 else (lambda x: x)
    out = np.zeros((H, d))
    for h in range(H):
        g = h // grp
        ck = rnd(O.truncate(ref["coef_k"][g], ref["ranks"]))
        cv = rnd(O.truncate(ref["coef_v"][g], ref["ranks"]))
        if keep is not None:
            ck, cv = ck[keep], cv[keep]
        s = ck @ (uk[g] @ q[h]) / np.sqrt(d)
        p = np.exp(s - s.max())
        out[h] = uv[g].T @ (rnd(p) @ cv) / p.sum()
    return rnd(out)


@pytest.fixture(scope="module")
def layer():
    wl = synth.workload("llama1", n_kv_heads=2, n_ctx=4096 + 37, n_layers=1)
    k, v, qw, bk, bv = synth.stack_inputs(wl)
    uk, uv = f64(bk[0]), f64(bv[0])
    ref = O.encode_layer(f64(qw[0, 0]), f64(k[0, 0]), f64(v[0, 0]), uk, uv, wl.group,
                         wl.budget_frac, wl.r_min)
    qs = [f64(q[0]) for q in synth.stack_decode_queries(wl, 0, 3)]
    wants = [O.decode_coef(q, ref["coef_k"], ref["coef_v"], ref["ranks"], uk, uv) for q in qs]
    cfg = V.make_config(1, wl.n_kv_heads, wl.group, wl.n_ctx, dtype=V.BF16)
    return dict(wl=wl, ref=ref, uk=uk, uv=uv, qs=qs, wants=wants, cfg=cfg)


def test_bf16_roundings_of_the_kernel_pass(layer):
    for q, want in zip(layer["qs"], layer["wants"]):
        got = _decode_variant(q, layer["ref"], layer["uk"], layer["uv"], bf16=True)
        rel, _ = decode_errors(got, want)
        assert decode_close(got, want, layer["cfg"]) and rel <= 2.0 ** -7, rel


def test_score_blind_and_zero_outputs_fail(layer):
    uni = uniform_weight_output(layer["ref"], layer["uv"], layer["wl"].group)
    for want in layer["wants"]:
        assert not decode_close(uni, want, layer["cfg"])
        assert not decode_close(np.zeros_like(want), want, layer["cfg"])
        assert decode_errors(uni, want)[0] > 0.3


def test_dropped_tokens_fail(layer):
    """A skipped rank bucket, a skipped exact window and a skipped last tile are each caught."""
    ranks = layer["ref"]["ranks"]
    n = ranks.size
    vals, counts = np.unique(ranks[: n - layer["wl"].window], return_counts=True)
    busiest = vals[np.argmax(counts)]
    masks = {"bucket": ranks != busiest,
             "exact window": np.arange(n) < n - layer["wl"].window,
             "last 128 tokens of a bucket": ~((ranks == busiest) &
                                               (np.cumsum(ranks == busiest) > counts.max() - 128))}
    for name, keep in masks.items():
        for q, want in zip(layer["qs"], layer["wants"]):
            got = _decode_variant(q, layer["ref"], layer["uk"], layer["uv"], keep=keep, bf16=True)
            assert not decode_close(got, want, layer["cfg"]), name
