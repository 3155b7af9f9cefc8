"""Shared helpers of the GPU parity tests: run the CUDA library through its C ABI and run the
oracle on the same drawn inputs."""
import numpy as np
import torch

import oracle as O
import synth
from paper_2607_15498_gb300 import varrate as V


def cfg_for(wl, mode=V.SALIENCE, budget_frac=None):
    return V.make_config(wl.n_layers, wl.n_kv_heads, wl.group, wl.n_ctx, batch=wl.batch,
                         budget_frac=wl.budget_frac if budget_frac is None else budget_frac,
                         r_min=wl.r_min, window=wl.window,
                         dtype=V.F32 if wl.dtype == "f32" else V.BF16, mode=mode)


def f64(t):
    return t.detach().to("cpu", torch.float64).numpy()


def gpu_encode(cfg, k, v, qw, bk, bv):
    """varrate_encode on device copies of the inputs; returns host copies of every output."""
    dev = "cuda"
    k, v, qw, bk, bv = (t.to(dev) for t in (k, v, qw, bk, bv))
    packed = V.PackedCache.allocate(cfg, dev)
    B, L, N, w = cfg.batch, cfg.n_layers, cfg.n_ctx, cfg.window
    sal = torch.full((B, L, N - w), float("nan"), dtype=torch.float32, device=dev)
    realized = torch.zeros((B, L), dtype=torch.int64, device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    ws = V.workspace(cfg, V.CALL_ENCODE, dev)
    V.check(V.varrate_encode(cfg, qw, k, v, bk, bv, sal, packed, realized, status, ws),
            "varrate_encode")
    torch.cuda.synchronize()
    return dict(packed=packed, sal=sal.cpu(), realized=realized.cpu(), status=int(status.item()),
                dev=(k, v, qw, bk, bv))


def gpu_allocate(cfg, sal32):
    sal = torch.as_tensor(np.asarray(sal32, dtype=np.float32)).reshape(
        cfg.batch, cfg.n_layers, cfg.n_ctx - cfg.window).cuda()
    ranks = torch.zeros((cfg.batch, cfg.n_layers, cfg.n_ctx), dtype=torch.uint8, device="cuda")
    realized = torch.zeros((cfg.batch, cfg.n_layers), dtype=torch.int64, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    V.check(V.varrate_allocate(cfg, sal, ranks, realized, status), "varrate_allocate")
    torch.cuda.synchronize()
    return ranks.cpu().numpy(), realized.cpu().numpy(), int(status.item())


def gpu_pack(cfg, ranks, k, v, bk, bv):
    packed = V.PackedCache.allocate(cfg, "cuda")
    packed.ranks.copy_(torch.as_tensor(np.asarray(ranks), dtype=torch.uint8).reshape(packed.ranks.shape))
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    V.check(V.varrate_pack(cfg, k.cuda(), v.cuda(), bk.cuda(), bv.cuda(), packed, status), "varrate_pack")
    torch.cuda.synchronize()
    return packed, int(status.item())


def gpu_decode(cfg, packed, bk, bv, q, layer, tail_k=None, tail_v=None):
    """One decode step for every sequence: q [B][H][d] -> out [B][H][d] (host float64)."""
    out = torch.empty_like(q, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    ws = V.workspace(cfg, V.CALL_DECODE, "cuda")
    n_tail = 0 if tail_k is None else tail_k.shape[2]
    V.check(V.varrate_decode_attn(cfg, packed, bk.cuda(), bv.cuda(), q.cuda(), layer,
                                  None if tail_k is None else tail_k.cuda(),
                                  None if tail_v is None else tail_v.cuda(), n_tail, out, status,
                                  ws), "varrate_decode_attn")
    torch.cuda.synchronize()
    return f64(out), int(status.item())


def coef_index(base_r, r, n8, p, j):
    """Element index of coefficient j of bucket slot p in the packed layout of include/varrate.h:
    128-slot tiles of r rows each, the 8-slot groups of row j rotated by j."""
    t0 = (p // 128) * 128
    tl = np.minimum(128, n8 - t0)
    ng = tl // 8
    grp = ((p - t0) // 8 + j) % ng
    return base_r + t0 * r + j * tl + grp * 8 + (p - t0) % 8


def unpack(packed, b, l, g, kv, ranks, count, base, pos, d=128):
    """Gather the coefficients of one stream from the device layout using the oracle's tables:
    [N][d] with zeros beyond each token's rank."""
    buf = f64(packed.coef[b, l, g, kv])
    ranks = np.asarray(ranks, dtype=np.int64)
    n8 = (np.asarray(count, dtype=np.int64) + 7) // 8 * 8
    j = np.arange(d)[None, :]
    rr = ranks[:, None]
    idx = coef_index(np.asarray(base)[rr], rr, n8[rr], np.asarray(pos, dtype=np.int64)[:, None], j)
    mask = j < rr
    out = np.zeros((ranks.size, d))
    out[mask] = buf[idx[mask]]
    return out


def oracle_layer(wl, k, v, qw, bk, bv, b, l, mode=O.SALIENCE, budget_frac=None):
    return O.encode_layer(f64(qw[b, l]) if qw is not None else None, f64(k[b, l]), f64(v[b, l]),
                          f64(bk[l]), f64(bv[l]), wl.group,
                          wl.budget_frac if budget_frac is None else budget_frac, wl.r_min,
                          mode=mode)


def salience_close(got, want):
    """|got - want| <= 1e-4 |want| + 1e-7 max(want): relative 1e-4, absolute floor far below
    every salient value."""
    got = np.asarray(got, dtype=np.float64)
    want = np.asarray(want, dtype=np.float64)
    tol = 1e-4 * np.abs(want) + 1e-7 * np.abs(want).max()
    bad = np.abs(got - want) > tol
    return (not bad.any()), int(bad.sum()), float(np.max(np.abs(got - want) / np.maximum(tol, 1e-30)))


def coef_tol(cfg):
    # fp32: accumulation error only; bf16: the stored coefficient is rounded to bf16 (unit roundoff
    # u = 2^-8, 8 significant bits) after an fp32 accumulation of exact bf16 products.
    return (1e-5, 1e-4) if cfg.dtype == V.F32 else (2.0 ** -8, 1e-3)


# Decode parity bar. Outer bound: 2e-2 max-abs (bf16) of the fp64 oracle, the stated requirement.
# That alone cannot fail at long context: there max|o| itself is 0.01-0.03, so an all-zero output
# or a score-blind one would pass. Inner bound, per output row (one sequence and query head, or one
# window query and head):
#     max_j |got_j - want_j| <= c * max_j |want_j|.
# Derivation for bf16 (unit roundoff u = 2^-8): o_j = sum_t alpha_t v_tj is a weighted sum of
# zero-mean terms, Var(o_j) = sum_t alpha_t^2 E[v_tj^2]. Each rounding source perturbs every term
# independently by at most u relative (the stored c^V, the bf16 weights P, and through the scores
# the stored c^K: a score error of ~u |q~||c^K|/sqrt(d) ~ u in log units), so each adds an error
# whose standard deviation is at most u std(o_j); with the bf16 output (u |o_j|) the four give ~2u
# in standard deviation, and the extremes of the 128 coordinates of error and output scale alike.
# Emulating these roundings in numpy gives a worst row of 1.5u on the llama shapes (N = 4133,
# 32768, 131072) and 2.3u on the qwen shape (group 7, N = 3005); the kernel measures the same.
# c = 4u = 2^-6. A score-blind output (uniform weights: the mean of v^) misses it by a factor of
# ~50 (relative error 0.84-1.0), which the negative controls check.
# fp32 path: no bf16 rounding anywhere, c = 1e-4 and 1e-4 max-abs.
DECODE_REL = {V.BF16: 2.0 ** -6, V.F32: 1e-4}
DECODE_ABS = {V.BF16: 2e-2, V.F32: 1e-4}


def decode_tol(cfg):
    return DECODE_ABS[cfg.dtype]


def decode_errors(got, want):
    """(worst per-row relative error, worst absolute error) over rows of the last axis."""
    got = np.asarray(got, dtype=np.float64)
    want = np.asarray(want, dtype=np.float64)
    err = np.abs(got - want).max(axis=-1)
    scale = np.abs(want).max(axis=-1)
    rel = err / np.maximum(scale, 1e-30)
    return float(rel.max()), float(err.max())


def decode_close(got, want, cfg):
    """True iff `got` meets both decode bars against the oracle output `want` ([..., d])."""
    rel, ab = decode_errors(got, want)
    return bool(np.isfinite(rel) and rel <= DECODE_REL[cfg.dtype] and ab <= DECODE_ABS[cfg.dtype])


def uniform_weight_output(ref, basis_v, group):
    """Negative control: the output of a decode that ignores the scores (every token weighted
    equally: the mean of the reconstructed values), per query head [H][d]."""
    G = ref["coef_v"].shape[0]
    out = []
    for g in range(G):
        mean_c = O.truncate(ref["coef_v"][g], ref["ranks"]).mean(axis=0)
        o = mean_c @ np.asarray(basis_v[g], dtype=np.float64)
        out.extend([o] * group)
    return np.stack(out)


__all__ = ["cfg_for", "gpu_encode", "gpu_allocate", "gpu_pack", "gpu_decode", "unpack",
           "oracle_layer", "salience_close", "coef_tol", "decode_tol", "decode_errors",
           "decode_close", "uniform_weight_output", "f64", "synth", "O", "V"]
