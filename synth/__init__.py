"""Seeded synthetic inputs for the VarRate hot path.

This module only draws random inputs; it holds none of the codec's arithmetic (no salience, no
allocation, no projection, no attention). Both the CUDA library's tests/bench and the CPU oracle
receive their inputs from here, so the two sides always see identical bytes.

Workloads (stand-ins for the paper's LongBench / NIAH prompts, whose models and data are not used):

* ``tiny``    1 layer, 1 KV head, group 4, d=128, N=2048, window 32, budget 0.20, r_min 16, fp32.
              Keys/values have singular spectrum sigma_i ~ 1/i; 5% of the coded tokens get 8x keys
              (salient outliers); 16 decode steps.
* ``llama1``  Llama-3.1-8B-shaped single layer: 8 KV heads, 32 query heads, d=128, N=32768, bf16,
              window 32, budget 0.20, r_min 16; low-rank-plus-noise K/V (rank 40, noise std 0.05,
              unit scale); 256 decode steps.
* ``llama32`` the same shape over a full 32-layer stack and 8 independent sequences.
* ``qwen``    Qwen2.5-7B-shaped: 28 layers, 4 KV heads, 28 query heads (group 7), sigma_i ~ i^-0.7,
              budgets 0.10/0.20/0.30/0.50.
* ``reuse``   Llama shape at N=131072, batch 1: encode once, then 16 query batches of
              (32 window queries + 128 decode steps).

Data model for one (sequence, layer, KV head, K-or-V) stream of N tokens:
    X = (Z * sigma * scale) @ F^T + noise_std * E,   Z, E ~ N(0, 1) i.i.d. [N, d]
where F is a seeded orthonormal d x d frame and ``scale`` makes the mean per-entry variance 1.
The per-head basis handed to the codec stands in for the paper's offline calibration (Sec. 3.1,
"Shared basis": the leading right singular vectors of calibration activations): the right singular
vectors, in fp64 (the eigenvectors of the Gram matrix), of a separate draw of CALIB_TOKENS tokens
from the same distribution (its own seeds), rows ordered by decreasing singular value, each row's
sign fixed so that its largest component is positive. Queries are N(0, 1).

Seeds are a pure function of (workload id, sequence, layer, head, stream kind); the same call on
the same device always returns the same tensor. CPU draws use torch's CPU generator, CUDA draws
torch's CUDA (Philox) generator, so a tensor drawn on CPU differs from one drawn on CUDA; a test
that compares two paths always feeds both the same drawn tensor.
"""
from __future__ import annotations

import functools
import math
from dataclasses import dataclass, field, replace

import numpy as np
import torch

__all__ = ["Workload", "WORKLOADS", "workload", "frames", "bases", "layer_kv", "window_queries",
           "decode_queries", "outlier_tokens", "seed_of"]

_KIND = {"k": 0, "v": 1, "qwin": 2, "qdec": 3, "outlier": 4, "frame": 5, "noise_k": 6,
         "noise_v": 7, "calib": 8}
CALIB_TOKENS = 2048   # tokens of the separate calibration draw the bases are fitted to


@dataclass(frozen=True)
class Workload:
    name: str
    wid: int
    n_layers: int
    n_kv_heads: int
    group: int
    head_dim: int
    n_ctx: int
    batch: int
    window: int
    budget_frac: float
    r_min: int
    dtype: str                 # "f32" or "bf16"
    spectrum: str              # "inv", "lowrank40", "pow0.7"
    noise_std: float = 0.0
    outlier_frac: float = 0.0
    outlier_scale: float = 1.0
    decode_steps: int = 16
    query_batches: int = 1
    budgets: tuple = field(default_factory=tuple)

    @property
    def n_q_heads(self) -> int:
        return self.n_kv_heads * self.group

    def with_(self, **kw) -> "Workload":
        return replace(self, **kw)


WORKLOADS = {
    "tiny": Workload("tiny", 1, 1, 1, 4, 128, 2048, 1, 32, 0.20, 16, "f32", "inv",
                     outlier_frac=0.05, outlier_scale=8.0, decode_steps=16),
    "llama1": Workload("llama1", 2, 1, 8, 4, 128, 32768, 1, 32, 0.20, 16, "bf16", "lowrank40",
                       noise_std=0.05, decode_steps=256),
    "llama32": Workload("llama32", 3, 32, 8, 4, 128, 32768, 8, 32, 0.20, 16, "bf16", "lowrank40",
                        noise_std=0.05, decode_steps=256),
    "qwen": Workload("qwen", 4, 28, 4, 7, 128, 32768, 1, 32, 0.20, 16, "bf16", "pow0.7",
                     noise_std=0.0, decode_steps=256, budgets=(0.10, 0.20, 0.30, 0.50)),
    "reuse": Workload("reuse", 5, 32, 8, 4, 128, 131072, 1, 32, 0.20, 16, "bf16", "lowrank40",
                      noise_std=0.05, decode_steps=128, query_batches=16),
}


def workload(name: str, **overrides) -> Workload:
    w = WORKLOADS[name]
    return w.with_(**overrides) if overrides else w


def seed_of(wl: Workload, kind: str, seq: int = 0, layer: int = 0, head: int = 0,
            extra: int = 0) -> int:
    """Deterministic 63-bit seed for one stream of one workload."""
    s = (((((wl.wid * 131 + _KIND[kind]) * 1_000_003 + seq) * 4099 + layer) * 257 + head)
         * 1_000_033 + extra)
    return s & ((1 << 63) - 1)


def _gen(seed: int, device) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    return g


def spectrum(wl: Workload) -> np.ndarray:
    """Singular spectrum sigma_1..sigma_d (non-increasing) of the synthetic K/V streams."""
    i = np.arange(1, wl.head_dim + 1, dtype=np.float64)
    if wl.spectrum == "inv":
        return 1.0 / i
    if wl.spectrum == "lowrank40":
        return (i <= 40).astype(np.float64)
    if wl.spectrum.startswith("pow"):
        return i ** (-float(wl.spectrum[3:]))
    raise ValueError(wl.spectrum)


def _scale(wl: Workload) -> float:
    sig = spectrum(wl)
    return math.sqrt((1.0 - wl.noise_std ** 2) * wl.head_dim / float(np.sum(sig ** 2)))


@functools.lru_cache(maxsize=256)
def _frames(wl: Workload, layer: int) -> np.ndarray:
    d = wl.head_dim
    out = np.empty((wl.n_kv_heads, 2, d, d))
    for g in range(wl.n_kv_heads):
        for kv in range(2):
            rng = np.random.Generator(np.random.Philox(seed_of(wl, "frame", 0, layer, g, kv)))
            a = rng.standard_normal((d, d))
            q, r = np.linalg.qr(a)
            q = q * np.sign(np.diag(r))[None, :]
            out[g, kv] = q
    out.setflags(write=False)
    return out


def frames(wl: Workload, layer: int) -> np.ndarray:
    """Orthonormal frames F [G][2][d][d] (fp64) for one layer: QR of a seeded Gaussian, with the
    diagonal of R made positive so the frame is unique for the seed."""
    return np.array(_frames(wl, layer))


@functools.lru_cache(maxsize=256)
def _bases(wl: Workload, layer: int) -> tuple[np.ndarray, np.ndarray]:
    d, n, G = wl.head_dim, CALIB_TOKENS, wl.n_kv_heads
    f = torch.from_numpy(frames(wl, layer).reshape(2 * G, d, d))   # stream 2 g + kv
    sig = torch.from_numpy(spectrum(wl) * _scale(wl))
    zs = torch.randn((2, 2 * G, n, d), generator=_gen(seed_of(wl, "calib", 0, layer), "cpu"),
                     dtype=torch.float32).double()
    x = (zs[0] * sig) @ f.transpose(1, 2)
    if wl.noise_std > 0:
        x += wl.noise_std * zs[1]
    # right singular vectors of each draw = eigenvectors of its Gram matrix, by decreasing eigenvalue
    vt = np.linalg.eigh((x.transpose(1, 2) @ x).numpy())[1][:, :, ::-1].transpose(0, 2, 1)
    lead = np.take_along_axis(vt, np.argmax(np.abs(vt), axis=2)[:, :, None], axis=2)
    vt = vt * np.sign(lead)
    out = np.ascontiguousarray(vt.reshape(G, 2, d, d).transpose(1, 0, 2, 3))
    out.setflags(write=False)
    return out[0], out[1]


def bases(wl: Workload, layer: int) -> tuple[np.ndarray, np.ndarray]:
    """Per-head bases U_K, U_V [G][d][d] (fp64), row j = basis vector j: the right singular vectors
    of a separate calibration draw (module docstring)."""
    uk, uv = _bases(wl, layer)
    return np.array(uk), np.array(uv)


def torch_dtype(wl: Workload) -> torch.dtype:
    return torch.float32 if wl.dtype == "f32" else torch.bfloat16


def outlier_tokens(wl: Workload, seq: int, layer: int) -> np.ndarray:
    """Sorted indices (within the coded set [0, N-w)) of tokens whose keys are scaled up."""
    n_coded = wl.n_ctx - wl.window
    n_out = int(round(wl.outlier_frac * n_coded))
    if n_out == 0:
        return np.zeros(0, dtype=np.int64)
    rng = np.random.Generator(np.random.Philox(seed_of(wl, "outlier", seq, layer)))
    return np.sort(rng.choice(n_coded, size=n_out, replace=False)).astype(np.int64)


def layer_kv(wl: Workload, seq: int, layer: int, device="cpu", out_dtype=None):
    """Keys and values of one (sequence, layer): two tensors [G][N][d] in the workload dtype
    (or ``out_dtype``), drawn on ``device``."""
    dt = out_dtype or torch_dtype(wl)
    d, n = wl.head_dim, wl.n_ctx
    sig = torch.tensor(spectrum(wl) * _scale(wl), dtype=torch.float32, device=device)
    f = torch.tensor(frames(wl, layer), dtype=torch.float32, device=device)  # [G][2][d][d]
    outs = []
    for kv, kind in ((0, "k"), (1, "v")):
        x = torch.empty((wl.n_kv_heads, n, d), dtype=dt, device=device)
        for g in range(wl.n_kv_heads):
            z = torch.randn((n, d), generator=_gen(seed_of(wl, kind, seq, layer, g), device),
                            device=device, dtype=torch.float32)
            y = (z * sig) @ f[g, kv].T
            if wl.noise_std > 0:
                e = torch.randn((n, d), device=device, dtype=torch.float32,
                                generator=_gen(seed_of(wl, "noise_" + kind, seq, layer, g), device))
                y.add_(e, alpha=wl.noise_std)
            x[g] = y.to(dt)
        outs.append(x)
    k, v = outs
    if wl.outlier_frac > 0:
        idx = torch.tensor(outlier_tokens(wl, seq, layer), device=device)
        k[:, idx] = (k[:, idx].float() * wl.outlier_scale).to(dt)
    return k, v


def window_queries(wl: Workload, seq: int, layer: int, device="cpu", out_dtype=None,
                   batch_index: int = 0) -> torch.Tensor:
    """Observation-window queries [w][H][d] of one (sequence, layer)."""
    dt = out_dtype or torch_dtype(wl)
    g = _gen(seed_of(wl, "qwin", seq, layer, 0, batch_index), device)
    return torch.randn((wl.window, wl.n_q_heads, wl.head_dim), generator=g, device=device,
                       dtype=torch.float32).to(dt)


def decode_queries(wl: Workload, seq: int, layer: int, n_steps: int, device="cpu",
                   out_dtype=None, batch_index: int = 0) -> torch.Tensor:
    """Decode-step queries [n_steps][H][d] of one (sequence, layer)."""
    dt = out_dtype or torch_dtype(wl)
    g = _gen(seed_of(wl, "qdec", seq, layer, 0, batch_index), device)
    return torch.randn((n_steps, wl.n_q_heads, wl.head_dim), generator=g, device=device,
                       dtype=torch.float32).to(dt)


def basis_tensors(wl: Workload, layer: int, device="cpu", out_dtype=None):
    """The per-head bases of one layer as [G][d][d] tensors in the workload dtype."""
    dt = out_dtype or torch_dtype(wl)
    uk, uv = bases(wl, layer)
    return (torch.tensor(uk, dtype=torch.float64).to(dt).to(device),
            torch.tensor(uv, dtype=torch.float64).to(dt).to(device))


def stack_inputs(wl: Workload, device="cpu", out_dtype=None, batch_index: int = 0):
    """All encode inputs of a workload, stacked in the library's layouts:
    k, v [B][L][G][N][d]; q_win [B][L][w][H][d]; basis_k, basis_v [L][G][d][d]."""
    dt = out_dtype or torch_dtype(wl)
    B, L, G, N, d = wl.batch, wl.n_layers, wl.n_kv_heads, wl.n_ctx, wl.head_dim
    k = torch.empty((B, L, G, N, d), dtype=dt, device=device)
    v = torch.empty_like(k)
    qw = torch.empty((B, L, wl.window, wl.n_q_heads, d), dtype=dt, device=device)
    for b in range(B):
        for l in range(L):
            kk, vv = layer_kv(wl, b, l, device=device, out_dtype=dt)
            k[b, l] = kk
            v[b, l] = vv
            qw[b, l] = window_queries(wl, b, l, device=device, out_dtype=dt, batch_index=batch_index)
    bk = torch.empty((L, G, d, d), dtype=dt, device=device)
    bv = torch.empty_like(bk)
    for l in range(L):
        a, c = basis_tensors(wl, l, device=device, out_dtype=dt)
        bk[l] = a
        bv[l] = c
    return k, v, qw, bk, bv


def stack_decode_queries(wl: Workload, layer: int, n_steps: int, device="cpu", out_dtype=None,
                         batch_index: int = 0) -> torch.Tensor:
    """Decode queries of every sequence for one layer: [n_steps][B][H][d]."""
    qs = [decode_queries(wl, b, layer, n_steps, device=device, out_dtype=out_dtype,
                         batch_index=batch_index) for b in range(wl.batch)]
    return torch.stack(qs, dim=1)
