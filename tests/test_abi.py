"""Host-side checks of the C ABI (no GPU needed): the library loads, exports every function that
include/varrate.h declares, and its host-only functions (budget, sizing, validation) agree with
the oracle and reject bad arguments before touching a device."""
import json
import os
import re
import subprocess

import pytest

import oracle as O

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "varrate.h")


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(varrate_\w+)\s*\(", text)))


A = 1 << 12   # a 16-byte aligned fake device pointer (never dereferenced: host-side checks only)


def test_header_declares_the_hot_path():
    names = declared_functions()
    for must in ("varrate_encode", "varrate_allocate", "varrate_pack", "varrate_decode_attn",
                 "varrate_salience"):
        assert must in names


def test_library_exports_every_declared_symbol(vlib):
    lib = vlib.lib()
    out = subprocess.run(["nm", "-D", "--defined-only", vlib.LIB_PATH], capture_output=True,
                         text=True).stdout
    exported = set(re.findall(r"\bT (varrate_\w+)", out))
    for name in declared_functions():
        assert name in exported, name
        assert hasattr(lib, name)
    assert set(vlib.EXPORTED) == set(declared_functions())


def test_version_and_status_strings(vlib):
    assert vlib.varrate_version() >= 10000
    for code in (0, 1, -1, -2, -3, -4, -5, -6):
        assert vlib.status_string(code) and vlib.status_string(code) != "unknown status"
    assert vlib.status_string(12345) == "unknown status"


def test_coded_budget_matches_oracle_golden(vlib):
    with open(os.path.join(ROOT, "tests", "golden", "budgets.json")) as f:
        for c in json.load(f)["cases"]:
            cfg = vlib.make_config(1, 1, 1, c["n_ctx"], budget_frac=c["budget_frac"],
                                   window=c["window"], head_dim=c["head_dim"])
            assert vlib.varrate_coded_budget(cfg) == c["B_c"] == O.coded_budget(
                c["n_ctx"], c["head_dim"], c["window"], c["budget_frac"])


@pytest.mark.parametrize("n_ctx,w,kappa,rmin", [(2048, 32, 0.2, 16), (32768, 32, 0.1, 16),
                                                (32768, 32, 1.0, 16), (100, 100, 0.5, 1),
                                                (1037, 5, 0.33, 7)])
def test_cap_bounds_oracle(vlib, n_ctx, w, kappa, rmin):
    cfg = vlib.make_config(1, 1, 1, n_ctx, budget_frac=kappa, window=w, r_min=rmin)
    cap = vlib.varrate_packed_cap_elems(cfg)
    assert cap % 8 == 0
    assert cap >= O.packed_cap_elems(n_ctx, 128, w, kappa, rmin)


@pytest.mark.parametrize("field,value,want", [
    ("head_dim", 64, -5), ("group", 9, -5), ("window", 0, -1), ("r_min", 0, -1),
    ("r_min", 129, -1), ("budget_frac", 0.0, -1), ("budget_frac", 1.5, -1), ("pool_len", 4, -1),
    ("dtype", 7, -1), ("mode", 3, -1), ("n_ctx", 16, -1), ("batch", 0, -1)])
def test_check_config_rejects(vlib, field, value, want):
    cfg = vlib.make_config(2, 8, 4, 32768)
    assert vlib.varrate_check_config(cfg) == 0
    setattr(cfg, field, value)
    assert vlib.varrate_check_config(cfg) == want
    assert vlib.varrate_coded_budget(cfg) == -(2 ** 63)
    assert vlib.varrate_packed_cap_elems(cfg) == -1
    assert vlib.varrate_workspace_bytes(cfg, vlib.CALL_ENCODE) == 0


def test_group_window_product_limit(vlib):
    cfg = vlib.make_config(1, 2, 8, 4096, window=32)
    assert vlib.varrate_check_config(cfg) == 0
    cfg.window = 33
    assert vlib.varrate_check_config(cfg) == vlib.ERR_UNSUPPORTED


def test_workspace_sizes_positive(vlib):
    cfg = vlib.make_config(32, 8, 4, 32768, batch=8)
    for which in (vlib.CALL_SALIENCE, vlib.CALL_ENCODE, vlib.CALL_DECODE):
        assert vlib.varrate_workspace_bytes(cfg, which) > 0
    assert vlib.varrate_workspace_bytes(cfg, vlib.CALL_PACK) == 0


def test_decode_workspace_holds_the_counter_block(vlib):
    """The decode workspace starts with a 33024-byte header (a call count and two alternating sets
    of 4096 arrival counters) whatever the shape, so one zero-filled workspace serves calls of any
    shape; the scratch follows it."""
    sizes = set()
    for dtype in (vlib.F32, vlib.BF16):
        for b, g in ((1, 1), (8, 8), (64, 8)):
            cfg = vlib.make_config(2, g, 4, 4096, batch=b, dtype=dtype)
            n = vlib.varrate_workspace_bytes(cfg, vlib.CALL_DECODE)
            assert n >= 33024 + 256 and n % 256 == 0
            sizes.add(n)
    assert len(sizes) > 1


def test_null_arguments_rejected_on_host(vlib):
    cfg = vlib.make_config(1, 1, 4, 2048, dtype=vlib.F32)
    L = vlib.lib()
    assert L.varrate_salience(vlib.ctypes.byref(cfg), None, None, None, None, 0, None) == vlib.ERR_ARG
    assert L.varrate_allocate(vlib.ctypes.byref(cfg), None, None, None, None, None) == vlib.ERR_ARG
    p = vlib.varrate_packed()
    assert L.varrate_pack(vlib.ctypes.byref(cfg), 1, 1, 1, 1, vlib.ctypes.byref(p), None, None, 0,
                          None) == vlib.ERR_ARG
    assert L.varrate_encode(vlib.ctypes.byref(cfg), 1, 1, 1, 1, 1, None, vlib.ctypes.byref(p), None,
                            None, None, 0, None) == vlib.ERR_ARG
    assert L.varrate_decode_attn(vlib.ctypes.byref(cfg), vlib.ctypes.byref(p), 1, 1, 1, 0, None,
                                 None, 0, 1, None, None, 0, None) == vlib.ERR_ARG


def test_small_workspace_and_bad_layer_rejected_on_host(vlib):
    cfg = vlib.make_config(2, 1, 4, 2048, dtype=vlib.F32)
    L = vlib.lib()
    cap = vlib.varrate_packed_cap_elems(cfg)
    p = vlib.varrate_packed(A, A, A, A, A, A, cap)
    assert L.varrate_decode_attn(vlib.ctypes.byref(cfg), vlib.ctypes.byref(p), A, A, A, 2, None,
                                 None, 0, A, None, A, 1 << 40, None) == vlib.ERR_ARG
    assert L.varrate_decode_attn(vlib.ctypes.byref(cfg), vlib.ctypes.byref(p), A, A, A, 0, None,
                                 None, 0, A, None, A, 16, None) == vlib.ERR_WORKSPACE
    assert L.varrate_decode_attn(vlib.ctypes.byref(cfg), vlib.ctypes.byref(p), A, A, A, 0, None,
                                 None, 5000, A, None, A, 1 << 40, None) == vlib.ERR_UNSUPPORTED
    p.cap_elems = cap - 8
    assert L.varrate_decode_attn(vlib.ctypes.byref(cfg), vlib.ctypes.byref(p), A, A, A, 0, None,
                                 None, 0, A, None, A, 1 << 40, None) == vlib.ERR_ARG
    assert L.varrate_encode(vlib.ctypes.byref(cfg), A, A, A, A, A, None,
                            vlib.ctypes.byref(vlib.varrate_packed(A, A, A, A, A, A, cap)), None,
                            None, A, 8, None) == vlib.ERR_WORKSPACE


def test_window_decode_rejected_on_host(vlib):
    """varrate_decode_window: bf16 only, 1 <= n_q <= n_tail, n_q * group <= 128, and a workspace of
    varrate_workspace_bytes(cfg, VARRATE_CALL_DECODE_WINDOW), all checked before any launch."""
    L = vlib.lib()
    cfg = vlib.make_config(2, 2, 4, 2048, batch=2, dtype=vlib.BF16)
    cap = vlib.varrate_packed_cap_elems(cfg)
    p = vlib.varrate_packed(A, A, A, A, A, A, cap)
    big = 1 << 40
    need = vlib.varrate_workspace_bytes(cfg, vlib.CALL_DECODE_WINDOW)
    assert need > 0 and need % 256 == 0

    def call(c=cfg, n_q=4, layer=0, n_tail=8, tk=A, ws=A, nbytes=big, q=A):
        return L.varrate_decode_window(vlib.ctypes.byref(c), vlib.ctypes.byref(p), A, A, q, n_q, layer,
                                       tk, tk, n_tail, A, A, ws, nbytes, None)

    assert call(tk=None) == vlib.ERR_ARG
    assert call(n_q=0) == vlib.ERR_ARG
    assert call(n_q=9, n_tail=8) == vlib.ERR_ARG
    assert call(layer=2) == vlib.ERR_ARG
    assert call(q=A + 2) == vlib.ERR_ARG
    assert call(n_q=33, n_tail=40) == vlib.ERR_UNSUPPORTED      # 132 query rows
    assert call(n_tail=5000) == vlib.ERR_UNSUPPORTED
    assert call(nbytes=need - 256) == vlib.ERR_WORKSPACE
    assert call(ws=None) == vlib.ERR_WORKSPACE
    f32 = vlib.make_config(2, 2, 4, 2048, batch=2, dtype=vlib.F32)
    assert call(c=f32) == vlib.ERR_UNSUPPORTED


def test_misaligned_pointers_rejected_on_host(vlib):
    """Bulk copies and TMA need 16-byte aligned addresses: a misaligned device pointer is an
    argument error found on the host, before anything is enqueued."""
    cfg = vlib.make_config(2, 1, 4, 2048, dtype=vlib.BF16)
    L = vlib.lib()
    cap = vlib.varrate_packed_cap_elems(cfg)
    p = vlib.varrate_packed(A, A, A, A, A, A, cap)
    args = [A, A, A]                       # basis_k, basis_v, q
    for i in range(3):
        bad = list(args)
        bad[i] = A + 2
        assert L.varrate_decode_attn(vlib.ctypes.byref(cfg), vlib.ctypes.byref(p), *bad, 0, None,
                                     None, 0, A, None, A, 1 << 40, None) == vlib.ERR_ARG
    q = vlib.varrate_packed(A + 8, A, A, A, A, A, cap)
    assert L.varrate_decode_attn(vlib.ctypes.byref(cfg), vlib.ctypes.byref(q), A, A, A, 0, None,
                                 None, 0, A, None, A, 1 << 40, None) == vlib.ERR_ARG
    assert L.varrate_pack(vlib.ctypes.byref(cfg), A + 4, A, A, A, vlib.ctypes.byref(p), None, None,
                          0, None) == vlib.ERR_ARG


def test_binding_fails_loudly_without_library(tmp_path, monkeypatch):
    from paper_2607_15498_gb300 import varrate as V
    monkeypatch.setattr(V, "_lib", None)
    monkeypatch.setattr(V, "LIB_PATH", str(tmp_path / "missing.so"))
    with pytest.raises(RuntimeError, match="no CPU fallback"):
        V.lib()


def test_packed_cache_and_workspace_helpers(vlib):
    """The binding's allocators give the documented shapes, 16-byte aligned buffers and a
    zero-filled workspace (allocated here on the host: only the layout is checked)."""
    cfg = vlib.make_config(2, 3, 4, 1000, batch=2, dtype=vlib.BF16)
    p = vlib.PackedCache.allocate(cfg, "cpu")
    cap = vlib.varrate_packed_cap_elems(cfg)
    assert p.cap_elems == cap and cap % 8 == 0
    assert tuple(p.coef.shape) == (2, 2, 3, 2, cap) and p.coef.dtype == vlib.torch.bfloat16
    assert tuple(p.bucket_count.shape) == (2, 2, 129) and tuple(p.bucket_base.shape) == (2, 2, 130)
    for t in (p.coef, p.bucket_count, p.bucket_base, p.perm, p.pos, p.ranks):
        assert t.data_ptr() % 16 == 0
    ws = vlib.workspace(cfg, vlib.CALL_DECODE, "cpu")
    assert ws.numel() >= vlib.varrate_workspace_bytes(cfg, vlib.CALL_DECODE)
    assert int(vlib.torch.count_nonzero(ws)) == 0


def test_selftest_wait_rejects_bad_arguments_on_host(vlib):
    """The bounded-wait self-test validates its arguments before anything is launched."""
    import ctypes
    buf = ctypes.create_string_buffer(16)
    base = ctypes.addressof(buf)
    aligned = base + ((-base) % 4)
    assert vlib.lib().varrate_selftest_wait_timeout(None, 8, None) == vlib.ERR_ARG
    assert vlib.lib().varrate_selftest_wait_timeout(ctypes.c_void_p(aligned), 0, None) == vlib.ERR_ARG
    assert vlib.lib().varrate_selftest_wait_timeout(ctypes.c_void_p(aligned), (1 << 24) + 1, None) == vlib.ERR_ARG
    assert vlib.lib().varrate_selftest_wait_timeout(ctypes.c_void_p(aligned + 1), 8, None) == vlib.ERR_ARG


def test_anchor_search_host_checks(vlib):
    """Workspace size of the nearest-anchor search and the argument checks made before any launch:
    anchors padded to 256 (ceil(1000 / 16) = 63 -> 256), 3 sequences x 2 layers, G = 8:
    anchors 6 * 2 * 8 * 256 * 128 * 2 B, their norms 6 * 256 * 4 B, token norms 6 * 1000 * 4 B,
    each rounded up to 256 B."""
    L = vlib.lib()
    cfg = vlib.make_config(2, 8, 4, 1000, batch=3, dtype=vlib.BF16)
    assert vlib.varrate_anchor_search_ws_bytes(cfg, 16) == 6291456 + 6144 + 24064
    assert vlib.varrate_anchor_search_ws_bytes(cfg, 0) == 0
    assert vlib.varrate_anchor_search_ws_bytes(cfg, 1001) == 0
    need = vlib.varrate_anchor_search_ws_bytes(cfg, 16)

    def call(c=cfg, k=A, v=A, stride=16, n=4, idx=A, dist=A, ws=A, nbytes=need):
        return L.varrate_anchor_search(vlib.ctypes.byref(c), k, v, stride, n, idx, dist, None, ws,
                                       nbytes, None)
    assert call(k=None) == vlib.ERR_ARG
    assert call(idx=None) == vlib.ERR_ARG
    assert call(stride=0) == vlib.ERR_ARG
    assert call(stride=1001) == vlib.ERR_ARG
    assert call(n=0) == vlib.ERR_ARG
    assert call(n=9) == vlib.ERR_UNSUPPORTED
    assert call(v=A + 8) == vlib.ERR_ARG
    assert call(dist=A + 4) == vlib.ERR_ARG
    assert call(nbytes=need - 1) == vlib.ERR_WORKSPACE
    assert call(ws=None) == vlib.ERR_WORKSPACE
    f32 = vlib.make_config(2, 8, 4, 1000, batch=3, dtype=vlib.F32)
    assert call(c=f32) == vlib.ERR_UNSUPPORTED


def test_anchor_residual_host_checks(vlib):
    """Argument checks of the residual entry point, made before any launch."""
    L = vlib.lib()
    cfg = vlib.make_config(2, 8, 4, 1000, batch=3, dtype=vlib.BF16)

    def call(c=cfg, k=A, v=A, stride=16, n=4, idx=A, e=A):
        return L.varrate_anchor_residual(vlib.ctypes.byref(c), k, v, stride, n, idx, e, None, None)
    assert call(k=None) == vlib.ERR_ARG
    assert call(idx=None) == vlib.ERR_ARG
    assert call(e=None) == vlib.ERR_ARG
    assert call(stride=0) == vlib.ERR_ARG
    assert call(stride=1001) == vlib.ERR_ARG
    assert call(n=0) == vlib.ERR_ARG
    assert call(n=9) == vlib.ERR_UNSUPPORTED
    assert call(e=A + 2) == vlib.ERR_ARG
    f32 = vlib.make_config(2, 8, 4, 1000, batch=3, dtype=vlib.F32)
    assert call(c=f32) == vlib.ERR_UNSUPPORTED
