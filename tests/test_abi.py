"""The C-ABI library loads, exports every symbol include/grkv.h declares, and
rejects bad arguments on the host with the documented codes (no GPU needed:
validation runs before any CUDA call)."""
import ctypes
import os
import re
import subprocess

import pytest

from paper_2605_31105_gb300 import binding as b
from paper_2605_31105_gb300 import build as build_mod

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    srcs = [os.path.join(build_mod.CSRC, f) for f in os.listdir(build_mod.CSRC)]
    srcs.append(os.path.join(ROOT, "include", "grkv.h"))
    if not os.path.exists(b.LIB_PATH) or any(
            os.path.getmtime(s) > os.path.getmtime(b.LIB_PATH) for s in srcs):
        build_mod.build()
    return b.load()


def declared_functions():
    with open(os.path.join(ROOT, "include", "grkv.h")) as f:
        text = f.read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(grkv_\w+)\s*\(", text)))


def test_every_declared_symbol_is_exported(lib):
    names = declared_functions()
    assert set(names) >= {"grkv_score", "grkv_select", "grkv_merge", "grkv_compress"}
    out = subprocess.run(["nm", "-D", "--defined-only", b.LIB_PATH], capture_output=True,
                         text=True, check=True).stdout
    exported = set(re.findall(r"\s[TW]\s+(grkv_\w+)$", out, flags=re.M))
    assert set(names) <= exported, set(names) - exported
    assert set(b.EXPORTS) == set(names)
    for n in names:
        assert hasattr(lib, n)


def test_params_init_defaults(lib):
    p = b.params(256, 4, 32768, 32, 2048)
    assert p.steps == 1 and p.step_tol == pytest.approx(1e-9)
    assert (p.d, p.pool_kernel, p.pool_type, p.n_sink, p.causal, p.dtype) == (128, 7, 0, 4, 1, 1)
    assert p.beta == pytest.approx(0.1) and p.lambda_v == pytest.approx(1e-2)


def test_workspace_size_and_validation(lib):
    p = b.params(8, 4, 8192, 32, 512)
    assert b.grkv_workspace_size(p) > 0
    bad = [dict(budget=16), dict(budget=9000), dict(pool_kernel=6), dict(pool_kernel=0),
           dict(beta=1.0), dict(beta=-0.1), dict(lambda_v=-1.0), dict(lambda_v=float("nan")),
           dict(causal=2), dict(dtype=7), dict(window_zero=True), dict(units=-1),
           dict(n_sink=-1), dict(flags=0x100), dict(pool_type=3), dict(scale=-1.0),
           dict(flags=b.GRKV_UPDATE_K, lambda_k=-1.0),
           dict(flags=b.GRKV_UPDATE_K, lambda_k=float("inf")),
           dict(flags=b.GRKV_UPDATE_K, lambda_k=float("nan")),
           dict(flags=b.GRKV_UPDATE_K, cg_iters=-1),
           dict(flags=b.GRKV_UPDATE_K, cg_iters=4097),
           dict(flags=b.GRKV_UPDATE_K, cg_tol=-1.0),
           dict(flags=b.GRKV_UPDATE_K, cg_tol=float("inf")),
           dict(steps=0), dict(steps=2), dict(flags=b.GRKV_UPDATE_K, steps=65),
           dict(step_tol=-1.0), dict(step_tol=float("inf"))]
    for kw in bad:
        q = b.params(8, 4, 8192, 32, 512)
        for key, val in kw.items():
            if key == "window_zero":
                q.window = 0
                q.group = 0
            else:
                setattr(q, key, val)
        with pytest.raises(b.GrkvError) as e:
            b.grkv_workspace_size(q)
        assert e.value.code == b.GRKV_ERR_INVALID_ARG, kw
    for kw in (dict(d=64), dict(group=9)):
        q = b.params(8, 4, 8192, 32, 512)
        for key, val in kw.items():
            setattr(q, key, val)
        with pytest.raises(b.GrkvError) as e:
            b.grkv_workspace_size(q)
        assert e.value.code == b.GRKV_ERR_UNSUPPORTED, kw
    # the key step adds its workspace; lambda_k and cg_iters are read only with it
    plain = b.grkv_workspace_size(b.params(8, 4, 8192, 32, 512))
    keyed = b.grkv_workspace_size(b.params(8, 4, 8192, 32, 512, flags=b.GRKV_UPDATE_K))
    assert keyed > plain
    assert b.grkv_workspace_size(b.params(8, 4, 8192, 32, 512, lambda_k=-1.0, cg_iters=-5)) == plain
    dp = b.params(1, 1, 64, 8, 16)
    assert dp.cg_iters == 512 and abs(dp.cg_tol - 1e-4) < 1e-9
    # lambda = +inf is valid: the value step leaves V0 unchanged
    assert b.grkv_workspace_size(b.params(8, 4, 8192, 32, 512, lambda_v=float("inf"))) > 0


def test_host_checks_before_any_launch(lib):
    p = b.params(2, 4, 1024, 32, 128)
    need = b.grkv_workspace_size(p)
    fake = 1 << 20   # never dereferenced: every check below fails on the host
    rc = b.grkv_compress(p, fake, fake, fake, fake, fake, fake, fake, need - 1, stream=0,
                         check=False)
    assert rc == b.GRKV_ERR_WORKSPACE_TOO_SMALL
    rc = b.grkv_compress(p, fake + 8, fake, fake, fake, fake, fake, fake, need, stream=0,
                         check=False)
    assert rc == b.GRKV_ERR_MISALIGNED
    rc = b.grkv_compress(p, 0, fake, fake, fake, fake, fake, fake, need, stream=0, check=False)
    assert rc == b.GRKV_ERR_INVALID_ARG
    rc = b.grkv_select(p, fake, fake, 0, need, stream=0, check=False)
    assert rc == b.GRKV_ERR_INVALID_ARG
    assert lib.grkv_compress(None, None, None, None, None, None, None, None, 0, None) == \
        b.GRKV_ERR_INVALID_ARG
    st = ctypes.c_int(0)
    assert lib.grkv_status(None, ctypes.byref(st), None) == b.GRKV_ERR_INVALID_ARG


def test_strerror(lib):
    assert b.strerror(0) == "ok"
    assert "Cholesky" in b.strerror(b.GRKV_ERR_NUMERIC)
    assert b.strerror(-99) == "unknown error"


def test_transfer_check_validation(lib):
    import ctypes as C
    p = b.params(8, 4, 8192, 32, 512)
    assert b.grkv_transfer_workspace_size(p, 32) > b.grkv_workspace_size(p) // 4
    n = C.c_size_t(0)
    L = b.load()
    assert L.grkv_transfer_workspace_size(C.byref(p), 0, C.byref(n)) == b.GRKV_ERR_INVALID_ARG
    assert L.grkv_transfer_workspace_size(C.byref(p), 513, C.byref(n)) == b.GRKV_ERR_INVALID_ARG
    assert L.grkv_transfer_workspace_size(C.byref(p), 65, C.byref(n)) == b.GRKV_ERR_UNSUPPORTED
    ws = (C.c_uint8 * 64)()
    z = C.c_void_p(16)
    rc = L.grkv_transfer_check(C.byref(p), 32, z, z, z, z, z, z, z, z, C.cast(ws, C.c_void_p), 64, None)
    assert rc in (b.GRKV_ERR_WORKSPACE_TOO_SMALL, b.GRKV_ERR_MISALIGNED)
