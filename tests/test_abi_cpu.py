"""C-ABI checks that need no GPU: the library builds, loads, exports every symbol
include/specdiff.h declares, and rejects bad arguments on the host (before any launch)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "specdiff.h")


@pytest.fixture(scope="module")
def lib():
    from paper_2606_13426_gb300 import binding, buildlib
    try:
        buildlib.build()
    except RuntimeError as e:  # no nvcc on this machine
        pytest.skip(str(e))
    return binding.load()


def declared_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(sdv_[a-z_0-9]+)\s*\(", src)))


def test_every_declared_symbol_is_exported_and_bound(lib):
    from paper_2606_13426_gb300 import binding
    names = declared_functions()
    assert len(names) >= 10
    for n in names:
        assert hasattr(lib, n), n
        assert n in binding.SIGNATURES, n
    assert set(binding.SIGNATURES) == set(names)


def test_version_and_errors(lib):
    from paper_2606_13426_gb300 import binding as B
    assert "sm_103a" in B.sdv_version()
    assert B.strerror(B.SDV_EINVAL) == "invalid argument"
    assert B.sdv_workspace_bytes(0, 4, 16, B.SDV_F32) == 0
    assert B.sdv_workspace_bytes(4, 65, 16, B.SDV_F32) == 0
    assert B.sdv_workspace_bytes(4, 4, 16, 7) == 0
    w1 = B.sdv_workspace_bytes(256, 8, 3072, B.SDV_F32)
    w2 = B.sdv_workspace_bytes(16, 32, 196608, B.SDV_F32)
    assert w1 > 0 and w2 > 0 and w1 % 256 == 0
    assert B.sdv_workspace_bytes(256, 8, 3072, B.SDV_BF16) <= w1


def _verify_ex(lib, **kw):
    a = dict(x=0x10000, mq=0x20000, mp=0x30000, sigma=0x40000, sstride=0, B=4, L=4, d=16,
             dtype=0, seed=0, mode=1, L_eff=0, mqb=0, sb=0, resid=0, omega=1.0,
             acc=0x50000, y=0x60000, lr=0, dn=0, st=0, aux=0, ws=0x70000, wsb=1 << 20)
    a.update(kw)
    return lib.sdv_verify_ex(a["x"], a["mq"], a["mp"], a["sigma"], a["sstride"], a["B"], a["L"],
                             a["d"], a["dtype"], a["seed"], a["mode"], a["L_eff"], a["mqb"],
                             a["sb"], a["resid"], a["omega"], a["acc"], a["y"], a["lr"], a["dn"],
                             a["st"], a["aux"], a["ws"], a["wsb"], None)


def test_host_validation_rejects_before_launch(lib):
    from paper_2606_13426_gb300 import binding as B
    assert _verify_ex(lib, x=0) == B.SDV_EINVAL
    assert _verify_ex(lib, B=0) == B.SDV_EINVAL
    assert _verify_ex(lib, L=0) == B.SDV_EINVAL
    assert _verify_ex(lib, L=65) == B.SDV_EINVAL
    assert _verify_ex(lib, d=0) == B.SDV_EINVAL
    assert _verify_ex(lib, dtype=3) == B.SDV_EINVAL
    assert _verify_ex(lib, mode=2) == B.SDV_EINVAL
    assert _verify_ex(lib, resid=5) == B.SDV_EINVAL
    assert _verify_ex(lib, resid=1, mode=1) == B.SDV_EINVAL      # reflection needs sample mode
    assert _verify_ex(lib, omega=0.0) == B.SDV_EINVAL
    assert _verify_ex(lib, omega=float("nan")) == B.SDV_EINVAL
    assert _verify_ex(lib, sstride=-1) == B.SDV_EINVAL
    assert _verify_ex(lib, acc=0) == B.SDV_EINVAL
    assert _verify_ex(lib, mqb=0x80000) == B.SDV_EINVAL           # bonus mean without sigma
    assert _verify_ex(lib, x=0x10002) == B.SDV_EALIGN              # fp32 needs 4-byte alignment
    assert _verify_ex(lib, x=0x10002, dtype=1) != B.SDV_EALIGN     # bf16 needs 2 bytes
    assert _verify_ex(lib, ws=0) == B.SDV_ENOWORKSPACE
    assert _verify_ex(lib, wsb=16) == B.SDV_ENOWORKSPACE
    assert _verify_ex(lib, ws=0x70010) == B.SDV_EALIGN
    assert lib.sdv_accept_scan(0, 0, 4, 4, 0, 0, 1, 1.0, 0, 0, None) == B.SDV_EINVAL
    assert lib.sdv_usample(0x100, 0x200, 0x300, -1, 0x400, 0, None) == B.SDV_EINVAL
    assert lib.sdv_usample(0x100, 0x200, 0x300, 0, 0x400, 0, None) == B.SDV_OK  # empty: no launch
    assert lib.sdv_philox(0x100, 0, 0, 0x208, None) == B.SDV_EALIGN
    assert lib.sdv_normals(0, 0, 16, 2, 0, 0x100, None) == B.SDV_EINVAL


def test_sampler_entry_points_validate_before_launch(lib):
    from paper_2606_13426_gb300 import binding as B
    sch = (8, 1.0, 40, 0.5, 0.1, 20.0, 1e-4)       # C, comp_var, K, churn, beta_min, beta_max, t_floor
    wsb = B.sdv_sampler_workspace_bytes(4, 4, 16)
    assert wsb > 0 and B.sdv_sampler_workspace_bytes(4, 65, 16) == 0

    def begin(**kw):
        a = dict(B=4, L=4, d=16, means=0x1000, lw=0x2000, ws=0x100000, wsb=wsb)
        a.update(kw)
        return lib.sdv_sampler_begin(a["B"], a["L"], a["d"], a["means"], a["lw"], *sch, 1, a["ws"],
                                     a["wsb"], None)

    def rnd(**kw):
        a = dict(B=4, L=4, d=16, mode=1, drafter=0, ws=0x100000, wsb=wsb)
        a.update(kw)
        return lib.sdv_sampler_round(a["B"], a["L"], a["d"], 0x1000, 0x2000, *sch, 1, a["mode"],
                                     a["drafter"], a["ws"], a["wsb"], None)

    assert begin(means=0) == B.SDV_EINVAL
    assert begin(B=0) == B.SDV_EINVAL
    assert begin(L=65) == B.SDV_EINVAL
    assert begin(ws=0) == B.SDV_ENOWORKSPACE
    assert begin(wsb=wsb - 1) == B.SDV_ENOWORKSPACE
    assert begin(ws=0x100010) == B.SDV_EALIGN
    assert rnd(mode=2) == B.SDV_EINVAL
    assert rnd(drafter=5) == B.SDV_EINVAL
    assert rnd(ws=0) == B.SDV_ENOWORKSPACE
    y = ctypes.c_int32(0)
    assert lib.sdv_sampler_end(4, 4, 16, 0x100000, wsb, 0, 0, 0, 0, ctypes.addressof(y), None) == B.SDV_EINVAL
    assert lib.sdv_sampler_end(4, 4, 16, 0, wsb, 0x3000, 0, 0, 0, ctypes.addressof(y), None) == \
        B.SDV_ENOWORKSPACE
    assert lib.sdv_sampler_end(0, 4, 16, 0x100000, wsb, 0x3000, 0, 0, 0, ctypes.addressof(y), None) == \
        B.SDV_EINVAL


def test_python_binding_raises_on_error(lib):
    from paper_2606_13426_gb300 import binding as B
    with pytest.raises(B.SDVError) as ei:
        B.sdv_accept_scan(0, 0, 4, 4, 0, 0, 1, 1.0, 0, 0, None)
    assert ei.value.code == B.SDV_EINVAL
