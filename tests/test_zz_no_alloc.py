"""sdv_verify_noalloc: the verification step for callers that cannot allocate device memory.

Some callers may not call cudaMalloc at all - plug-ins inside a host program that owns
every device allocation, or real-time loops where cudaMalloc's implicit
synchronisation and possible failure are not allowed.  sdv_verify_noalloc takes no
workspace and uses a static device array of the library instead.  This test calls it
through the C ABI twice in a row (so the second call starts from the first call's
leftover scratch) and checks each result against sdv_verify with a caller-provided
workspace, within the tolerances of the other parity tests.  The file is named so that
pytest collects it last.
"""
import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu


def _dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def _run(B_, fn_name, inp, seed, mode, ws=None):
    Bn, L, d = inp["x_draft"].shape
    x, mq, mp, sg = (_dev(inp[k]) for k in ("x_draft", "mu_target", "mu_draft", "sigma"))
    acc = torch.empty(Bn, dtype=torch.int32, device="cuda")
    y = torch.empty(Bn, d, dtype=torch.float32, device="cuda")
    lr = torch.empty(Bn, L, dtype=torch.float32, device="cuda")
    dn = torch.empty(Bn, L, dtype=torch.float32, device="cuda")
    st = torch.empty(Bn, dtype=torch.int32, device="cuda")
    stream = torch.cuda.current_stream().cuda_stream
    args = (x.data_ptr(), mq.data_ptr(), mp.data_ptr(), sg.data_ptr(), L, Bn, L, d, B_.SDV_F32,
            seed, mode, acc.data_ptr(), y.data_ptr(), lr.data_ptr(), dn.data_ptr(), st.data_ptr())
    if fn_name == "sdv_verify":
        B_.sdv_verify(*args, ws.data_ptr(), ws.numel(), stream)
    else:
        B_.sdv_verify_noalloc(*args, stream)
    torch.cuda.synchronize()
    return acc.cpu().numpy(), y.cpu().numpy(), lr.cpu().numpy(), st.cpu().numpy()


def test_noalloc_matches_workspace_entry_point_twice():
    import __graft_entry__ as g
    g.build()
    import workloads as W
    from paper_2606_13426_gb300 import api
    from paper_2606_13426_gb300 import binding as B_

    cases = [(W.make_verify_inputs("pixel", B=96, L=8, d=3072, per_chain_sigma=True), 21,
              B_.SDV_MODE_BLOCK),
             (W.make_verify_inputs("tiny", B=40, L=5, d=37, per_chain_sigma=True), 22,
              B_.SDV_MODE_SAMPLE)]
    # two calls in a row through the static scratch, then the reference calls
    got = [_run(B_, "sdv_verify_noalloc", inp, seed, mode) for inp, seed, mode in cases]
    for (inp, seed, mode), (acc, y, lr, st) in zip(cases, got):
        Bn, L, d = inp["x_draft"].shape
        ws = api.make_workspace(Bn, L, d)
        acc_r, y_r, lr_r, st_r = _run(B_, "sdv_verify", inp, seed, mode, ws)
        np.testing.assert_array_equal(acc, acc_r)
        np.testing.assert_array_equal(st, st_r)
        assert np.all(np.abs(lr - lr_r) <= 1e-5 * np.maximum(1.0, np.abs(lr_r)))
        assert np.max(np.abs(y - y_r)) <= 1e-5


def test_noalloc_rejects_problems_beyond_its_scratch():
    import __graft_entry__ as g
    g.build()
    from paper_2606_13426_gb300 import binding as B_
    assert B_.sdv_workspace_bytes(16, 32, 196608, B_.SDV_F32) <= B_.SDV_NOALLOC_SCRATCH_BYTES
    big = (4096, 64, 65536)            # needs more than SDV_NOALLOC_SCRATCH_BYTES of scratch
    assert B_.sdv_workspace_bytes(*big, B_.SDV_F32) > B_.SDV_NOALLOC_SCRATCH_BYTES
    lib = B_.load()
    rc = lib.sdv_verify_noalloc(0x1000, 0x2000, 0x3000, 0x4000, 0, big[0], big[1], big[2],
                                B_.SDV_F32, 0, 1, 0x5000, 0x6000, 0, 0, 0, None)
    assert rc == B_.SDV_ENOWORKSPACE
