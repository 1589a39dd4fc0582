"""bench.py's host-side accounting, checked on the CPU: launches per call, algorithmic
bytes of a call, the shared workload name of both arms, and the lookup of a
profile's traffic (only for the workload's full batch and a matching source hash)."""
import os
import re

import bench
import workloads as W


class _Args:
    def __init__(self, workload, mode):
        self.workload, self.mode = workload, mode


def test_launches_per_pipelined_call():
    assert bench.launches_per_step(256, 3072, True) == 2     # k_tiles + k_finish, overlapping
    assert bench.launches_per_step(64, 16384, True) == 2     # k_finish with 256 threads
    assert bench.launches_per_step(16, 196608, True) == 4    # + the long-row kernels, all overlapping
    assert bench.kernels_of_step(256, 3072, True) == ["k_tiles", "k_finish"]


def test_launches_per_call():
    assert bench.launches_per_step(32, 3072) == 1       # fused kernel (fewer than 64 chains)
    assert bench.launches_per_step(256, 3072) == 2      # k_tiles + k_finish
    assert bench.launches_per_step(64, 16384) == 2      # plain: k_tiles + 256-thread k_finish
    assert bench.launches_per_step(16, 196608) == 3     # + long-row dot and write
    assert bench.launches_per_step(1024, 3072) == 2     # k_tiles + k_finish
    assert bench.launches_per_step(1024, 16384) == 4    # k_finish caches up to 4096 elements


def test_algorithmic_bytes_of_a_call():
    # window read once, plus the rejected rows (m^q, m^p re-read) and y written, per chain
    assert bench.call_bytes(256, 8, 3072, "f32") == 3 * 256 * 8 * 3072 * 4 + 3 * 256 * 3072 * 4
    assert bench.call_bytes(64, 16, 16384, "bf16") == 3 * 64 * 16 * 16384 * 2 + 3 * 64 * 16384 * 2


def test_both_arms_name_the_workload_alike():
    cfg = W.VERIFY_CONFIGS["pixel"]
    name = bench.workload_name(_Args("pixel", "block"), cfg["B"], cfg["L"], cfg["d"], cfg["dtype"])
    assert name == "pixel verify (B=256, L=8, d=3072 f32), block mode"


def test_profile_traffic_lookup():
    path = os.path.join(bench.ROOT, "profiles", "verify_pixel_pipelined.md")
    txt = open(path).read()
    recorded = float(re.search(r"traffic_bytes_per_call:\s*([0-9.eE+]+)", txt).group(1))
    digest = re.search(r"kernel_source_sha256:\s*([0-9a-f]+)", txt).group(1)
    got = bench.profile_traffic("pixel", True, True)
    assert got == (recorded if digest == bench.kernel_sources_digest() else None)
    assert bench.profile_traffic("pixel", False, True) is None     # not the workload's full batch
    assert bench.profile_traffic("tiny", True, True) is None       # no summary for this workload
    # traffic, when reported, is the window plus at most the rejected rows and y
    if got is not None:
        assert 3 * 256 * 8 * 3072 * 4 <= got <= 1.02 * bench.call_bytes(256, 8, 3072, "f32")
