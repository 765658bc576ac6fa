"""Host-side parts of bench.py that need no GPU: the DRAM-traffic records of the roofline objects.

A record holds the ncu DRAM bytes of one launch of one kernel source (sha256 prefix), captured on
a small case (L_capture blocks at the workload's own N and d); the bench scales it by the number
of blocks and reports it only while the source and the shape still match, and null otherwise.
"""

import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402


def test_gram_traffic_record_scales_with_blocks_and_checks_shape():
    rec = bench.GRAM_TC_TRAFFIC
    got = bench.recorded_traffic(rec, "gram_tc.cu", rec["L_capture"], N=rec["N"], d=rec["d"])
    if got is not None:  # None only while the kernel source differs from the captured one
        assert got == float(rec["read"] + rec["write"])
        assert bench.recorded_traffic(rec, "gram_tc.cu", 28, N=rec["N"], d=rec["d"]) == 14 * got
    assert bench.recorded_traffic(rec, "gram_tc.cu", 28, N=rec["N"] // 2, d=rec["d"]) is None


def test_kspace_traffic_record_checks_k_and_source():
    rec = bench.KSPACE_TRAFFIC
    shape = dict(N=rec["N"], d=rec["d"], k=rec["k"])
    got = bench.recorded_traffic(rec, "kspace.cu", rec["L_capture"], **shape)
    if got is not None:
        assert got == float(rec["read"] + rec["write"])
        # the record covers the X read once: more than X, by less than 1%
        x_bytes = 2.0 * rec["L_capture"] * rec["N"] * rec["d"]
        assert x_bytes < got < 1.01 * x_bytes
    assert bench.recorded_traffic(rec, "kspace.cu", rec["L_capture"], **dict(shape, k=32)) is None
    stale = dict(rec, sha256="0000000000000000")
    assert bench.recorded_traffic(stale, "kspace.cu", rec["L_capture"], **shape) is None


def test_targets_traffic_record_is_the_write_of_T():
    rec = bench.TARGETS_TRAFFIC
    got = bench.recorded_traffic(rec, "targets.cu", rec["L_capture"], N=rec["N"], d=rec["d"], r=rec["r"])
    if got is not None:
        t_bytes = 2.0 * rec["L_capture"] * rec["N"] * rec["d"]
        # the write of T (part of it may still sit in L2 when the kernel ends) and a few reads
        assert 0.95 * t_bytes < got < 1.01 * t_bytes
