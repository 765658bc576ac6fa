"""Host-side parts of bench.py that need no GPU: the DRAM-traffic records of the roofline objects.

A record holds the ncu DRAM bytes of one launch for one kernel source (sha256 prefix) and one
workload shape; the bench reports them only while both still match, and null otherwise.
"""

import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402


def test_gram_traffic_record_holds_read_plus_write_for_its_shape():
    rec = bench.GRAM_TC_TRAFFIC
    got = bench.recorded_traffic(rec, "gram_tc.cu", L=rec["L"], N=rec["N"], d=rec["d"])
    if got is not None:  # None only while the kernel source differs from the captured one
        assert got == float(rec["read"] + rec["write"])
    assert bench.recorded_traffic(rec, "gram_tc.cu", L=rec["L"], N=rec["N"] // 2, d=rec["d"]) is None


def test_kspace_traffic_record_checks_k_and_source():
    rec = bench.KSPACE_TRAFFIC
    shape = dict(L=rec["L"], N=rec["N"], d=rec["d"], k=rec["k"])
    got = bench.recorded_traffic(rec, "kspace.cu", **shape)
    if got is not None:
        assert got == float(rec["read"] + rec["write"])
        # the record covers the X read once: more than X, by less than 1%
        x_bytes = 2.0 * rec["L"] * rec["N"] * rec["d"]
        assert x_bytes < got < 1.01 * x_bytes
    assert bench.recorded_traffic(rec, "kspace.cu", **dict(shape, k=32)) is None
    stale = dict(rec, sha256="0000000000000000")
    assert bench.recorded_traffic(stale, "kspace.cu", **shape) is None
