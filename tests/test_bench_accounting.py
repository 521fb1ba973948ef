"""bench.py's byte accounting, on CPU.

The roofline fraction divides algorithmic bytes by measured time, so the
bytes must be the definition's: every cached K and V row attended to once
(the new token's included), the queries and the outputs, and the new row the
fused step writes (Eq. (attn); Sec. III-C appends the token uncompressed).
The rows come from the workload's lengths through the oracle's compressed
length (speech pooled in windows of w from l0 on, Eq. (pool)).  The
committed ncu traffic figures feed roofline.traffic only while they were
taken on the current decode-kernel source.
"""
import glob
import os
import shlex
import sys
import types

import pytest

from paper_2607_06827_gb300 import inputs
from tests import harness as H

sys.path.insert(0, H.ROOT)
import bench  # noqa: E402


def _traffic_file():
    kv = {}
    with open(bench.PROFILE_TRAFFIC) as f:
        for line in f:
            if "=" in line and not line.startswith("#"):
                k, v = line.strip().split("=", 1)
                kv[k.strip()] = v.strip()
    return kv


def _expected_bytes(wl, rows_per_req):
    s = 2  # bf16
    kv = sum(rows_per_req) * wl.H_kv * wl.d * 2 * s
    q_and_out = 2 * wl.B * wl.H_q * wl.d * s
    new_rows = wl.B * wl.H_kv * wl.d * 2 * s
    return kv + q_and_out + new_rows


def test_profiled_traffic_is_for_the_current_kernel_source():
    assert os.path.exists(bench.PROFILE_TRAFFIC)
    assert _traffic_file()["kernel_sha256_16"] == bench.kernel_hash(), (
        "decode kernel sources changed since the committed ncu traffic capture; "
        "recapture it (roofline.traffic is reported as null meanwhile)")


def test_attn_bytes_reproduce_the_profiled_launches(oracle):
    """The captured launches were pooled layer 8 and full-resolution layer 0
    of the 20 min / w = 4 / batch 8 workload (64 tokens already generated),
    three decode steps into the run: 3881 and 15131 rows per request."""
    wl = inputs.qwen_long_audio(20, 4, generated=bench.GENERATED)
    kv = _traffic_file()
    me = types.SimpleNamespace(wl=wl)
    for kind, layer in (("pooled", wl.l0), ("full", 0)):
        rows = [oracle.compressed_len(wl.P[b], wl.T[b], wl.N[b], wl.G[b], wl.w, layer, wl.l0) + 3
                for b in range(wl.B)]
        assert rows == [3881 if kind == "pooled" else 15131] * wl.B
        got = bench.DecodeModel.attn_bytes(me, rows, fused=True)
        assert got == _expected_bytes(wl, rows) == int(kv[f"{kind}_algorithmic_bytes"])
        # the unfused attention launch does not write the new row
        assert bench.DecodeModel.attn_bytes(me, rows, fused=False) == \
            got - wl.B * wl.H_kv * wl.d * 2 * 2


def test_traffic_scales_each_kind_by_its_own_ratio():
    kv = _traffic_file()
    res = {"n_compressed_layers": 20, "n_full_layers": 8,
           "attn_bytes_per_launch_compressed": 100.0, "attn_bytes_per_launch_full": 400.0}
    rp = float(kv["pooled_dram_bytes_per_launch"]) / float(kv["pooled_algorithmic_bytes"])
    rf = float(kv["full_dram_bytes_per_launch"]) / float(kv["full_algorithmic_bytes"])
    assert 1.0 <= rp < 1.1 and 1.0 <= rf < 1.1
    assert bench.profiled_traffic(res) == round((20 * rp * 100.0 + 8 * rf * 400.0) / 28)


def test_profile_commands_parse(monkeypatch):
    """Each ncu summary under profiles/ names the bench command it captured;
    every such command must still be accepted by the bench's arguments."""
    cmds = []
    for path in sorted(glob.glob(os.path.join(H.ROOT, "profiles", "*"))):
        for line in open(path):
            line = line.strip().rstrip("\\").strip()
            at = line.find("python bench.py")
            if at >= 0:
                cmds.append((os.path.basename(path), line[at + len("python bench.py"):]))
    assert len(cmds) >= 6
    for name, argv in cmds:
        monkeypatch.setattr(sys, "argv", ["bench.py", *shlex.split(argv)])
        try:
            bench.parse_args()
        except SystemExit:
            pytest.fail(f"{name}: bench.py rejects {argv!r}")
