"""Host logic of bench.py on CPU: the byte counts, the roofline of the dominant
call, and the committed ncu summaries it reads its DRAM traffic from.

The workload's throughput is algorithmic bytes (kept values + stored offsets +
row metadata + X read once + Y written once) over time against the HBM peak;
work a kernel executes beyond that (the zeros and the two bf16 parts of X that
the tensor-core path multiplies) may be reported beside it, never as achieved.
"""
import os
import re
import sys
import types

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402

# FC6 as encoded by the bench workload's shapes: 4096 x 9216 bf16, a made-up
# kept count with 4-bit offsets for a third of the blocks
FC6 = {"rows": 4096, "cols": 9216, "wtype": 1, "nnzb": 1_470_000,
       "value_bytes": 2 * 1_470_000, "offset_bytes": 490_000 // 2 + 980_000, "meta_bytes": 4096 * 6}


def test_spmm_bytes_count_what_the_product_must_move():
    b = 256
    want = (FC6["value_bytes"] + FC6["offset_bytes"] + FC6["meta_bytes"]
            + FC6["cols"] * b * 4 + FC6["rows"] * b * 4)
    assert bench.spmm_bytes(FC6, b) == want
    # the dense work the format avoids is not counted: far below a dense bf16 W
    assert bench.spmm_bytes(FC6, 1) < FC6["rows"] * FC6["cols"] * 2 / 10


def test_encode_bytes_are_dense_w_plus_the_encoding():
    assert bench.encode_bytes(FC6) == (FC6["rows"] * FC6["cols"] * 2 + FC6["value_bytes"]
                                       + FC6["offset_bytes"] + FC6["meta_bytes"])


def _workload(path):
    wl = types.SimpleNamespace()
    b = 256
    wl.calls = [("spmm", 0, b, bench.spmm_bytes(FC6, b))]
    wl.paths = [(path, 2 if path == "tensor" else 1)]
    wl.mats = [{"rows": FC6["rows"], "cols": FC6["cols"], "info": FC6}]
    return wl


@pytest.mark.parametrize("path", ["tensor", "cuda"])
def test_roofline_of_the_dominant_call_is_algorithmic_bytes_over_hbm(path):
    wl = _workload(path)
    ms = 0.040
    achieved = wl.calls[0][3] / (ms * 1e-3) / 1e9
    r = bench.roofline(wl, 0, "fc6_spmm_b256", ms, achieved, 6790.0, "measured", 1900.0, "measured",
                       12345, 0.18, 40000.0)
    assert r["bound"] == "hbm" and r["unit"] == "GB/s"
    assert r["achieved"] == pytest.approx(achieved, abs=0.1)
    assert r["frac"] == pytest.approx(achieved / 6790.0, abs=1e-4)
    assert r["traffic"] == 12345
    assert r["share_of_step"] == pytest.approx(0.040 / 0.18, abs=1e-3)
    if path == "tensor":
        ex = r["tensor_executed"]
        # the executed densified product, reported as context: 2 x 2 x rows x cols x batch
        assert ex["flops_per_call"] == 2 * 2 * FC6["rows"] * FC6["cols"] * 256
        assert ex["algorithmic_flops_per_call"] == 2 * FC6["nnzb"] * 256
        assert ex["frac"] == pytest.approx(ex["tflops"] / 1900.0, abs=1e-3)
        assert "binding" in r and 0.0 < r["gather_equiv_frac"]
    else:
        assert "tensor_executed" not in r


PROFILES = os.path.join(ROOT, "profiles")
SUMMARIES = sorted(f for f in os.listdir(PROFILES) if f.endswith((".md", ".txt"))) if os.path.isdir(PROFILES) else []


@pytest.mark.parametrize("name", SUMMARIES)
def test_profile_summaries_name_a_committed_command(name):
    text = open(os.path.join(PROFILES, name)).read()
    cmds = [ln for ln in text.splitlines() if ln.startswith("ncu ")]
    assert cmds, "a summary gives the full command that made it"
    for c in cmds:
        assert "--clock-control none" in c
        assert "_work" not in c
        assert not any(tok.startswith("/") for tok in c.split()), "relative paths only (runs from the repository root)"
        for script in re.findall(r"python (\S+\.py)", c):
            assert os.path.exists(os.path.join(ROOT, script)), script
    assert len(text) < 16 * 1024, "a short summary, not a raw report"


@pytest.mark.parametrize("name", SUMMARIES)
def test_traffic_lines_parse(name):
    for ln in open(os.path.join(PROFILES, name)):
        parts = ln.strip().strip("`").split()
        if parts and parts[0] == "traffic:":
            assert len(parts) == 4 and int(parts[2]) > 0 and re.fullmatch(r"src=[0-9a-f]{12}", parts[3])
            call = parts[1]
            assert bench.call_sources(call), call
            # a line taken on the current sources is the one the bench reports
            if parts[3] == f"src={bench.library_source_hash(call)}":
                assert bench.profiled_traffic(call) == int(parts[2])


def test_nvml_reason_bits_name_the_rejecting_reasons():
    p = bench.NvmlPoller.__new__(bench.NvmlPoller)   # no NVML needed: summarise given samples
    p.max_mhz = 2070.0
    p.samples = [(2070.0, 0x0), (2055.0, 0x4), (1900.0, 0x8 | 0x40), (2070.0, 0x1)]
    s = p.summary()
    assert s["reasons"] == ["hw_slowdown", "hw_thermal_slowdown", "sw_power_cap"]
    assert s["sm_mhz"] == pytest.approx(2062.5) and s["sm_max_mhz"] == 2070.0 and s["samples"] == 4
    p.samples = []
    assert p.summary() is None


def test_nvidia_smi_lines_parse():
    c = bench.ClockSampler(0)
    c.lines = ["2070, 2070, 900.5, 0x0000000000000000, Not Active, Not Active, Not Active, Not Active",
               "1980, 2070, 1390.0, 0x0000000000000004, Not Active, Not Active, Not Active, Active",
               "garbage"]
    s = c.summary()
    assert s["reasons"] == ["sw_power_cap"] and s["samples"] == 2 and s["sm_mhz"] == pytest.approx(2025.0)
