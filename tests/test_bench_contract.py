"""Host logic of ``bench.py`` on the CPU: the algorithmic work each kernel's
roofline divides by, the roofline arithmetic, the source-hash gating of the
DRAM traffic figures and the workload description of the JSON line."""
import hashlib
import os
import shutil

import pytest

import bench


class _Shape:
    """The fields of a layer that the bench's models read."""

    def __init__(self, name, din, dout, g, bits, K):
        self.name, self.din, self.dout, self.g, self.bits, self.K = name, din, dout, g, bits, K


Q_PROJ = _Shape(bench.WORKLOAD, 4096, 4096, 128, 3, 10)


def test_kernel_work_closed_forms():
    p, d, g = 4096, 4096, 128
    G = d // g
    # phase product: one (p x d) x (d x g) product of useful work, four digit planes issued
    m = bench.kernel_model("target", Q_PROJ)
    assert m["bound"] == "tensor" and m["work"] == 2.0 * p * g * d == 4294967296.0
    assert m["issued"] == 4 * m["work"]
    # Gram: the G (G + 1) / 2 blocks h <= i of c_h^T H_hi c_i, 2 p g^2 each
    m = bench.kernel_model("gram", Q_PROJ)
    assert m["work"] == 2.0 * p * g * g * G * (G + 1) / 2 == 70866960384.0
    # target projection P = W H and its 18 digit pairs
    m = bench.kernel_model("proj", Q_PROJ)
    assert m["work"] == 2.0 * p * d * d and m["issued"] == 18 * m["work"]
    # Babai: the dense triangular back substitution, g^2 flops per (row, group)
    assert bench.kernel_model("babai", Q_PROJ) == {"bound": "alu", "work": 1.0 * g * g * p}
    # the scale solve moves each row's float64 Gram matrix once
    m = bench.kernel_model("scale_solve", Q_PROJ)
    assert m["bound"] == "hbm" and m["work"] >= 8.0 * p * G * G
    assert bench.kernel_model("no_such_kernel", Q_PROJ) is None


def test_roofline_arithmetic():
    pk = {"hbm_gbs": 6789.0, "bf16_tflops": 1942.2, "bf16_tflops_sustained": 1736.3}
    # 10 launches of 35 us each
    e = bench.roofline_entry("target", {"launches": 10, "total_ms": 0.35}, Q_PROJ, pk, "measured")
    achieved = 2.0 * 4096 * 128 * 4096 / 35e-6 / 1e12
    assert e["bound"] == "tensor" and e["unit"] == "TFLOP/s"
    assert e["achieved"] == pytest.approx(achieved) and e["peak"] == 1736.3
    assert e["frac"] == pytest.approx(achieved / 1736.3)
    assert e["issued_frac"] == pytest.approx(4 * e["frac"])
    assert e["avg_us"] == pytest.approx(35.0)
    # an HBM-bound kernel against the copy bandwidth
    e = bench.roofline_entry("rhs", {"launches": 2, "total_ms": 0.08}, Q_PROJ, pk, "measured")
    assert e["unit"] == "GB/s" and e["peak"] == 6789.0
    assert e["frac"] == pytest.approx(e["achieved"] / 6789.0)
    # Babai against the float32 FMA rate of 152 SMs at 2070 MHz
    e = bench.roofline_entry("babai", {"launches": 1, "total_ms": 0.0186}, Q_PROJ, pk, "measured")
    assert e["bound"] == "alu"
    assert e["peak"] == pytest.approx(152 * 128 * 2 * 2070e6 / 1e12)
    # no launches, no entry
    assert bench.roofline_entry("target", {"launches": 0, "total_ms": 0.0}, Q_PROJ, pk, "x") is None


def test_traffic_is_reported_only_for_an_unchanged_source(tmp_path, monkeypatch):
    # with the committed sources, a figure is either the committed one (hash
    # matches) or absent; never a different number
    for k, (fname, sha, val) in bench.TRAFFIC.items():
        path = os.path.join(bench.ROOT, "paper_2609_38599_gb300", "csrc", fname)
        cur = hashlib.sha1(open(path, "rb").read()).hexdigest()[:12]
        assert bench.traffic_for(k) == (val if cur == sha else None)
    # a changed source file withdraws its figure
    csrc = tmp_path / "paper_2609_38599_gb300" / "csrc"
    csrc.mkdir(parents=True)
    fname = bench.TRAFFIC["target"][0]
    shutil.copy(os.path.join(bench.ROOT, "paper_2609_38599_gb300", "csrc", fname), csrc / fname)
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    unchanged = bench.traffic_for("target")
    with open(csrc / fname, "a") as fh:
        fh.write("\n// changed\n")
    assert bench.traffic_for("target") is None
    assert unchanged in (None, bench.TRAFFIC["target"][2])
    assert bench.traffic_for("not_in_table") is None


def test_roofline_traffic_only_for_the_main_workload():
    pk = {"hbm_gbs": 6789.0, "bf16_tflops": 1942.2, "bf16_tflops_sustained": 1736.3}
    other = _Shape("llama2_7b_down_proj_4096x11008_g128_w4", 11008, 4096, 128, 4, 10)
    e = bench.roofline_entry("target", {"launches": 1, "total_ms": 0.07}, other, pk, "measured")
    assert e["traffic"] is None


def test_config_names_the_workload_and_its_l2_note():
    c = bench.config_dict(Q_PROJ)
    assert c["workload"] == bench.WORKLOAD
    assert (c["din"], c["dout"], c["group_size"], c["bits"], c["K"]) == (4096, 4096, 128, 3, 10)
    assert c["early_stop"] is False and c["host"] == "RTN"
    # W 64 MB, P and the folded P 128 MB each, digit planes 448 MB: all larger than L2
    assert "W 64 MB" in c["l2"] and "128 MB" in c["l2"] and "448 MB" in c["l2"]
    assert bench.config_dict(Q_PROJ, note="x")["note"] == "x"
