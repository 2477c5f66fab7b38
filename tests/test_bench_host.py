"""Host-side bookkeeping of bench.py's roofline object (CPU only).

* algorithmic bytes: the expert weights counted per stage add up to the
  layer's |U| * 6 d F (Sec. 2.1: gate, up and down matrices of d x F bf16);
* the recorded ncu traffic (profiles/traffic.json) scales with the units a
  launch processes and is refused when it was captured from other kernel
  sources;
* the committed record is plausible: DRAM traffic per used expert within a
  few percent of the algorithmic bytes of one expert's weights.
"""
import json
import os
import shutil

import pytest

import bench
from paper_2602_07265_gb300 import workloads as W

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.mark.parametrize("w", [W.TINY, W.OLMOE, W.QWEN3, W.DSR1], ids=lambda w: w.name)
@pytest.mark.parametrize("n_shared", [0, 1])
def test_stage_bytes_add_up_to_the_layer(w, n_shared):
    n_used, n_pairs = 24, w.B * w.k
    a = bench.algorithmic_bytes(w, n_used, n_pairs, n_shared)
    per_expert = 6 * w.d * w.F                     # 3 matrices of d x F bf16
    n_exp = n_used + n_shared
    rows = n_pairs + n_shared * w.B
    weights_gu = a["ffn_gate_up"] - rows * w.d * 2 - rows * w.F * 2
    weights_dn = a["ffn_down"] - rows * w.F * 2 - rows * w.d * 4
    assert weights_gu + weights_dn == n_exp * per_expert
    assert a["layer"] == n_exp * per_expert + w.N * w.d * 4 + 2 * w.B * w.d * 2
    assert a["router"] == w.N * w.d * 4 + w.B * w.d * 2 + w.B * w.N * 4


def _tree(tmp_path, record):
    """A copy of the kernel sources and a traffic record under tmp_path."""
    src = os.path.join(ROOT, "paper_2602_07265_gb300", "csrc")
    dst = tmp_path / "paper_2602_07265_gb300" / "csrc"
    shutil.copytree(src, dst)
    (tmp_path / "profiles").mkdir()
    if record is not None:
        (tmp_path / "profiles" / "traffic.json").write_text(json.dumps(record))
    return tmp_path


def test_recorded_traffic_scales_and_checks_sources(tmp_path, monkeypatch):
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    _tree(tmp_path, None)
    assert bench.recorded_traffic("ffn_gate_up", 10) is None          # no record
    h = bench.kernel_source_hash("ffn_gate_up")
    rec = {"ffn_gate_up": {"bytes_per_unit": 1000.0, "source_hash": h}}
    (tmp_path / "profiles" / "traffic.json").write_text(json.dumps(rec))
    assert bench.recorded_traffic("ffn_gate_up", 10) == 10000.0
    assert bench.recorded_traffic("ffn_gate_up", 43.5) == 43500.0
    assert bench.recorded_traffic("router", 1) is None                 # no such stage
    # Any change to a kernel source invalidates the record.
    f = tmp_path / "paper_2602_07265_gb300" / "csrc" / "ffn_tc.cu"
    f.write_text(f.read_text() + "\n// changed\n")
    assert bench.kernel_source_hash("ffn_gate_up") != h
    assert bench.recorded_traffic("ffn_gate_up", 10) is None
    (tmp_path / "profiles" / "traffic.json").write_text("not json")
    assert bench.recorded_traffic("ffn_gate_up", 10) is None


def test_committed_traffic_record_is_plausible():
    """The record was taken on DeepSeek-R1 shapes (d = 7168, F = 2048, 32
    tokens): per used expert the gate/up kernel must move 2 d F bf16 of
    weights and the down kernel d F, plus a few MB of token rows per launch."""
    with open(os.path.join(ROOT, "profiles", "traffic.json")) as f:
        rec = json.load(f)
    d, F = W.DSR1.d, W.DSR1.F
    for stage, weights in (("ffn_gate_up", 2 * d * F * 2), ("ffn_down", d * F * 2)):
        r = rec[stage]
        assert r["unit"] == "bytes per used expert"
        assert 1.0 <= r["bytes_per_unit"] / weights <= 1.05, stage
        assert os.path.exists(os.path.join(ROOT, r["capture"]))
