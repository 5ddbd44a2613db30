"""Host-side logic of bench.py that needs no GPU: where the roofline's DRAM
traffic figure comes from, the peaks it divides by, and the bytes a step
reads (the L2 rule of the timing)."""
import hashlib
import json
import os

import bench


def test_traffic_record_of_the_roofline_kernel_matches_its_source():
    """The committed ncu record of the attention kernel the roofline names was
    taken on the current source of that kernel (else the line would carry no
    traffic figure)."""
    rec = json.load(open(os.path.join(bench.ROOT, "profiles",
                                      f"attn_tc2_{bench.WORKLOAD}.json")))
    src = os.path.join(bench.ROOT, "paper_2505_23970_gb300", "csrc", "attn_tc2.cu")
    assert rec["src_sha"] == hashlib.sha256(open(src, "rb").read()).hexdigest()[:16]
    assert rec["dram_bytes_per_launch"] == rec["dram_bytes_read"] + rec["dram_bytes_write"]
    assert bench.traffic_record("attn_tc2", bench.WORKLOAD) == rec["dram_bytes_per_launch"]


def test_stale_traffic_record_is_not_reported(tmp_path, monkeypatch):
    """A record whose source hash no longer matches reads as None."""
    root = tmp_path
    os.makedirs(root / "profiles")
    os.makedirs(root / "paper_2505_23970_gb300" / "csrc")
    src = root / "paper_2505_23970_gb300" / "csrc" / "attn_tc2.cu"
    src.write_text("// kernel v1\n")
    sha = hashlib.sha256(src.read_bytes()).hexdigest()[:16]
    (root / "profiles" / "attn_tc2_w.json").write_text(
        json.dumps({"src_sha": sha, "dram_bytes_per_launch": 1234}))
    monkeypatch.setattr(bench, "ROOT", str(root))
    assert bench.traffic_record("attn_tc2", "w") == 1234
    src.write_text("// kernel v2\n")
    assert bench.traffic_record("attn_tc2", "w") is None
    assert bench.traffic_record("attn_tc2", "no-such-workload") is None


def test_restore_traffic_record_follows_its_own_source(tmp_path, monkeypatch):
    """The restore kernel's record is checked against kv_copy.cu, not an
    attention source."""
    root = tmp_path
    os.makedirs(root / "profiles")
    os.makedirs(root / "paper_2505_23970_gb300" / "csrc")
    kv = root / "paper_2505_23970_gb300" / "csrc" / "kv_copy.cu"
    kv.write_text("// copies\n")
    (root / "paper_2505_23970_gb300" / "csrc" / "attn_tc2.cu").write_text("// other\n")
    sha = hashlib.sha256(kv.read_bytes()).hexdigest()[:16]
    (root / "profiles" / "restore_bulk_w.json").write_text(
        json.dumps({"src_sha": sha, "dram_bytes_per_launch": 77}))
    monkeypatch.setattr(bench, "ROOT", str(root))
    assert bench.traffic_record("restore_bulk", "w") == 77


def test_peaks_measured_or_fallback(tmp_path, monkeypatch):
    """MEASURED_PEAKS.json when present (source "measured"), the recipe's
    fallback figures otherwise."""
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    pk = bench.peaks()
    assert pk["source"] == "fallback" and pk["hbm_gbs"] == 6800.0 and pk["bf16_tflops"] == 1900.0
    (tmp_path / "MEASURED_PEAKS.json").write_text(
        json.dumps({"hbm_gbs": 6790.0, "bf16_tflops": 1909.5, "bf16_tflops_sustained": 1724.2}))
    pk = bench.peaks()
    assert pk == {"hbm_gbs": 6790.0, "bf16_tflops": 1909.5, "bf16_tflops_sustained": 1724.2,
                  "source": "measured"}


def test_70b_layer_step_reads_more_than_twice_the_l2():
    """The timing rule: the 70B layer's step reads q, the new K/V, the
    restore's staging image and the pool pages it writes, and every context
    row of K and V, far more than twice the 129 MB L2, so the bench needs no
    flush between its steps and says so in `config`."""
    w = bench.make_workload("70b", 0)
    q = w.T_new * w.Hq * w.d * 2
    kv_new = 2 * w.T_new * w.Hkv * w.d * 2
    ctx = int(w.total_lens.sum()) * 2 * w.Hkv * w.d * 2
    got = bench.step_input_bytes(w)
    assert got > q + kv_new + ctx > 2 * 129 * 2**20
    cfg = bench.arm_config(w, 1)
    assert cfg["l2"].startswith("inputs larger than L2") and cfg["parallelism"] == "single"
    assert bench.arm_config(w, 4)["parallelism"] == "replicas"
