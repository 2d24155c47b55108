"""Host-side arithmetic of bench.py's roofline figures (no GPU).

The algorithmic bytes and FLOPs of each stage are checked against hand
computation from the workload shapes, and the per-stage roofline against the
slower of the two peaks."""
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
from paper_2506_07416_gb300 import inputs  # noqa: E402

PK = {"hbm_gbs": 6794.5, "bf16_tflops": 1926.9, "bf16_tflops_sustained": 1718.2, "source": "measured"}


def test_single_workload_algorithmic_work():
    # one request: 1536 visual + 64 text tokens, 16 heads x 128, bf16, keep floor(0.3f * 1536) = 460,
    # gathers the hidden rows (2048 bf16 = 4096 B)
    alg = bench.algorithmic(inputs.workload("single"))
    assert alg["kept"] == [460]
    assert alg["score_bytes"] == 1536 * 16 * 128 * 2 + 64 * 16 * 128 * 2 + 4 * 1536
    assert alg["score_flops"] == 2 * 16 * 64 * 1536 * 128
    assert alg["topk_bytes"] == 4 * 1536 + 4 * 460
    assert alg["compact_bytes"] == 2 * 460 * alg["row_total"] + 4 * 460


def test_stage_rooflines_take_the_slower_peak():
    alg = {"score_flops": 4e9, "score_bytes": 1e6, "topk_bytes": 2e4, "compact_bytes": 6.7945e6}
    st = {"score": 10.0, "topk": 4.0, "compact": 2.0, "timing": "text"}
    r = bench.stage_rooflines(alg, st, 20.0, PK, "bf16")
    t_score = 4e9 / 1926.9e12 * 1e6          # 2.076 us of tensor work > 0.147 us of bytes
    assert r["score"]["bound"] == "tensor"
    assert r["score"]["roofline_us"] == pytest.approx(t_score)
    assert r["score"]["frac"] == pytest.approx(t_score / 10.0)
    assert r["topk"]["bound"] == "hbm"
    assert r["compact"]["roofline_us"] == pytest.approx(1.0)
    assert r["compact"]["frac"] == pytest.approx(0.5)
    total = t_score + 2e4 / 6794.5e9 * 1e6 + 1.0
    assert r["step"]["roofline_us"] == pytest.approx(total)
    assert r["step"]["frac"] == pytest.approx(total / 20.0)
    # e4m3: twice the bf16 tensor peak, so the same FLOPs take half the time
    r8 = bench.stage_rooflines(alg, st, 20.0, PK, "e4m3")
    assert r8["score"]["roofline_us"] == pytest.approx(t_score / 2)


def test_workload_bounds_match_their_intensity():
    # highres (GQA 7:1, 128 text tokens) is tensor-bound; single is HBM-bound
    for name, bound in (("highres", "tensor"), ("single", "hbm")):
        alg = bench.algorithmic(inputs.workload(name))
        r = bench.stage_rooflines(alg, {"score": 1.0, "topk": 1.0, "compact": 1.0}, 3.0, PK, "bf16")
        assert r["score"]["bound"] == bound
        assert r["topk"]["bound"] == "hbm" and r["compact"]["bound"] == "hbm"


@pytest.mark.parametrize("ratio,k", [(0.1, 345), (0.2, 691), (0.3, 1036), (0.5, 1728)])
def test_sweep_keep_counts_follow_the_floor_reading(ratio, k):
    # k = floor((double)(float)r * N) with N = 3456: 0.1f * 3456 = 345.6..., 0.2f -> 691.2..., 0.3f -> 1036.8...
    class A:
        workload, batch = "sweep", None
    A.ratio = ratio
    w = bench.workload_for(A())
    alg = bench.algorithmic(w)
    assert alg["kept"] == [k] * 128
    assert sum(alg["kept"]) == 128 * k


def test_batch_option_takes_the_first_requests():
    class A:
        workload, ratio, batch = "fp8_ragged", None, 5
    w = bench.workload_for(A())
    full = inputs.workload("fp8_ragged")
    assert w.batch == 5 and list(w.n_vis) == list(full.n_vis[:5]) and list(w.n_txt) == list(full.n_txt[:5])


def test_committed_traffic_follows_the_workloads_own_kernel(tmp_path, monkeypatch):
    """A DRAM figure is reported only while the files of the kernel that serves
    the workload still hash to the recorded kernel_sha; a change to the other
    kernel's source leaves it valid."""
    prof = tmp_path / "profiles"
    prof.mkdir()
    csrc = tmp_path / "paper_2506_07416_gb300" / "csrc"
    csrc.mkdir(parents=True)
    for f in bench.KERNEL_SOURCES:
        (tmp_path / f).write_text("source of " + os.path.basename(f))
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    res, tc = bench.kernel_source_sha("score_res"), bench.kernel_source_sha("score_tc")
    assert res != tc
    import json
    (prof / "score_traffic.json").write_text(json.dumps({
        "sweep": {"kernel": "score_res_kernel<256, 0, 64, 1, 0>", "kernel_sha": res, "dram_bytes_per_launch": 7},
        "highres": {"kernel": "score_tc_kernel<256, 0, 128>", "kernel_sha": tc, "dram_bytes_per_launch": 9}}))
    assert bench.committed_traffic("sweep") == 7 and bench.committed_traffic("highres") == 9
    assert bench.committed_traffic("single") is None  # no entry
    # the re-read kernel's source changes: its figure goes stale, the resident kernel's stays
    (tmp_path / bench.KERNEL_SOURCES[0]).write_text("changed score_tc.cu")
    assert bench.committed_traffic("highres") is None and bench.committed_traffic("sweep") == 7
    # a shared header changes: both go stale
    (tmp_path / bench.KERNEL_SOURCES[2]).write_text("changed pipe.cuh")
    assert bench.committed_traffic("sweep") is None
