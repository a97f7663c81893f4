"""Host-side arithmetic of bench.py: the algorithmic work a step is credited with, the
rows a cached step computes, and the inputs and bounds of the acceptance workload.
"""
import os
import subprocess
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
import synthetic as syn  # noqa: E402


def test_step_work_of_the_llada8b_shape():
    """Batch 1, prompt 256, gen 256: 7.147 TFLOP of linear layers, 0.137 of attention
    (4 T^2 h H per layer), 0.265 of LM head over the 256 generation rows; 13.96 GB of layer
    weights plus the 1.036 GB LM head streamed once per step."""
    _, total, bytes_ = bench.step_work(syn.SHAPES["llada8b"], 1, 256, 256)
    linear = sum(v for k, v in total.items() if k.startswith("gemm") and k != "gemm_lmhead")
    assert linear == pytest.approx(7.147e12, rel=1e-3)
    assert total["attention"] == pytest.approx(4 * 512 ** 2 * 128 * 32 * 32, rel=1e-12)
    assert total["attention"] == pytest.approx(0.137e12, rel=5e-3)  # a 3-digit figure
    assert total["gemm_lmhead"] == pytest.approx(0.265e12, rel=2e-3)
    assert sum(total.values()) == pytest.approx(7.55e12, rel=2e-3)
    lm = 2.0 * 126464 * 4096
    assert lm == pytest.approx(1.036e9, rel=1e-3)
    assert bytes_ - lm == pytest.approx(13.96e9 + 2 * 512 * 4096, rel=2e-3)


def test_cached_rows_follow_the_refresh_rule():
    """N = 4, M = 8, block 4: step 1 refreshes (all 12 rows, 8 at generation positions),
    step 2 stays in the block [4, 8) and computes rows 4.., step 3 crosses into the next
    block and refreshes again; a finished row computes nothing."""
    out = bench.cached_rows([np.array([1]), np.array([3]), np.array([4])], 4, 8, 4)
    assert out == [(12, 8), (8, 8), (12, 8)]
    out = bench.cached_rows([np.array([8, 1]), np.array([0, 1])], 4, 8, 4)
    assert out == [(24, 16), (8, 8)]


def test_accept_inputs_and_their_uncommitted_rows():
    wl = bench.WORKLOADS["accept"]
    d, rows = bench._accept_data(wl, 0, nseq=2)
    P, V = wl["positions"], wl["vocab"]
    assert d["logits_bf16"].shape == (wl["batch"], P, V)
    assert rows == int((P - d["committed"][:2]).sum())
    # only the sampled sequences carry logits; their realised top-1 sits at the drawn index
    assert not d["logits_bf16"][2:].any()
    for b in range(2):
        for i in range(P):
            z = syn.bf16_to_f32(d["logits_bf16"][b, i])
            assert int(np.argmax(z)) == int(d["top_index"][b, i])
    assert bench._accept_oracle_seconds(wl, d, 2) > 0
    cfg = bench._accept_config(wl, type("A", (), {"gpus": 1})())
    assert cfg["global_batch"] == 64 and cfg["seq_len"] == 32 and cfg["parallelism"] == "single"


def test_accept_algorithmic_bytes():
    """The acceptance pass must read every uncommitted logit row once: for the seeded
    workload 948 of the 2048 positions, 948 x 126464 x 2 B = 239.8 MB (35.3 us at the
    measured 6793.8 GB/s)."""
    wl = bench.WORKLOADS["accept"]
    d, rows = bench._accept_data(wl, 0, nseq=1)  # committed prefixes of all 64 sequences
    total = int((wl["positions"] - d["committed"]).sum())
    assert total == 948
    assert total * wl["vocab"] * 2 == pytest.approx(239.8e6, rel=1e-3)


def test_traffic_comes_only_from_counters_of_the_current_source(tmp_path, monkeypatch):
    """The roofline's `traffic` is the ncu DRAM byte count of the kernel as it stands: the
    acceptance pass's figure covers at least the rows it must read, and any change to the
    kernel's source file turns the figure into null."""
    algo = 948 * bench.WORKLOADS["accept"]["vocab"] * 2
    t = bench._traffic_from_profiles("accept_stats", "kernels.cu")
    assert t is not None and algo <= t < 1.05 * algo
    assert bench._traffic_from_profiles("gemm_mlp") is not None
    assert bench._traffic_from_profiles("no_such_kernel") is None
    csrc = tmp_path / "paper_2607_20467_gb300" / "csrc"
    csrc.mkdir(parents=True)
    (tmp_path / "profiles").mkdir()
    with open(os.path.join(bench.ROOT, "profiles", "traffic.txt")) as f:
        (tmp_path / "profiles" / "traffic.txt").write_text(f.read())
    with open(os.path.join(bench.ROOT, "paper_2607_20467_gb300", "csrc", "kernels.cu")) as f:
        (csrc / "kernels.cu").write_text(f.read() + "// edited\n")
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench._traffic_from_profiles("accept_stats", "kernels.cu") is None


def test_sweep_refuses_the_acceptance_workload():
    r = subprocess.run([sys.executable, "bench.py", "--workload", "accept", "--sweep"], cwd=ROOT,
                       capture_output=True, text=True, timeout=120)
    assert r.returncode == 2 and "decoding workloads" in r.stderr


def test_k_histogram_counts_active_rows_only():
    kper = [np.array([3, 1]), np.array([1, 2]), np.array([0, 2]), np.array([0, 5])]
    assert bench.k_histogram(kper) == {"1": 2, "2": 2, "3": 1, "5": 1}
    assert bench.k_histogram([]) == {}
    # the histogram's tokens are the trajectory's tokens
    h = bench.k_histogram(kper)
    assert sum(int(k) * n for k, n in h.items()) == sum(int(v.sum()) for v in kper)


def test_l2_note_follows_the_weight_bytes():
    assert "streams all weights" in bench._l2_note(bench.WORKLOADS["llada8b"])
    assert "stay in the 129 MB L2" in bench._l2_note(bench.WORKLOADS["tiny"])


def test_oracle_whole_generation_of_the_tiny_workload():
    """The tiny workload's CPU baseline runs the oracle's Algorithm 1 to completion."""
    s, steps, n = bench.oracle_generation(bench.WORKLOADS["tiny"], 0.0)
    assert s > 0 and n == 1 and 1 <= steps <= 64


def test_step_work_of_a_cached_suffix_step():
    """LLaDA-8B shape, prompt 512 + gen 1024, a cached step over 32 suffix rows: 6.98e9
    linear weights per row (2 flops each), attention 4 q T h H per layer, and the stored
    keys / values of all T = 1536 positions read once: 0.524 MB per position = 805 MB."""
    sh = syn.SHAPES["llada8b"]
    _, total, b_cached = bench.step_work(sh, 1, 512, 1024, rows=32, lm_rows=32, cached=True)
    _, _, b_plain = bench.step_work(sh, 1, 512, 1024, rows=32, lm_rows=32, cached=False)
    linear = sum(v for k, v in total.items() if k.startswith("gemm") and k != "gemm_lmhead")
    assert linear == pytest.approx(2 * 6.98e9 * 32, rel=1e-3)
    assert total["attention"] == 4.0 * 32 * 1536 * 4096 * 32
    assert total["gemm_lmhead"] == 2.0 * 32 * 4096 * 126464
    assert b_cached - b_plain == pytest.approx(0.524e6 * 1536, rel=1e-3)
    assert b_cached - b_plain == pytest.approx(805e6, rel=1e-3)


def test_steps_by_rows_groups_and_grades_each_row_count():
    """Cached trajectories are graded per computed-row count: a refresh (all rows) and the
    suffix steps are separate groups, each with the median of its steps and the roofline
    of its own work (the larger of its tensor and HBM times)."""
    shape = syn.SHAPES["llada8b"]
    N, M = 512, 1024
    rl = [(1536, 1024), (1024, 1024), (1024, 1024), (1536, 1024), (1024, 1024)]
    works = [bench.step_work(shape, 1, N, M, r, l, True) for r, l in rl]
    ms = [20.0, 12.0, 13.0, 19.0, 14.0]
    peaks = {"bf16_tflops_sustained": 1699.7, "hbm_gbs": 6793.8}
    out = bench.steps_by_rows(rl, works, ms, peaks)
    assert [g["rows"] for g in out] == [1536, 1024]
    assert [g["steps"] for g in out] == [2, 3]
    assert out[0]["ms"] == pytest.approx(19.5) and out[1]["ms"] == pytest.approx(13.0)
    for g, w in zip(out, (works[0], works[1])):
        t_t = sum(w[1].values()) / 1699.7e12
        t_h = w[2] / 6793.8e9
        assert g["t_roof_ms"] == pytest.approx(1e3 * max(t_t, t_h))
        assert g["bound"] == ("hbm" if t_h >= t_t else "tensor")
        assert g["frac"] == pytest.approx(g["t_roof_ms"] / g["ms"])
    # 32 suffix rows at batch 1 stream 15 GB of weights for far fewer flops: HBM-bound
    small = bench.steps_by_rows([(32, 32)], [bench.step_work(shape, 1, N, M, 32, 32, True)], [6.0], peaks)
    assert small[0]["bound"] == "hbm"


def test_cached_rows_of_the_dual_cache():
    """N = 4, M = 8, block 4, dual cache: the first step refreshes (12 rows), the second
    stays in the block [4, 8) and computes only that block (4 rows, all generation rows),
    the third crosses into [8, 12) and refreshes."""
    out = bench.cached_rows([np.array([1]), np.array([3]), np.array([4])], 4, 8, 4, dual=True)
    assert out == [(12, 8), (4, 4), (12, 8)]
    # two rows: at the second step row 0 crosses into [8, 12) and refreshes, row 1 stays in
    # [4, 8) and computes that block
    out = bench.cached_rows([np.array([5, 1]), np.array([1, 8])], 4, 8, 4, dual=True)
    assert out == [(24, 16), (4 + 12, 4 + 8)]
