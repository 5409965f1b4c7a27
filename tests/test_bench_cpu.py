"""The bench's bookkeeping, without a GPU: algorithmic work per launch and the use of the
recorded DRAM traffic."""
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
import workloads as wk  # noqa: E402


def test_phase_b_algorithmic_bytes_per_launch():
    # one segment of 8 chains of the 16-layer shape: 18 B per parameter of state (W and
    # momentum read and written in fp32, the bf16 operand copy written), U and Y in bf16,
    # dH and At in bf16
    wl = wk.WORKLOADS["l16_d2048_128k"]
    params = wl.d_hid * (wl.d_in + wl.d_out)
    per_chain = params * 18 + wl.seg_T * (wl.d_in + wl.d_out) * 2 + wl.seg_T * wl.d_hid * 2 * 2
    flops, byts = bench.kernel_work(wl, "phase_b", 8)
    assert byts == pytest.approx(8 * per_chain)
    assert byts == pytest.approx(494.5e6, rel=1e-3)
    assert flops == pytest.approx(8 * 2 * wl.seg_T * wl.d_hid * (wl.d_in + wl.d_out))


def test_recorded_traffic_applies_only_to_its_shape(tmp_path, monkeypatch):
    # a record for this source of the kernel, taken on one segment of 8 chains of the 16-layer
    # shape at T = 512, in a scratch copy of the layout bench.py reads
    src = open(os.path.join(ROOT, "paper_2608_17616_gb300", "csrc", "ttl_tc.cu")).read()
    (tmp_path / "paper_2608_17616_gb300" / "csrc").mkdir(parents=True)
    (tmp_path / "paper_2608_17616_gb300" / "csrc" / "ttl_tc.cu").write_text(src)
    (tmp_path / "profiles").mkdir()
    sha = bench.kernel_source_sha(src, "phase_b")
    shape = bench.shape_key(wk.WORKLOADS["l16_d2048_128k"])
    (tmp_path / "profiles" / "ncu_traffic.txt").write_text(
        f"# test record\nkernel=phase_b source_sha={sha} shape={shape} bytes_per_launch=400000000 chains=8\n")
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    got = {n: bench.ncu_traffic("phase_b", 8.0, wk.WORKLOADS[n])[0]
           for n in ("l16_d2048_128k", "l16_d2048_32k", "ctx8_l16_T512", "ctx8_l16_T1024", "l28_d3072_128k",
                     "swiglu_l24_d896_32k")}
    assert got["l16_d2048_128k"] == pytest.approx(4e8)
    assert got["l16_d2048_32k"] == got["l16_d2048_128k"] and got["ctx8_l16_T512"] == got["l16_d2048_128k"]
    for other in ("ctx8_l16_T1024", "l28_d3072_128k", "swiglu_l24_d896_32k"):
        assert got[other] is None, other
    # scaled in proportion to the chains of a launch
    assert bench.ncu_traffic("phase_b", 16.0, wk.WORKLOADS["l16_d2048_128k"])[0] == pytest.approx(8e8)
    # a record of another version of the kernel is not used
    banner = "// ------------------------------------------------------------------ phase B"
    (tmp_path / "paper_2608_17616_gb300" / "csrc" / "ttl_tc.cu").write_text(
        src.replace(banner, banner + "\n// edited", 1))
    assert bench.ncu_traffic("phase_b", 8.0, wk.WORKLOADS["l16_d2048_128k"])[0] is None


def test_resident_kernel_work_counts_inputs_per_segment_and_state_per_launch():
    # the resident fp32 kernel covers a window of segments in one launch: U and Y (fp32) stream once
    # per segment, W (and mu in paper mode) cross HBM once per launch
    wl = wk.WORKLOADS["tiny_f32"]
    S = wl.S
    flops, byts = bench.kernel_work(wl, "resident", wl.chains * S)
    assert flops == wl.N * 4 * (256 * 512 + 512 * 256)
    assert byts == wl.N * (256 + 256) * 4 + 512 * (256 + 256) * 8      # plain mode: W read and write
    paper = wl.replace(mode=wk.PAPER)
    assert bench.kernel_work(paper, "resident", wl.chains * S)[1] == byts + 512 * (256 + 256) * 8  # + momentum


def test_dominant_roofline_is_the_tensor_work_of_the_path():
    # phase B of the 16-layer shape: 2 T d_hid (d_in + d_out) flops per chain-segment, 8 chains a
    # launch; the per-launch and busy-time figures of a 20-step run (116.79 us a launch, 850.4 ms
    # busy over 20 x 256 segments of all 16 chains) against the measured bf16 peaks
    wl = wk.WORKLOADS["l16_d2048_128k"]
    per_chain = 2 * wl.seg_T * wl.d_hid * (wl.d_in + wl.d_out)
    assert per_chain == 2 * 512 * 1024 * 3072
    d = {"chains_per_launch": 8.0, "avg_us": 116.79}
    pk = (6681.8, 1909.7, 1723.2, "measured")
    roof = bench.dominant_roofline(wl, "phase_b", d, 850.4, 20 * 256, 20 * 54.17, pk)
    assert roof["bound"] == "tensor" and roof["unit"] == "TFLOP/s" and roof["peak"] == 1723.2
    assert roof["achieved"] == pytest.approx(8 * per_chain / 116.79e-6 / 1e12)
    assert roof["achieved"] == pytest.approx(220.6, rel=1e-3)
    assert roof["frac_of_burst"] == pytest.approx(0.1155, abs=5e-4)
    assert roof["busy"]["achieved"] == pytest.approx(16 * per_chain * 20 * 256 / 0.8504 / 1e12)
    assert roof["busy"]["frac_of_burst"] == pytest.approx(0.1625, abs=5e-4)
    # the state-inclusive HBM view of the same launch stays beside it
    assert roof["hbm"]["bytes_per_launch"] == pytest.approx(494.5e6, rel=1e-3)
    assert roof["hbm"]["frac"] == pytest.approx(494.5e6 / 116.79e-6 / 1e9 / 6681.8, rel=1e-3)


def test_e2e_breakdown_separates_the_link_from_the_pipeline():
    # 26 gathers of 4 ms each, busy 104 ms of a 110 ms step, 20.8 GB over the link: the step is
    # bound by the link (96% of it has a gather running), which ran at 200 GB/s
    out = bench.e2e_breakdown(20.8e9, 104.0, 26, 104.0, 110.0)
    assert out["h2d_gbs"] == pytest.approx(200.0)
    assert out["gathers_per_step"] == 26 and out["gather_ms_mean"] == pytest.approx(4.0)
    assert out["gather_share_of_step"] == pytest.approx(104.0 / 110.0)
    # overlapping gathers (busy below the summed time): the rate uses the busy time
    out = bench.e2e_breakdown(10e9, 80.0, 10, 50.0, 100.0)
    assert out["h2d_gbs"] == pytest.approx(200.0) and out["gather_share_of_step"] == pytest.approx(0.5)
