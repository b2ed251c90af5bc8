"""The benchmark's roofline arithmetic on the CPU: the algorithmic bytes and
flops it credits per launch, which roof bounds each workload, which peak a
fraction is taken against (the measured copy bandwidth, the measured bf16
burst rate, twice that for e4m3 x e4m3 on the f8f6f4 pipe) and the issued
fraction beside the algorithmic one (hi/lo planes for fp32 activations);
and one entry of the configuration block assembled around fake timings,
with the committed DRAM traffic of its call.  The expected figures are
built from their physical terms, not from the benchmark's own
expressions."""
from types import SimpleNamespace

import pytest

import bench

PEAKS = {"hbm_gbs": 6691.1, "bf16_tflops": 1903.6, "bf16_tflops_sustained": 1696.8}


def head(rows, n_keep, d, d_l, w_dtype="bf16"):
    return SimpleNamespace(rows=rows, n_keep=n_keep, d=d, d_l=d_l, d_h=d - d_l,
                           w_dtype=w_dtype)


DECODE = head(32, 12000, 4096, 256)
SWEEP = dict(n_keep=256000, d=5120, d_l=512)
FP8 = head(256, 152064, 8192, 1024, "fp8")


def test_decode_cloud_call_is_hbm_bound_on_its_algorithmic_bytes():
    kept_rows = 12000 * 3840 * 2       # the kept W_h rows, bf16, read once
    h = 32 * 3840 * 4                  # h_cloud, fp32
    ids = 12000 * 4                    # the kept-id list, int32
    codes, scales = 32 * 12000, 32 * 4  # the payload: int8 codes + fp32 row scales
    alg = kept_rows + h + ids + codes + scales
    assert alg == 93_083_648
    r = bench.roofline(DECODE, "fp32", 0.03938, PEAKS)
    assert r["bound"] == "hbm" and r["unit"] == "GB/s" and r["peak"] == PEAKS["hbm_gbs"]
    assert r["algorithmic_bytes"] == alg
    # 93.08 MB in 39.38 us against 6691.1 GB/s
    assert r["frac"] == pytest.approx(0.3533, abs=1e-4)
    assert r["achieved"] == pytest.approx(alg / 39.38e-6 / 1e9, rel=1e-3)
    assert "issued_frac" not in r


@pytest.mark.parametrize("act,planes", [("fp32", 2), ("bf16", 1)])
def test_headline_is_tensor_bound_against_the_burst_rate(act, planes):
    w = head(1024, **SWEEP)
    flops = 2 * 1024 * 256000 * 4608   # one multiply-add per (row, kept id, cloud column)
    r = bench.roofline(w, act, 2.977, PEAKS)
    assert r["bound"] == "tensor" and r["unit"] == "TFLOP/s"
    assert r["algorithmic_flops"] == flops
    # the burst peak for a kernel timed on its own, not the sustained one
    assert r["peak"] == pytest.approx(PEAKS["bf16_tflops"])
    assert r["frac"] == pytest.approx(flops / 2.977e-3 / 1e12 / 1903.6, rel=1e-3)
    assert r["frac"] == pytest.approx(0.426, abs=1e-3)
    # fp32 activations issue a hi and a lo plane per algorithmic MMA
    assert r["issued_frac"] == pytest.approx(planes * r["frac"], rel=1e-3)


def test_the_bound_is_the_roof_that_takes_longer():
    # one row over the full vocabulary streams 2.36 GB for 2.4 GFLOP: HBM;
    # 1024 rows do 2.4 TFLOP over 2.37 GB: tensor pipe
    assert bench.roofline(head(1, **SWEEP), "fp32", 0.376, PEAKS)["bound"] == "hbm"
    assert bench.roofline(head(1024, **SWEEP), "fp32", 2.977, PEAKS)["bound"] == "tensor"
    for R in (1, 8, 64, 256, 1024):
        r = bench.roofline(head(R, **SWEEP), "fp32", 1.0, PEAKS)
        t_hbm = r["algorithmic_bytes"] / (PEAKS["hbm_gbs"] * 1e9)
        t_tc = r["algorithmic_flops"] / (PEAKS["bf16_tflops"] * 1e12)
        assert r["bound"] == ("tensor" if t_tc > t_hbm else "hbm"), R


@pytest.mark.parametrize("act,planes", [("fp32", 4), ("bf16", 2)])
def test_e4m3_head_is_credited_at_twice_the_bf16_rate(act, planes):
    r = bench.roofline(FP8, act, 0.760, PEAKS)
    # one byte a weight plus one fp32 scale per kept row
    kept = 152064 * 7168 * 1 + 152064 * 4
    assert r["algorithmic_bytes"] == kept + 256 * 7168 * 4 + 152064 * 4 + 256 * 152064 + 256 * 4
    assert r["bound"] == "hbm"
    assert r["tensor"]["peak"] == pytest.approx(2 * PEAKS["bf16_tflops"], abs=0.1)
    assert r["tensor"]["planes"] == planes
    assert r["tensor"]["issued_frac"] == pytest.approx(planes * r["tensor"]["frac"], rel=1e-3)


def test_whole_step_adds_the_endpoint_half():
    w = head(1024, **SWEEP)
    cloud = bench.roofline(w, "fp32", 3.0, PEAKS)
    step = bench.roofline(w, "fp32", 3.0, PEAKS, mode="fused")
    end_bytes = (256000 * 512 * 2 + 1024 * 512 * 4 + 1024 * 256000 + 1024 * 4
                 + 256000 * 4 + 1024 * 4)   # W_l rows, h_local, codes, scales, ids, tokens
    assert step["algorithmic_bytes"] == cloud["algorithmic_bytes"] + end_bytes
    assert step["algorithmic_flops"] == 2 * 1024 * 256000 * (4608 + 512)
    # both halves on bf16 weights: the combined peak is the bf16 rate
    assert step["tensor"]["peak"] == pytest.approx(PEAKS["bf16_tflops"], abs=0.1)
    assert step["tensor"]["issued_frac"] is None


def test_unsplit_head_reads_the_whole_hidden_state():
    r = bench.roofline(DECODE, "fp32", 0.05, PEAKS, mode="nosplit")
    assert r["algorithmic_bytes"] == 12000 * 4096 * 2 + 32 * 4096 * 4 + 12000 * 4 + 32 * 4
    assert r["algorithmic_flops"] == 2 * 32 * 12000 * 4096
    assert r["tensor"]["planes"] == 1 and r["tensor"]["issued_frac"] is None


class _FakeRunner:
    """Stands in for the GPU step: config_entry's host logic only."""
    gsteps = 16

    def __init__(self, sph, wl, w, dev, act="fp32", mode="split", chunk=0, **kw):
        self.nchunk = 1 if not chunk else -(-w.n_keep // chunk)

    def step(self, i, events=None):
        pass

    def close(self):
        pass


@pytest.mark.parametrize("mode,has_traffic", [("split", True), ("fused", False)])
def test_configuration_entry_carries_the_committed_traffic(monkeypatch, mode, has_traffic):
    # the decode entry of the block reports the DRAM bytes of its cloud call
    # from the committed record (the two-call step only); the GPU pieces are
    # replaced by fakes that return fixed timings
    import torch
    from paper_2607_13093_gb300 import workloads as wl
    monkeypatch.setattr(bench, "Runner", _FakeRunner)
    monkeypatch.setattr(bench, "timed_run", lambda r, steps, warmup, **kw: dict(
        ms=steps * 0.05, unit=[0.03938] * 64, timing="fake", launches_per_step=6.0))
    monkeypatch.setattr(bench, "e2e_run", lambda r, steps: {
        "value": 1.0, "direct_calls": {"value": 0.5}})
    monkeypatch.setattr(torch.cuda, "synchronize", lambda *a, **k: None)
    monkeypatch.setattr(torch.cuda, "empty_cache", lambda: None)
    e = bench.config_entry(None, wl, torch.device("cpu"), "decode", None, None, None, "fp32",
                           PEAKS, 0.0, with_cpu=False, mode=mode)
    assert e["workload"].startswith("decode: d=4096 (d_l=256, d_h=3840), V=32000, R=32")
    assert e["payload_bytes_per_step"] == 32 * 12000 + 4 * 32
    if has_traffic:
        assert e["roofline"]["traffic"] == 95_321_216
        assert e["roofline"]["frac"] == pytest.approx(0.3533, abs=1e-4)
        assert e["cloud_us"] == pytest.approx(39.38)
    else:
        assert e["roofline"]["traffic"] is None and "step_call_us" in e
    assert e["e2e_rows_per_s"] == 1.0 and e["e2e_direct_rows_per_s"] == 0.5
