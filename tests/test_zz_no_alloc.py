"""The allocation-free cloud call agrees with the oracle and with the regular
call, and allocates nothing once set up.

sph_partial_logits_noalloc exists for callers that cannot allocate device
memory while they run (a foreign or locked allocator, a fixed-size pool, a
serving loop that must not call cudaMalloc); it keeps its scratch in a fixed
device array inside the library.  This file is collected last so that a
failure here never hides the rest of the suite; it also passes when run on
its own in a fresh process."""
import numpy as np
import pytest
import torch

from paper_2607_13093_gb300 import workloads as wl
from _parity import assert_close, assert_codes, np_, oracle_cloud

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def sph():
    from paper_2607_13093_gb300 import build_lib
    build_lib.build()
    from paper_2607_13093_gb300 import sph as mod
    return mod


def regular(sph, ctx, w, act):
    part = torch.empty(w.rows, w.n_keep, device="cuda")
    codes, scale, pb = ctx.partial_logits(w.h_cloud, w.W_h, keep_ids=w.keep_ids,
                                          clip=w.clip, w_row_scale=w.w_scale,
                                          bias=w.bias, partial_out=part,
                                          act_mode=act)
    return codes, scale, part, pb


def no_alloc(sph, w, act):
    codes = torch.full((w.rows, w.n_keep), 99, dtype=torch.int8, device="cuda")
    scale = torch.full((w.rows,), -1.0, device="cuda")
    part = torch.full((w.rows, w.n_keep), float("nan"), device="cuda")
    pb = sph.sph_partial_logits_noalloc(w.h_cloud, w.W_h, codes=codes,
                                        row_scale=scale, keep_ids=w.keep_ids,
                                        clip=w.clip, w_row_scale=w.w_scale,
                                        bias=w.bias, partial_out=part,
                                        act_mode=act)
    return codes, scale, part, pb


def compare(a, b):
    assert_close(np_(b[2]), np_(a[2]).astype(np.float64), "partial logits")
    assert_codes(np_(b[0]), np_(a[0]))
    assert_close(np_(b[1]) * 127.0, np_(a[1]).astype(np.float64) * 127.0, "row absmax")
    assert a[3] == b[3]


def against_oracle(w, got, act_name):
    ref = oracle_cloud(w, act_name)
    assert_close(np_(got[2]), ref["y"], "partial logits vs oracle")
    assert_codes(np_(got[0]), ref["codes"], "codes vs oracle")
    assert_close(np_(got[1]).astype(np.float64) * 127.0,
                 ref["row_scale"].astype(np.float64) * 127.0, "row absmax vs oracle")
    assert got[3] == ref["payload_bytes"]


def padded(W, mult):
    """W [V, d_h] as a view of a buffer whose rows are padded to a multiple of
    `mult` elements (the 16-byte row stride the calls require), so that a
    d_h that is not a multiple of the GEMV's 16-byte vector reaches its
    scalar tail."""
    V, dh = W.shape
    ld = (dh + mult - 1) // mult * mult
    buf = torch.zeros(V, ld, dtype=W.dtype, device=W.device)
    buf[:, :dh] = W
    return buf[:, :dh]


# (kwargs of the seeded workload, activation mode): bf16 and e4m3 heads,
# both activation modes, a kept-id subset and the full vocabulary, hidden
# widths that are and are not multiples of the 16-byte vector (the GEMV's
# scalar tail: 1023 bf16 and 595 e4m3 columns, in padded row strides)
CASES = [
    (dict(V=6000, d=1024, d_l=128, rows=32, n_keep=2500, seed=501), "fp32"),
    (dict(V=3000, d=776, d_l=8, rows=7, n_keep=3000, seed=502, with_bias=True,
          clip=0.4), "fp32"),
    (dict(V=2500, d=1280, d_l=256, rows=5, n_keep=2500, seed=504, w_dtype="fp8",
          clip=40.0), "fp32"),
    (dict(V=4000, d=1100, d_l=77, rows=3, n_keep=1700, seed=505), "bf16"),
    (dict(V=2048, d=600, d_l=5, rows=9, n_keep=900, seed=506, w_dtype="fp8",
          clip=40.0), "bf16"),
]


@pytest.mark.parametrize("kw,act", CASES,
                         ids=[f"{c[0].get('w_dtype', 'bf16')}-{c[1]}-{c[0]['rows']}r-"
                              f"{c[0]['d'] - c[0]['d_l']}dh" for c in CASES])
def test_no_alloc_matches_oracle_and_regular_call_twice(sph, kw, act):
    mode = sph.SPH_ACT_BF16 if act == "bf16" else sph.SPH_ACT_FP32
    ctx = sph.Context(0)
    try:
        w = wl.make_workload(device="cuda", **kw)
        w.W_h = padded(w.W_h, 16 if w.w_dtype == "fp8" else 8)
        ref = regular(sph, ctx, w, mode)
        # two calls in a row: the shared scratch keeps the first call's
        # contents (row maxima included), which must not leak into the second
        for _ in range(2):
            got = no_alloc(sph, w, mode)
            torch.cuda.synchronize()
            compare(ref, got)
            against_oracle(w, got, act)
    finally:
        ctx.close()


def test_no_alloc_calls_in_a_row_with_different_inputs(sph):
    ctx = sph.Context(0)
    try:
        w1 = wl.make_workload(V=6000, d=1024, d_l=128, rows=32, n_keep=2500,
                              seed=511, device="cuda")
        w2 = wl.make_workload(V=3000, d=776, d_l=8, rows=7, n_keep=3000,
                              seed=512, device="cuda", with_bias=True, clip=0.4)
        for w in (w1, w2, w1):
            got = no_alloc(sph, w, sph.SPH_ACT_FP32)
            torch.cuda.synchronize()
            compare(regular(sph, ctx, w, sph.SPH_ACT_FP32), got)
            against_oracle(w, got, "fp32")
    finally:
        ctx.close()


def test_no_alloc_allocates_nothing_after_its_first_call(sph):
    w = wl.make_workload(V=5000, d=900, d_l=100, rows=12, n_keep=2000, seed=513,
                         device="cuda")
    codes = torch.empty(w.rows, w.n_keep, dtype=torch.int8, device="cuda")
    scale = torch.empty(w.rows, device="cuda")
    part = torch.empty(w.rows, w.n_keep, device="cuda")

    def call():
        sph.sph_partial_logits_noalloc(w.h_cloud, w.W_h, codes=codes, row_scale=scale,
                                       keep_ids=w.keep_ids, clip=w.clip, partial_out=part)
    call()                                     # set-up call: modules load here
    torch.cuda.synchronize()
    free0, _ = torch.cuda.mem_get_info()
    torch_alloc0 = torch.cuda.memory_allocated()
    for _ in range(5):
        call()
    torch.cuda.synchronize()
    free1, _ = torch.cuda.mem_get_info()
    assert free1 == free0, f"device free memory moved by {free0 - free1} bytes"
    assert torch.cuda.memory_allocated() == torch_alloc0
    against_oracle(w, (codes, scale, part, sph.sph_payload_bytes(w.rows, w.n_keep)), "fp32")


def test_no_alloc_rejects_oversized_calls(sph):
    limit = sph.NOALLOC_SCRATCH_BYTES
    rows = 64
    n = limit // (4 * rows) + 1                  # one column over the limit
    w = wl.make_workload(V=n, d=16, d_l=8, rows=rows, n_keep=n, seed=503,
                         device="cuda")
    codes = torch.empty(rows, n, dtype=torch.int8, device="cuda")
    scale = torch.empty(rows, device="cuda")
    with pytest.raises(sph.SphError) as e:
        sph.sph_partial_logits_noalloc(w.h_cloud, w.W_h, codes=codes,
                                       row_scale=scale, clip=30.0)
    assert e.value.status == 2 and "fixed scratch" in str(e.value)


def test_no_alloc_binding_checks_output_shapes(sph):
    w = wl.make_workload(V=1000, d=300, d_l=44, rows=4, n_keep=500, seed=514,
                         device="cuda")
    good = dict(codes=torch.empty(4, 500, dtype=torch.int8, device="cuda"),
                row_scale=torch.empty(4, device="cuda"))
    bad = [dict(good, codes=torch.empty(4, 499, dtype=torch.int8, device="cuda")),
           dict(good, codes=torch.empty(500, 4, dtype=torch.int8, device="cuda").t()),
           dict(good, row_scale=torch.empty(3, device="cuda")),
           dict(good, partial_out=torch.empty(4, 1000, device="cuda")[:, :500])]
    for kw in bad:
        with pytest.raises(ValueError):
            sph.sph_partial_logits_noalloc(w.h_cloud, w.W_h, keep_ids=w.keep_ids,
                                           clip=w.clip, **kw)
