"""The allocation-free cloud call agrees with the regular one.

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
from _parity import assert_close, assert_codes, np_

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def sph():
    from paper_2607_13093_gb300 import build_lib
    build_lib.build()
    from paper_2607_13093_gb300 import sph as mod
    return mod


def regular(sph, ctx, w):
    part = torch.empty(w.rows, w.n_keep, device="cuda")
    codes, scale, pb = ctx.partial_logits(w.h_cloud, w.W_h, keep_ids=w.keep_ids,
                                          clip=w.clip, w_row_scale=w.w_scale,
                                          bias=w.bias, partial_out=part)
    return codes, scale, part, pb


def no_alloc(sph, w):
    codes = torch.full((w.rows, w.n_keep), 99, dtype=torch.int8, device="cuda")
    scale = torch.full((w.rows,), -1.0, device="cuda")
    part = torch.full((w.rows, w.n_keep), float("nan"), device="cuda")
    pb = sph.sph_partial_logits_noalloc(w.h_cloud, w.W_h, codes=codes,
                                        row_scale=scale, keep_ids=w.keep_ids,
                                        clip=w.clip, w_row_scale=w.w_scale,
                                        bias=w.bias, partial_out=part)
    return codes, scale, part, pb


def compare(a, b):
    assert_close(np_(b[2]), np_(a[2]).astype(np.float64), "partial logits")
    assert_codes(np_(b[0]), np_(a[0]))
    assert_close(np_(b[1]) * 127.0, np_(a[1]).astype(np.float64) * 127.0, "row absmax")
    assert a[3] == b[3]


def test_no_alloc_matches_regular_call_twice(sph):
    ctx = sph.Context(0)
    try:
        # two calls in a row with different inputs: the shared scratch keeps
        # the first call's contents, which must not leak into the second
        w1 = wl.make_workload(V=6000, d=1024, d_l=128, rows=32, n_keep=2500,
                              seed=501, device="cuda")
        w2 = wl.make_workload(V=3000, d=776, d_l=8, rows=7, n_keep=3000,
                              seed=502, device="cuda", with_bias=True, clip=0.4)
        for w in (w1, w2):
            ref = regular(sph, ctx, w)
            got = no_alloc(sph, w)
            torch.cuda.synchronize()
            compare(ref, got)
    finally:
        ctx.close()


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
