"""A context moved to another stream (sph_set_stream, which the Python
Context does whenever torch's current stream changes) orders the new
stream after the work already issued on the old one: the next call reuses
the context's scratch.  Needs a GPU (marked gpu)."""
import numpy as np
import pytest
import torch

from paper_2607_13093_gb300 import workloads as wl
from _parity import assert_close, assert_codes, np_, oracle_cloud

pytestmark = pytest.mark.gpu
DEV = "cuda"
SENTINEL = -128          # never a code: |code| <= 127 (Eq. 18 with b = 8)
SLEEP_CYCLES = 200_000_000   # about 0.1 s of GPU clock: far longer than the host's enqueue


@pytest.fixture(scope="module")
def ctx():
    from paper_2607_13093_gb300 import build_lib
    build_lib.build()
    from paper_2607_13093_gb300 import sph
    c = sph.Context(0)
    yield c
    c.close()


def cloud(ctx, w, codes=None, scale=None):
    return ctx.partial_logits(w.h_cloud, w.W_h, keep_ids=w.keep_ids, clip=w.clip,
                              codes=codes, row_scale=scale)[:2]


@pytest.mark.parametrize("rows", [32, 2], ids=["tensor-core", "gemv"])
def test_new_stream_waits_for_the_old_one(ctx, rows):
    w1 = wl.make_workload(V=4000, d=1024, d_l=128, rows=rows, n_keep=2500, seed=611,
                          device=DEV)
    w2 = wl.make_workload(V=4000, d=1024, d_l=128, rows=rows, n_keep=2500, seed=612,
                          device=DEV)
    a, b = torch.cuda.Stream(device=DEV), torch.cuda.Stream(device=DEV)
    codes1 = torch.full((rows, w1.n_keep), SENTINEL, dtype=torch.int8, device=DEV)
    scale1 = torch.empty(rows, device=DEV)
    with torch.cuda.stream(a):
        a.wait_stream(torch.cuda.default_stream())
        cloud(ctx, w1)                        # warm-up: scratch sized, modules loaded
        torch.cuda.synchronize()
        torch.cuda._sleep(SLEEP_CYCLES)       # call 1 waits behind ~0.1 s on stream a
        cloud(ctx, w1, codes1, scale1)
    with torch.cuda.stream(b):
        codes2, scale2 = cloud(ctx, w2)       # the context moves to b: b waits for a
        snap = codes1.clone()                 # on b, after call 2
    torch.cuda.synchronize()
    ctx.sync()
    # b ran after a's call 1: the snapshot holds its codes, not the sentinel
    assert not (snap == SENTINEL).any()
    assert torch.equal(snap, codes1)
    for w, codes, scale in ((w1, codes1, scale1), (w2, codes2, scale2)):
        ref = oracle_cloud(w)
        assert_codes(np_(codes), ref["codes"])
        assert_close(np_(scale).astype(np.float64) * 127.0,
                     ref["row_scale"].astype(np.float64) * 127.0, "row absmax")
