"""Failure detection on the GPU without a GPU fault (needs a GPU; marked gpu).

Every device-side wait of the tensor-core kernel is bounded by the context's
spin limit.  With a limit of one clock cycle the first wait that is not
already satisfied gives up: the kernel records the timeout in the context's
error word, lets the copies and MMAs it issued land, releases its tensor
memory and returns.  The host reads SPH_ERR_TIMEOUT at sync, and the same
context then computes correct results again."""
import pytest

from paper_2607_13093_gb300 import workloads as wl
from _parity import check_cloud, check_endpoint, oracle_cloud

pytestmark = pytest.mark.gpu

DEV = "cuda"
STATUS_TIMEOUT = 4


@pytest.fixture(scope="module")
def ctx():
    from paper_2607_13093_gb300 import build_lib
    build_lib.build()
    from paper_2607_13093_gb300 import sph
    c = sph.Context(0)
    yield c
    c.close()


def _expect_timeout(ctx, enqueue):
    from paper_2607_13093_gb300 import sph
    ctx.set_option(sph.SPH_OPT_SPIN_LIMIT, 1)
    try:
        enqueue()
        with pytest.raises(sph.SphError) as err:
            ctx.sync()
        assert err.value.status == STATUS_TIMEOUT, str(err.value)
    finally:
        ctx.set_option(sph.SPH_OPT_SPIN_LIMIT, 1 << 34)
    ctx.sync()                      # reported once, then cleared


def test_cloud_wait_timeout_is_reported_and_context_recovers(ctx):
    w = wl.make_workload(V=6000, d=1024, d_l=128, rows=64, n_keep=3000, device=DEV, seed=91)
    _expect_timeout(ctx, lambda: ctx.partial_logits(w.h_cloud, w.W_h, keep_ids=w.keep_ids,
                                                    clip=w.clip))
    check_cloud(ctx, w)


def test_endpoint_wait_timeout_is_reported_and_context_recovers(ctx):
    import torch
    w = wl.make_workload(V=6000, d=1024, d_l=128, rows=48, n_keep=3000, device=DEV, seed=92)
    ref = oracle_cloud(w)
    codes = torch.from_numpy(ref["codes"])
    scale = torch.from_numpy(ref["row_scale"])
    _expect_timeout(ctx, lambda: ctx.fuse_sample(codes.to(DEV), scale.to(DEV), w.h_local,
                                                 w.W_l, keep_ids=w.keep_ids,
                                                 temperature=w.tau, seed=w.seed))
    check_endpoint(ctx, w, codes, scale)
