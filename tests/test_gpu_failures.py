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


@pytest.mark.parametrize("gather", [True, False])
def test_pair_wait_timeout_is_reported_and_context_recovers(ctx, gather):
    # CTA pairs: a wait that gives up in either CTA winds both down (every
    # wait bounded, the odd CTA's in-flight copies given time to land, both
    # CTAs meet at the end before freeing tensor memory)
    from paper_2607_13093_gb300 import sph
    w = wl.make_workload(V=6000, d=1024, d_l=128, rows=200, n_keep=3000 if gather else 6000,
                         device=DEV, seed=94)
    ctx.set_option(sph.SPH_OPT_TC_PAIR, 1)
    try:
        assert ctx.plan(0, w.rows, w.n_keep, w.d_h, gather=gather)["pair"] == 1
        _expect_timeout(ctx, lambda: ctx.partial_logits(w.h_cloud, w.W_h, keep_ids=w.keep_ids,
                                                        clip=w.clip))
        check_cloud(ctx, w)
    finally:
        ctx.set_option(sph.SPH_OPT_TC_PAIR, 0)


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


def test_bad_arguments_are_rejected_before_any_launch(ctx):
    # each call fails on the host with SPH_ERR_INVALID_ARG before it
    # launches anything; the context then computes correct results
    import torch
    from paper_2607_13093_gb300 import sph
    w = wl.make_workload(V=600, d=136, d_l=8, rows=4, n_keep=300, device=DEV, seed=93)
    codes, scale = (t.to(DEV) for t in wl.make_payload(4, 300, seed=3))
    target = torch.zeros(4, 300, device=DEV)
    drafts = w.keep_ids[:2].view(2, 1).contiguous()
    W36 = torch.zeros(600, 36, dtype=torch.bfloat16, device=DEV)   # 72-byte rows
    h36 = torch.zeros(4, 36, device=DEV)
    W8 = w.W_h.float().to(torch.float8_e4m3fn)
    nan = float("nan")
    cloud = dict(keep_ids=w.keep_ids, clip=30.0)
    cases = {
        "NaN clip": lambda: ctx.partial_logits(w.h_cloud, w.W_h, keep_ids=w.keep_ids, clip=nan),
        "zero clip": lambda: ctx.partial_logits(w.h_cloud, w.W_h, keep_ids=w.keep_ids, clip=0.0),
        "no kept id": lambda: ctx.partial_logits(w.h_cloud, w.W_h, keep_ids=w.keep_ids[:0],
                                                 clip=30.0),
        "more kept ids than V": lambda: ctx.partial_logits(w.h_cloud, w.W_h[:100], **cloud),
        "unaligned weight rows": lambda: ctx.partial_logits(h36, W36, **cloud),
        "fp8 weights without scales": lambda: ctx.partial_logits(w.h_cloud, W8, **cloud),
        "no row": lambda: ctx.partial_logits(w.h_cloud[:0], w.W_h, **cloud),
        "negative temperature": lambda: ctx.fuse_sample(codes, scale, w.h_local, w.W_l,
                                                        keep_ids=w.keep_ids, temperature=-1.0),
        "NaN temperature": lambda: ctx.fuse_sample(codes, scale, w.h_local, w.W_l,
                                                   keep_ids=w.keep_ids, temperature=nan),
        "codes without scales": lambda: ctx.fuse_sample(codes, None, w.h_local, w.W_l,
                                                        keep_ids=w.keep_ids),
        "no draft position": lambda: ctx.verify_draft(target, 4, 0, drafts[:, :0],
                                                      keep_ids=w.keep_ids),
        "no session": lambda: ctx.verify_draft(target[:0], 0, 1, drafts[:0],
                                               keep_ids=w.keep_ids),
        "negative verification temperature": lambda: ctx.verify_draft(
            target, 2, 1, drafts, keep_ids=w.keep_ids, temperature=-0.5),
        "tile height 64": lambda: ctx.set_option(sph.SPH_OPT_TC_TILE_M, 64),
        "row block of 20": lambda: ctx.set_option(sph.SPH_OPT_TC_MAX_BN, 20),
        "one stage": lambda: ctx.set_option(sph.SPH_OPT_TC_STAGES, 1),
        "sampler 2": lambda: ctx.set_option(sph.SPH_OPT_SAMPLER, 2),
        "spin limit 0": lambda: ctx.set_option(sph.SPH_OPT_SPIN_LIMIT, 0),
        "unknown option": lambda: ctx.set_option(99, 0),
        "gemv_quantize 2": lambda: ctx.set_option(sph.SPH_OPT_GEMV_QUANTIZE, 2),
    }
    for name, call in cases.items():
        with pytest.raises(sph.SphError) as err:
            call()
        assert err.value.status == 1, (name, str(err.value))
    ctx.sync()
    check_cloud(ctx, w)
