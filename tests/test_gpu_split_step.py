"""The one-call split step (sph_split_step) against the oracle's chained
split step: the payload that would cross (codes and scales, per chunk), the
fused logits and the tokens, on both kernel paths, with one chunk (the
endpoint quantizes the cloud's partials in its own epilogue) and with a
block-streamed payload on two streams.  Needs a GPU (marked gpu)."""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_13093_gb300 import workloads as wl
from _parity import (ATOL, MARGIN, RTOL, GREEDY_GAP, assert_codes, bits, np_)

pytestmark = pytest.mark.gpu
DEV = "cuda"
PATHS = {"tc": 1, "gemv": 1 << 40}


@pytest.fixture(scope="module")
def ctx():
    from paper_2607_13093_gb300 import build_lib
    build_lib.build()
    from paper_2607_13093_gb300 import sph
    c = sph.Context(0)
    yield c
    c.close()


@pytest.fixture(params=sorted(PATHS))
def path_ctx(request, ctx):
    from paper_2607_13093_gb300 import sph
    ctx.set_option(sph.SPH_OPT_TC_MIN_ROWS, PATHS[request.param])
    yield ctx
    ctx.set_option(sph.SPH_OPT_TC_MIN_ROWS, 4)


def small(**kw):
    kw.setdefault("seed", 301)
    return wl.make_workload(device=DEV, **kw)


def run_gpu(ctx, w, chunk, act="fp32", store_z=True):
    """The split step; store_z False: no z output and z never stored
    (SPH_OPT_ENDPOINT_Z = 2), z returned as None."""
    from paper_2607_13093_gb300 import sph
    z = torch.empty(w.rows, w.n_keep, device=DEV) if store_z else None
    ctx.set_option(sph.SPH_OPT_ENDPOINT_Z, 0 if store_z else 2)
    try:
        codes, scales, tok, pb = ctx.split_step(
            w.h, w.d_l, w.W_h, w.W_l, keep_ids=w.keep_ids, clip=w.clip,
            w_row_scale=w.w_scale, bias=w.bias,
            act_mode=sph.SPH_ACT_BF16 if act == "bf16" else sph.SPH_ACT_FP32,
            temperature=w.tau, seed=w.seed, offset=w.offset, chunk=chunk, fused_logits_out=z)
    finally:
        ctx.set_option(sph.SPH_OPT_ENDPOINT_Z, 0)
    ctx.sync()
    R, n = w.rows, w.n_keep
    b = oracle.chunk_bounds(n, chunk)
    flat = np_(codes)
    c = np.empty((R, n), dtype=np.int8)
    for q, (j0, j1) in enumerate(b):         # chunk-major -> [R, n]
        c[:, j0:j1] = flat[j0 * R: j0 * R + R * (j1 - j0)].reshape(R, j1 - j0)
    s = np_(scales)[: len(b) * R].reshape(len(b), R)
    return c, s, np_(tok), (np_(z) if store_z else None), pb


def oracle_split(w, chunk, act="fp32", rows=None):
    """The oracle's split step on rows `rows` (all by default), drawing with
    each row's own uniform."""
    sel = np.arange(w.rows) if rows is None else np.asarray(rows)
    h = np_(w.h)[sel]
    ids = np_(w.keep_ids)
    c = oracle.partial_logits(h[:, w.d_l:], bits(w.W_h), w_dtype=w.w_dtype,
                              w_scale=np_(w.w_scale), bias=np_(w.bias), keep_ids=ids,
                              clip=w.clip, act_mode=act)
    codes, scales = oracle.quantize_chunks(c["y"], w.clip, chunk)
    vocab = np.arange(w.V) if ids is None else ids
    zl = oracle.local_partial(h[:, :w.d_l], bits(w.W_l), vocab)
    z = oracle.fuse_chunks(codes, scales, zl, chunk)
    if w.tau == 0:
        j, margin = oracle.greedy_rows(z)
        margin = np.where(margin >= GREEDY_GAP, 1.0, 0.0)
    else:
        u = oracle.philox_uniform(w.seed, sel, 0, w.offset)
        j, margin = oracle.sample_rows(z, w.tau, u)
    return dict(codes=codes, scales=scales, z=z, tokens=vocab[j], margin=margin,
                payload=oracle.payload_bytes_chunked(w.rows, w.n_keep, chunk), sel=sel,
                vocab=vocab)


def check_split(ctx, w, chunk, act="fp32", rows=None):
    c, s, tok, z, pb = run_gpu(ctx, w, chunk, act)
    ref = oracle_split(w, chunk, act, rows)
    sel = ref["sel"]
    assert pb == ref["payload"]
    assert_codes(c[sel], ref["codes"])
    assert np.allclose(s[:, sel].astype(np.float64) * 127, ref["scales"].astype(np.float64) * 127,
                       rtol=RTOL, atol=ATOL)
    # fused logits: within the tolerance, plus one quantization step where
    # the GPU's code is the other rounding of a quotient on a half-integer
    # (which the code bar allows)
    diff = c[sel].astype(np.int64) != ref["codes"].astype(np.int64)
    step = np.zeros_like(ref["z"])
    for q, (j0, j1) in enumerate(oracle.chunk_bounds(w.n_keep, chunk)):
        step[:, j0:j1] = ref["scales"][q].astype(np.float64)[:, None]
    allow = ATOL + RTOL * np.abs(ref["z"]) + np.where(diff, step * (1 + 1e-6), 0.0)
    excess = np.abs(z[sel].astype(np.float64) - ref["z"]) - allow
    assert excess.max() <= 0, f"fused logits off by {excess.max()}"
    # tokens: identical wherever the draw's margin exceeds what the codes
    # that differ (by one step, as the bar allows) can move it.  Moving
    # logits j in M by at most one step s changes their weights by a factor
    # within exp(+-s/tau), so no CDF value moves by more than
    # 2 sum_{j in M} p_j (exp(s/tau) - 1) (to first order; 2.2 with slack);
    # for greedy draws the top-two gap must exceed two steps.
    need = np.full(len(sel), MARGIN)
    for i in np.nonzero(diff.any(axis=1))[0]:
        m = diff[i]
        s_max = float(step[i][m].max())
        if w.tau == 0:
            gap = np.sort(ref["z"][i])[-2:]
            need[i] = MARGIN if gap[1] - gap[0] > 2 * s_max + GREEDY_GAP else np.inf
        else:
            p = oracle.softmax_rows(ref["z"][i][None, :], w.tau)[0]
            need[i] = max(MARGIN, 2.2 * float(p[m].sum()) * np.expm1(s_max / w.tau))
    check = ref["margin"] >= need
    bad = check & (tok[sel] != ref["tokens"])
    assert not bad.any(), f"tokens differ at rows {sel[bad]}"
    assert np.isin(tok, ref["vocab"]).all(), "a masked id was sampled"
    assert check.any()
    if chunk == 0:
        # the same step without storing z: the same payload bit for bit, and
        # tokens under the same rule
        c2, s2, tok2, _, pb2 = run_gpu(ctx, w, chunk, act, store_z=False)
        assert pb2 == pb and np.array_equal(c2, c) and np.array_equal(s2, s)
        bad = check & (tok2[sel] != ref["tokens"])
        assert not bad.any(), f"tokens (z recomputed) differ at rows {sel[bad]}"
        assert np.isin(tok2, ref["vocab"]).all(), "a masked id was sampled (z recomputed)"
    return c, s, tok, z


ONE_CHUNK = [
    ("decode-small", dict(V=4000, d=1024, d_l=128, rows=32, n_keep=1500, tau=0.8)),
    ("rows3", dict(V=2000, d=312, d_l=40, rows=3, n_keep=700)),
    ("full-vocab-bias", dict(V=3000, d=776, d_l=8, rows=7, n_keep=3000, with_bias=True,
                             clip=0.5)),
    ("fp8", dict(V=3000, d=1280, d_l=256, rows=16, n_keep=3000, w_dtype="fp8", clip=40.0)),
    ("rows130", dict(V=1500, d=392, d_l=8, rows=130, n_keep=1300)),
    ("greedy", dict(V=4000, d=1024, d_l=256, rows=24, n_keep=1500, tau=0.0)),
]


@pytest.mark.parametrize("name,kw", ONE_CHUNK, ids=[c[0] for c in ONE_CHUNK])
def test_split_step_one_chunk(path_ctx, name, kw):
    check_split(path_ctx, small(**kw), 0)


@pytest.mark.parametrize("name,kw", [c for c in ONE_CHUNK if c[0] != "fp8"],
                         ids=[c[0] for c in ONE_CHUNK if c[0] != "fp8"])
@pytest.mark.parametrize("quantize", [1, 2])
@pytest.mark.parametrize("rows_m", [1, 2])
def test_split_step_pairs(ctx, name, kw, quantize, rows_m):
    # both contractions on CTA pairs, the endpoint quantizing in its epilogue
    # (1) or after a separate pass (2), with the rows as the MMA's M (1) or
    # the ids (2)
    from paper_2607_13093_gb300 import sph
    ctx.set_option(sph.SPH_OPT_TC_MIN_ROWS, 1)
    ctx.set_option(sph.SPH_OPT_TC_PAIR, 1)
    ctx.set_option(sph.SPH_OPT_SPLIT_QUANTIZE, quantize)
    ctx.set_option(sph.SPH_OPT_ENDPOINT_ROWS_M, rows_m)
    try:
        w = small(**kw)
        pe = ctx.plan(1, w.rows, w.n_keep, w.d_l, gather=w.keep_ids is not None)
        assert pe["pair"] == 1 and pe["rows_m"] == (rows_m == 1)
        check_split(ctx, w, 0)
    finally:
        ctx.set_option(sph.SPH_OPT_ENDPOINT_ROWS_M, 0)
        ctx.set_option(sph.SPH_OPT_SPLIT_QUANTIZE, 0)
        ctx.set_option(sph.SPH_OPT_TC_PAIR, 0)
        ctx.set_option(sph.SPH_OPT_TC_MIN_ROWS, 4)


@pytest.mark.parametrize("rows", [2, 40])
def test_split_step_bf16_activations(path_ctx, rows):
    check_split(path_ctx, small(V=3000, d=776, d_l=64, rows=rows, n_keep=1200), 0, act="bf16")


@pytest.mark.parametrize("where", [1, 2], ids=["epilogue", "pass"])
def test_split_step_equals_the_two_calls(ctx, where):
    # one chunk: the fused epilogue rounds exactly as the quantize kernel,
    # and the endpoint's contraction is the same, so the payload, the fused
    # logits and the tokens are bit-identical to the two calls', whether the
    # quantization runs in the endpoint's epilogue or as its own pass
    from paper_2607_13093_gb300 import sph
    for kw in (dict(V=4000, d=1024, d_l=128, rows=32, n_keep=1500, tau=0.8),
               dict(V=2000, d=312, d_l=40, rows=3, n_keep=700),
               dict(V=6000, d=2112, d_l=64, rows=160, n_keep=5000)):
        w = small(**kw)
        ctx.set_option(sph.SPH_OPT_SPLIT_QUANTIZE, where)
        try:
            c, s, tok, z, _ = run_gpu(ctx, w, 0)
        finally:
            ctx.set_option(sph.SPH_OPT_SPLIT_QUANTIZE, 0)
        codes2, scale2, _ = ctx.partial_logits(w.h_cloud, w.W_h, keep_ids=w.keep_ids,
                                               clip=w.clip)
        z2 = torch.empty(w.rows, w.n_keep, device=DEV)
        tok2 = ctx.fuse_sample(codes2, scale2, w.h_local, w.W_l, keep_ids=w.keep_ids,
                               temperature=w.tau, seed=w.seed, offset=w.offset,
                               fused_logits_out=z2)
        ctx.sync()
        assert np.array_equal(c, np_(codes2))
        assert np.array_equal(s[0], np_(scale2))
        assert np.array_equal(z, np_(z2))
        assert np.array_equal(tok, np_(tok2))


CHUNKED = [
    ("decode-small-1024", dict(V=4000, d=1024, d_l=128, rows=32, n_keep=2500, tau=0.8), 1024),
    ("ragged-700", dict(V=3000, d=600, d_l=72, rows=20, n_keep=2100), 700),
    ("gemv-rows", dict(V=2000, d=312, d_l=40, rows=3, n_keep=1700), 512),
    ("full-vocab-bias", dict(V=3000, d=776, d_l=8, rows=9, n_keep=3000, with_bias=True), 1000),
    ("fp8-full-vocab", dict(V=3000, d=1280, d_l=256, rows=16, n_keep=3000, w_dtype="fp8",
                            clip=40.0), 768),
    ("one-id-chunks", dict(V=40, d=96, d_l=16, rows=5, n_keep=7, run_lo=1, run_hi=3), 1),
    ("greedy", dict(V=4000, d=1024, d_l=256, rows=24, n_keep=2500, tau=0.0), 1024),
    # 160-row blocks over d_l = 64: the endpoint's transposed epilogue, with
    # chunk offsets that keep z's rows 16-byte aligned (1000) or not (1002)
    ("rows160-1000", dict(V=5000, d=1088, d_l=64, rows=160, n_keep=4000), 1000),
    ("rows160-1002", dict(V=5000, d=1088, d_l=64, rows=160, n_keep=4000), 1002),
]


@pytest.mark.parametrize("name,kw,chunk", CHUNKED, ids=[c[0] for c in CHUNKED])
def test_split_step_chunked(path_ctx, name, kw, chunk):
    check_split(path_ctx, small(**kw), chunk)


def test_split_step_chunked_on_a_callers_stream(ctx):
    w = small(V=4000, d=1024, d_l=128, rows=32, n_keep=2500, tau=0.8)
    es = torch.cuda.Stream()
    from paper_2607_13093_gb300 import sph
    z = torch.empty(w.rows, w.n_keep, device=DEV)
    codes, scales, tok, _ = ctx.split_step(w.h, w.d_l, w.W_h, w.W_l, keep_ids=w.keep_ids,
                                           clip=w.clip, temperature=w.tau, seed=w.seed,
                                           chunk=1024, endpoint_stream=es.cuda_stream,
                                           fused_logits_out=z)
    # the call's work is ordered on the context's stream: read without syncing es
    got = np_(tok)
    c, s, tok2, z2, _ = run_gpu(ctx, w, 1024)
    assert np.array_equal(got, tok2) and np.array_equal(np_(z), z2)
    # the context's own stream: the chunks one after another, same results
    z3 = torch.empty(w.rows, w.n_keep, device=DEV)
    codes3, scales3, tok3, _ = ctx.split_step(
        w.h, w.d_l, w.W_h, w.W_l, keep_ids=w.keep_ids, clip=w.clip, temperature=w.tau,
        seed=w.seed, chunk=1024, endpoint_stream=torch.cuda.current_stream().cuda_stream,
        fused_logits_out=z3)
    assert np.array_equal(np_(tok3), got) and np.array_equal(np_(z3), np_(z))
    assert np.array_equal(np_(codes3), np_(codes)) and np.array_equal(np_(scales3), np_(scales))


@pytest.mark.parametrize("name,rows,keep,chunk", [("decode", None, None, 0),
                                                  ("decode", None, None, 4096),
                                                  ("dend", None, 0.4, 15000),
                                                  ("sweep", 64, 0.5, 0)])
def test_split_step_full_size(ctx, name, rows, keep, chunk):
    w = wl.workload(name, device=DEV, rows=rows, keep_frac=keep)
    sample = list(range(w.rows)) if w.rows <= 32 else sorted(
        set(np.linspace(0, w.rows - 1, 16).round().astype(int).tolist()))
    check_split(ctx, w, chunk, rows=sample)
