"""GPU <-> oracle parity through the C-ABI (needs a GPU; marked gpu).

Small cases span several tiles and ragged tails; the five named workloads
run at full size in the launch configuration the benchmark times, with the
oracle checking sampled rows."""
import numpy as np
import pytest
import torch

from paper_2607_13093_gb300 import workloads as wl
import oracle
from _parity import (GREEDY_GAP, MARGIN, assert_close, bits, check_cloud, check_endpoint,
                     check_verify, np_, oracle_cloud)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ctx():
    from paper_2607_13093_gb300 import build_lib
    build_lib.build()
    from paper_2607_13093_gb300 import sph
    c = sph.Context(0)
    yield c
    c.close()


DEV = "cuda"
PATHS = {"tc": 1, "gemv": 1 << 40}      # SPH_OPT_TC_MIN_ROWS per kernel path


@pytest.fixture(params=sorted(PATHS))
def path_ctx(request, ctx):
    from paper_2607_13093_gb300 import sph
    ctx.set_option(sph.SPH_OPT_TC_MIN_ROWS, PATHS[request.param])
    yield ctx
    ctx.set_option(sph.SPH_OPT_TC_MIN_ROWS, 4)


def small(**kw):
    kw.setdefault("seed", 77)
    return wl.make_workload(device=DEV, **kw)


# ---------------------------------------------------------------------------
# cloud call: shapes x paths
# ---------------------------------------------------------------------------

CLOUD_CASES = [
    # name, kwargs
    ("tiny-full", dict(V=8192, d=512, d_l=64, rows=1, n_keep=2048)),
    ("decode-small", dict(V=4000, d=1024, d_l=128, rows=32, n_keep=1500, tau=0.8)),
    ("spec-small", dict(V=6000, d=640, d_l=128, rows=20, n_keep=2400, sessions=4, k=4)),
    ("fp8-small", dict(V=3000, d=1280, d_l=256, rows=16, n_keep=3000, w_dtype="fp8", clip=40.0)),
    ("rows3", dict(V=2000, d=300, d_l=44, rows=3, n_keep=700)),
    ("rows17", dict(V=2000, d=300, d_l=44, rows=17, n_keep=701)),
    ("rows64", dict(V=3000, d=520, d_l=8, rows=64, n_keep=1000)),
    ("rows130", dict(V=1500, d=392, d_l=8, rows=130, n_keep=1300)),
    ("keep1", dict(V=500, d=136, d_l=8, rows=2, n_keep=1, run_lo=1, run_hi=1)),
    ("keep7", dict(V=500, d=136, d_l=8, rows=5, n_keep=7, run_lo=1, run_hi=3)),
    ("keep127", dict(V=500, d=136, d_l=8, rows=9, n_keep=127, run_lo=2, run_hi=9)),
    ("bias", dict(V=1000, d=264, d_l=8, rows=4, n_keep=400, with_bias=True)),
]


@pytest.mark.parametrize("name,kw", CLOUD_CASES, ids=[c[0] for c in CLOUD_CASES])
def test_cloud_parity(path_ctx, name, kw):
    w = small(**kw)
    check_cloud(path_ctx, w)


@pytest.mark.parametrize("rows", [1, 8, 40, 300])
def test_cloud_bf16_activation_mode(path_ctx, rows):
    w = small(V=3000, d=776, d_l=8, rows=rows, n_keep=1200)
    check_cloud(path_ctx, w, act_mode="bf16")


def test_cloud_clipping_bites(path_ctx):
    w = small(V=2000, d=1032, d_l=8, rows=6, n_keep=900, clip=0.5)
    codes, scale, part = check_cloud(path_ctx, w)
    assert (np_(part).__abs__() > 0.5).any()          # clip was exercised
    assert np.allclose(np_(scale), np.float32(0.5 / 127))


def test_cloud_zero_row_and_edge_ids(path_ctx):
    ctx = path_ctx
    w = small(V=1000, d=264, d_l=8, rows=5, n_keep=300)
    w.h[2].zero_()
    ids = w.keep_ids.clone()
    ids[0] = 0
    ids[-1] = w.V - 1
    w.keep_ids = torch.unique(ids).to(torch.int32)
    codes, scale, _ = check_cloud(ctx, w)
    assert np_(scale)[2] == 0 and not np_(codes)[2].any()


def test_cloud_tiny_row_scales(path_ctx):
    # row scales below 2^-64 quantize like ordinary rows
    w = small(V=3000, d=264, d_l=8, rows=4, n_keep=2500)
    w.h[1] *= 1e-21
    w.h[3] *= 1e-24
    codes, scale, _ = check_cloud(path_ctx, w)
    ref = oracle_cloud(w, "fp32", None)
    s = np_(scale).astype(np.float64)
    for r in (1, 3):
        assert 0 < s[r] < 2.0 ** -64
        assert abs(s[r] - ref["row_scale"][r]) <= 1e-3 * ref["row_scale"][r]
        assert np.abs(np_(codes)[r]).max() == 127


GUARD_BYTES = 256              # keeps every output view 256-byte aligned
SENTINEL = 0xA5


def guarded(shape, dtype):
    """An output tensor inside a larger buffer whose GUARD_BYTES margins on
    each side hold a sentinel byte."""
    n = int(np.prod(shape))
    g = GUARD_BYTES // torch.empty((), dtype=dtype).element_size()
    buf = torch.empty(n + 2 * g, dtype=dtype, device=DEV)
    buf.view(torch.uint8).fill_(SENTINEL)
    return buf, buf[g:g + n].view(shape)


def guards_intact(buf):
    b = buf.view(torch.uint8)
    return bool((b[:GUARD_BYTES] == SENTINEL).all()) and bool((b[-GUARD_BYTES:] == SENTINEL).all())


@pytest.mark.parametrize("w_dtype", ["bf16", "fp8"])
@pytest.mark.parametrize("n_keep", [1301, 1304])
def test_outputs_stay_inside_their_buffers(path_ctx, w_dtype, n_keep):
    # every output of the three calls sits between sentinel margins; a write
    # past either end of any output (a vector store rounded up to a tile, a
    # ragged tail) shows up as a changed margin byte
    ctx = path_ctx
    S, k = 6, 2
    w = small(V=3000, d=1048, d_l=40, rows=S * (k + 1), n_keep=n_keep, w_dtype=w_dtype,
              clip=40.0 if w_dtype == "fp8" else 30.0, sessions=S, k=k, tau=0.9)
    R, n = w.rows, w.n_keep
    outs = {}
    outs["codes"], codes = guarded((R, n), torch.int8)
    outs["row_scale"], scale = guarded((R,), torch.float32)
    outs["partial_out"], part = guarded((R, n), torch.float32)
    ctx.partial_logits(w.h_cloud, w.W_h, keep_ids=w.keep_ids, clip=w.clip,
                       w_row_scale=w.w_scale, codes=codes, row_scale=scale,
                       partial_out=part)
    for tau in (w.tau, 0.0):
        outs[f"tokens {tau}"], tok = guarded((R,), torch.int32)
        outs[f"z {tau}"], z = guarded((R, n), torch.float32)
        ctx.fuse_sample(codes, scale, w.h_local, w.W_l, keep_ids=w.keep_ids,
                        temperature=tau, seed=w.seed, tokens=tok, fused_logits_out=z)
        outs[f"n_accepted {tau}"], acc = guarded((S,), torch.int32)
        outs[f"next_token {tau}"], nxt = guarded((S,), torch.int32)
        ctx.verify_draft(z, S, k, w.draft_tokens, keep_ids=w.keep_ids,
                         draft_probs=w.draft_probs if tau > 0 else None, temperature=tau,
                         seed=w.seed, n_accepted=acc, next_token=nxt)
        ctx.sync()
        assert set(np_(tok).tolist()) <= set(np_(w.keep_ids).tolist())
        assert ((np_(acc) >= 0) & (np_(acc) <= k)).all()
    ctx.sync()
    assert np.abs(np_(codes).astype(int)).max() == 127 and (np_(scale) > 0).all()
    for name, buf in outs.items():
        assert guards_intact(buf), name


GEMV_Q = [
    # rows, n_keep, d, w_dtype, act, bias
    (1, 2048, 512, "bf16", "fp32", False),     # the tiny workload's shape
    (2, 2000, 1032, "bf16", "bf16", True),
    (4, 700, 296, "fp8", "fp32", False),
    (8, 512, 776, "bf16", "fp32", False),      # 2^12 entries, the most it takes
    (1, 4001, 520, "bf16", "fp32", False),     # a ragged last batch
]


@pytest.mark.parametrize("rows,n_keep,d,w_dtype,act,bias", GEMV_Q,
                         ids=[f"{c[0]}x{c[1]}-{c[3]}-{c[4]}" for c in GEMV_Q])
def test_gemv_last_block_quantize(ctx, rows, n_keep, d, w_dtype, act, bias):
    """The cloud GEMV whose last block quantizes the payload itself: codes,
    scales and partials bit-identical to the separate quantize pass and
    within the parity bar of the oracle; calls in a row (different inputs,
    then the first again) find the row maxima and the arrival count cleared."""
    from paper_2607_13093_gb300 import sph
    ws = [small(V=5 * n_keep, d=d, d_l=8, rows=rows, n_keep=n_keep, w_dtype=w_dtype,
                clip=40.0 if w_dtype == "fp8" else 30.0, with_bias=bias, seed=s)
          for s in (701, 702)]
    ws[1].h[rows - 1].zero_()                    # an all-zero row (scale 0)
    ctx.set_option(sph.SPH_OPT_TC_MIN_ROWS, 1 << 40)
    try:
        got = {}
        for mode in (1, 0):                       # separate pass, then the last block
            ctx.set_option(sph.SPH_OPT_GEMV_QUANTIZE, mode)
            for i in (0, 1, 0):
                codes, scale, part = check_cloud(ctx, ws[i], act_mode=act)
                got.setdefault((mode, i), (np_(codes), np_(scale), np_(part)))
        for i in (0, 1):
            for a, b in zip(got[(0, i)], got[(1, i)]):
                assert np.array_equal(a.view(np.uint8), b.view(np.uint8))
    finally:
        ctx.set_option(sph.SPH_OPT_TC_MIN_ROWS, 4)
        ctx.set_option(sph.SPH_OPT_GEMV_QUANTIZE, 0)


def test_cloud_odd_hidden_width_and_strides(path_ctx):
    ctx = path_ctx
    # d_h = 37 (not a multiple of anything) inside a padded weight stride
    base = small(V=900, d=45, d_l=8, rows=7, n_keep=350)
    Wpad = torch.zeros(base.V, 40, dtype=torch.bfloat16, device=DEV)
    Wpad[:, :37] = base.W_h
    base.W_h = Wpad[:, :37]
    check_cloud(ctx, base)


# ---------------------------------------------------------------------------
# endpoint call: fuse + mask + softmax + sample on the oracle's payload
# ---------------------------------------------------------------------------

ENDPOINT_CASES = [
    ("tiny-full", dict(V=8192, d=512, d_l=64, rows=1, n_keep=2048)),
    ("decode-small", dict(V=4000, d=1024, d_l=256, rows=32, n_keep=1500, tau=0.8)),
    ("rows17-keep7", dict(V=500, d=136, d_l=40, rows=17, n_keep=7, run_lo=1, run_hi=3)),
    ("full-vocab", dict(V=3000, d=1280, d_l=264, rows=16, n_keep=3000)),
    ("rows70", dict(V=2500, d=600, d_l=72, rows=70, n_keep=1100)),
]


@pytest.mark.parametrize("name,kw", ENDPOINT_CASES, ids=[c[0] for c in ENDPOINT_CASES])
def test_endpoint_parity(path_ctx, name, kw):
    ctx = path_ctx
    w = small(**kw)
    ref = oracle_cloud(w)
    codes = torch.from_numpy(ref["codes"])
    scale = torch.from_numpy(ref["row_scale"])
    for off in (0, 1, 12345):
        w.offset = off
        check_endpoint(ctx, w, codes, scale)


FUSE_ONLY = [
    ("decode-small", dict(V=4000, d=1024, d_l=256, rows=32, n_keep=1500, tau=0.8)),
    ("spec-like", dict(V=6000, d=640, d_l=128, rows=160, n_keep=2400, sessions=32, k=4)),
    ("full-vocab", dict(V=3000, d=1280, d_l=264, rows=16, n_keep=3000)),
    ("rows3", dict(V=2000, d=300, d_l=40, rows=3, n_keep=700)),
]


@pytest.mark.parametrize("name,kw", FUSE_ONLY, ids=[c[0] for c in FUSE_ONLY])
def test_endpoint_fuse_only(path_ctx, name, kw):
    # no tokens: z alone (no statistics, no draw), bit-identical to the z of
    # the drawing call and within tolerance of the oracle; the verification
    # of drafted rows on it matches the oracle
    ctx = path_ctx
    w = small(**kw)
    ref = oracle_cloud(w)
    codes = torch.from_numpy(ref["codes"]).to(DEV)
    scale = torch.from_numpy(ref["row_scale"]).to(DEV)
    z_draw = torch.empty(w.rows, w.n_keep, device=DEV)
    z_only = torch.full((w.rows, w.n_keep), float("nan"), device=DEV)
    ctx.fuse_sample(codes, scale, w.h_local, w.W_l, keep_ids=w.keep_ids, temperature=w.tau,
                    seed=w.seed, fused_logits_out=z_draw)
    assert ctx.fuse_sample(codes, scale, w.h_local, w.W_l, keep_ids=w.keep_ids,
                           temperature=w.tau, seed=w.seed, fused_logits_out=z_only,
                           draw=False) is None
    ctx.sync()
    assert torch.equal(z_draw.view(torch.int32), z_only.view(torch.int32))
    zl = oracle.local_partial(np_(w.h_local), bits(w.W_l), np_(w.keep_ids))
    assert_close(np_(z_only), oracle.fuse(ref["codes"], ref["row_scale"], zl), "fused logits")
    if w.sessions:
        check_verify(ctx, w, z_only.cpu())


def test_endpoint_fuse_only_needs_z(ctx):
    from paper_2607_13093_gb300 import sph
    w = small(V=600, d=136, d_l=8, rows=4, n_keep=300)
    codes, scale = (t.to(DEV) for t in wl.make_payload(4, 300, seed=3))
    with pytest.raises(ValueError):
        ctx.fuse_sample(codes, scale, w.h_local, w.W_l, keep_ids=w.keep_ids, draw=False)
    # through the C ABI: neither tokens nor z is INVALID_ARG, before any launch
    st = sph.lib.sph_fuse_sample(ctx.handle, codes.data_ptr(), scale.data_ptr(), 4,
                                 w.h_local.data_ptr(), w.h_local.stride(0),
                                 w.W_l.data_ptr(), w.V, w.d_l, w.W_l.stride(0),
                                 w.keep_ids.data_ptr(), 300, 1.0, 0, 0, None, None)
    assert st == 1
    ctx.sync()


@pytest.mark.parametrize("tau", [0.05, 0.8, 3.0])
def test_endpoint_temperatures(ctx, tau):
    w = small(V=2000, d=300, d_l=64, rows=24, n_keep=800, tau=tau)
    codes, scale = wl.make_payload(w.rows, w.n_keep, seed=5)
    check_endpoint(ctx, w, codes, scale)


def test_endpoint_masked_ids_never_sampled(ctx):
    w = small(V=3000, d=200, d_l=64, rows=64, n_keep=300, tau=5.0)
    codes, scale = wl.make_payload(w.rows, w.n_keep, seed=6)
    ids = set(np_(w.keep_ids).tolist())
    seen = set()
    for off in range(50):
        tok = ctx.fuse_sample(codes.to(DEV), scale.to(DEV), w.h_local, w.W_l,
                              keep_ids=w.keep_ids, temperature=w.tau,
                              seed=w.seed, offset=off)
        seen.update(np_(tok).tolist())
    assert seen <= ids and len(seen) > 50


# ---------------------------------------------------------------------------
# verification
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("S,k,n,greedy", [(4, 4, 2400, False), (9, 1, 300, False),
                                          (5, 3, 1000, True), (64, 4, 5000, False)])
def test_verify_parity(ctx, S, k, n, greedy):
    w = small(V=3 * n, d=96, d_l=8, rows=S * (k + 1), n_keep=n, sessions=S, k=k)
    if greedy:
        w.draft_probs = None
    for seed in (3, 4):
        target = wl.make_target_logits(w.rows, w.n_keep, seed=seed, std=1.0)
        w.offset = seed
        check_verify(ctx, w, target)


@pytest.mark.parametrize("n", [1, 31, 33, 1025, 16 * 1024 + 5, 40000])
def test_row_kernels_ragged_sizes(ctx, n):
    # edges of the 32-id segment, the 1024-id chunk and the 16-chunk pass of
    # the statistics and draw kernels; rows 2 and 6 take the CUDA-core and
    # the tensor-core endpoint paths
    for rows in (2, 6):
        w = small(V=n + 7, d=96, d_l=16, rows=rows, n_keep=n, tau=0.7)
        codes, scale = wl.make_payload(w.rows, w.n_keep, seed=n % 97)
        for off in (0, 5):
            w.offset = off
            check_endpoint(ctx, w, codes, scale)
    S, k = 3, 2
    for tau, greedy in ((1.0, False), (0.1, True)):
        w = small(V=n + 7, d=96, d_l=8, rows=S * (k + 1), n_keep=n, sessions=S, k=k,
                  tau=tau)
        if greedy:
            w.draft_probs = None
        target = wl.make_target_logits(w.rows, n, seed=n % 89, std=1.0)
        check_verify(ctx, w, target)


def test_verify_many_sessions(ctx):
    S, k, n = 1000, 1, 200
    w = small(V=3 * n, d=96, d_l=8, rows=S * (k + 1), n_keep=n, sessions=S, k=k)
    target = wl.make_target_logits(w.rows, n, seed=21, std=2.0)
    n_acc, _, _ = check_verify(ctx, w, target)
    a = np_(n_acc)
    assert 0 < (a == 0).sum() < S and 0 < (a == 1).sum() < S


GREEDY_ENDPOINT = [
    ("decode-like", dict(V=4000, d=1024, d_l=256, rows=32, n_keep=1500)),
    ("gemv-rows", dict(V=3000, d=600, d_l=72, rows=3, n_keep=3000)),
    ("stats-pass", dict(V=60000, d=640, d_l=128, rows=160, n_keep=40000)),
]


@pytest.mark.parametrize("name,kw", GREEDY_ENDPOINT, ids=[c[0] for c in GREEDY_ENDPOINT])
def test_endpoint_greedy(path_ctx, name, kw):
    # temperature 0: the first argmax of the fused logits
    w = small(tau=0.0, **kw)
    ref = oracle_cloud(w)
    codes = torch.from_numpy(ref["codes"])
    scale = torch.from_numpy(ref["row_scale"])
    check_endpoint(path_ctx, w, codes, scale)


@pytest.mark.parametrize("S,k,n", [(16, 4, 3000), (64, 2, 51302), (5, 1, 40)])
def test_verify_greedy(ctx, S, k, n):
    # temperature 0: drafts that follow the target's argmax for a random
    # number of positions, then deviate
    w = small(V=2 * n, d=96, d_l=8, rows=S * (k + 1), n_keep=n, sessions=S, k=k, tau=0.0)
    target = wl.make_target_logits(w.rows, n, seed=S + k, std=2.0)
    a = np.argmax(np_(target).astype(np.float64), axis=1).reshape(S, k + 1)
    rng = np.random.default_rng(S)
    ids = np_(w.keep_ids)
    vocab = np.arange(w.V) if ids is None else ids
    drafts = np.empty((S, k), dtype=np.int32)
    for s in range(S):
        cut = rng.integers(0, k + 1)
        for i in range(k):
            j = a[s, i] if i < cut else (a[s, i] + 1 + rng.integers(0, n - 1)) % n
            drafts[s, i] = vocab[j]
    w.draft_tokens = torch.from_numpy(drafts).to(DEV)
    w.draft_probs = None
    n_acc, _, ref = check_verify(ctx, w, target)
    assert 0 < (np_(n_acc) > 0).sum() or S < 8


def test_verify_accepts_drafts_equal_to_target(ctx):
    # q == p  =>  every draft accepted (r < 1 = p/q), bonus from p_k
    S, k, n = 6, 3, 500
    w = small(V=2 * n, d=96, d_l=8, rows=S * (k + 1), n_keep=n, sessions=S, k=k)
    target = wl.make_target_logits(w.rows, n, seed=8, std=1.0)
    p = torch.softmax(target.double(), dim=1).float().view(S, k + 1, n)
    w.draft_probs = p[:, :k].contiguous().to(DEV)
    n_acc, _, _ = check_verify(ctx, w, target)
    assert (np_(n_acc) == k).all()


# ---------------------------------------------------------------------------
# full-size workloads, sampled rows
# ---------------------------------------------------------------------------

FULL = [("tiny", None, None, "fp32"), ("decode", None, None, "fp32"),
        ("decode", None, None, "bf16"), ("spec", None, None, "fp32"),
        ("spec", None, None, "bf16"), ("fp8", None, None, "fp32"),
        ("fp8", None, None, "bf16"), ("sweep", 1, 0.1, "fp32"),
        ("sweep", 8, 1.0, "fp32"), ("sweep", 64, 0.5, "fp32"),
        ("sweep", 256, 1.0, "fp32"), ("sweep", 1024, 1.0, "fp32"),
        ("sweep", 1024, 1.0, "bf16"),
        # the kept-fraction grid of the benchmark (--sweep-grid)
        ("sweep", 8, 0.1, "fp32"), ("sweep", 64, 0.1, "fp32"),
        ("sweep", 256, 0.5, "fp32"), ("sweep", 1024, 0.1, "fp32"),
        ("sweep", 1024, 0.5, "fp32")]


def rows_to_check(ctx, w, act, want=16):
    """Rows of a full-size launch to compare with the oracle: every row when
    there are at most 32, else at least `want`, with at least two from every
    row block of the cloud and the endpoint plans (the block's last row and
    one at an offset that moves with the block, so that different 16-row
    epilogue chunks and lanes are hit), plus rows spread evenly."""
    from paper_2607_13093_gb300 import sph
    R = w.rows
    if R <= 32:
        return list(range(R))
    gather = w.keep_ids is not None
    wdt = sph.SPH_DTYPE_FP8_E4M3 if w.w_dtype == "fp8" else sph.SPH_DTYPE_BF16
    plans = [ctx.plan(0, R, w.n_keep, w.d_h, w_dtype=wdt, gather=gather,
                      act_mode=sph.SPH_ACT_BF16 if act == "bf16" else sph.SPH_ACT_FP32),
             ctx.plan(1, R, w.n_keep, w.d_l, gather=gather)]
    sel = {0, R - 1}
    for p in plans:
        if not p["tensor_core"]:
            continue
        BN = p["block_rows"]
        for b in range(p["row_blocks"]):
            lo, hi = b * BN, min(R, (b + 1) * BN)
            if lo >= R:
                continue
            sel.add(lo + (23 * b + 7) % (hi - lo))
            sel.add(hi - 1)
    for r in np.linspace(0, R - 1, want).round().astype(int):
        sel.add(int(r))
    return sorted(sel)


@pytest.mark.parametrize("name,rows,keep,act", FULL,
                         ids=[f"{n}-{r}-{k}-{a}" for n, r, k, a in FULL])
def test_full_size_sampled_rows(ctx, name, rows, keep, act):
    w = wl.workload(name, device=DEV, rows=rows, keep_frac=keep)
    sample = rows_to_check(ctx, w, act)
    assert len(sample) >= min(16, w.rows)
    codes, scale, _ = check_cloud(ctx, w, act_mode=act, rows=sample)
    # endpoint on a synthetic payload of the same shape (an input shared by
    # both sides), full launch, sampled rows checked
    pc, ps = wl.make_payload(w.rows, w.n_keep, seed=11, device=DEV)
    check_endpoint(ctx, w, pc, ps, rows=sample)
    if w.sessions:
        target = wl.make_target_logits(w.rows, w.n_keep, seed=12, device=DEV)
        check_verify(ctx, w, target.cpu())


def test_full_size_plans_are_covered(ctx):
    # the C5 1024-row plan has several row blocks, and the sampled rows hit
    # every one of them
    from paper_2607_13093_gb300 import sph
    w = wl.workload("sweep", device=DEV, rows=1024, keep_frac=1.0)
    p = ctx.plan(0, 1024, w.n_keep, w.d_h, gather=False)
    assert p["tensor_core"] and p["row_blocks"] >= 4
    sample = rows_to_check(ctx, w, "fp32")
    hit = {r // p["block_rows"] for r in sample}
    assert hit == set(range(p["row_blocks"]))
    assert len({(r % p["block_rows"]) // 16 for r in sample}) >= 4


# ---------------------------------------------------------------------------
# the paper's split-dimension study (Sec. "Sensitivity to Split Dimension"):
# D = 4096, V = 150000, 32 rows, language subsets of 40 % and 30 %, every
# d_l of its table; all rows compared
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("keep", [0.4, 0.3])
@pytest.mark.parametrize("d_l", [48, 96, 128, 256, 512])
def test_split_dimension_study_shapes(ctx, d_l, keep):
    w = wl.workload("dend", device=DEV, keep_frac=keep, d_l=d_l)
    assert (w.d, w.V, w.rows, w.n_keep) == (4096, 150000, 32, round(keep * 150000))
    check_cloud(ctx, w)
    # the endpoint on the oracle's own payload (an input both sides share)
    ref = oracle_cloud(w)
    check_endpoint(ctx, w, torch.from_numpy(ref["codes"]), torch.from_numpy(ref["row_scale"]))


# ---------------------------------------------------------------------------
# maximum sizes: the API's 2^20 rows, and a kept set past the fused
# sampler's 4096 chunks (4.19M ids), where the chunk statistics take their
# own pass
# ---------------------------------------------------------------------------

def test_max_rows(ctx):
    w = small(V=600, d=128, d_l=64, rows=1 << 20, n_keep=40, run_lo=4, run_hi=12, seed=1201)
    sample = [0, 1, 777_777, (1 << 20) - 1]
    check_cloud(ctx, w, rows=sample)
    pc, ps = wl.make_payload(w.rows, w.n_keep, seed=13, device=DEV)
    check_endpoint(ctx, w, pc, ps, rows=sample)


def test_kept_set_past_the_fused_sampler(ctx):
    n = 4096 * 1024 + 5000
    w = small(V=n + 7000, d=96, d_l=32, rows=4, n_keep=n, run_lo=200, run_hi=4000,
              seed=1202)
    check_cloud(ctx, w, rows=[0, 3])
    pc, ps = wl.make_payload(w.rows, w.n_keep, seed=14, device=DEV)
    check_endpoint(ctx, w, pc, ps)


# ---------------------------------------------------------------------------
# tensor-core kernel variants: pipeline k-block width x work schedule
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("block_k", [64, 128, 256])
@pytest.mark.parametrize("schedule", [1, 2])
@pytest.mark.parametrize("keep", [700, 2000])
def test_tensor_core_variants(ctx, block_k, schedule, keep):
    from paper_2607_13093_gb300 import sph
    ctx.set_option(sph.SPH_OPT_TC_MIN_ROWS, 1)
    ctx.set_option(sph.SPH_OPT_TC_BLOCK_K, block_k)
    ctx.set_option(sph.SPH_OPT_TC_SCHEDULE, schedule)
    try:
        # K = 1000 (not a multiple of any k-block), ragged vocabulary tail
        w = small(V=2000, d=1072, d_l=72, rows=24, n_keep=keep, seed=91 + block_k)
        check_cloud(ctx, w)
        ref = oracle_cloud(w)
        check_endpoint(ctx, w, torch.from_numpy(ref["codes"]),
                       torch.from_numpy(ref["row_scale"]))
    finally:
        ctx.set_option(sph.SPH_OPT_TC_MIN_ROWS, 4)
        ctx.set_option(sph.SPH_OPT_TC_BLOCK_K, 0)
        ctx.set_option(sph.SPH_OPT_TC_SCHEDULE, 0)


# ---------------------------------------------------------------------------
# the unsplit head (no payload, whole hidden state and head): the comparator
# of the paper's "no split projection" ablation
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("kw", [dict(V=4000, d=1024, d_l=128, rows=32, n_keep=1500, tau=0.8),
                                dict(V=3000, d=600, d_l=40, rows=3, n_keep=3000),
                                dict(V=6000, d=1088, d_l=64, rows=20, n_keep=2400, tau=0.0)])
def test_unsplit_head(path_ctx, kw):
    w = small(seed=611, **kw)
    W_full = torch.cat([w.W_l, w.W_h], dim=1).contiguous()
    z = torch.empty(w.rows, w.n_keep, device=DEV)
    tok = path_ctx.fuse_sample(None, None, w.h, W_full, keep_ids=w.keep_ids,
                               temperature=w.tau, seed=w.seed, offset=3, fused_logits_out=z)
    path_ctx.sync()
    ids = np_(w.keep_ids)
    ids = np.arange(w.V) if ids is None else ids
    zref = oracle.fuse(None, None, oracle.local_partial(np_(w.h), bits(W_full), ids))
    assert_close(np_(z), zref, "unsplit logits")
    if w.tau == 0:
        j, gap = oracle.greedy_rows(zref)
        ok = gap >= GREEDY_GAP
    else:
        j, margin = oracle.sample_rows(zref, w.tau, oracle.philox_uniform(w.seed, np.arange(w.rows), 0, 3))
        ok = margin >= MARGIN
    got = np_(tok)
    assert not ((got != ids[j]) & ok).any()


GUMBEL_GAP = 2e-4     # Gumbel-max: top-two key gap of the fp64 keys


@pytest.mark.parametrize("kw", [dict(V=4000, d=1024, d_l=128, rows=32, n_keep=1500, tau=0.8),
                                dict(V=3000, d=600, d_l=40, rows=3, n_keep=3000, tau=1.3),
                                dict(V=9000, d=900, d_l=96, rows=40, n_keep=4001, tau=0.5)])
def test_gumbel_sampler(path_ctx, kw):
    from paper_2607_13093_gb300 import sph
    w = small(seed=733, **kw)
    pc, ps = wl.make_payload(w.rows, w.n_keep, seed=9, device=DEV)
    z = torch.empty(w.rows, w.n_keep, device=DEV)
    path_ctx.set_option(sph.SPH_OPT_SAMPLER, sph.SPH_SAMPLER_GUMBEL)
    try:
        tok = path_ctx.fuse_sample(pc, ps, w.h_local, w.W_l, keep_ids=w.keep_ids,
                                   temperature=w.tau, seed=w.seed, offset=11, fused_logits_out=z)
        path_ctx.sync()
    finally:
        path_ctx.set_option(sph.SPH_OPT_SAMPLER, sph.SPH_SAMPLER_CDF)
    ids = np_(w.keep_ids)
    ids = np.arange(w.V) if ids is None else ids
    zref = oracle.fuse(np_(pc), np_(ps), oracle.local_partial(np_(w.h_local), bits(w.W_l), ids))
    assert_close(np_(z), zref, "fused logits")
    u = oracle.gumbel_uniforms(w.seed, w.rows, w.n_keep, 11)
    j, gap = oracle.gumbel_rows(zref, w.tau, u)
    got = np_(tok)
    bad = (got != ids[j]) & (gap >= GUMBEL_GAP)
    assert not bad.any(), f"rows {np.nonzero(bad)[0]}: {got[bad]} vs {ids[j][bad]}"


def test_payload_arguments_together(ctx):
    from paper_2607_13093_gb300 import sph
    w = small(V=2000, d=512, d_l=64, rows=4, n_keep=800)
    with pytest.raises(sph.SphError):
        ctx.fuse_sample(None, torch.ones(w.rows, device=DEV), w.h_local, w.W_l,
                        keep_ids=w.keep_ids)


@pytest.mark.parametrize("schedule", [1, 2])
def test_tensor_core_256_tiles_one_accumulator(ctx, schedule):
    """256-id tiles over row blocks of more than 128 rows: one accumulator."""
    from paper_2607_13093_gb300 import sph
    ctx.set_option(sph.SPH_OPT_TC_MIN_ROWS, 1)
    ctx.set_option(sph.SPH_OPT_TC_TILE_M, 256)
    ctx.set_option(sph.SPH_OPT_TC_MAX_BN, 192)
    ctx.set_option(sph.SPH_OPT_TC_SCHEDULE, schedule)
    try:
        w = small(V=5000, d=1096, d_l=72, rows=300, n_keep=3100, seed=950 + schedule)
        check_cloud(ctx, w, rows=[0, 150, 299])
        ref = oracle_cloud(w)
        check_endpoint(ctx, w, torch.from_numpy(ref["codes"]),
                       torch.from_numpy(ref["row_scale"]), rows=[0, 150, 299])
    finally:
        ctx.set_option(sph.SPH_OPT_TC_MIN_ROWS, 4)
        ctx.set_option(sph.SPH_OPT_TC_TILE_M, 0)
        ctx.set_option(sph.SPH_OPT_TC_MAX_BN, 0)
        ctx.set_option(sph.SPH_OPT_TC_SCHEDULE, 0)


# ---------------------------------------------------------------------------
# split tiles: the designated finisher and the count-in fallback agree bit
# for bit (the partials are added in the same CTA order on both paths)
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("n_keep", [3000, 6000, 20000])
@pytest.mark.parametrize("rows", [24, 130])
def test_split_tile_finisher_matches_count_in(ctx, n_keep, rows):
    from paper_2607_13093_gb300 import sph
    w = small(V=24000, d=2000, d_l=1000, rows=rows, n_keep=n_keep, seed=500 + rows)
    ctx.set_option(sph.SPH_OPT_TC_MIN_ROWS, 1)
    ctx.set_option(sph.SPH_OPT_TC_SCHEDULE, 2)
    ctx.set_option(sph.SPH_OPT_TC_BLOCK_K, 64)
    outs = []
    try:
        for wait in (1 << 15, 0):
            ctx.set_option(sph.SPH_OPT_TC_FINISH_WAIT, wait)
            part = torch.empty(w.rows, w.n_keep, dtype=torch.float32, device=DEV)
            codes, scale, _ = ctx.partial_logits(w.h_cloud, w.W_h, keep_ids=w.keep_ids,
                                                 clip=w.clip, partial_out=part)
            z = torch.empty(w.rows, w.n_keep, dtype=torch.float32, device=DEV)
            tok = ctx.fuse_sample(codes, scale, w.h_local, w.W_l, keep_ids=w.keep_ids,
                                  temperature=w.tau, seed=w.seed, fused_logits_out=z)
            ctx.sync()
            outs.append((part, codes, scale, z, tok))
        for a, b in zip(*outs):
            assert torch.equal(a, b)
        # and the finisher's results are the oracle's
        ctx.set_option(sph.SPH_OPT_TC_FINISH_WAIT, 1 << 15)
        check_cloud(ctx, w, rows=sorted({0, rows // 2, rows - 1}))
    finally:
        ctx.set_option(sph.SPH_OPT_TC_FINISH_WAIT, 1 << 15)
        ctx.set_option(sph.SPH_OPT_TC_MIN_ROWS, 4)
        ctx.set_option(sph.SPH_OPT_TC_SCHEDULE, 0)
        ctx.set_option(sph.SPH_OPT_TC_BLOCK_K, 0)


# ---------------------------------------------------------------------------
# 256-id tensor-core tiles (two M = 128 MMAs per hidden-state stage)
# ---------------------------------------------------------------------------

TILE256_CASES = [
    # full vocabulary, K = 1000: one 2-D copy per (atom, tile half), ragged tail
    ("full-k1000", dict(V=3000, d=1072, d_l=72, rows=24, n_keep=3000)),
    # full vocabulary, K = 1024: one 3-D copy of all atoms per stage
    ("full-k1024", dict(V=3000, d=1096, d_l=72, rows=40, n_keep=3000)),
    # kept runs longer than 128 ids: two row boxes per run
    ("long-runs", dict(V=4000, d=1072, d_l=72, rows=24, n_keep=2000, run_lo=150, run_hi=400)),
    # isolated ids (one-row boxes) and two row blocks of 80 rows
    ("isolated", dict(V=2000, d=1072, d_l=72, rows=130, n_keep=700, run_lo=1, run_hi=3)),
]


@pytest.mark.parametrize("name,kw", TILE256_CASES, ids=[c[0] for c in TILE256_CASES])
@pytest.mark.parametrize("schedule", [1, 2])
@pytest.mark.parametrize("act", ["fp32", "bf16"])
def test_tensor_core_256_tiles(ctx, name, kw, schedule, act):
    from paper_2607_13093_gb300 import sph
    ctx.set_option(sph.SPH_OPT_TC_MIN_ROWS, 1)
    ctx.set_option(sph.SPH_OPT_TC_TILE_M, 256)
    ctx.set_option(sph.SPH_OPT_TC_SCHEDULE, schedule)
    try:
        w = small(seed=400 + len(name) + schedule, **kw)
        check_cloud(ctx, w, act_mode=act)
        if act == "fp32":
            ref = oracle_cloud(w)
            check_endpoint(ctx, w, torch.from_numpy(ref["codes"]),
                           torch.from_numpy(ref["row_scale"]))
    finally:
        ctx.set_option(sph.SPH_OPT_TC_MIN_ROWS, 4)
        ctx.set_option(sph.SPH_OPT_TC_TILE_M, 0)
        ctx.set_option(sph.SPH_OPT_TC_SCHEDULE, 0)


# ---------------------------------------------------------------------------
# fp8 (e4m3) weights on the tensor cores
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("rows,keep,act", [(16, 3000, "fp32"), (40, 1100, "fp32"),
                                           (200, 2000, "fp32"), (24, 900, "bf16"),
                                           (7, 3000, "fp32")])
def test_fp8_tensor_core(ctx, rows, keep, act):
    from paper_2607_13093_gb300 import sph
    ctx.set_option(sph.SPH_OPT_TC_MIN_ROWS, 1)
    try:
        # d_h = 1008: a ragged last 64-wide k-block
        w = small(V=3000, d=1048, d_l=40, rows=rows, n_keep=keep, w_dtype="fp8",
                  clip=40.0, seed=321 + rows, with_bias=(rows == 40))
        check_cloud(ctx, w, act_mode=act)
        if rows == 7:
            # d_h = 1000 inside a 1008-byte row stride: the last 16-byte
            # chunk of every row is only partly valid
            Wp = torch.zeros(w.V, 1008, dtype=torch.float8_e4m3fn, device=DEV)
            Wp.view(torch.uint8)[:, :1000] = w.W_h.view(torch.uint8)[:, :1000]
            Wp.view(torch.uint8)[:, 1000:] = 0x7E          # junk past the end (448)
            w.W_h = Wp[:, :1000]
            w.h = w.h[:, :w.d_l + 1000].contiguous()
            w.d = w.d_l + 1000
            check_cloud(ctx, w, act_mode=act)
    finally:
        ctx.set_option(sph.SPH_OPT_TC_MIN_ROWS, 4)


@pytest.mark.parametrize("schedule", [1, 2])
@pytest.mark.parametrize("tile_m", [128, 256])
@pytest.mark.parametrize("act", ["fp32", "bf16"])
def test_fp8_tile_heights(ctx, tile_m, act, schedule):
    """e4m3 weights with both tile heights and both schedules (whole tiles;
    stream-K split tiles), gathered and full vocabulary, K = 2048 (16 e4m3
    atoms), ragged vocabulary tails."""
    from paper_2607_13093_gb300 import sph
    ctx.set_option(sph.SPH_OPT_TC_MIN_ROWS, 1)
    ctx.set_option(sph.SPH_OPT_TC_TILE_M, tile_m)
    ctx.set_option(sph.SPH_OPT_TC_SCHEDULE, schedule)
    try:
        for keep in (2900, 3000):
            w = small(V=3000, d=2304, d_l=256, rows=150, n_keep=keep, w_dtype="fp8",
                      clip=40.0, seed=808 + keep)
            check_cloud(ctx, w, act_mode=act)
    finally:
        ctx.set_option(sph.SPH_OPT_TC_MIN_ROWS, 4)
        ctx.set_option(sph.SPH_OPT_TC_TILE_M, 0)
        ctx.set_option(sph.SPH_OPT_TC_SCHEDULE, 0)


# ---------------------------------------------------------------------------
# CUDA-graph capture (as the benchmark times the step) = direct calls
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("rows_kw", [dict(rows=20, sessions=4, k=4), dict(rows=3, sessions=1, k=2)])
def test_graph_capture_matches_direct_calls(ctx, rows_kw):
    w = small(V=6000, d=640, d_l=128, n_keep=2400, **rows_kw)
    ctx.reserve(w.rows, w.n_keep, max(w.d_h, w.d_l))
    target = wl.make_target_logits(w.rows, w.n_keep, seed=31, std=1.0).to(DEV)
    R, n, S = w.rows, w.n_keep, w.sessions
    codes = torch.empty(R, n, dtype=torch.int8, device=DEV)
    scale = torch.empty(R, device=DEV)
    tokens = torch.empty(R, dtype=torch.int32, device=DEV)
    z = torch.empty(R, n, device=DEV)
    n_acc = torch.empty(S, dtype=torch.int32, device=DEV)
    nxt = torch.empty(S, dtype=torch.int32, device=DEV)

    def step():
        ctx.partial_logits(w.h_cloud, w.W_h, keep_ids=w.keep_ids, clip=w.clip, codes=codes,
                           row_scale=scale)
        ctx.fuse_sample(codes, scale, w.h_local, w.W_l, keep_ids=w.keep_ids, temperature=w.tau,
                        seed=w.seed, offset=7, tokens=tokens, fused_logits_out=z)
        ctx.verify_draft(target, S, w.k, w.draft_tokens, keep_ids=w.keep_ids,
                         draft_probs=w.draft_probs, temperature=w.tau, seed=w.seed, offset=9,
                         n_accepted=n_acc, next_token=nxt)

    step()
    ctx.sync()
    ref = [t.clone() for t in (codes, scale, tokens, z, n_acc, nxt)]
    for t in (codes, scale, tokens, z, n_acc, nxt):
        t.zero_()
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    cs = torch.cuda.Stream(device=DEV)
    cs.wait_stream(torch.cuda.current_stream())
    with torch.cuda.graph(g, stream=cs):
        step()
    g.replay()
    g.replay()
    torch.cuda.synchronize()
    ctx.sync()
    for a, b in zip(ref, (codes, scale, tokens, z, n_acc, nxt)):
        assert torch.equal(a, b)


def test_tracing_times_each_call_class_once(ctx):
    # one cloud, one endpoint and one verification call under tracing: one
    # timed group per class with positive device time, and every kernel
    # counted; enabling again starts from zero
    S, k = 6, 2
    w = small(V=3000, d=1048, d_l=40, rows=S * (k + 1), n_keep=1301, sessions=S, k=k, tau=0.9)
    z = torch.empty(w.rows, w.n_keep, device=DEV)
    ctx.profile_enable(True)
    codes, scale, _ = ctx.partial_logits(w.h_cloud, w.W_h, keep_ids=w.keep_ids, clip=w.clip)
    ctx.fuse_sample(codes, scale, w.h_local, w.W_l, keep_ids=w.keep_ids, temperature=w.tau,
                    seed=w.seed, fused_logits_out=z)
    ctx.verify_draft(z, S, k, w.draft_tokens, keep_ids=w.keep_ids, draft_probs=w.draft_probs,
                     temperature=w.tau, seed=w.seed)
    p = ctx.profile_read()
    ctx.profile_enable(True)
    fresh = ctx.profile_read()
    ctx.profile_enable(False)
    for c in ("cloud_gemm", "quantize", "local_gemm", "sample", "verify"):
        assert p["calls"][c] == 1 and p["ms"][c] > 0, (c, p)
    assert p["launches"] >= 7          # split + contraction, quantize, endpoint, draw, verification
    assert fresh["launches"] == 0 and not any(fresh["calls"].values())


# ---------------------------------------------------------------------------
# CTA pairs (SPH_OPT_TC_PAIR): each 256-id tile one M = 256 MMA over two
# CTAs, each holding 128 ids and half of the hidden-state rows
# ---------------------------------------------------------------------------

PAIR_CASES = [
    ("decode-like", dict(V=4000, d=1024, d_l=128, rows=32, n_keep=1500)),
    ("full-vocab", dict(V=3000, d=1280, d_l=256, rows=48, n_keep=3000)),
    ("ragged-K", dict(V=2000, d=1072, d_l=72, rows=24, n_keep=700)),
    ("rows300", dict(V=3000, d=776, d_l=8, rows=300, n_keep=2000)),
    ("rows1000-bias", dict(V=6000, d=2112, d_l=64, rows=1000, n_keep=5000, with_bias=True)),
]


@pytest.mark.parametrize("name,kw", PAIR_CASES, ids=[c[0] for c in PAIR_CASES])
@pytest.mark.parametrize("schedule", [1, 2])
@pytest.mark.parametrize("act", ["fp32", "bf16"])
def test_tensor_core_pairs(ctx, name, kw, schedule, act):
    from paper_2607_13093_gb300 import sph
    ctx.set_option(sph.SPH_OPT_TC_MIN_ROWS, 1)
    ctx.set_option(sph.SPH_OPT_TC_PAIR, 1)
    ctx.set_option(sph.SPH_OPT_TC_SCHEDULE, schedule)
    try:
        w = small(seed=707, **kw)
        p = ctx.plan(0, w.rows, w.n_keep, w.d_h, gather=w.keep_ids is not None,
                     act_mode=sph.SPH_ACT_BF16 if act == "bf16" else sph.SPH_ACT_FP32)
        assert p["pair"] == 1 and p["grid"] % 2 == 0 and p["block_rows"] % 32 == 0
        check_cloud(ctx, w, act_mode=act)
        # the endpoint on pairs too (z stored and not)
        pe = ctx.plan(1, w.rows, w.n_keep, w.d_l, gather=w.keep_ids is not None)
        assert pe["pair"] == 1 and pe["grid"] % 2 == 0
        ref = oracle_cloud(w)
        check_endpoint(ctx, w, torch.from_numpy(ref["codes"]), torch.from_numpy(ref["row_scale"]))
    finally:
        ctx.set_option(sph.SPH_OPT_TC_PAIR, 0)
        ctx.set_option(sph.SPH_OPT_TC_SCHEDULE, 0)
        ctx.set_option(sph.SPH_OPT_TC_MIN_ROWS, 4)


@pytest.mark.parametrize("n_keep", [3000, 20000])
def test_tensor_core_pairs_split_tiles_without_finisher(ctx, n_keep):
    # stream-K split tiles finished by the last contributor to count in
    from paper_2607_13093_gb300 import sph
    ctx.set_option(sph.SPH_OPT_TC_PAIR, 1)
    ctx.set_option(sph.SPH_OPT_TC_SCHEDULE, 2)
    ctx.set_option(sph.SPH_OPT_TC_FINISH_WAIT, 0)
    try:
        w = small(V=n_keep + 4000, d=2112, d_l=64, rows=130, n_keep=n_keep, seed=708)
        check_cloud(ctx, w)
    finally:
        ctx.set_option(sph.SPH_OPT_TC_FINISH_WAIT, 1 << 15)
        ctx.set_option(sph.SPH_OPT_TC_SCHEDULE, 0)
        ctx.set_option(sph.SPH_OPT_TC_PAIR, 0)


def test_tensor_core_pairs_full_size_sweep(ctx):
    # the 1024-row sweep point in the pair plan, rows from every row block
    from paper_2607_13093_gb300 import sph
    ctx.set_option(sph.SPH_OPT_TC_PAIR, 1)
    try:
        w = wl.workload("sweep", device=DEV, rows=1024, keep_frac=1.0)
        sample = rows_to_check(ctx, w, "fp32")
        p = ctx.plan(0, 1024, w.n_keep, w.d_h, gather=False)
        assert p["pair"] == 1
        assert {r // p["block_rows"] for r in sample} == set(range(p["row_blocks"]))
        check_cloud(ctx, w, rows=sample)
    finally:
        ctx.set_option(sph.SPH_OPT_TC_PAIR, 0)


@pytest.mark.parametrize("rows,keep", [(40, 1100), (200, 3000), (256, 2500)])
@pytest.mark.parametrize("schedule", [1, 2])
@pytest.mark.parametrize("act", ["fp32", "bf16"])
def test_fp8_tensor_core_pairs(ctx, rows, keep, schedule, act):
    # e4m3 weights on CTA pairs (kind::f8f6f4, M = 256 over two CTAs);
    # d_h = 1008: a ragged last k-block
    from paper_2607_13093_gb300 import sph
    ctx.set_option(sph.SPH_OPT_TC_PAIR, 1)
    ctx.set_option(sph.SPH_OPT_TC_SCHEDULE, schedule)
    try:
        w = small(V=3000, d=1048, d_l=40, rows=rows, n_keep=keep, w_dtype="fp8", clip=40.0,
                  seed=331 + rows, with_bias=(rows == 40))
        p = ctx.plan(0, w.rows, w.n_keep, w.d_h, w_dtype=sph.SPH_DTYPE_FP8_E4M3,
                     gather=w.keep_ids is not None)
        assert p["pair"] == 1
        check_cloud(ctx, w, act_mode=act)
    finally:
        ctx.set_option(sph.SPH_OPT_TC_SCHEDULE, 0)
        ctx.set_option(sph.SPH_OPT_TC_PAIR, 0)


@pytest.mark.parametrize("n_keep", [2004, 3000, 3002, 3001])
@pytest.mark.parametrize("payload", [True, False])
def test_endpoint_transposed_epilogue(ctx, n_keep, payload):
    # row blocks of >= 128 rows over a short hidden dimension finish the
    # endpoint through shared memory when rows are 2-element aligned (2004:
    # 8-byte code loads on every other row, a ragged last window; 3000: all
    # 16-byte aligned; 3002: rows alternately 8- and 16-byte aligned, 2-byte
    # code loads; 3001: odd, the per-lane path)
    w = small(V=n_keep + 1500, d=1088, d_l=64, rows=160, n_keep=n_keep, seed=909)
    if payload:
        ref = oracle_cloud(w)
        check_endpoint(ctx, w, torch.from_numpy(ref["codes"]), torch.from_numpy(ref["row_scale"]))
    else:
        W_full = torch.cat([w.W_l, w.W_h], dim=1).contiguous()
        z = torch.empty(w.rows, w.n_keep, device=DEV)
        tok = ctx.fuse_sample(None, None, w.h, W_full, keep_ids=w.keep_ids, temperature=w.tau,
                              seed=w.seed, fused_logits_out=z)
        ctx.sync()
        zref = oracle.local_partial(np_(w.h), bits(W_full), np_(w.keep_ids))
        assert_close(np_(z), zref, "unsplit fused logits")
        assert np.isin(np_(tok), np_(w.keep_ids)).all()


# ---------------------------------------------------------------------------
# the endpoint without a stored z: the contraction's epilogue keeps the
# 32-id segment statistics and the draw recomputes z for the segment it
# lands in (SPH_OPT_ENDPOINT_Z = 2)
# ---------------------------------------------------------------------------

UNSTORED = [
    # name, workload, extra elements per W_l row (a padded row stride)
    ("aligned", dict(V=6000, d=640, d_l=128, rows=40, n_keep=3000), 0),
    ("even", dict(V=6000, d=640, d_l=128, rows=40, n_keep=3002), 0),
    ("odd", dict(V=6000, d=640, d_l=128, rows=40, n_keep=3001), 0),
    ("short", dict(V=500, d=136, d_l=16, rows=9, n_keep=7, run_lo=1, run_hi=3), 0),
    ("k-tail", dict(V=3000, d=302, d_l=44, rows=20, n_keep=1111), 4),
    ("row-blocks", dict(V=30000, d=640, d_l=64, rows=300, n_keep=20000), 0),
    ("full-vocab", dict(V=3000, d=1280, d_l=264, rows=16, n_keep=3000), 0),
]


@pytest.mark.parametrize("tau", [0.8, 0.0])
@pytest.mark.parametrize("payload", [True, False])
@pytest.mark.parametrize("name,kw,pad", UNSTORED, ids=[c[0] for c in UNSTORED])
def test_endpoint_unstored_z(ctx, name, kw, pad, payload, tau):
    # tokens of the unstored path and of the stored one against the oracle
    # (margin rule), on rows whose hidden states are 8- or 16-byte aligned
    # ("k-tail": d = 302; a hidden dimension of 44 = 5 x 8 + 4 over a padded
    # weight row stride)
    from paper_2607_13093_gb300 import sph
    from _parity import fuse_sample_unstored
    w = small(seed=1301, tau=tau, **kw)
    W_l = w.W_l
    if pad:
        buf = torch.zeros(w.V, w.d_l + pad, dtype=torch.bfloat16, device=DEV)
        buf[:, :w.d_l] = w.W_l
        W_l = buf[:, :w.d_l]
    pc, ps = wl.make_payload(w.rows, w.n_keep, seed=21, device=DEV) if payload else (None, None)
    ids = np_(w.keep_ids)
    vocab = np.arange(w.V) if ids is None else ids
    zref = oracle.fuse(np_(pc), np_(ps), oracle.local_partial(np_(w.h_local), bits(w.W_l), vocab))
    ctx.set_option(sph.SPH_OPT_TC_MIN_ROWS, 1)
    try:
        for off in (0, 5):
            z = torch.empty(w.rows, w.n_keep, device=DEV)
            t1 = ctx.fuse_sample(pc, ps, w.h_local, W_l, keep_ids=w.keep_ids, temperature=tau,
                                 seed=w.seed, offset=off, fused_logits_out=z)
            t2 = fuse_sample_unstored(ctx, pc, ps, w.h_local, W_l, keep_ids=w.keep_ids,
                                      temperature=tau, seed=w.seed, offset=off)
            ctx.sync()
            assert_close(np_(z), zref, "fused logits")
            if tau == 0:
                j, gap = oracle.greedy_rows(zref)
                ok = gap >= GREEDY_GAP
            else:
                u = oracle.philox_uniform(w.seed, np.arange(w.rows), 0, off)
                j, margin = oracle.sample_rows(zref, tau, u)
                ok = margin >= MARGIN
            assert ok.mean() > 0.5
            for t, what in ((t1, "stored"), (t2, "unstored")):
                got = np_(t)
                bad = (got != vocab[j]) & ok
                assert not bad.any(), f"{what}: rows {np.nonzero(bad)[0]}"
                assert np.isin(got, vocab).all()
    finally:
        ctx.set_option(sph.SPH_OPT_TC_MIN_ROWS, 4)


def test_endpoint_z_option_values(ctx):
    from paper_2607_13093_gb300 import sph
    for v in (0, 1, 2):
        ctx.set_option(sph.SPH_OPT_ENDPOINT_Z, v)
    for v in (-1, 3):
        with pytest.raises(sph.SphError):
            ctx.set_option(sph.SPH_OPT_ENDPOINT_Z, v)
    ctx.set_option(sph.SPH_OPT_ENDPOINT_Z, 0)


# ---------------------------------------------------------------------------
# the endpoint on CTA pairs with the hidden-state rows as the MMA's M
# (SPH_OPT_ENDPOINT_ROWS_M = 1): 256-row blocks, a lane per row, the
# segment statistics from the epilogue
# ---------------------------------------------------------------------------

ROWS_M = [
    ("few-rows", dict(V=4000, d=1024, d_l=128, rows=40, n_keep=1500, tau=0.8)),
    ("ragged-n", dict(V=6000, d=640, d_l=64, rows=300, n_keep=3001)),
    ("even-n", dict(V=6000, d=640, d_l=64, rows=256, n_keep=2002)),
    ("aligned", dict(V=9000, d=600, d_l=72, rows=520, n_keep=4096)),
    ("full-vocab", dict(V=3000, d=1280, d_l=256, rows=200, n_keep=3000)),
    ("short", dict(V=500, d=136, d_l=16, rows=33, n_keep=7, run_lo=1, run_hi=3)),
    ("greedy", dict(V=5000, d=768, d_l=128, rows=260, n_keep=2500, tau=0.0)),
]


@pytest.mark.parametrize("payload", [True, False])
@pytest.mark.parametrize("name,kw", ROWS_M, ids=[c[0] for c in ROWS_M])
def test_endpoint_rows_as_m(ctx, name, kw, payload):
    from paper_2607_13093_gb300 import sph
    ctx.set_option(sph.SPH_OPT_TC_MIN_ROWS, 1)
    ctx.set_option(sph.SPH_OPT_TC_PAIR, 1)
    ctx.set_option(sph.SPH_OPT_ENDPOINT_ROWS_M, 1)
    try:
        w = small(seed=1401, **kw)
        pe = ctx.plan(1, w.rows, w.n_keep, w.d_l, gather=w.keep_ids is not None)
        assert pe["pair"] == 1 and pe["rows_m"] == 1 and pe["block_rows"] == 256
        assert pe["epilogue_stats"] == 1
        if payload:
            pc, ps = wl.make_payload(w.rows, w.n_keep, seed=31)
        else:
            pc = ps = None
        if payload:
            check_endpoint(ctx, w, pc, ps)
        else:
            # no payload: z is the local partial alone
            from _parity import fuse_sample_unstored
            z = torch.empty(w.rows, w.n_keep, device=DEV)
            t1 = ctx.fuse_sample(None, None, w.h_local, w.W_l, keep_ids=w.keep_ids,
                                 temperature=w.tau, seed=w.seed, fused_logits_out=z)
            t2 = fuse_sample_unstored(ctx, None, None, w.h_local, w.W_l, keep_ids=w.keep_ids,
                                      temperature=w.tau, seed=w.seed)
            ctx.sync()
            ids = np_(w.keep_ids)
            vocab = np.arange(w.V) if ids is None else ids
            zref = oracle.local_partial(np_(w.h_local), bits(w.W_l), vocab)
            assert_close(np_(z), zref, "local partial logits")
            if w.tau == 0:
                j, gap = oracle.greedy_rows(zref)
                ok = gap >= GREEDY_GAP
            else:
                j, margin = oracle.sample_rows(
                    zref, w.tau, oracle.philox_uniform(w.seed, np.arange(w.rows), 0, 0))
                ok = margin >= MARGIN
            for t in (t1, t2):
                assert not ((np_(t) != vocab[j]) & ok).any()
    finally:
        ctx.set_option(sph.SPH_OPT_ENDPOINT_ROWS_M, 0)
        ctx.set_option(sph.SPH_OPT_TC_PAIR, 0)
        ctx.set_option(sph.SPH_OPT_TC_MIN_ROWS, 4)


def test_endpoint_rows_as_m_option_values(ctx):
    from paper_2607_13093_gb300 import sph
    for v in (0, 1, 2):
        ctx.set_option(sph.SPH_OPT_ENDPOINT_ROWS_M, v)
    for v in (-1, 3):
        with pytest.raises(sph.SphError):
            ctx.set_option(sph.SPH_OPT_ENDPOINT_ROWS_M, v)
    ctx.set_option(sph.SPH_OPT_ENDPOINT_ROWS_M, 0)
    # stream-K schedules keep the transposed (ids as M) endpoint
    ctx.set_option(sph.SPH_OPT_TC_SCHEDULE, 2)
    try:
        assert ctx.plan(1, 1024, 256000, 512, gather=False)["rows_m"] == 0
    finally:
        ctx.set_option(sph.SPH_OPT_TC_SCHEDULE, 0)
    assert ctx.plan(1, 1024, 256000, 512, gather=False)["rows_m"] == 1
