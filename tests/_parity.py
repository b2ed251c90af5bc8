"""Helpers shared by the GPU parity tests: run the CUDA path through the
C-ABI binding and the oracle on the same seeded inputs, and compare with the
tolerances of the method (fp32 partials within 1e-3 relative + 1e-3
absolute; int8 codes within 1 LSB on at most 0.1 % of entries; tokens and
accept decisions identical unless the oracle's margin is below 1e-5)."""
import numpy as np
import torch

import oracle

RTOL = 1e-3
ATOL = 1e-3
CODE_FRAC = 1e-3
MARGIN = 1e-5
GREEDY_GAP = 1e-4      # greedy decoding: top-two gap of the fp64 logits


def bits(t: torch.Tensor) -> np.ndarray:
    t = t.detach().contiguous().cpu()
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).numpy().view(np.uint16)
    if t.dtype == torch.float8_e4m3fn:
        return t.view(torch.uint8).numpy()
    raise TypeError(t.dtype)


def np_(t):
    return None if t is None else t.detach().cpu().numpy()


def assert_close(got, ref, what, rtol=RTOL, atol=ATOL):
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert got.shape == ref.shape, (what, got.shape, ref.shape)
    excess = np.abs(got - ref) - (atol + rtol * np.abs(ref))
    if excess.size and excess.max() > 0:
        i = np.unravel_index(np.argmax(excess), excess.shape)
        raise AssertionError(f"{what}: |{got[i]} - {ref[i]}| over tolerance at {i}")


def assert_codes(got, ref, what="codes"):
    d = np.abs(np.asarray(got, np.int64) - np.asarray(ref, np.int64))
    assert d.max(initial=0) <= 1, f"{what}: a code differs by {d.max()}"
    frac = (d > 0).mean() if d.size else 0.0
    assert frac <= CODE_FRAC, f"{what}: {frac:.2e} of codes differ"


def oracle_cloud(w, act_mode="fp32", rows=None):
    """Oracle cloud call on the workload (optionally a subset of rows)."""
    h = np_(w.h_cloud)
    if rows is not None:
        h = h[rows]
    return oracle.partial_logits(
        h, bits(w.W_h), w_dtype=w.w_dtype, w_scale=np_(w.w_scale),
        bias=np_(w.bias), keep_ids=np_(w.keep_ids), clip=w.clip,
        act_mode=act_mode)


def check_cloud(ctx, w, act_mode="fp32", rows=None):
    """GPU cloud call over all rows; compare (the sampled) rows with the
    oracle.  Returns the GPU outputs."""
    from paper_2607_13093_gb300 import sph
    dev = w.h.device
    part = torch.empty(w.rows, w.n_keep, device=dev)
    codes, scale, pb = ctx.partial_logits(
        w.h_cloud, w.W_h, keep_ids=w.keep_ids, clip=w.clip,
        w_row_scale=w.w_scale, bias=w.bias, partial_out=part,
        act_mode=sph.SPH_ACT_BF16 if act_mode == "bf16" else sph.SPH_ACT_FP32)
    ctx.sync()
    ref = oracle_cloud(w, act_mode, rows)
    sel = slice(None) if rows is None else rows
    assert_close(np_(part)[sel], ref["y"], "partial logits")
    assert_codes(np_(codes)[sel], ref["codes"])
    a_ref = ref["row_scale"].astype(np.float64) * 127.0
    assert_close(np_(scale)[sel].astype(np.float64) * 127.0, a_ref, "row absmax")
    assert pb == oracle.payload_bytes(w.rows, w.n_keep)
    return codes, scale, part


def fuse_sample_unstored(ctx, *a, **kw):
    """sph_fuse_sample without a z output and with z never stored
    (SPH_OPT_ENDPOINT_Z = 2: the draw recomputes the z it visits)."""
    from paper_2607_13093_gb300 import sph
    ctx.set_option(sph.SPH_OPT_ENDPOINT_Z, 2)
    try:
        return ctx.fuse_sample(*a, **kw)
    finally:
        ctx.set_option(sph.SPH_OPT_ENDPOINT_Z, 0)


def check_endpoint(ctx, w, codes, scale, rows=None, unstored=True):
    """GPU fuse+sample on a given payload (a host-side input shared with the
    oracle); compare fused logits and tokens (margin rule).  unstored: also
    draw without storing z (the tokens under the same rule)."""
    dev = w.h.device
    z = torch.empty(w.rows, w.n_keep, device=dev)
    tok = ctx.fuse_sample(codes.to(dev), scale.to(dev), w.h_local, w.W_l,
                          keep_ids=w.keep_ids, temperature=w.tau, seed=w.seed,
                          offset=w.offset, fused_logits_out=z)
    toks = [tok]
    if unstored:
        toks.append(fuse_sample_unstored(ctx, codes.to(dev), scale.to(dev), w.h_local, w.W_l,
                                         keep_ids=w.keep_ids, temperature=w.tau,
                                         seed=w.seed, offset=w.offset))
    ctx.sync()
    c = np_(codes)
    s = np_(scale)
    hl = np_(w.h_local)
    sel = np.arange(w.rows) if rows is None else np.asarray(rows)
    ids = np_(w.keep_ids)
    zl = oracle.local_partial(hl[sel], bits(w.W_l), ids)
    zref = oracle.fuse(c[sel], s[sel], zl)
    assert_close(np_(z)[sel], zref, "fused logits")
    if w.tau == 0:
        # greedy: identical unless the top-two gap of the exact logits is
        # within the fused logits' own rounding (GREEDY_GAP)
        j, gap = oracle.greedy_rows(zref)
        ok = gap >= GREEDY_GAP
    else:
        u = oracle.philox_uniform(w.seed, sel, 0, w.offset)
        j, margin = oracle.sample_rows(zref, w.tau, u)
        ok = margin >= MARGIN
    vocab = np.arange(w.V) if ids is None else ids
    want = vocab[j]
    for t, what in zip(toks, ("z stored", "z recomputed")):
        got = np_(t)[sel]
        bad = (got != want) & ok
        assert not bad.any(), f"tokens ({what}) differ at rows {sel[bad]}: {got[bad]} vs {want[bad]}"
        assert np.isin(np_(t), vocab).all(), f"a masked id was sampled ({what})"
    return tok, z


def check_verify(ctx, w, target, rows_sessions=None):
    """GPU verification on given fused target logits (fp32, host input)."""
    dev = w.h.device
    n_acc, nxt = ctx.verify_draft(target.to(dev), w.sessions, w.k, w.draft_tokens,
                                  keep_ids=w.keep_ids, draft_probs=w.draft_probs,
                                  temperature=w.tau, seed=w.seed, offset=w.offset)
    ctx.sync()
    ref = oracle.verify_draft(np_(target), w.sessions, w.k, keep_ids=np_(w.keep_ids),
                              V=w.V, tau=w.tau, draft_tokens=np_(w.draft_tokens),
                              draft_probs=np_(w.draft_probs), seed=w.seed,
                              offset=w.offset)
    a_ok = ref["accept_margin"] >= MARGIN
    bad_a = a_ok & (np_(n_acc) != ref["n_accepted"])
    assert not bad_a.any(), f"accept counts differ: {np_(n_acc)[bad_a]} vs {ref['n_accepted'][bad_a]}"
    t_ok = a_ok & (ref["draw_margin"] >= MARGIN)
    bad_t = t_ok & (np_(nxt) != ref["next_token"])
    assert not bad_t.any(), f"next tokens differ: {np_(nxt)[bad_t]} vs {ref['next_token'][bad_t]}"
    return n_acc, nxt, ref
