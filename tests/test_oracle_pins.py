"""Pins of the CPU oracle against what the paper and mathematics fix.

None of these re-type the oracle's formulas: each compares the oracle with a
brute-force definition on a tiny case, a library routine (torch's number
format conversions, scipy's softmax, Triton's Philox), a closed form, an
invariant, or a value printed in the paper (tests/golden/).
"""
import itertools
import json
import os
import subprocess
import sys
import textwrap

import numpy as np
import pytest
import torch

import oracle
from paper_2607_13093_gb300 import workloads as wl

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def bits16(t):
    return t.contiguous().view(torch.int16).numpy().view(np.uint16)


def bits8(t):
    return t.contiguous().view(torch.uint8).numpy()


def tiny(with_bias=True, w_dtype="bf16", seed=7, V=37, d=13, d_l=5, rows=3,
         n_keep=20, sessions=0, k=0):
    return wl.make_workload(V=V, d=d, d_l=d_l, rows=rows, n_keep=n_keep,
                            seed=seed, with_bias=with_bias, w_dtype=w_dtype,
                            run_lo=2, run_hi=5, sessions=sessions, k=k)


# ---------------------------------------------------------------------------
# Eq. 9-13: split partial logits add up to the full head, bias once
# ---------------------------------------------------------------------------

def brute_full_head(h, W_full, bias):
    """z[r, v] = sum_c h[r, c] W[v, c] + b[v] with explicit loops (Eq. 9)."""
    R, d = h.shape
    V = W_full.shape[0]
    z = np.zeros((R, V))
    for r in range(R):
        for v in range(V):
            acc = 0.0
            for c in range(d):
                acc += float(h[r, c]) * float(W_full[v, c])
            z[r, v] = acc + (float(bias[v]) if bias is not None else 0.0)
    return z


@pytest.mark.parametrize("act_mode", ["fp32", "bf16"])
def test_split_partials_equal_full_head(act_mode):
    w = tiny()
    ids = w.keep_ids.numpy()
    h = w.h.numpy().astype(np.float64)
    if act_mode == "bf16":
        # the cloud half sees h rounded to bf16 (torch's conversion)
        h[:, w.d_l:] = w.h[:, w.d_l:].to(torch.bfloat16).double().numpy()
    W_full = torch.cat([w.W_l, w.W_h], dim=1).double().numpy()
    z_full = brute_full_head(h, W_full, w.bias.numpy())[:, ids]
    cloud = oracle.partial_logits(w.h_cloud.numpy(), bits16(w.W_h),
                                  bias=w.bias.numpy(), keep_ids=ids,
                                  clip=1e30, act_mode=act_mode)
    local = oracle.local_partial(w.h_local.numpy(), bits16(w.W_l), ids)
    np.testing.assert_allclose(cloud["y"] + local, z_full, rtol=1e-12, atol=1e-14)
    # the bias enters exactly once: without it the sum drops by b[ids]
    cloud0 = oracle.partial_logits(w.h_cloud.numpy(), bits16(w.W_h),
                                   keep_ids=ids, clip=1e30, act_mode=act_mode)
    np.testing.assert_allclose(cloud0["y"] + local + w.bias.numpy()[ids],
                               z_full, rtol=1e-12, atol=1e-14)


def test_unsplit_endpoint_call_is_full_head():
    """Without a payload the endpoint call over the whole hidden state and
    head computes the unsplit head (Eq. 9) -- the comparator of the paper's
    "no split projection" ablation -- and samples from it."""
    w = tiny(with_bias=False)
    ids = w.keep_ids.numpy()
    h = w.h.numpy().astype(np.float64)
    W_full = torch.cat([w.W_l, w.W_h], dim=1)
    z_full = brute_full_head(h, W_full.double().numpy(), None)[:, ids]
    out = oracle.fuse_sample(None, None, w.h.numpy(), bits16(W_full.contiguous()),
                             keep_ids=ids, tau=1.0, seed=5, offset=2)
    np.testing.assert_allclose(out["z"], z_full, rtol=1e-12, atol=1e-14)
    u = oracle.philox_uniform(5, np.arange(w.rows), 0, 2)
    j, _ = oracle.sample_rows(z_full, 1.0, u)
    assert (out["tokens"] == ids[j]).all()


def test_fused_logits_within_dequantization_bound():
    """z = code * s + z_end reproduces the full head (Eq. 13) to within half
    a quantization step (Eq. 18) when nothing is clipped."""
    w = tiny(with_bias=False)
    ids = w.keep_ids.numpy()
    h = w.h.numpy().astype(np.float64)
    W_full = torch.cat([w.W_l, w.W_h], dim=1).double().numpy()
    z_full = brute_full_head(h, W_full, None)[:, ids]
    cloud = oracle.partial_logits(w.h_cloud.numpy(), bits16(w.W_h), keep_ids=ids,
                                  clip=1e30)
    zl = oracle.local_partial(w.h_local.numpy(), bits16(w.W_l), ids)
    z = oracle.fuse(cloud["codes"], cloud["row_scale"], zl)
    half = cloud["row_scale"].astype(np.float64)[:, None] / 2
    assert np.all(np.abs(z - z_full) <= half * (1 + 1e-9))
    assert np.any(np.abs(z - z_full) > half * 0.5)     # the bound is not slack


def test_fp8_partials_equal_full_head():
    w = tiny(with_bias=False, w_dtype="fp8")
    ids = w.keep_ids.numpy()
    Wh = (w.W_h.float().double() * w.w_scale.double()[:, None]).numpy()  # torch decode
    h = w.h.numpy().astype(np.float64)
    z_ref = brute_full_head(h[:, w.d_l:], Wh, None)[:, ids]
    cloud = oracle.partial_logits(w.h_cloud.numpy(), bits8(w.W_h), w_dtype="fp8",
                                  w_scale=w.w_scale.numpy(), keep_ids=ids,
                                  clip=1e30)
    np.testing.assert_allclose(cloud["y"], z_ref, rtol=1e-12, atol=1e-14)


def test_full_vocab_reduces_to_plain_matmul():
    """keep_ids=None (mixed-language mode) is the plain GEMM over all V."""
    w = tiny(with_bias=False, n_keep=37)
    assert w.keep_ids is None
    ref = w.h_cloud.double() @ w.W_h.double().T
    out = oracle.partial_logits(w.h_cloud.numpy(), bits16(w.W_h), clip=1e30)
    np.testing.assert_allclose(out["y"], ref.numpy(), rtol=1e-12)
    assert out["codes"].shape == (w.rows, w.V)


# ---------------------------------------------------------------------------
# Eq. 18 with b = 8: quantizer invariants and closed forms
# ---------------------------------------------------------------------------

def test_quantizer_closed_form():
    # s = 127/127 = 1 exactly; rint is half-to-even: -63.5 -> -64, 0.5 -> 0,
    # 1.5 -> 2, 2.5 -> 2
    y = np.array([[127.0, -63.5, 0.5, 1.5, 2.5, -127.0]])
    codes, s = oracle.quantize_rows(y, clip=1e9)
    assert s[0] == np.float32(1.0)
    assert codes.tolist() == [[127, -64, 0, 2, 2, -127]]
    # clipping happens before the row maximum: s = fl32(c/127)
    codes, s = oracle.quantize_rows(np.array([[100.0, -5.0, 29.0]]), clip=30.0)
    assert s[0] == np.float32(30.0 / 127.0)
    assert codes[0, 0] == 127
    # an all-zero row
    codes, s = oracle.quantize_rows(np.zeros((1, 5)), clip=30.0)
    assert s[0] == 0 and not codes.any()


def test_quantizer_invariants():
    rng = np.random.default_rng(3)
    y = rng.normal(size=(64, 301)) * rng.uniform(0.01, 60, size=(64, 1))
    y[5] = 0.0
    clip = 30.0
    codes, s = oracle.quantize_rows(y, clip)
    yc = np.clip(y, -clip, clip)
    s64 = s.astype(np.float64)
    assert codes.dtype == np.int8
    assert codes.min() >= -127 and codes.max() <= 127
    err = np.abs(codes * s64[:, None] - yc)
    assert np.all(err <= s64[:, None] / 2 * (1 + 1e-6) + 1e-300)
    nz = np.any(yc != 0, axis=1)
    assert np.all(np.abs(codes[nz]).max(axis=1) == 127)
    assert s[5] == 0 and not codes[5].any()
    # re-quantizing the dequantized payload reproduces it exactly
    codes2, s2 = oracle.quantize_rows(codes * s64[:, None], clip)
    assert np.array_equal(codes2, codes)
    np.testing.assert_allclose(s2, s, rtol=1e-6)


# ---------------------------------------------------------------------------
# Eq. 21 payload model against the numbers the paper prints
# ---------------------------------------------------------------------------

def test_payload_matches_paper():
    g = json.load(open(os.path.join(GOLDEN, "payload_eq21.json")))
    V = g["V"]
    code_bytes = oracle.payload_bytes(1, V) - 4          # minus the row scale
    assert code_bytes == V * g["b"] // 8
    assert round(code_bytes / 1024, 1) == g["full_logits_KB"]
    for row in g["rows"]:
        pct = 100 * (1 - row["downlink_KB"] / g["full_logits_KB"])
        assert abs(pct - row["compression_pct"]) < 0.051, row
        # the measured payload exceeds the bare clipped-logit bytes of the
        # kept fraction (tags, metadata and padding come on top)
        keep = g["keep_fractions"][row["mode"]]
        bare = (oracle.payload_bytes(1, round(keep * V)) - 4) / 1024
        assert bare < row["downlink_KB"] < bare + 10


# ---------------------------------------------------------------------------
# number formats against torch's conversions (exhaustive)
# ---------------------------------------------------------------------------

def test_bf16_decode_exhaustive():
    allbits = np.arange(65536, dtype=np.uint32).astype(np.uint16)
    ours = oracle.decode_bf16(allbits)
    ref = torch.from_numpy(allbits.view(np.int16)).view(torch.bfloat16).double().numpy()
    both_nan = np.isnan(ours) & np.isnan(ref)
    assert np.all(both_nan | (ours == ref))


def test_e4m3_decode_exhaustive():
    allbits = np.arange(256, dtype=np.uint8)
    ours = oracle.decode_e4m3(allbits)
    ref = torch.from_numpy(allbits).view(torch.float8_e4m3fn).double().numpy()
    both_nan = np.isnan(ours) & np.isnan(ref)
    assert np.all(both_nan | (ours == ref))
    assert np.nanmax(ours) == 448.0


def test_bf16_rounding_matches_torch():
    rng = np.random.default_rng(11)
    x = rng.normal(size=200000).astype(np.float32) * 10 ** rng.uniform(-6, 6, 200000).astype(np.float32)
    # exact ties: low 16 bits = 0x8000 with both parities of the kept lsb
    hi = rng.integers(0, 2 ** 15, 1000, dtype=np.uint32) << np.uint32(17)
    tb = (hi & np.uint32(0x00FE0000)) | np.uint32(0x3F000000)
    ties = np.concatenate([tb | np.uint32(0x8000), tb | np.uint32(0x18000)]).view(np.float32)
    x = np.concatenate([x, ties])
    assert np.all(np.isfinite(x))
    ours = oracle.round_fp32_to_bf16(x)
    ref = torch.from_numpy(x).to(torch.bfloat16).double().numpy()
    assert np.array_equal(ours, ref, equal_nan=True)


# ---------------------------------------------------------------------------
# Philox4x32-10 against an independent library implementation + statistics
# ---------------------------------------------------------------------------

_TRITON_PHILOX = textwrap.dedent("""
    import os, sys, json
    os.environ["TRITON_INTERPRET"] = "1"
    import numpy as np, torch, triton, triton.language as tl

    @triton.jit
    def k(seed, a, b, c, d, o0, o1, o2, o3, N: tl.constexpr):
        i = tl.arange(0, N)
        r0, r1, r2, r3 = tl.philox(seed, tl.load(a + i), tl.load(b + i),
                                   tl.load(c + i), tl.load(d + i), 10)
        tl.store(o0 + i, r0); tl.store(o1 + i, r1)
        tl.store(o2 + i, r2); tl.store(o3 + i, r3)

    spec = json.loads(sys.stdin.read())
    N = len(spec["c0"])
    cs = [torch.from_numpy(np.array(spec[n], dtype=np.uint32)) for n in ("c0","c1","c2","c3")]
    outs = [torch.empty(N, dtype=torch.uint32) for _ in range(4)]
    k[(1,)](spec["seed"], *cs, *outs, N=N)
    print(json.dumps([o.numpy().astype(np.int64).tolist() for o in outs]))
""")


def test_philox_known_answers():
    # the published known-answer outputs of Philox4x32-10
    # (tests/golden/philox4x32_10_kat.json)
    with open(os.path.join(GOLDEN, "philox4x32_10_kat.json")) as f:
        kat = json.load(f)
    for v in kat["vectors"]:
        c = [np.array([int(x, 16)], dtype=np.uint64) for x in v["counter"]]
        k0, k1 = (int(x, 16) for x in v["key"])
        out = oracle.philox4x32_10(*c, k0, k1)
        got = [int(np.asarray(o).ravel()[0]) for o in out]
        assert got == [int(x, 16) for x in v["output"]]


def test_philox_matches_triton_interpreter():
    pytest.importorskip("triton")
    rng = np.random.default_rng(5)
    N = 64
    c = [rng.integers(0, 2 ** 32, N, dtype=np.uint64) for _ in range(4)]
    c[0][:4] = [0, 1, 2, 0xFFFFFFFF]
    c[1][:4] = 0
    for seed in (0, 1234567, (0xDEADBEEF << 32) | 0x01234567):
        spec = dict(seed=seed, **{f"c{i}": c[i].tolist() for i in range(4)})
        res = subprocess.run([sys.executable, "-c", _TRITON_PHILOX],
                             input=json.dumps(spec), capture_output=True,
                             text=True, timeout=300)
        if res.returncode != 0:
            pytest.skip("triton interpreter unavailable: " + res.stderr[-300:])
        ref = json.loads(res.stdout.strip().splitlines()[-1])
        ours = oracle.philox4x32_10(*c, seed & 0xFFFFFFFF, seed >> 32)
        for w in range(4):
            assert np.array_equal(ours[w].astype(np.int64), np.array(ref[w])), (seed, w)


def test_philox_uniform_statistics():
    n = 1 << 20
    u = oracle.philox_uniform(99, np.arange(n), 0, 7)
    assert u.min() >= 0.0 and u.max() < 1.0
    # 24-bit grid: every value is an exact multiple of 2^-24
    assert np.all(u * 2 ** 24 == np.floor(u * 2 ** 24))
    hist = np.bincount((u * 256).astype(np.int64), minlength=256)
    chi2 = ((hist - n / 256) ** 2 / (n / 256)).sum()
    assert chi2 < 255 + 6 * np.sqrt(2 * 255)
    # neighbouring counters are uncorrelated; other purposes/offsets differ
    assert abs(np.corrcoef(u[:-1], u[1:])[0, 1]) < 5e-3
    u2 = oracle.philox_uniform(99, np.arange(n), 1, 7)
    u3 = oracle.philox_uniform(99, np.arange(n), 0, 8)
    assert abs(np.corrcoef(u, u2)[0, 1]) < 5e-3 and np.mean(u == u3) < 1e-3


# ---------------------------------------------------------------------------
# Eq. 14-15: masked softmax and the draw
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("tau", [0.5, 1.0, 2.0])
def test_sampling_distribution(tau):
    from scipy.special import softmax
    rng = np.random.default_rng(int(tau * 10))
    z = rng.normal(size=16) * 2
    P = softmax(z / tau)
    # stratified uniforms: the histogram must match P to within 1/G per bin
    G = 1 << 16
    u = (np.arange(G) + 0.5) / G
    idx, _ = oracle.sample_rows(np.broadcast_to(z, (G, 16)), tau, u)
    hist = np.bincount(idx, minlength=16) / G
    assert np.max(np.abs(hist - P)) <= 1.0 / G + 1e-12
    # Philox uniforms: chi-square goodness of fit
    n = 200000
    u = oracle.philox_uniform(3, np.arange(n), 0, int(tau * 100))
    idx, _ = oracle.sample_rows(np.broadcast_to(z, (n, 16)), tau, u)
    hist = np.bincount(idx, minlength=16)
    exp = P * n
    chi2 = ((hist - exp) ** 2 / exp).sum()
    assert chi2 < 15 + 6 * np.sqrt(30)


def test_small_temperature_is_argmax_and_edges():
    z = np.array([[0.1, 3.0, 2.999, -5.0]])
    for u in (0.0, 0.3, 0.999999):
        j, _ = oracle.sample_rows(z, 1e-5, [u])
        assert j[0] == 1
    # u = 0 draws the first id with nonzero probability; margins are >= 0
    P = np.array([0.0, 0.25, 0.75])
    assert oracle.inverse_cdf(P, 0.0)[0] == 1
    assert oracle.inverse_cdf(P, 0.25)[0] == 2
    j, m = oracle.inverse_cdf(P, 0.2)
    assert j == 1 and abs(m - 0.05) < 1e-15


def test_masked_ids_never_sampled():
    w = wl.make_workload(V=300, d=24, d_l=8, rows=4, n_keep=90, seed=21,
                         run_lo=3, run_hi=9)
    ids = w.keep_ids.numpy()
    cloud = oracle.partial_logits(w.h_cloud.numpy(), bits16(w.W_h), keep_ids=ids,
                                  clip=30.0)
    seen = set()
    for off in range(400):
        out = oracle.fuse_sample(cloud["codes"], cloud["row_scale"],
                                 w.h_local.numpy(), bits16(w.W_l), keep_ids=ids,
                                 tau=3.0, seed=w.seed, offset=off)
        seen.update(out["tokens"].tolist())
    assert seen <= set(ids.tolist())
    assert len(seen) > 30            # the draw does move around the subset


# ---------------------------------------------------------------------------
# speculative verification: exhaustive enumeration on a tiny vocabulary
# ---------------------------------------------------------------------------

def _rand_dist(rng, n, zero_some=False):
    p = rng.uniform(0.05, 1.0, size=n)
    if zero_some:
        p[rng.integers(0, n)] = 0.0
    return p / p.sum()


@pytest.mark.parametrize("n,seed", [(4, 0), (5, 1), (6, 2)])
def test_verify_preserves_target_k1(n, seed):
    """Standard speculative sampling emits its first token with exactly the
    target distribution p_0, whatever the draft distribution q_0."""
    rng = np.random.default_rng(seed)
    p = np.stack([_rand_dist(rng, n), _rand_dist(rng, n)])
    q = _rand_dist(rng, n, zero_some=True)[None, :]
    G = 1 << 10
    grid = (np.arange(G) + 0.5) / G
    dist = np.zeros(n)
    for x in range(n):
        if q[0, x] == 0:
            continue
        for r in grid:
            for u in grid[::8]:
                a, j, _, _ = oracle.verify_core(p, q, [x], [r], u)
                first = x if a >= 1 else j
                dist[first] += q[0, x] / (G * (G // 8))
    assert np.max(np.abs(dist - p[0])) < 4 * n / G


def test_verify_preserves_target_k2():
    """k = 2: the first token follows p_0 and, once x_0 is accepted, the
    second emitted token follows p_1."""
    rng = np.random.default_rng(9)
    n = 4
    p = np.stack([_rand_dist(rng, n) for _ in range(3)])
    q = np.stack([_rand_dist(rng, n) for _ in range(2)])
    G = 1 << 5
    grid = (np.arange(G) + 0.5) / G
    first = np.zeros(n)
    second = np.zeros(n)
    acc0 = 0.0
    for x0, x1 in itertools.product(range(n), range(n)):
        wq = q[0, x0] * q[1, x1]
        for r0, r1, u in itertools.product(grid, grid, grid):
            a, j, _, _ = oracle.verify_core(p, q, [x0, x1], [r0, r1], u)
            w = wq / G ** 3
            first[x0 if a >= 1 else j] += w
            if a >= 1:
                acc0 += w
                second[x1 if a >= 2 else j] += w
    assert np.max(np.abs(first - p[0])) < 6 * n / G
    assert np.max(np.abs(second / acc0 - p[1])) < 12 * n / G


def test_verify_greedy_is_one_hot_q_and_identical_drafts_accept():
    rng = np.random.default_rng(4)
    n, k = 5, 3
    p = np.stack([_rand_dist(rng, n) for _ in range(k + 1)])
    x = rng.integers(0, n, size=k)
    onehot = np.zeros((k, n))
    onehot[np.arange(k), x] = 1.0
    for _ in range(500):
        r = rng.uniform(size=k)
        u = rng.uniform()
        a1, j1, _, _ = oracle.verify_core(p, None, x, r, u)
        a2, j2, _, _ = oracle.verify_core(p, onehot, x, r, u)
        assert (a1, j1) == (a2, j2)
    # a draft that equals the target is always accepted (r < 1 = p/q)
    for _ in range(200):
        xs = rng.integers(0, n, size=k)
        a, _, _, _ = oracle.verify_core(p, p[:k], xs, rng.uniform(size=k), 0.5)
        assert a == k


def test_verify_draft_end_to_end_tiny():
    w = tiny(with_bias=False, V=60, d=16, d_l=4, rows=6, n_keep=25,
             sessions=2, k=2)
    ids = w.keep_ids.numpy()
    cloud = oracle.partial_logits(w.h_cloud.numpy(), bits16(w.W_h), keep_ids=ids,
                                  clip=30.0)
    z = oracle.fuse_sample(cloud["codes"], cloud["row_scale"], w.h_local.numpy(),
                           bits16(w.W_l), keep_ids=ids, tau=1.0,
                           seed=w.seed)["z"]
    out = oracle.verify_draft(z.astype(np.float32), 2, 2, keep_ids=ids, V=w.V,
                              tau=1.0, draft_tokens=w.draft_tokens.numpy(),
                              draft_probs=w.draft_probs.numpy(), seed=w.seed)
    assert set(out["next_token"].tolist()) <= set(ids.tolist())
    assert np.all((out["n_accepted"] >= 0) & (out["n_accepted"] <= 2))


def test_verify_draft_preserves_each_sessions_target_distribution():
    # End to end through verify_draft's own row, draft and uniform wiring:
    # drafts drawn from q (numpy's generator, independent of Philox), then
    # over many offsets the first emitted token of session s follows
    # softmax(z_{s,0} / tau), and after an accepted first draft the second
    # follows softmax(z_{s,1} / tau) -- the defining property of
    # speculative sampling.  Rows differ per session and position, ids are
    # a masked subset of V, so a wrong row, draft-probability or id mapping
    # shows up as a distribution mismatch.
    from scipy.stats import chisquare
    S, k, n, tau = 2, 2, 5, 0.7
    V = 9
    keep = np.array([0, 2, 3, 6, 8])
    g = np.random.default_rng(2024)
    Z = g.normal(0.0, 1.2, size=(S * (k + 1), n)).astype(np.float32)
    q = g.dirichlet(np.ones(n), size=(S, k))
    P = np.exp(Z.astype(np.float64) / tau)
    P /= P.sum(axis=1, keepdims=True)
    trials = 3000
    first = np.zeros((S, n))
    second = np.zeros((S, n))
    pos = {int(v): i for i, v in enumerate(keep)}
    for t in range(trials):
        x = np.array([[g.choice(n, p=q[s, i]) for i in range(k)] for s in range(S)])
        out = oracle.verify_draft(Z, S, k, keep_ids=keep, V=V, tau=tau,
                                  draft_tokens=keep[x], draft_probs=q, seed=11,
                                  offset=t)
        for s in range(S):
            a = int(out["n_accepted"][s])
            nxt = pos[int(out["next_token"][s])]
            first[s, x[s, 0] if a >= 1 else nxt] += 1
            if a >= 1:
                second[s, x[s, 1] if a >= 2 else nxt] += 1
    for s in range(S):
        assert chisquare(first[s], P[s * (k + 1)] * trials).pvalue > 1e-3
        m = second[s].sum()
        assert m > trials / 10
        assert chisquare(second[s], P[s * (k + 1) + 1] * m).pvalue > 1e-3


def test_compact_index_brute_force():
    ids = np.array([2, 3, 7, 11, 12])
    toks = np.array([0, 2, 3, 4, 7, 12, 13, 11, -1])
    exp = [next((i for i, v in enumerate(ids) if v == t), -1) for t in toks]
    assert oracle.compact_index(ids, 14, toks).tolist() == exp
    assert oracle.compact_index(None, 5, np.array([0, 4, 5, -1])).tolist() == [0, 4, -1, -1]


# ---------------------------------------------------------------------------
# greedy decoding (temperature 0)
# ---------------------------------------------------------------------------

def test_greedy_rows_first_maximum_by_brute_force():
    rng = np.random.default_rng(41)
    z = rng.integers(-3, 4, size=(200, 9)).astype(np.float64)   # many ties
    j, gap = oracle.greedy_rows(z)
    for r in range(z.shape[0]):
        m = max(z[r])
        first = min(i for i in range(z.shape[1]) if z[r, i] == m)
        assert j[r] == first
        rest = sorted(z[r])[-2]
        assert gap[r] == m - rest
    assert (gap[np.array([np.sum(z[r] == z[r].max()) > 1 for r in range(200)])] == 0).all()


def test_greedy_is_the_small_temperature_limit_of_sampling():
    # well separated maxima: softmax(z / tau) puts all mass on the argmax for
    # tiny tau, so every uniform draws it
    rng = np.random.default_rng(42)
    z = rng.normal(size=(50, 300)) * 3
    j, gap = oracle.greedy_rows(z)
    keep = gap > 0.05
    u = rng.random(50)
    js, _ = oracle.sample_rows(z, 1e-4, u)
    assert (js[keep] == j[keep]).all()


def test_fuse_sample_tau_zero_is_argmax_of_fused_logits():
    rng = np.random.default_rng(43)
    V, dl, R, n = 300, 12, 5, 120
    ids = np.sort(rng.choice(V, n, replace=False))
    W = rng.normal(size=(V, dl)) * 0.02
    Wb = (np.asarray(W, dtype=np.float32).view(np.uint32) >> 16).astype(np.uint16)
    codes = rng.integers(-127, 128, size=(R, n)).astype(np.int8)
    scale = (rng.random(R) * 0.2 + 0.01).astype(np.float32)
    h = rng.normal(size=(R, dl)).astype(np.float32)
    out = oracle.fuse_sample(codes, scale, h, Wb, keep_ids=ids, tau=0)
    z = oracle.fuse(codes, scale, oracle.local_partial(h, Wb, ids))
    assert (out["tokens"] == ids[np.argmax(z, axis=1)]).all()


def test_greedy_verify_matches_its_closed_form_and_the_small_tau_limit():
    rng = np.random.default_rng(44)
    S, k, n = 40, 3, 50
    Z = (rng.normal(size=(S * (k + 1), n)) * 4).astype(np.float32)
    a = np.argmax(Z.astype(np.float64), axis=1).reshape(S, k + 1)
    # drafts: the argmax for a random prefix, then something else
    drafts = np.empty((S, k), dtype=np.int64)
    for s in range(S):
        cut = rng.integers(0, k + 1)
        for i in range(k):
            drafts[s, i] = a[s, i] if i < cut else (a[s, i] + 1 + rng.integers(0, n - 1)) % n
    out = oracle.verify_draft(Z, S, k, tau=0, draft_tokens=drafts, draft_probs=None)
    for s in range(S):
        i = 0
        while i < k and drafts[s, i] == a[s, i]:
            i += 1
        assert out["n_accepted"][s] == i
        assert out["next_token"][s] == a[s, i]
        # the stochastic rule at a tiny temperature reaches the same result
        # (greedy one-hot drafts; p is one-hot up to exp(-gap / tau))
        P = oracle.softmax_rows(Z[s * (k + 1):(s + 1) * (k + 1)].astype(np.float64), 1e-3)
        acc, j, _, _ = oracle.verify_core(P, None, drafts[s], np.full(k, 0.5), 0.5)
        gaps = oracle.greedy_rows(Z[s * (k + 1):(s + 1) * (k + 1)])[1]
        if gaps.min() > 0.05:
            assert acc == i and j == a[s, i]


# ---------------------------------------------------------------------------
# Gumbel-max sampling (the alternative single-pass sampler)
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("tau", [0.7, 1.0, 2.0])
def test_gumbel_max_draws_follow_softmax(tau):
    """argmax(z/tau + Gumbel noise) is a draw from softmax(z/tau): a chi-square
    test over 60000 independent rows of the same logits."""
    z0 = np.array([0.3, -1.2, 2.0, 0.0, 1.1, -0.4])
    N, n = 60000, z0.size
    u = oracle.gumbel_uniforms(seed=77, rows=N, n=n, offset=5)
    j, _ = oracle.gumbel_rows(np.tile(z0, (N, 1)), tau, u)
    counts = np.bincount(j, minlength=n)
    p = np.exp(z0 / tau) / np.exp(z0 / tau).sum()
    chi2 = ((counts - N * p) ** 2 / (N * p)).sum()
    assert chi2 < 25.7          # df = 5, upper tail 1e-4


def test_gumbel_uniforms_are_strictly_inside_the_unit_interval():
    u = oracle.gumbel_uniforms(seed=3, rows=64, n=4099, offset=2 ** 40 + 7)
    assert u.min() > 0.0 and u.max() < 1.0
    # 23 random bits per value, on the grid (k + 1/2) 2^-23
    k = u * 2.0 ** 23 - 0.5
    assert np.all(k == np.round(k))
    # indices 4q .. 4q+3 use the four words of one Philox block
    w = oracle.philox4x32_10(np.uint64(5), np.uint64(oracle.GUMBEL_TAG | 1), np.uint64(2 ** 40 + 7 & 0xFFFFFFFF),
                             np.uint64((2 ** 40 + 7) >> 32), 3, 0)
    assert [int(x) >> 9 for x in w] == [int(v) for v in k[5, 4:8]]


def test_gumbel_max_small_temperature_is_greedy():
    rng = np.random.default_rng(4)
    z = rng.normal(size=(16, 300))
    u = oracle.gumbel_uniforms(seed=1, rows=16, n=300, offset=0)
    j, _ = oracle.gumbel_rows(z, 1e-9, u)
    g, gap = oracle.greedy_rows(z)
    assert (gap > 1e-6).all() and (j == g).all()


# ---------------------------------------------------------------------------
# block streaming of the payload (Eq. 3 blocks, Eq. 18 per block, Eq. 21):
# a chunked quantizer, its payload count, fusion, and the whole split step
# ---------------------------------------------------------------------------

def test_one_chunk_is_the_row_quantizer():
    rng = np.random.default_rng(11)
    y = rng.normal(size=(7, 533)) * 20.0
    codes, s = oracle.quantize_rows(y, 30.0)
    for chunk in (0, 533, 534, 10 ** 6):
        c2, s2 = oracle.quantize_chunks(y, 30.0, chunk)
        assert np.array_equal(c2, codes) and s2.shape == (1, 7)
        assert np.array_equal(s2[0], s)
        assert oracle.payload_bytes_chunked(7, 533, chunk) == oracle.payload_bytes(7, 533)


def test_chunk_bounds_cover_the_ids_in_order():
    assert oracle.chunk_bounds(10, 4) == [(0, 4), (4, 8), (8, 10)]
    assert oracle.chunk_bounds(8, 4) == [(0, 4), (4, 8)]
    assert oracle.chunk_bounds(5, 0) == [(0, 5)]
    for n, L in ((1, 1), (1000, 7), (1024, 256), (150000, 37500)):
        b = oracle.chunk_bounds(n, L)
        assert b[0][0] == 0 and b[-1][1] == n
        assert all(b[i][1] == b[i + 1][0] for i in range(len(b) - 1))
        assert all(j1 - j0 == L for j0, j1 in b[:-1]) and 0 < b[-1][1] - b[-1][0] <= L


def test_chunked_quantizer_closed_form():
    # chunk q's largest |entry| is 127 * 2^-q exactly, so its scale is 2^-q
    # and every entry of the form m * 2^-q quantizes to m; the all-zero
    # chunk has scale 0 and codes 0
    L = 5
    y = np.zeros((1, 4 * L))
    ms = np.array([127, -3, 64, 0, 5])
    for q in range(3):
        y[0, q * L:(q + 1) * L] = ms * 2.0 ** -q
    codes, s = oracle.quantize_chunks(y, 1e9, L)
    assert s[:, 0].tolist() == [1.0, 0.5, 0.25, 0.0]
    for q in range(3):
        assert codes[0, q * L:(q + 1) * L].tolist() == ms.tolist()
    assert not codes[0, 3 * L:].any()
    assert oracle.payload_bytes_chunked(1, 4 * L, L) == 4 * L + 16


def test_chunked_quantizer_invariants():
    # every chunk obeys the row quantizer's invariants with its own scale;
    # the chunk scales never exceed the row scale and their maximum is it,
    # so the chunked payload is never coarser than one scale per row
    rng = np.random.default_rng(12)
    R, n, L, clip = 9, 1000, 128, 30.0
    y = rng.normal(size=(R, n)) * rng.uniform(0.01, 60, size=(1, n))
    y[2, 256:384] = 0.0
    codes, s = oracle.quantize_chunks(y, clip, L)
    _, s_row = oracle.quantize_rows(y, clip)
    yc = np.clip(y, -clip, clip)
    b = oracle.chunk_bounds(n, L)
    assert s.shape == (len(b), R) and len(b) == 8
    for q, (j0, j1) in enumerate(b):
        sq = s[q].astype(np.float64)[:, None]
        err = np.abs(codes[:, j0:j1] * sq - yc[:, j0:j1])
        assert np.all(err <= sq / 2 * (1 + 1e-6) + 1e-300)
        nz = np.any(yc[:, j0:j1] != 0, axis=1)
        assert np.all(np.abs(codes[nz, j0:j1]).max(axis=1) == 127)
        assert np.all(s[q] <= s_row)
    assert s[2, 2] == 0 and not codes[2, 256:384].any()
    assert np.array_equal(s.max(axis=0), s_row)
    assert oracle.payload_bytes_chunked(R, n, L) == R * n + 4 * R * 8
    # the paper's CPU endpoint streams N_b = 4 blocks: 16 bytes of scales
    # per row on top of Eq. 21's one byte per kept logit
    assert oracle.payload_bytes_chunked(1, 150000, 37500) == 150000 + 16


def test_chunked_fusion_within_each_chunks_bound():
    """z from a chunked payload reproduces the full head (Eq. 13) to within
    half of each chunk's own quantization step, and that bound is tighter
    than one scale per row gives."""
    w = tiny(with_bias=False, V=60, n_keep=40, rows=4)
    ids = w.keep_ids.numpy()
    h = w.h.numpy().astype(np.float64)
    W_full = torch.cat([w.W_l, w.W_h], dim=1).double().numpy()
    z_full = brute_full_head(h, W_full, None)[:, ids]
    y = oracle.partial_logits(w.h_cloud.numpy(), bits16(w.W_h), keep_ids=ids, clip=1e30)["y"]
    L = 8
    codes, s = oracle.quantize_chunks(y, 1e30, L)
    zl = oracle.local_partial(w.h_local.numpy(), bits16(w.W_l), ids)
    z = oracle.fuse_chunks(codes, s, zl, L)
    for q, (j0, j1) in enumerate(oracle.chunk_bounds(40, L)):
        half = s[q].astype(np.float64)[:, None] / 2
        assert np.all(np.abs(z[:, j0:j1] - z_full[:, j0:j1]) <= half * (1 + 1e-9))
    _, s_row = oracle.quantize_rows(y, 1e30)
    assert np.any(s < s_row[None, :])


@pytest.mark.parametrize("chunk", [0, 8])
def test_split_step_chains_cloud_and_endpoint(chunk):
    # one chunk: exactly the cloud call followed by the endpoint call on its
    # payload; chunks: the fused logits stay within each chunk's bound of
    # the brute-force full head (Eq. 9) and the draw comes from them
    w = tiny(with_bias=True, V=60, n_keep=40, rows=5)
    ids = w.keep_ids.numpy()
    out = oracle.split_step(w.h.numpy(), w.d_l, bits16(w.W_h), bits16(w.W_l),
                            bias=w.bias.numpy(), keep_ids=ids, clip=1e30, tau=0.9,
                            seed=5, offset=3, chunk=chunk)
    if chunk == 0:
        c = oracle.partial_logits(w.h_cloud.numpy(), bits16(w.W_h), bias=w.bias.numpy(),
                                  keep_ids=ids, clip=1e30)
        e = oracle.fuse_sample(c["codes"], c["row_scale"], w.h_local.numpy(), bits16(w.W_l),
                               keep_ids=ids, tau=0.9, seed=5, offset=3)
        assert np.array_equal(out["codes"], c["codes"])
        assert np.array_equal(out["scales"][0], c["row_scale"])
        assert np.array_equal(out["draw"]["z"], e["z"])
        assert np.array_equal(out["draw"]["tokens"], e["tokens"])
        assert out["payload_bytes"] == c["payload_bytes"]
    h = w.h.numpy().astype(np.float64)
    W_full = torch.cat([w.W_l, w.W_h], dim=1).double().numpy()
    z_full = brute_full_head(h, W_full, w.bias.numpy())[:, ids]
    b = oracle.chunk_bounds(40, chunk)
    for q, (j0, j1) in enumerate(b):
        half = out["scales"][q].astype(np.float64)[:, None] / 2
        assert np.all(np.abs(out["draw"]["z"][:, j0:j1] - z_full[:, j0:j1]) <= half * (1 + 1e-9))
    assert out["payload_bytes"] == 5 * 40 + 4 * 5 * len(b)
    assert np.isin(out["draw"]["tokens"], ids).all()
