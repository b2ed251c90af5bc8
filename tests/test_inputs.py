"""The seeded input recipe shared by the oracle and the CUDA path: the
generators produce what the recipe states (no GPU needed).  These inputs stand
in for the paper's prompts, model and tokenizer subsets (Sec. "Experimental
Setup")."""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_13093_gb300 import workloads as wl


def runs_of(ids):
    """Maximal runs of consecutive ids: list of lengths."""
    breaks = np.nonzero(np.diff(ids) != 1)[0]
    edges = np.concatenate([[-1], breaks, [ids.size - 1]])
    return np.diff(edges)


@pytest.mark.parametrize("V,n", [(8192, 2048), (32000, 12000), (128256, 51302),
                                 (150000, 45000), (1000, 999), (500, 7), (64, 1)])
def test_keep_ids_are_sorted_unique_runs_with_the_exact_count(V, n):
    rng = np.random.default_rng(V + n)
    ids = wl.keep_id_runs(V, n, rng)
    assert ids.dtype == np.int32 and ids.size == n
    assert ids[0] >= 0 and ids[-1] < V
    assert np.all(np.diff(ids) > 0)
    lens = runs_of(ids.astype(np.int64))
    if (V - n) >= lens.size:            # room for separated runs
        assert lens.max() <= 256
        # every run but possibly one reaches the lower bound (the last run
        # absorbs the remainder only where the others have no slack)
        assert (lens < 16).sum() <= 1 or n < 16


def test_keep_ids_full_vocabulary_is_no_mask_and_bad_counts_raise():
    rng = np.random.default_rng(0)
    assert wl.keep_id_runs(100, 100, rng) is None
    for n in (0, 101):
        with pytest.raises(ValueError):
            wl.keep_id_runs(100, n, rng)


def test_keep_ids_are_seeded():
    a = wl.keep_id_runs(32000, 12000, np.random.default_rng(5))
    b = wl.keep_id_runs(32000, 12000, np.random.default_rng(5))
    c = wl.keep_id_runs(32000, 12000, np.random.default_rng(6))
    assert np.array_equal(a, b) and not np.array_equal(a, c)


def test_hidden_states_are_rms_normalised():
    h = wl.make_hidden(16, 4096, wl._gen("cpu", 3), "cpu").double()
    rms = torch.sqrt((h * h).mean(dim=1))
    assert torch.allclose(rms, torch.ones_like(rms), atol=1e-6)
    assert abs(float(h.mean())) < 0.02


def test_weights_are_bf16_normal_with_the_stated_spread():
    W = wl.make_weights(4096, 256, wl._gen("cpu", 4), "cpu")
    assert W.dtype == torch.bfloat16
    std = float(W.float().std())
    assert abs(std - 0.02) < 0.0005


def test_drafts_are_distributions_over_the_kept_ids():
    keep = torch.tensor([2, 3, 5, 7, 11, 13, 17], dtype=torch.int32)
    tok, q = wl.make_drafts(6, 3, keep.numel(), keep, 20, wl._gen("cpu", 9), "cpu")
    assert tok.shape == (6, 3) and q.shape == (6, 3, keep.numel())
    assert torch.allclose(q.double().sum(dim=2), torch.ones(6, 3, dtype=torch.float64),
                          atol=1e-5)
    assert set(tok.view(-1).tolist()) <= set(keep.tolist())


def test_e4m3_head_rows_decode_to_the_weights_within_e4m3_precision():
    W = wl.make_weights(300, 96, wl._gen("cpu", 8), "cpu")
    codes, scale = wl.to_e4m3_rows(W)
    dec = oracle.decode_e4m3(codes.view(torch.uint8).numpy()) * scale.numpy()[:, None]
    w = W.float().numpy()
    # e4m3 keeps 3 mantissa bits: relative error <= 2^-4 for normal codes,
    # absolute <= half the smallest subnormal step (2^-10 of the scale)
    tol = np.maximum(np.abs(w) * 2.0 ** -4, scale.numpy()[:, None] * 2.0 ** -10)
    assert np.all(np.abs(dec - w) <= tol)
    # each row's largest magnitude maps to the e4m3 maximum, 448
    assert np.allclose(np.abs(dec).max(axis=1), np.abs(w).max(axis=1), rtol=1e-6)


def test_named_workloads_follow_the_papers_setting():
    # the split-dimension study is the paper's own setup: D = 4096,
    # V = 150,000, D_end = 96, a 40 % language subset
    d = wl.WORKLOADS["dend"]
    assert (d["d"], d["V"], d["d_l"], d["n_keep"]) == (4096, 150000, 96, 60000)
    for name, cfg in wl.WORKLOADS.items():
        assert 1 <= cfg["d_l"] < cfg["d"], name
        assert 1 <= cfg["n_keep"] <= cfg["V"], name
        if "sessions" in cfg:
            assert cfg["rows"] == cfg["sessions"] * (cfg["k"] + 1), name
    assert wl.WORKLOADS["spec"]["n_keep"] == round(0.4 * 128256)
    assert [c["num"] for c in wl.WORKLOADS.values()] == list(range(1, len(wl.WORKLOADS) + 1))


def test_small_workloads_regenerate_identically():
    a = wl.make_workload(V=500, d=64, d_l=8, rows=6, n_keep=200, seed=77,
                         sessions=2, k=2)
    b = wl.make_workload(V=500, d=64, d_l=8, rows=6, n_keep=200, seed=77,
                         sessions=2, k=2)
    for x, y in ((a.h, b.h), (a.W_h, b.W_h), (a.keep_ids, b.keep_ids),
                 (a.draft_tokens, b.draft_tokens), (a.draft_probs, b.draft_probs)):
        assert torch.equal(x, y)
    assert a.seed == b.seed
