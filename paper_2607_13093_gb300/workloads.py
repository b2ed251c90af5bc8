"""Seeded synthetic inputs for the split-head vocabulary projection.

This module only *generates inputs*; it holds none of the method's arithmetic
(no partial logits, no clipping, no quantization of logits, no fusing, no
sampling rule, no acceptance rule).  Both the CUDA path's tests/benchmark and
the CPU oracle draw their inputs from here, so the two sides see identical
bytes.

Shapes follow the paper's setting (Sec. "Experimental Setup": a 7B-class
decoder, D=4096, V=150,000, language subsets keeping 40 % / 30 % / 100 % of
the vocabulary) and the five workloads used throughout this package:

  tiny      d=512  (d_l=64,   d_h=448),  V=8192,   R=1,    keep 2048 ids
  decode    d=4096 (d_l=256,  d_h=3840), V=32000,  R=32,   keep 12000 ids, tau 0.8
  spec      d=4096 (d_l=512,  d_h=3584), V=128256, S=64 sessions x (k=4 + 1)
  fp8       d=8192 (d_l=1024, d_h=7168), V=152064, R=256, full vocab, W_h e4m3
  sweep     d=5120 (d_l=512,  d_h=4608), V=256000, R in {1,8,64,256,1024},
            keep in {10 %, 50 %, 100 %}
  dend      d=4096 (d_l in {48, 96, 128, 256, 512}), V=150000, R=32,
            keep 40 % or 30 % (the paper's split-dimension study)

Input recipe (every workload):
  * W_lm is stored vocab-major, W[V, d] ~ N(0, 0.02) rounded to bf16 (RNE);
    W_l = W[:, :d_l], W_h = W[:, d_l:] (Eq. 10 splits the hidden dimension).
  * fp8 workload: per-vocab-row scale w_scale[v] = max_c |W_h[v,c]| / 448 and
    e4m3 = RNE(W_h / w_scale) (saturated to +-448) -- input preparation only.
  * h ~ N(0,1) fp32 over the full d, RMS-normalised over d (h / sqrt(mean h^2),
    no gain, no epsilon), computed in fp64 and stored fp32.
  * keep_ids: sorted unique int32 vocabulary ids laid out as seeded runs of
    length U{16..256} separated by seeded gaps, hitting n_keep exactly; a keep
    fraction of 100 % means "no mask" (keep_ids = None).
  * speculative drafts: per session and draft position, logits ~ N(0, std 2)
    over the kept ids, q = softmax(logits) stored fp32, draft token drawn from
    q; target rows are the fused logits of the S*(k+1) verification rows.
  * seeds: workload seed = 1000 + workload number (tiny=1 ... dend=6).
"""
from __future__ import annotations

import dataclasses
import math
from typing import Optional

import numpy as np
import torch

# ---------------------------------------------------------------------------
# workload table
# ---------------------------------------------------------------------------

WORKLOADS = {
    "tiny": dict(num=1, d=512, d_l=64, V=8192, rows=1, n_keep=2048, clip=30.0,
                 tau=1.0, w_dtype="bf16"),
    "decode": dict(num=2, d=4096, d_l=256, V=32000, rows=32, n_keep=12000,
                   clip=30.0, tau=0.8, w_dtype="bf16"),
    "spec": dict(num=3, d=4096, d_l=512, V=128256, sessions=64, k=4,
                 rows=320, n_keep=round(0.4 * 128256), clip=30.0, tau=1.0,
                 w_dtype="bf16"),
    "fp8": dict(num=4, d=8192, d_l=1024, V=152064, rows=256, n_keep=152064,
                clip=40.0, tau=1.0, w_dtype="fp8"),
    "sweep": dict(num=5, d=5120, d_l=512, V=256000, rows=64, n_keep=256000,
                  clip=30.0, tau=1.0, w_dtype="bf16"),
    "dend": dict(num=6, d=4096, d_l=96, V=150000, rows=32, n_keep=round(0.4 * 150000),
                 clip=30.0, tau=1.0, w_dtype="bf16"),
}
SWEEP_ROWS = (1, 8, 64, 256, 1024)
SWEEP_KEEP = (0.10, 0.50, 1.00)


@dataclasses.dataclass
class Workload:
    """All inputs of one split-head projection step (tensors on `device`)."""
    name: str
    V: int
    d: int
    d_l: int
    rows: int
    clip: float
    tau: float
    w_dtype: str                      # "bf16" | "fp8"
    h: torch.Tensor                   # fp32 [rows, d]; h_local = h[:, :d_l]
    W_l: torch.Tensor                 # bf16 [V, d_l]
    W_h: torch.Tensor                 # bf16 [V, d_h] or float8_e4m3fn [V, d_h]
    w_scale: Optional[torch.Tensor]   # fp32 [V] for fp8 W_h, else None
    bias: Optional[torch.Tensor]      # fp32 [V] or None
    keep_ids: Optional[torch.Tensor]  # int32 [n_keep] sorted, or None = full
    seed: int                         # Philox key for sampling
    offset: int                       # Philox counter offset (decode step)
    sessions: int = 0                 # speculative workloads only
    k: int = 0
    draft_tokens: Optional[torch.Tensor] = None   # int32 [S, k] vocab ids
    draft_probs: Optional[torch.Tensor] = None    # fp32 [S, k, n_keep]

    @property
    def d_h(self) -> int:
        return self.d - self.d_l

    @property
    def n_keep(self) -> int:
        return self.V if self.keep_ids is None else int(self.keep_ids.numel())

    @property
    def h_local(self) -> torch.Tensor:
        return self.h[:, : self.d_l]

    @property
    def h_cloud(self) -> torch.Tensor:
        return self.h[:, self.d_l:]


# ---------------------------------------------------------------------------
# building blocks
# ---------------------------------------------------------------------------

def keep_id_runs(V: int, n_keep: int, rng: np.random.Generator,
                 run_lo: int = 16, run_hi: int = 256) -> Optional[np.ndarray]:
    """Sorted unique ids in [0, V): seeded runs of U{run_lo..run_hi} kept ids
    separated by seeded gaps of >= 1 dropped id; exactly n_keep ids.
    Returns None when n_keep == V (no mask)."""
    if not 1 <= n_keep <= V:
        raise ValueError("need 1 <= n_keep <= V")
    if n_keep == V:
        return None
    lengths = []
    total = 0
    while total < n_keep:
        L = int(rng.integers(run_lo, run_hi + 1))
        lengths.append(L)
        total += L
    lengths[-1] -= total - n_keep
    # keep every run >= run_lo where the other runs have slack to give
    i = len(lengths) - 2
    while lengths[-1] < run_lo and i >= 0:
        give = min(run_lo - lengths[-1], lengths[i] - run_lo)
        if give > 0:
            lengths[i] -= give
            lengths[-1] += give
        i -= 1
    n_runs = len(lengths)
    gaps_total = V - n_keep
    interior = n_runs - 1
    if gaps_total < interior:           # too dense for separated runs
        ids = np.sort(rng.choice(V, size=n_keep, replace=False))
        return ids.astype(np.int32)
    rest = gaps_total - interior
    cuts = np.sort(rng.integers(0, rest + 1, size=n_runs))
    gaps = np.diff(np.concatenate([[0], cuts, [rest]]))
    gaps[1:-1] += 1
    ids = np.empty(n_keep, dtype=np.int64)
    pos = int(gaps[0])
    o = 0
    for r, L in enumerate(lengths):
        ids[o:o + L] = np.arange(pos, pos + L)
        o += L
        pos += L + int(gaps[r + 1])
    assert o == n_keep and ids[-1] < V
    return ids.astype(np.int32)


def _gen(device, seed: int) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    return g


def make_weights(V: int, d: int, g: torch.Generator, device,
                 std: float = 0.02, chunk_rows: int = 16384) -> torch.Tensor:
    """W[V, d] ~ N(0, std) rounded to bf16, generated in row chunks."""
    W = torch.empty(V, d, dtype=torch.bfloat16, device=device)
    for r0 in range(0, V, chunk_rows):
        r1 = min(V, r0 + chunk_rows)
        W[r0:r1] = (torch.randn(r1 - r0, d, generator=g, device=device,
                                dtype=torch.float32) * std).to(torch.bfloat16)
    return W


def to_e4m3_rows(W: torch.Tensor, chunk_rows: int = 16384):
    """Input preparation for the fp8 head: per-row scale amax/448 and the
    e4m3 codes of W/scale (torch's float8_e4m3fn conversion, saturated)."""
    V, dh = W.shape
    codes = torch.empty(V, dh, dtype=torch.float8_e4m3fn, device=W.device)
    scale = torch.empty(V, dtype=torch.float32, device=W.device)
    for r0 in range(0, V, chunk_rows):
        r1 = min(V, r0 + chunk_rows)
        w = W[r0:r1].float()
        amax = w.abs().amax(dim=1)
        s = torch.where(amax > 0, amax / 448.0, torch.ones_like(amax))
        scale[r0:r1] = s
        codes[r0:r1] = (w / s[:, None]).clamp(-448.0, 448.0).to(torch.float8_e4m3fn)
    return codes, scale


def make_hidden(rows: int, d: int, g: torch.Generator, device) -> torch.Tensor:
    """h ~ N(0,1) fp32, RMS-normalised over the full hidden dimension."""
    h = torch.randn(rows, d, generator=g, device=device, dtype=torch.float32)
    h64 = h.double()
    rms = torch.sqrt((h64 * h64).mean(dim=1, keepdim=True))
    rms = torch.where(rms > 0, rms, torch.ones_like(rms))
    return (h64 / rms).float().contiguous()


def make_drafts(sessions: int, k: int, n_keep: int, keep_ids, V: int,
                g: torch.Generator, device, std: float = 2.0):
    """Draft distributions q (softmax of N(0, std) logits over the kept ids)
    and draft tokens drawn from q; tokens are vocabulary ids."""
    logits = torch.randn(sessions * k, n_keep, generator=g, device=device,
                         dtype=torch.float32) * std
    q = torch.softmax(logits.double(), dim=1).float()
    idx = torch.multinomial(q, 1, generator=g).view(sessions, k)
    if keep_ids is None:
        tok = idx.to(torch.int32)
    else:
        tok = keep_ids.to(device).long()[idx].to(torch.int32)
    return tok.contiguous(), q.view(sessions, k, n_keep).contiguous()


# ---------------------------------------------------------------------------
# workloads
# ---------------------------------------------------------------------------

def make_workload(name: str = "custom", *, V: int, d: int, d_l: int, rows: int,
                  n_keep: int, clip: float = 30.0, tau: float = 1.0,
                  w_dtype: str = "bf16", seed: int = 1000, device="cpu",
                  sessions: int = 0, k: int = 0, with_bias: bool = False,
                  run_lo: int = 16, run_hi: int = 256,
                  offset: int = 0) -> Workload:
    """Generate one workload from explicit sizes (see the module docstring
    for the recipe).  `sessions`/`k` > 0 adds speculative drafts, in which
    case rows must equal sessions * (k + 1)."""
    if not 1 <= d_l < d:
        raise ValueError("need 1 <= d_l < d")
    if sessions:
        if rows != sessions * (k + 1):
            raise ValueError("speculative workload needs rows == S*(k+1)")
    rng = np.random.default_rng(seed)
    ids = keep_id_runs(V, n_keep, rng, run_lo, run_hi)
    keep = None if ids is None else torch.from_numpy(ids).to(device)
    g = _gen(device, seed)
    W = make_weights(V, d, g, device)
    W_l = W[:, :d_l].contiguous()
    W_h = W[:, d_l:].contiguous()
    del W
    w_scale = None
    if w_dtype == "fp8":
        W_h, w_scale = to_e4m3_rows(W_h)
    elif w_dtype != "bf16":
        raise ValueError(w_dtype)
    h = make_hidden(rows, d, g, device)
    bias = None
    if with_bias:
        bias = (torch.randn(V, generator=g, device=device,
                            dtype=torch.float32) * 0.5).contiguous()
    tok = probs = None
    if sessions:
        tok, probs = make_drafts(sessions, k, n_keep, keep, V, g, device)
    return Workload(name=name, V=V, d=d, d_l=d_l, rows=rows, clip=clip,
                    tau=tau, w_dtype=w_dtype, h=h, W_l=W_l, W_h=W_h,
                    w_scale=w_scale, bias=bias, keep_ids=keep,
                    seed=(seed * 2654435761) & 0xFFFFFFFFFFFFFFFF,
                    offset=offset, sessions=sessions, k=k,
                    draft_tokens=tok, draft_probs=probs)


def workload(name: str, device="cpu", rows: Optional[int] = None,
             keep_frac: Optional[float] = None, d_l: Optional[int] = None,
             V: Optional[int] = None) -> Workload:
    """One of the named workloads at full size.  For "sweep" and "dend",
    `rows` and `keep_frac` pick the grid point (defaults: sweep 64 rows,
    100 %; dend 32 rows, 40 %), and for "dend" `d_l` the split dimension
    (default 96, the paper's D_end).  `V` shrinks the vocabulary of "sweep"
    or "dend" (the kept fraction stays), for small profiling captures of the
    same kernel plan."""
    cfg = dict(WORKLOADS[name])
    num = cfg.pop("num")
    sessions = cfg.pop("sessions", 0)
    k = cfg.pop("k", 0)
    if name in ("sweep", "dend"):
        if V is not None:
            frac = cfg["n_keep"] / cfg["V"]
            cfg["V"] = int(V)
            cfg["n_keep"] = round(frac * cfg["V"])
        if rows is not None:
            cfg["rows"] = rows
        if keep_frac is not None:
            cfg["n_keep"] = round(keep_frac * cfg["V"])
    if name == "dend" and d_l is not None:
        cfg["d_l"] = d_l
    return make_workload(name, seed=1000 + num, device=device,
                         sessions=sessions, k=k, **cfg)


def algorithmic_bytes_cloud(R: int, n: int, d_h: int, w_bytes: int,
                            fp8_scales: bool = False, bias: bool = False,
                            partial_out: bool = False) -> int:
    """Bytes the cloud call must move at minimum: the kept W_h rows once,
    h_cloud, the id list, the int8 codes and the row scales."""
    b = n * d_h * w_bytes + 4 * R * d_h + 4 * n + R * n + 4 * R
    if fp8_scales:
        b += 4 * n
    if bias:
        b += 4 * n
    if partial_out:
        b += 4 * R * n
    return b


def algorithmic_bytes_endpoint(R: int, n: int, d_l: int) -> int:
    """Bytes of the endpoint fuse+sample call: kept W_l rows, h_local, codes,
    scales, ids and the sampled tokens."""
    return n * d_l * 2 + 4 * R * d_l + R * n + 4 * R + 4 * n + 4 * R


def algorithmic_flops(R: int, n: int, d: int) -> int:
    return 2 * R * n * d


def rows_per_second(rows: int, seconds: float) -> float:
    return rows / seconds if seconds > 0 else math.inf


def make_payload(rows: int, n: int, seed: int, device="cpu"):
    """A synthetic cloud payload (int8 codes in [-127, 127] and positive fp32
    row scales) for exercising the endpoint call on its own."""
    g = _gen(device, seed)
    codes = torch.randn(rows, n, generator=g, device=device) * 40.0
    codes = codes.round().clamp(-127, 127).to(torch.int8)
    scale = (torch.rand(rows, generator=g, device=device) * 0.05 + 0.01).float()
    return codes.contiguous(), scale.contiguous()


def make_target_logits(rows: int, n: int, seed: int, device="cpu",
                       std: float = 1.5):
    """Synthetic fused target logits for exercising verification alone."""
    g = _gen(device, seed)
    return (torch.randn(rows, n, generator=g, device=device) * std).contiguous()
