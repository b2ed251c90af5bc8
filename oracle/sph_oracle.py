"""CPU oracle for the split-head vocabulary projection (fp64, numpy).

TEST INFRASTRUCTURE ONLY.  Only the test suite (tests/), the smoke check in
__graft_entry__.smoke() and bench.py's cpu_baseline / reference leg may
import, call or run anything in this package.  The product path (the CUDA
library and its Python binding) never does, and shares no code with it.

What it computes is the paper's definition, written out plainly:
  * Eq. 9-13   full head z = h' W_lm + b split along the hidden dimension
               into an endpoint part (first d_l dims) and a cloud part;
               the two partial logits are added (the bias once, cloud side).
  * Sec. "Distributed Vocabulary Projection" / Eq. 14: only the ids of the
               language subset V_l are computed and returned, "after clipping,
               quantization"; everything else is -inf before the softmax.
  * Eq. 15     p = softmax(z~ / tau), a token is drawn from p.
  * Eq. 18     Q_b with b = 8 (INT8 payloads, Sec. "Experimental Setup").
  * Eq. 21     downlink payload ~ |V_l| * b/8 (+ tag/meta/pad, 0 here).
  * Sec. "Endpoint Speculative Decoding and Cloud Verification" and
               Algorithm 1: the cloud verifies the endpoint's draft tokens;
               the acceptance rule is standard speculative sampling (the
               paper cites Leviathan et al. 2023 and Chen et al. 2023).

Readings where the paper is silent (each also listed in the design notes):
  * Q_8 is symmetric per row: s_r = fl32(max_j |clip(y_rj)| / 127), code =
    round-half-even(clip(y)/s_r) clamped to [-127, 127]; an all-zero row has
    s_r = 0 and all codes 0.
  * clip(y) = min(max(y, -c), c) is applied before the row maximum.
  * Sampling is the inverse CDF in ascending vocabulary-id order with one
    uniform u in [0,1): the token is the first kept id whose CDF exceeds u
    (the last kept id if rounding leaves CDF_last <= u).
  * Uniforms come from Philox4x32-10 (Salmon et al., SC'11): key = (seed lo,
    seed hi), counter = (row or session, purpose, offset lo, offset hi),
    u = (x0 >> 8) * 2^-24.  purpose 0: the fuse-sample draw of a row;
    purpose 1+i: acceptance uniform of draft position i; purpose 1+k: the
    single final draw of a verification (residual or bonus token).
  * In act_mode "bf16" the cloud hidden state is first rounded to bf16 (RNE).

Every stored input is decoded exactly (bf16 and e4m3 values are exact in
fp64; fp32 h is exact in fp64) and all arithmetic is fp64.
"""
from __future__ import annotations

import numpy as np

# ---------------------------------------------------------------------------
# exact decoding of the stored number formats
# ---------------------------------------------------------------------------

def decode_bf16(bits) -> np.ndarray:
    """bf16 is the upper half of an IEEE-754 binary32: value = float32 with
    the 16 stored bits as its high half and zeros below."""
    b = np.asarray(bits).view(np.uint16).astype(np.uint32) << np.uint32(16)
    with np.errstate(invalid="ignore"):
        return b.view(np.float32).astype(np.float64)


def _e4m3_table() -> np.ndarray:
    """The 256 values of OCP FP8 E4M3 ('fn' variant): 1 sign bit, 4 exponent
    bits with bias 7, 3 mantissa bits; exponent field 0 is subnormal
    (2^-6 * m/8); S.1111.111 is NaN; there are no infinities."""
    t = np.empty(256, dtype=np.float64)
    for code in range(256):
        sign = -1.0 if code & 0x80 else 1.0
        e = (code >> 3) & 0xF
        m = code & 0x7
        if e == 0xF and m == 0x7:
            t[code] = np.nan
        elif e == 0:
            t[code] = sign * (m / 8.0) * 2.0 ** (-6)
        else:
            t[code] = sign * (1.0 + m / 8.0) * 2.0 ** (e - 7)
    return t


E4M3_VALUES = _e4m3_table()


def decode_e4m3(bits) -> np.ndarray:
    return E4M3_VALUES[np.asarray(bits).view(np.uint8)]


def round_fp32_to_bf16(x) -> np.ndarray:
    """Round-to-nearest-even of binary32 to bf16, returned as fp64 values.
    (Finite inputs: add 0x7FFF plus the lowest kept bit, truncate.)"""
    u = np.asarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    lsb = (u >> np.uint64(16)) & np.uint64(1)
    r = ((u + np.uint64(0x7FFF) + lsb) >> np.uint64(16)) & np.uint64(0xFFFF)
    return decode_bf16(r.astype(np.uint16))


# ---------------------------------------------------------------------------
# Philox4x32-10 (Salmon, Moraes, Dror, Shaw: "Parallel random numbers: as
# easy as 1, 2, 3", SC'11) -- the counter-based generator for every uniform
# ---------------------------------------------------------------------------

PHILOX_M0 = 0xD2511F53
PHILOX_M1 = 0xCD9E8D57
PHILOX_W0 = 0x9E3779B9
PHILOX_W1 = 0xBB67AE85
_MASK32 = 0xFFFFFFFF


def philox4x32_10(c0, c1, c2, c3, k0, k1):
    """Vectorised Philox4x32 with 10 rounds.  Each round multiplies c0 by M0
    and c2 by M1 (64-bit products split into hi/lo words), and outputs
    (hi(M1*c2) ^ c1 ^ k0, lo(M1*c2), hi(M0*c0) ^ c3 ^ k1, lo(M0*c0)); the key
    is bumped by (W0, W1) between rounds."""
    c = [np.asarray(v, dtype=np.uint64) & _MASK32 for v in (c0, c1, c2, c3)]
    k0 = np.uint64(int(k0) & _MASK32)
    k1 = np.uint64(int(k1) & _MASK32)
    m0 = np.uint64(PHILOX_M0)
    m1 = np.uint64(PHILOX_M1)
    mask = np.uint64(_MASK32)
    for rnd in range(10):
        if rnd:
            k0 = (k0 + np.uint64(PHILOX_W0)) & mask
            k1 = (k1 + np.uint64(PHILOX_W1)) & mask
        p0 = m0 * c[0]
        p1 = m1 * c[2]
        hi0, lo0 = p0 >> np.uint64(32), p0 & mask
        hi1, lo1 = p1 >> np.uint64(32), p1 & mask
        c = [hi1 ^ c[1] ^ k0, lo1, hi0 ^ c[3] ^ k1, lo0]
    return tuple(v.astype(np.uint32) for v in c)


def philox_uniform(seed: int, index, purpose, offset: int) -> np.ndarray:
    """u in [0,1) with 24 random bits from output word 0 for the counter
    (index, purpose, offset lo, offset hi) under key (seed lo, seed hi)."""
    index = np.asarray(index, dtype=np.uint64)
    purpose = np.broadcast_to(np.asarray(purpose, dtype=np.uint64), index.shape)
    off = int(offset)
    x0, _, _, _ = philox4x32_10(index, purpose,
                                np.full(index.shape, off & _MASK32, np.uint64),
                                np.full(index.shape, (off >> 32) & _MASK32, np.uint64),
                                int(seed) & _MASK32, (int(seed) >> 32) & _MASK32)
    return (x0 >> np.uint32(8)).astype(np.float64) * 2.0 ** -24


# ---------------------------------------------------------------------------
# cloud side: Eq. 12 over V_l, clipping, Eq. 18 with b = 8, Eq. 21
# ---------------------------------------------------------------------------

def _ids(keep_ids, V: int) -> np.ndarray:
    if keep_ids is None:
        return np.arange(V, dtype=np.int64)
    return np.asarray(keep_ids, dtype=np.int64)


def _decoded_rows(W_bits, w_dtype: str, w_scale, ids: np.ndarray) -> np.ndarray:
    """Exact fp64 values of the vocabulary rows `ids` of a stored weight."""
    if w_dtype == "bf16":
        return decode_bf16(W_bits[ids])
    if w_dtype == "fp8":
        sc = np.asarray(w_scale, dtype=np.float32).astype(np.float64)[ids]
        return decode_e4m3(W_bits[ids]) * sc[:, None]
    raise ValueError(w_dtype)


def gathered_matvec(H: np.ndarray, W_bits, w_dtype: str, w_scale,
                    ids: np.ndarray, chunk_elems: int = 1 << 25) -> np.ndarray:
    """y[r, j] = sum_c H[r, c] * W[ids[j], c] in fp64 (Eq. 11 / Eq. 12
    restricted to V_l).  The vocabulary is visited in chunks only to bound
    memory; every output is one complete fp64 dot product."""
    R = H.shape[0]
    dcols = W_bits.shape[1]
    y = np.empty((R, ids.size), dtype=np.float64)
    step = max(1, chunk_elems // max(1, dcols))
    for j0 in range(0, ids.size, step):
        j1 = min(ids.size, j0 + step)
        Wc = _decoded_rows(W_bits, w_dtype, w_scale, ids[j0:j1])
        y[:, j0:j1] = H @ Wc.T
    return y


def quantize_rows(y: np.ndarray, clip: float):
    """Clip to [-c, c], then the symmetric per-row INT8 quantizer Q_8
    (Eq. 18): s_r = fl32(max|clip(y)| / 127), code = rint_even(clip(y)/s_r)
    clamped to [-127, 127]; s_r = 0 and codes 0 for an all-zero row."""
    yc = np.clip(y, -clip, clip)
    a = np.max(np.abs(yc), axis=1) if yc.shape[1] else np.zeros(yc.shape[0])
    s = (a / 127.0).astype(np.float32)
    s64 = s.astype(np.float64)
    codes = np.zeros(yc.shape, dtype=np.int8)
    nz = s64 > 0
    if np.any(nz):
        q = np.rint(yc[nz] / s64[nz, None])
        codes[nz] = np.clip(q, -127, 127).astype(np.int8)
    return codes, s


def payload_bytes(rows: int, n_keep: int) -> int:
    """Eq. 21 with b = 8 and B_tag = B_meta = B_pad = 0: one byte per kept
    logit plus the fp32 scale of each row."""
    return int(rows) * int(n_keep) * 1 + 4 * int(rows)


def partial_logits(h_cloud, W_h_bits, *, w_dtype="bf16", w_scale=None,
                   bias=None, keep_ids=None, clip=30.0, act_mode="fp32"):
    """Cloud call: y = h_cloud W_h[V_l]^T (+ b[V_l]) (Eq. 12 over the subset
    of Eq. 14), then clip and INT8 (Eq. 18).  Returns a dict with the
    unclipped fp64 `y`, `codes` int8 [R, n], `row_scale` fp32 [R] and
    `payload_bytes` (Eq. 21)."""
    h = np.asarray(h_cloud, dtype=np.float32)
    H = round_fp32_to_bf16(h) if act_mode == "bf16" else h.astype(np.float64)
    ids = _ids(keep_ids, W_h_bits.shape[0])
    y = gathered_matvec(H, W_h_bits, w_dtype, w_scale, ids)
    if bias is not None:
        y = y + np.asarray(bias, dtype=np.float32).astype(np.float64)[ids][None, :]
    codes, s = quantize_rows(y, clip)
    return dict(y=y, codes=codes, row_scale=s,
                payload_bytes=payload_bytes(h.shape[0], ids.size))


# ---------------------------------------------------------------------------
# endpoint side: Eq. 11, Eq. 13, Eq. 14, Eq. 15 and the draw
# ---------------------------------------------------------------------------

def local_partial(h_local, W_l_bits, keep_ids=None) -> np.ndarray:
    """z_end[V_l] = h_end W_end (Eq. 11) over the kept ids, fp64."""
    H = np.asarray(h_local, dtype=np.float32).astype(np.float64)
    ids = _ids(keep_ids, W_l_bits.shape[0])
    return gathered_matvec(H, W_l_bits, "bf16", None, ids)


def fuse(codes, row_scale, z_local) -> np.ndarray:
    """z = dequant(z_cloud) + z_end (Eq. 13); dequant(code) = code * s_r.
    Without a payload (codes and row_scale None) z is z_end alone: given
    the whole hidden state and head, the unsplit head of Eq. 9."""
    if codes is None and row_scale is None:
        return np.asarray(z_local, dtype=np.float64)
    s = np.asarray(row_scale, dtype=np.float32).astype(np.float64)
    return np.asarray(codes).astype(np.float64) * s[:, None] + z_local


def softmax_rows(z, tau: float) -> np.ndarray:
    """p = softmax(z / tau) over the kept ids (Eq. 15); ids outside V_l carry
    -inf (Eq. 14) and so probability exactly 0 -- they are simply absent
    from the compacted rows."""
    z = np.asarray(z, dtype=np.float64)
    m = np.max(z, axis=-1, keepdims=True)
    w = np.exp((z - m) / tau)
    return w / np.sum(w, axis=-1, keepdims=True)


def inverse_cdf(P: np.ndarray, u: float):
    """First index j with C_j = sum_{i<=j} P_i > u (ascending id order);
    the last index if rounding leaves C_last <= u.  Returns (j, margin)
    with margin = distance of u to the nearer CDF boundary of j."""
    C = np.cumsum(P)
    j = int(np.searchsorted(C, u, side="right"))
    if j >= C.size:
        j = C.size - 1
    lo = C[j - 1] if j > 0 else 0.0
    return j, float(min(abs(u - lo), abs(C[j] - u)))


def sample_rows(z, tau: float, u):
    """Draw one compact index per row of z by the inverse CDF of Eq. 15."""
    P = softmax_rows(z, tau)
    out = np.empty(P.shape[0], dtype=np.int64)
    margin = np.empty(P.shape[0], dtype=np.float64)
    for r in range(P.shape[0]):
        out[r], margin[r] = inverse_cdf(P[r], float(u[r]))
    return out, margin


def greedy_rows(z):
    """Greedy decoding (temperature 0; the argmax decoding the paper's draft
    model uses, Eq. 17): per row the first index of the maximum, that is the
    lowest kept id on ties.  Returns (index, margin) with margin = the gap
    between the largest and the second-largest value (0 on a tie)."""
    z = np.asarray(z, dtype=np.float64)
    j = np.argmax(z, axis=-1)
    if z.shape[-1] < 2:
        return j, np.full(z.shape[0], np.inf)
    top2 = np.sort(z, axis=-1)[:, -2:]
    return j, top2[:, 1] - top2[:, 0]


# Gumbel-max sampling: an alternative single-pass sampler (reading listed
# in the design notes).  Index j of row r gets its own uniform: word j mod 4
# of the Philox output for counter (r, 2^31 + j div 4, offset lo, offset hi)
# under key (seed lo, seed hi), u = ((x >> 9) + 1/2) * 2^-23, which lies in
# (0, 1) and is exact in fp32 and fp64.
GUMBEL_TAG = 0x80000000


def gumbel_uniforms(seed: int, rows: int, n: int, offset: int) -> np.ndarray:
    """The [rows, n] uniforms of Gumbel-max sampling (see GUMBEL_TAG)."""
    g = (n + 3) // 4
    r = np.repeat(np.arange(rows, dtype=np.uint64), g)
    q = np.tile(np.arange(g, dtype=np.uint64), rows) | np.uint64(GUMBEL_TAG)
    off = int(offset)
    words = philox4x32_10(r, q, np.full(r.shape, off & _MASK32, np.uint64),
                          np.full(r.shape, (off >> 32) & _MASK32, np.uint64),
                          int(seed) & _MASK32, (int(seed) >> 32) & _MASK32)
    x = np.stack(words, axis=-1).reshape(rows, 4 * g)[:, :n]
    return ((x >> np.uint32(9)).astype(np.float64) + 0.5) * 2.0 ** -23


def gumbel_rows(z, tau: float, u):
    """Gumbel-max draw: per row the first index of the largest
    z_j / tau - log(-log u_j), a sample from softmax(z / tau) (the Gumbel-max
    property).  Returns (index, margin = top-two key gap)."""
    key = np.asarray(z, dtype=np.float64) / tau - np.log(-np.log(u))
    return greedy_rows(key)


def draw(z, ids, *, tau=1.0, seed=0, offset=0, sampler="cdf"):
    """The endpoint's draw from fused logits z (Eq. 15): one Philox uniform
    per row (purpose 0) and the inverse CDF; tau = 0 is greedy decoding (no
    uniform); sampler="gumbel" draws by Gumbel-max instead (gumbel_rows).
    Returns vocabulary-id `tokens`, the `margin` of each draw (CDF distance,
    or for greedy and Gumbel-max the top-two gap) and `z` itself."""
    R = z.shape[0]
    u = philox_uniform(seed, np.arange(R), 0, offset)
    if tau == 0:
        j, margin = greedy_rows(z)
    elif sampler == "gumbel":
        u = gumbel_uniforms(seed, R, z.shape[1], offset)
        j, margin = gumbel_rows(z, tau, u)
    else:
        j, margin = sample_rows(z, tau, u)
    return dict(tokens=ids[j].astype(np.int32), margin=margin, z=z, u=u,
                index=j)


def fuse_sample(codes, row_scale, h_local, W_l_bits, *, keep_ids=None,
                tau=1.0, seed=0, offset=0, sampler="cdf"):
    """Endpoint call: local partial, fuse, mask, softmax(./tau), draw (see
    `draw`)."""
    V = W_l_bits.shape[0]
    ids = _ids(keep_ids, V)
    zl = local_partial(h_local, W_l_bits, ids)
    z = fuse(codes, row_scale, zl)
    return draw(z, ids, tau=tau, seed=seed, offset=offset, sampler=sampler)


# ---------------------------------------------------------------------------
# block streaming of the payload (Sec. "Device-Adaptive Feature
# Preparation", Eq. 3: a tensor cut by columns into blocks that travel, and
# are processed, one after another; Eq. 18 quantizes each transmitted
# tensor; Eq. 21 counts its bytes).  Reading: the compacted logits are cut
# into chunks of L consecutive kept ids, chunk q = ids q*L .. (q+1)*L - 1
# (the last one shorter), and each chunk is quantized as a tensor of its
# own, with one scale per row and chunk.
# ---------------------------------------------------------------------------

def chunk_bounds(n: int, chunk: int):
    """[(j0, j1)] of the chunks of `chunk` kept ids (one chunk for chunk = 0
    or chunk >= n)."""
    L = n if (chunk <= 0 or chunk >= n) else int(chunk)
    return [(j0, min(n, j0 + L)) for j0 in range(0, n, L)]


def quantize_chunks(y: np.ndarray, clip: float, chunk: int):
    """Q_8 of Eq. 18 applied to every chunk as its own tensor: codes [R, n]
    (compacted id order) and scales [nchunk, R]."""
    R, n = y.shape
    b = chunk_bounds(n, chunk)
    codes = np.zeros((R, n), dtype=np.int8)
    scales = np.zeros((len(b), R), dtype=np.float32)
    for q, (j0, j1) in enumerate(b):
        codes[:, j0:j1], scales[q] = quantize_rows(y[:, j0:j1], clip)
    return codes, scales


def payload_bytes_chunked(rows: int, n_keep: int, chunk: int) -> int:
    """Eq. 21 with b = 8 for a chunked payload: every kept logit's byte plus
    one fp32 scale per row and chunk (the chunks' metadata B_meta); tag and
    padding 0."""
    return int(rows) * int(n_keep) + 4 * int(rows) * len(chunk_bounds(int(n_keep), chunk))


def fuse_chunks(codes, scales, z_local, chunk: int) -> np.ndarray:
    """Eq. 13 on a chunked payload: each chunk dequantized with its own
    scales, plus the local partial."""
    codes = np.asarray(codes)
    z = np.array(z_local, dtype=np.float64)
    for q, (j0, j1) in enumerate(chunk_bounds(codes.shape[1], chunk)):
        s = np.asarray(scales[q], dtype=np.float32).astype(np.float64)
        z[:, j0:j1] += codes[:, j0:j1].astype(np.float64) * s[:, None]
    return z


def split_step(h, d_l: int, W_h_bits, W_l_bits, *, w_dtype="bf16", w_scale=None,
               bias=None, keep_ids=None, clip=30.0, act_mode="fp32", tau=1.0,
               seed=0, offset=0, chunk=0, sampler="cdf"):
    """The whole split step from the full hidden state (Algorithm 1's cloud
    projection, then the endpoint's fusion and sampling): the cloud partial
    of h[:, d_l:] (Eq. 12) clipped and quantized per chunk (Eq. 18; one
    chunk = the whole row), the payload that would cross (Eq. 21), then the
    local partial of h[:, :d_l] (Eq. 11), the fusion (Eq. 13) and the draw
    (Eqs. 14-15).  Returns the cloud dict of `partial_logits` with the
    chunked `codes`/`scales`, and the draw's dict under "draw"."""
    h = np.asarray(h, dtype=np.float32)
    c = partial_logits(h[:, d_l:], W_h_bits, w_dtype=w_dtype, w_scale=w_scale, bias=bias,
                       keep_ids=keep_ids, clip=clip, act_mode=act_mode)
    codes, scales = quantize_chunks(c["y"], clip, chunk)
    ids = _ids(keep_ids, W_h_bits.shape[0])
    zl = local_partial(h[:, :d_l], W_l_bits, ids)
    z = fuse_chunks(codes, scales, zl, chunk)
    return dict(y=c["y"], codes=codes, scales=scales,
                payload_bytes=payload_bytes_chunked(h.shape[0], ids.size, chunk),
                draw=draw(z, ids, tau=tau, seed=seed, offset=offset, sampler=sampler))


# ---------------------------------------------------------------------------
# speculative verification (standard rejection sampling)
# ---------------------------------------------------------------------------

def verify_core(p, q, x, r, u):
    """One session with explicit uniforms.
      p: [k+1, n] target probabilities (rows 0..k), q: [k, n] draft
      probabilities or None (greedy one-hot drafts at x), x: [k] compact
      indices of the draft tokens (-1 = not in V_l), r: [k] acceptance
      uniforms, u: the final uniform.
    For i = 0..k-1: accept x_i iff r_i * q_i(x_i) < p_i(x_i).  At the first
    rejection draw from max(0, p_i - q_i) renormalised (from p_i if that is
    all zero); if all k are accepted draw the bonus token from p_k.
    Returns (n_accepted, compact index of the drawn token, accept margin,
    draw margin); the accept margin is min_i |r_i - p_i(x_i)/q_i(x_i)|."""
    p = np.asarray(p, dtype=np.float64)
    k = p.shape[0] - 1
    acc_margin = np.inf
    for i in range(k):
        xi = int(x[i])
        px = p[i, xi] if xi >= 0 else 0.0
        if q is None:
            qx = 1.0 if xi >= 0 else 0.0
        else:
            qx = float(q[i][xi]) if xi >= 0 else 0.0
        if qx > 0:
            acc_margin = min(acc_margin, abs(float(r[i]) - px / qx))
        if float(r[i]) * qx < px:
            continue
        if q is None:
            res = p[i].copy()
            if xi >= 0:
                res[xi] = 0.0
        else:
            res = np.maximum(0.0, p[i] - np.asarray(q[i], dtype=np.float64))
        tot = res.sum()
        dist = res / tot if tot > 0 else p[i]
        j, m = inverse_cdf(dist, float(u))
        return i, j, acc_margin, m
    j, m = inverse_cdf(p[k], float(u))
    return k, j, acc_margin, m


def compact_index(keep_ids, V: int, tokens) -> np.ndarray:
    """Position of each vocabulary id in the sorted id list (-1 if absent)."""
    tokens = np.asarray(tokens, dtype=np.int64)
    if keep_ids is None:
        return np.where((tokens >= 0) & (tokens < V), tokens, -1)
    ids = np.asarray(keep_ids, dtype=np.int64)
    pos = np.searchsorted(ids, tokens)
    pos_c = np.minimum(pos, ids.size - 1)
    return np.where((pos < ids.size) & (ids[pos_c] == tokens), pos_c, -1)


def verify_draft(target_logits, sessions: int, k: int, *, keep_ids=None,
                 V=None, tau=1.0, draft_tokens, draft_probs=None, seed=0,
                 offset=0):
    """Cloud verification of k drafts per session.  target_logits
    [S*(k+1), n] are fused logits (row s*(k+1)+i is the target at draft
    position i, row s*(k+1)+k the bonus position); p_i = softmax(. / tau),
    tau = 0 greedy.  Uniforms: r_i = Philox(session, 1+i),
    u = Philox(session, 1+k)."""
    Z = np.asarray(target_logits, dtype=np.float32).astype(np.float64)
    n = Z.shape[1]
    if V is None:
        V = n
    ids = _ids(keep_ids, V)
    n_acc = np.empty(sessions, dtype=np.int32)
    nxt = np.empty(sessions, dtype=np.int32)
    am = np.empty(sessions)
    dm = np.empty(sessions)
    xs = compact_index(keep_ids, V, np.asarray(draft_tokens).reshape(sessions, k))
    if tau == 0:
        # greedy verification, the tau -> 0 limit of the rule in verify_core
        # with ties resolved to the lowest id: p_i is one-hot at a_i =
        # argmax z_i, so x_i is accepted iff x_i == a_i (r_i q_i(x_i) < 1
        # always holds), the residual at the first rejection is one-hot at
        # a_i (or, all zero, falls back to p_i), and the bonus token is a_k.
        for s in range(sessions):
            a, gap = greedy_rows(Z[s * (k + 1):(s + 1) * (k + 1)])
            i = 0
            while i < k and xs[s][i] == a[i]:
                i += 1
            n_acc[s] = i
            nxt[s] = ids[a[i]]
            am[s] = np.min(gap[:i + 1])
            dm[s] = gap[i]
        return dict(n_accepted=n_acc, next_token=nxt, accept_margin=am,
                    draw_margin=dm)
    for s in range(sessions):
        P = softmax_rows(Z[s * (k + 1):(s + 1) * (k + 1)], tau)
        r = philox_uniform(seed, np.full(k, s), 1 + np.arange(k), offset)
        u = float(philox_uniform(seed, np.array([s]), 1 + k, offset)[0])
        q = None if draft_probs is None else np.asarray(draft_probs)[s]
        a, j, am[s], dm[s] = verify_core(P, q, xs[s], r, u)
        n_acc[s] = a
        nxt[s] = ids[j]
    return dict(n_accepted=n_acc, next_token=nxt, accept_margin=am,
                draw_margin=dm)
