"""MM-ShiftKV prefill-only KV selection, CPU oracle (test infrastructure).

Only the tests, ``__graft_entry__.smoke()`` and the benchmark's CPU-baseline
leg use this module; the product library never imports or runs it.

Everything is float64 numpy, one request, one KV head and one proxy group at a
time, in the order of the paper's Algorithm 1 (Appendix B). Each function cites
the passage it restates. Readings of points the paper leaves open are marked
"Reading:"; they are the same readings the CUDA path implements.

Notation: T prompt length, W observation window, Hq / Hkv query / KV heads,
r = Hq / Hkv, d head_dim, N_p proxies per query head (the paper's N), G groups
of g = N_p / G proxies, C the per-KV-head budget.
"""
from __future__ import annotations

import math
from typing import Dict, List, Optional, Sequence

import numpy as np

# §4.1 "Implementation and Hyperparameters": N=512 proxies in G=32 groups of
# g=16, gamma=10, tau=0.95, lambda=1.
DEFAULTS = dict(n_proxies=512, n_groups=32, gamma=10.0, tau=0.95, lam=1.0)

SCORE_VOTE = 0   # §3.2.2-3.2.3: group-wise tau-coverage vote + last-query anchor
SCORE_MASS = 1   # Table 5 "+ Var. Exp." row: rank by aggregated mass, no vote

BF16 = "bf16"
F32 = "f32"

__all__ = [
    "DEFAULTS", "SCORE_VOTE", "SCORE_MASS", "BF16", "F32", "philox4x64_10", "uniforms_from_bits",
    "proxy_normals", "window_stats", "prefill_stats", "rope_rotate", "round_to",
    "build_proxies", "build_proxies_from_stats", "hidden_normals", "hidden_proxies",
    "softmax_rows", "group_masses", "anchor_attention", "cover_sets", "votes",
    "scores", "select_topk", "select_topk_heads", "gather", "attention_coverage", "select_request", "select",
]

# ---------------------------------------------------------------------------
# Counter-based normal generator.
#
# The paper samples proxies from a Gaussian but does not fix a generator.
# Reading: Philox4x64-10 (Salmon, Moraes, Dror, Shaw, "Parallel random numbers:
# as easy as 1, 2, 3", SC'11) keyed by the seed, with one counter per
# (request, query head, proxy, quad of dimensions), and the Box-Muller
# transform (Box & Muller 1958) turning two uniforms into two normals.
# ---------------------------------------------------------------------------
_PHILOX_M0 = np.uint64(0xD2E7470EE14C6C93)
_PHILOX_M1 = np.uint64(0xCA5A826395121157)
_PHILOX_W0 = np.uint64(0x9E3779B97F4A7C15)   # golden ratio
_PHILOX_W1 = np.uint64(0xBB67AE8584CAA73B)   # sqrt(3) - 1
_M32 = np.uint64(0xFFFFFFFF)
_S32 = np.uint64(32)


def _mulhilo64(a: np.ndarray, b: np.uint64):
    """(high, low) 64-bit halves of the 128-bit product a*b, from 32-bit limbs."""
    a0, a1 = a & _M32, a >> _S32
    b0, b1 = b & _M32, b >> _S32
    p00, p01, p10, p11 = a0 * b0, a0 * b1, a1 * b0, a1 * b1
    mid = (p00 >> _S32) + (p01 & _M32) + (p10 & _M32)
    hi = p11 + (p01 >> _S32) + (p10 >> _S32) + (mid >> _S32)
    lo = a * b                      # wraps modulo 2**64
    return hi, lo


def philox4x64_10(ctr: np.ndarray, key: Sequence[int]) -> np.ndarray:
    """Philox4x64 with 10 rounds. ctr: uint64 [..., 4]; key: two uint64 words.

    One round maps (c0, c1, c2, c3) to
    (hi(M1*c2) ^ c1 ^ k0, lo(M1*c2), hi(M0*c0) ^ c3 ^ k1, lo(M0*c0)),
    and the key is bumped by the Weyl constants (W0, W1) between rounds.
    """
    c = [np.array(ctr[..., i], dtype=np.uint64) for i in range(4)]
    k0, k1 = np.uint64(key[0]), np.uint64(key[1])
    with np.errstate(over="ignore"):
        for rnd in range(10):
            if rnd:
                k0 = np.uint64((int(k0) + int(_PHILOX_W0)) & 0xFFFFFFFFFFFFFFFF)
                k1 = np.uint64((int(k1) + int(_PHILOX_W1)) & 0xFFFFFFFFFFFFFFFF)
            hi0, lo0 = _mulhilo64(c[0], _PHILOX_M0)
            hi1, lo1 = _mulhilo64(c[2], _PHILOX_M1)
            c = [hi1 ^ c[1] ^ k0, lo1, hi0 ^ c[3] ^ k1, lo0]
    return np.stack(c, axis=-1)


def uniforms_from_bits(x: np.ndarray) -> np.ndarray:
    """uint32 words -> float64 uniforms in (0, 1): ((x >> 9) + 1/2) * 2**-23
    (24 significant bits: exact in float32 too)."""
    return ((np.asarray(x, dtype=np.uint64) >> np.uint64(9)).astype(np.float64) + 0.5) * 2.0 ** -23


def proxy_normals(seed: int, layer_id: int, b: int, n_q_heads: int,
                  n_proxies: int, head_dim: int, stream: int = 0) -> np.ndarray:
    """Standard normals z[hq, i, j] for request b of layer ``layer_id``.

    One Philox4x64-10 draw with counter (i * d/8 + q, hq, b, layer_id) and key
    (seed, stream) covers dims 4q..4q+3 and d/2+4q..d/2+4q+3 of proxy i of
    query head hq (stream 0: query-space proxies; stream 1: hidden-space
    proxies, see hidden_normals). Its four 64-bit outputs, split low word first, give eight 32-bit
    words w0..w7 and uniforms u_k = ((w_k >> 9) + 1/2) 2^-23; Box-Muller turns
    each pair (u_2m, u_2m+1) into sqrt(-2 ln u_2m) (cos, sin)(2 pi u_2m+1).
    Pairs 0, 1 fill dims 4q..4q+3; pairs 2, 3 fill d/2+4q..d/2+4q+3.
    """
    assert head_dim % 8 == 0
    nq = head_dim // 8
    hq, i, q = np.meshgrid(np.arange(n_q_heads, dtype=np.uint64),
                           np.arange(n_proxies, dtype=np.uint64),
                           np.arange(nq, dtype=np.uint64), indexing="ij")
    ctr = np.stack([i * np.uint64(nq) + q, hq,
                    np.full_like(q, np.uint64(b)),
                    np.full_like(q, np.uint64(layer_id))], axis=-1)
    x = philox4x64_10(ctr, (seed & 0xFFFFFFFFFFFFFFFF, stream))  # [Hq, Np, d/8, 4]
    words = np.stack([x & _M32, x >> _S32], axis=-1).reshape(x.shape[:-1] + (8,))
    u = uniforms_from_bits(words)                               # [Hq, Np, d/8, 8]
    r = np.sqrt(-2.0 * np.log(u[..., 0::2]))                    # [.., 4]
    ang = 2.0 * np.pi * u[..., 1::2]
    zc, zs = r * np.cos(ang), r * np.sin(ang)
    z = np.empty(u.shape, dtype=np.float64)                      # [.., 8]
    z[..., 0::2] = zc
    z[..., 1::2] = zs
    out = np.empty((n_q_heads, n_proxies, head_dim), dtype=np.float64)
    half = head_dim // 2
    for k in range(4):
        out[:, :, 4 * np.arange(nq) + k] = z[..., k]
        out[:, :, half + 4 * np.arange(nq) + k] = z[..., 4 + k]
    return out


# ---------------------------------------------------------------------------
# Step 1: query proxies (§3.2.1; Appendix A.4; Algorithm 1, first three steps)
# ---------------------------------------------------------------------------
def window_stats(qwin: np.ndarray):
    """Element-wise mean and standard deviation of the prefill queries.

    §3.2.1 defines mu_pre = mean(h), sigma_pre = std(h) per feature across
    prompt tokens. Reading (query-space form of Appendix A.4): the statistics
    are taken per (query head, dimension) over the W observation-window
    queries, with the unbiased (W - 1) estimator.
    qwin: [W, Hq, d] -> (mu, sigma), each [Hq, d] float64.
    """
    q = np.asarray(qwin, dtype=np.float64)
    w = q.shape[0]
    mu = q.sum(axis=0) / w
    var = ((q - mu) ** 2).sum(axis=0) / (w - 1)
    return mu, np.sqrt(var)


def prefill_stats(qfull: np.ndarray):
    """Statistics over the whole prefill (§3.2.1: mu_pre and sigma_pre are taken
    across all prompt tokens).

    Reading: in query space, per (query head, dimension) over all T prompt
    queries of the request, with the unbiased (T - 1) estimator (0 for T = 1).
    qfull: [T, Hq, d] -> (mu, sigma), each [Hq, d] float64. The same
    statistics of hidden states [T, d_model] (the paper's own space) give
    [d_model] vectors for hidden_proxies.
    """
    q = np.asarray(qfull, dtype=np.float64)
    t = q.shape[0]
    mu = q.sum(axis=0) / t
    if t < 2:
        return mu, np.zeros_like(mu)
    var = ((q - mu) ** 2).sum(axis=0) / (t - 1)
    return mu, np.sqrt(var)


def rope_rotate(x: np.ndarray, pos: float, theta: float) -> np.ndarray:
    """Rotary embedding at position ``pos`` (rotate-half pairing).

    Pairs (x_j, x_{j+d/2}) for j < d/2 are rotated by pos * theta**(-2j/d).
    §3.2.1 assigns proxies a synthetic future position; keys keep theirs.
    """
    x = np.asarray(x, dtype=np.float64)
    half = x.shape[-1] // 2
    freq = theta ** (-2.0 * np.arange(half, dtype=np.float64) / x.shape[-1])
    ang = pos * freq
    c, s = np.cos(ang), np.sin(ang)
    a, b = x[..., :half], x[..., half:]
    return np.concatenate([a * c - b * s, b * c + a * s], axis=-1)


def round_to(x: np.ndarray, dtype: str) -> np.ndarray:
    """Round float64 values to bf16 or float32 (round to nearest, ties to
    even), returned as float64. bf16 keeps 8 significant bits."""
    x = np.asarray(x, dtype=np.float64)
    if dtype == F32:
        return x.astype(np.float32).astype(np.float64)
    m, e = np.frexp(x)                       # x = m * 2**e, 0.5 <= |m| < 1
    ulp = np.ldexp(1.0, e - 8)
    out = np.rint(x / ulp) * ulp             # np.rint rounds half to even
    return np.where(x == 0.0, 0.0, out)


def build_proxies(qwin: np.ndarray, z: np.ndarray, gamma: float, t_len: int,
                  dtype: str, rope_theta: float = 0.0, rope_pos_offset: int = 0):
    """Variance-expanded query proxies for one request.

    §3.2.1 / Appendix A.4: q~ ~ N(mu_q, gamma^2 Sigma_q) with diagonal Sigma_q,
    i.e. q~[hq, i, j] = mu[hq, j] + gamma * sigma[hq, j] * z[hq, i, j].
    Reading: RoPE, when enabled, rotates every proxy to the first decode
    position T + rope_pos_offset. Reading: proxies are rounded to the input
    dtype before they meet the keys, as in a bf16 inference stack.
    qwin: [W, Hq, d]; z: [Hq, N_p, d] -> [Hq, N_p, d] float64 (dtype-exact).
    """
    mu, sigma = window_stats(qwin)
    return build_proxies_from_stats(mu, sigma, z, gamma, t_len, dtype, rope_theta, rope_pos_offset)


def build_proxies_from_stats(mu: np.ndarray, sigma: np.ndarray, z: np.ndarray, gamma: float,
                             t_len: int, dtype: str, rope_theta: float = 0.0,
                             rope_pos_offset: int = 0):
    """The same expansion from given statistics (e.g. prefill_stats):
    q~[hq, i, j] = mu[hq, j] + gamma * sigma[hq, j] * z[hq, i, j], then the
    optional RoPE rotation and rounding of build_proxies.
    mu, sigma: [Hq, d]; z: [Hq, N_p, d] -> [Hq, N_p, d] float64 (dtype-exact).
    """
    q = mu[:, None, :] + gamma * sigma[:, None, :] * z
    if rope_theta > 0.0:
        q = rope_rotate(q, float(t_len + rope_pos_offset), rope_theta)
    return round_to(q, dtype)


def hidden_normals(seed: int, layer_id: int, b: int, n_proxies: int, d_model: int) -> np.ndarray:
    """Standard normals z[i, j] of the N proxy hidden states of request b
    (§3.2.1: H~_i ~ N(mu_pre, diag((gamma sigma_pre)^2)) in the model's
    hidden space). Reading: the generator of proxy_normals with key
    (seed, 1) and one 'head' of width d_model: counter
    (i * d_model/8 + q, 0, b, layer_id) covers dims 4q..4q+3 and
    d_model/2+4q..d_model/2+4q+3. -> [N, d_model] float64.
    """
    return proxy_normals(seed, layer_id, b, 1, n_proxies, d_model, stream=1)[0]


def hidden_proxies(mu: np.ndarray, sigma: np.ndarray, z: np.ndarray, w_q: np.ndarray,
                   bias: Optional[np.ndarray], gamma: float, n_q_heads: int, pos: float,
                   dtype: str, rope_theta: float = 0.0) -> np.ndarray:
    """Query proxies from proxy hidden states (§3.2.1, Algorithm 1's first
    steps): H~_i = mu + gamma * sigma * z_i in the hidden space, projected by
    the query projection q~_i^(h) = W_Q^(h) H~_i, then placed at a future
    position with RoPE.

    mu, sigma: [d_model] statistics of the prefill hidden states
    (prefill_stats over [T, d_model]); z: [N, d_model] (hidden_normals);
    w_q: [Hq*d, d_model] (row f of the projection gives output feature f =
    hq*d + j); bias: [Hq*d] or None; pos: the proxies' position.
    Reading: H~ is rounded to the input dtype before the projection (the
    model's projection consumes hidden states in that dtype); the projection,
    the bias (Qwen-style query projections carry one) and RoPE are exact
    (float64) and the proxies are rounded once at the end, as in
    build_proxies. -> [Hq, N, d] float64 (dtype-exact).
    """
    h = round_to(mu[None, :] + gamma * sigma[None, :] * z, dtype)      # [N, d_model]
    q = h @ np.asarray(w_q, dtype=np.float64).T                        # [N, Hq*d]
    if bias is not None:
        q = q + np.asarray(bias, dtype=np.float64)[None, :]
    n = q.shape[0]
    q = q.reshape(n, n_q_heads, -1).transpose(1, 0, 2)                 # [Hq, N, d]
    if rope_theta > 0.0:
        q = rope_rotate(q, float(pos), rope_theta)
    return round_to(q, dtype)


# ---------------------------------------------------------------------------
# Step 2: importance estimation (§3.2.2; Appendix B)
# ---------------------------------------------------------------------------
def softmax_rows(logits: np.ndarray) -> np.ndarray:
    """Row softmax over the last axis (max-subtracted, float64)."""
    m = logits.max(axis=-1, keepdims=True)
    e = np.exp(logits - m)
    return e / e.sum(axis=-1, keepdims=True)


def group_masses(proxies: np.ndarray, keys: np.ndarray, n_groups: int,
                 scale: float) -> np.ndarray:
    """Group attention mass abar[h, g, t].

    §3.2.2: a_t(q~_i) = softmax_t(q~_i . k_t / sqrt(d)) over all T prompt keys,
    and abar^(g)_t = sum over the proxies i of group g of a_t(q~_i).
    §4.1 / Appendix B (GQA): the scores of the r query heads that share KV head
    h are aggregated, so group g of KV head h sums over those r heads too.
    Reading: group g holds proxies g*(N_p/G) .. (g+1)*(N_p/G) - 1.
    proxies: [Hq, N_p, d]; keys: [T, Hkv, d] -> [Hkv, G, T] float64.
    """
    hq, n_p, d = proxies.shape
    t_len, hkv, _ = keys.shape
    r = hq // hkv
    out = np.zeros((hkv, n_groups, t_len), dtype=np.float64)
    if n_groups == 0:
        return out
    gs = n_p // n_groups
    for h in range(hkv):
        k = np.asarray(keys[:, h, :], dtype=np.float64)            # [T, d]
        for g in range(n_groups):
            rows = proxies[h * r:(h + 1) * r, g * gs:(g + 1) * gs, :].reshape(-1, d)
            a = softmax_rows((rows @ k.T) * scale)                  # [r*gs, T]
            out[h, g] = a.sum(axis=0)
    return out


def anchor_attention(q_last: np.ndarray, keys: np.ndarray, scale: float) -> np.ndarray:
    """Last-query anchor alpha[h, t] (§3.2.3).

    a_t(q_last) is the softmax attention of the last real prefill query.
    Reading (GQA): alpha for KV head h is the mean over its r query heads, so
    it stays within one vote step, as §3.2.3 requires of the anchor.
    q_last: [Hq, d]; keys: [T, Hkv, d] -> [Hkv, T] float64.
    """
    hq = q_last.shape[0]
    t_len, hkv, d = keys.shape
    r = hq // hkv
    out = np.zeros((hkv, t_len), dtype=np.float64)
    for h in range(hkv):
        k = np.asarray(keys[:, h, :], dtype=np.float64)
        a = softmax_rows((np.asarray(q_last[h * r:(h + 1) * r], dtype=np.float64) @ k.T) * scale)
        out[h] = a.mean(axis=0)
    return out


def cover_sets(abar: np.ndarray, tau: float) -> np.ndarray:
    """tau-coverage sets S_g (§3.2.2).

    Keys are ranked by descending abar^(g)_t; S_g is the smallest prefix of that
    ranking whose mass is at least tau times the group's total mass.
    Reading: equal masses are ranked by ascending t; the total is the sum over
    the same ranking (so tau = 1 is reachable).
    abar: [G, T] -> bool [G, T].
    """
    n_groups, t_len = abar.shape
    member = np.zeros((n_groups, t_len), dtype=bool)
    t_idx = np.arange(t_len)
    for g in range(n_groups):
        order = np.lexsort((t_idx, -abar[g]))        # mass desc, then t asc
        csum = np.cumsum(abar[g][order])
        target = tau * csum[-1]
        k = int(np.argmax(csum >= target)) + 1
        member[g, order[:k]] = True
    return member


def votes(member: np.ndarray) -> np.ndarray:
    """vote(t) = sum_g 1[t in S_g] (§3.2.2). member: [G, T] -> [T]."""
    return member.sum(axis=0).astype(np.float64)


def scores(mode: int, abar: np.ndarray, alpha: np.ndarray, tau: float,
           lam: float) -> np.ndarray:
    """Per-key importance S_t for one KV head.

    VOTE (§3.2.3): S_t = vote(t) + lambda * alpha_t.
    MASS (Table 5, "+ Var. Exp." row): S_t = sum_g abar^(g)_t.
    abar: [G, T]; alpha: [T] -> [T].
    """
    if mode == SCORE_MASS:
        return abar.sum(axis=0)
    return votes(cover_sets(abar, tau)) + lam * alpha


def select_topk(s: np.ndarray, budget: int) -> np.ndarray:
    """Budgeted selection for one KV head (§3.2.3; Algorithm 1, last steps).

    The most recent token T-1 is always kept; the other C-1 are the largest
    S_t among t < T-1; the kept indices are returned in temporal order.
    Reading: equal scores are ranked by ascending t; C >= T keeps everything.
    s: [T] -> int64 [min(C, T)].
    """
    t_len = s.shape[0]
    if budget >= t_len:
        return np.arange(t_len, dtype=np.int64)
    cand = np.arange(t_len - 1)
    order = np.lexsort((cand, -s[:t_len - 1]))       # score desc, then t asc
    kept = np.concatenate([order[:budget - 1], [t_len - 1]])
    return np.sort(kept).astype(np.int64)


def select_topk_heads(s: np.ndarray, head_budgets: Sequence[int], capacity: int):
    """Selection with a budget per KV head (§3.1: the budget C_{l,h} is set per
    layer and KV head; §4.1 uses one value everywhere; §4.3 pairs the method
    with allocators that spread budgets over layers and heads). Head h keeps
    select_topk(s[h], C_h). Reading: every head's rows are padded to the
    request's capacity min(C_max, T) with -1, C_max >= C_h >= 1 being the
    request's largest budget. s: [Hkv, T] -> (idx [min(C_max, T), Hkv] int64,
    counts [Hkv] = min(C_h, T))."""
    hkv, t_len = s.shape
    rows = min(capacity, t_len)
    idx = np.full((rows, hkv), -1, dtype=np.int64)
    counts = np.zeros(hkv, dtype=np.int64)
    for h in range(hkv):
        c = int(head_budgets[h])
        assert 1 <= c <= capacity
        kept = select_topk(s[h], c)
        idx[:kept.shape[0], h] = kept
        counts[h] = kept.shape[0]
    return idx, counts


def gather(keys: np.ndarray, values: np.ndarray, idx: np.ndarray):
    """Compacted cache (Appendix B): row c of KV head h is token idx[c, h];
    padding rows (idx -1, per-head budgets) are zero.
    keys/values: [T, Hkv, d]; idx: [C', Hkv] -> two [C', Hkv, d] arrays."""
    h = np.arange(idx.shape[1])[None, :]
    pad = (idx < 0)[..., None]
    safe = np.where(idx < 0, 0, idx)
    return np.where(pad, 0.0, keys[safe, h]), np.where(pad, 0.0, values[safe, h])


# ---------------------------------------------------------------------------
# Quality metric: attention-mass coverage of the kept set (§1, Fig. 1b)
# ---------------------------------------------------------------------------
def attention_coverage(keys: np.ndarray, dec_queries: np.ndarray, idx: np.ndarray,
                       scale: float) -> np.ndarray:
    """Fraction of decode-time attention probability that lands on the kept
    prompt entries (§1, Fig. 1b's attention mass coverage).

    Reading: for decode query q of query head hq, the softmax of
    scale * q.k_t over the T prompt keys of KV head h = hq // r (the prompt
    part of the decode-time attention, renormalised over the prompt), summed
    over the kept indices idx[:, h].
    keys: [T, Hkv, d]; dec_queries: [n, Hq, d]; idx: [C', Hkv] -> [Hq, n].
    """
    keys = np.asarray(keys, dtype=np.float64)
    dq = np.asarray(dec_queries, dtype=np.float64)
    t_len, hkv, _ = keys.shape
    n, hq, _ = dq.shape
    r = hq // hkv
    out = np.zeros((hq, n))
    for q in range(hq):
        h = q // r
        p = softmax_rows(scale * (dq[:, q, :] @ keys[:, h, :].T))     # [n, T]
        out[q] = p[:, np.asarray(idx)[:, h]].sum(axis=1)
    return out


# ---------------------------------------------------------------------------
# Whole method (Algorithm 1) for one request and for a batch.
# ---------------------------------------------------------------------------
def select_request(keys, values, qwin, budget: int, *, n_proxies=512, n_groups=32,
                   gamma=10.0, tau=0.95, lam=1.0, seed=0, layer_id=0, b=0,
                   score_mode=SCORE_VOTE, softmax_scale=0.0, rope_theta=0.0,
                   rope_pos_offset=0, dtype=BF16, proxies=None,
                   qfull=None, head_budgets=None) -> Dict[str, np.ndarray]:
    """Algorithm 1 for one request of one layer.

    keys/values: [T, Hkv, d]; qwin: [W, Hq, d] (its last row is the last real
    prefill query). ``proxies`` ([Hq, N_p, d]) replaces the sampled proxies
    when given. ``qfull`` ([T, Hq, d], all prompt queries), when given, is the
    source of the proxies' statistics (prefill_stats) instead of the window.
    ``head_budgets`` ([Hkv], each in [1, budget]) gives every KV head its own
    budget (select_topk_heads); ``budget`` is then the request's largest.
    Returns proxies, group masses, anchor, mass, scores, indices ([C', Hkv],
    ascending per head, -1 padded with head budgets), the kept count per head
    and the gathered cache.
    """
    keys = np.asarray(keys, dtype=np.float64)
    values = np.asarray(values, dtype=np.float64)
    qwin = np.asarray(qwin, dtype=np.float64)
    t_len, hkv, d = keys.shape
    hq = qwin.shape[1]
    scale = softmax_scale if softmax_scale > 0.0 else 1.0 / math.sqrt(d)
    if proxies is None:
        z = proxy_normals(seed, layer_id, b, hq, n_proxies, d)
        if qfull is None:
            proxies = build_proxies(qwin, z, gamma, t_len, dtype, rope_theta, rope_pos_offset)
        else:
            mu, sigma = prefill_stats(qfull)
            proxies = build_proxies_from_stats(mu, sigma, z, gamma, t_len, dtype, rope_theta,
                                               rope_pos_offset)
    else:
        proxies = np.asarray(proxies, dtype=np.float64)
    abar = group_masses(proxies, keys, n_groups, scale)            # [Hkv, G, T]
    alpha = anchor_attention(qwin[-1], keys, scale)                # [Hkv, T]
    mass = abar.sum(axis=1)                                         # [Hkv, T]
    s = np.stack([scores(score_mode, abar[h], alpha[h], tau, lam) for h in range(hkv)])
    if head_budgets is None:
        idx = np.stack([select_topk(s[h], budget) for h in range(hkv)], axis=1)
        count = np.full(hkv, idx.shape[0], dtype=np.int64)
    else:
        idx, count = select_topk_heads(s, head_budgets, budget)
    out_k, out_v = gather(keys, values, idx)
    return dict(proxies=proxies, group_mass=abar, anchor=alpha, mass=mass,
                scores=s, idx=idx, count=count, out_k=out_k, out_v=out_v)


def select(keys, values, qwin, cu_seqlens: Sequence[int], budgets: Sequence[int],
           proxies=None, **kw) -> List[Dict[str, np.ndarray]]:
    """Batch of requests packed as [total_T, Hkv, d] with prefix offsets
    ``cu_seqlens``; qwin [B, W, Hq, d]; optional proxies [B, Hq, N_p, d].
    One result dict per request."""
    res = []
    for b in range(len(budgets)):
        lo, hi = int(cu_seqlens[b]), int(cu_seqlens[b + 1])
        res.append(select_request(keys[lo:hi], values[lo:hi], qwin[b], int(budgets[b]),
                                  b=b, proxies=None if proxies is None else proxies[b],
                                  **kw))
    return res
