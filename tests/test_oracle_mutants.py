"""Plant plausible mistakes in the oracle (on the CPU) and check that the
pins of test_oracle_pins catch every one of them: the pins are only worth
something if a dropped term, a wrong sign, a swapped index or an off-by-one
in the oracle makes at least one of them fail."""
import math

import numpy as np
import pytest

from oracle import mmshift_oracle as O
from tests import test_oracle_pins as P


def _window_stats_ddof0(qwin):
    q = np.asarray(qwin, dtype=np.float64)
    mu = q.mean(axis=0)
    return mu, q.std(axis=0)


def _prefill_stats_ddof0(qfull):
    q = np.asarray(qfull, dtype=np.float64)
    return q.mean(axis=0), q.std(axis=0)


def _proxies_from_stats_sigma_squared(mu, sigma, z, gamma, t_len, dtype, rope_theta=0.0,
                                      rope_pos_offset=0):
    return O.round_to(mu[:, None, :] + gamma * (sigma ** 2)[:, None, :] * z, dtype)


def _build_proxies_no_gamma(qwin, z, gamma, t_len, dtype, rope_theta=0.0, rope_pos_offset=0):
    mu, sigma = O.window_stats(qwin)
    return O.round_to(mu[:, None, :] + sigma[:, None, :] * z, dtype)


def _group_masses_wrong_gqa(proxies, keys, n_groups, scale):
    hq, n_p, d = proxies.shape
    t_len, hkv, _ = keys.shape
    out = np.zeros((hkv, n_groups, t_len))
    gs = n_p // n_groups
    for h in range(hkv):
        for g in range(n_groups):
            rows = proxies[h::hkv, g * gs:(g + 1) * gs].reshape(-1, d)   # hq % Hkv mapping
            out[h, g] = O.softmax_rows((rows @ keys[:, h].T) * scale).sum(axis=0)
    return out


_orig_group_masses = O.group_masses
_orig_anchor = O.anchor_attention
_orig_cover = O.cover_sets
_orig_topk = O.select_topk
_orig_normals = O.proxy_normals
_orig_rope = O.rope_rotate
_orig_philox = O.philox4x64_10


def _group_masses_no_scale(proxies, keys, n_groups, scale):
    return _orig_group_masses(proxies, keys, n_groups, 1.0)


def _anchor_sum(q_last, keys, scale):
    r = q_last.shape[0] // keys.shape[1]
    return _orig_anchor(q_last, keys, scale) * r


def _anchor_first_query(q_last, keys, scale):
    # mistake planted in select_request's choice of query: use a different row
    return _orig_anchor(q_last[::-1].copy(), keys, scale)


def _cover_strict(abar, tau):
    n_groups, t_len = abar.shape
    member = np.zeros((n_groups, t_len), dtype=bool)
    for g in range(n_groups):
        order = np.lexsort((np.arange(t_len), -abar[g]))
        csum = np.cumsum(abar[g][order])
        k = int(np.argmax(csum > tau * csum[-1])) + 1
        member[g, order[:k]] = True
    return member


def _topk_forgets_last(s, budget):
    t_len = s.shape[0]
    if budget >= t_len:
        return np.arange(t_len)
    order = np.lexsort((np.arange(t_len), -s))
    return np.sort(order[:budget])


def _topk_high_t_ties(s, budget):
    t_len = s.shape[0]
    if budget >= t_len:
        return np.arange(t_len)
    cand = np.arange(t_len - 1)
    order = np.lexsort((-cand, -s[:t_len - 1]))
    return np.sort(np.concatenate([order[:budget - 1], [t_len - 1]]))


def _normals_no_two(seed, layer_id, b, n_q_heads, n_proxies, head_dim):
    return _orig_normals(seed, layer_id, b, n_q_heads, n_proxies, head_dim) / math.sqrt(2.0)


def _rope_wrong_sign(x, pos, theta):
    return _orig_rope(x, -pos, theta)


def _round_truncate(x, dtype):
    x = np.asarray(x, dtype=np.float64)
    if dtype == O.F32:
        return x.astype(np.float32).astype(np.float64)
    m, e = np.frexp(x)
    ulp = np.ldexp(1.0, e - 8)
    return np.trunc(x / ulp) * ulp


def _philox_9_rounds(ctr, key):
    c = [np.array(ctr[..., i], dtype=np.uint64) for i in range(4)]
    k0, k1 = np.uint64(key[0]), np.uint64(key[1])
    with np.errstate(over="ignore"):
        for rnd in range(9):
            if rnd:
                k0 = np.uint64((int(k0) + int(O._PHILOX_W0)) & 0xFFFFFFFFFFFFFFFF)
                k1 = np.uint64((int(k1) + int(O._PHILOX_W1)) & 0xFFFFFFFFFFFFFFFF)
            hi0, lo0 = O._mulhilo64(c[0], O._PHILOX_M0)
            hi1, lo1 = O._mulhilo64(c[2], O._PHILOX_M1)
            c = [hi1 ^ c[1] ^ k0, lo1, hi0 ^ c[3] ^ k1, lo0]
    return np.stack(c, axis=-1)


def _hidden_proxies_transposed(mu, sigma, z, w_q, bias, gamma, n_q_heads, pos, dtype,
                               rope_theta=0.0):
    h = O.round_to(mu[None, :] + gamma * sigma[None, :] * z, dtype)
    q = h @ np.asarray(w_q, dtype=np.float64)
    if bias is not None:
        q = q + bias[None, :]
    q = q.reshape(q.shape[0], n_q_heads, -1).transpose(1, 0, 2)
    return O.round_to(q, dtype)


def _hidden_proxies_no_bias(mu, sigma, z, w_q, bias, gamma, n_q_heads, pos, dtype, rope_theta=0.0):
    h = O.round_to(mu[None, :] + gamma * sigma[None, :] * z, dtype)
    q = (h @ np.asarray(w_q, dtype=np.float64).T)
    q = q.reshape(q.shape[0], n_q_heads, -1).transpose(1, 0, 2)
    return O.round_to(q, dtype)


def _hidden_proxies_unrounded_hidden(mu, sigma, z, w_q, bias, gamma, n_q_heads, pos, dtype,
                                     rope_theta=0.0):
    h = mu[None, :] + gamma * sigma[None, :] * z
    q = h @ np.asarray(w_q, dtype=np.float64).T
    if bias is not None:
        q = q + bias[None, :]
    q = q.reshape(q.shape[0], n_q_heads, -1).transpose(1, 0, 2)
    return O.round_to(q, dtype)


def _hidden_normals_query_stream(seed, layer_id, b, n_proxies, d_model):
    return O.proxy_normals(seed, layer_id, b, 1, n_proxies, d_model)[0]


def _coverage_modulo_heads(keys, dec_queries, idx, scale):
    keys = np.asarray(keys, dtype=np.float64)
    dq = np.asarray(dec_queries, dtype=np.float64)
    hkv, hq = keys.shape[1], dq.shape[1]
    out = np.zeros((hq, dq.shape[0]))
    for q in range(hq):
        h = q % hkv
        p = O.softmax_rows(scale * (dq[:, q, :] @ keys[:, h, :].T))
        out[q] = p[:, idx[:, h]].sum(axis=1)
    return out


def _coverage_no_scale(keys, dec_queries, idx, scale):
    keys = np.asarray(keys, dtype=np.float64)
    dq = np.asarray(dec_queries, dtype=np.float64)
    hkv, hq = keys.shape[1], dq.shape[1]
    r = hq // hkv
    out = np.zeros((hq, dq.shape[0]))
    for q in range(hq):
        p = O.softmax_rows(dq[:, q, :] @ keys[:, q // r, :].T)
        out[q] = p[:, idx[:, q // r]].sum(axis=1)
    return out


def _coverage_renormalised_on_kept(keys, dec_queries, idx, scale):
    keys = np.asarray(keys, dtype=np.float64)
    dq = np.asarray(dec_queries, dtype=np.float64)
    hkv, hq = keys.shape[1], dq.shape[1]
    r = hq // hkv
    out = np.zeros((hq, dq.shape[0]))
    for q in range(hq):
        h = q // r
        p = O.softmax_rows(scale * (dq[:, q, :] @ keys[idx[:, h], h, :].T))
        out[q] = p.sum(axis=1)
    return out


def _topk_heads_capacity_everywhere(s, head_budgets, capacity):
    hkv, t_len = s.shape
    idx = np.stack([O.select_topk(s[h], capacity) for h in range(hkv)], axis=1)
    return idx, np.full(hkv, idx.shape[0], dtype=np.int64)


def _topk_heads_drops_last_token(s, head_budgets, capacity):
    hkv, t_len = s.shape
    rows = min(capacity, t_len)
    idx = np.full((rows, hkv), -1, dtype=np.int64)
    counts = np.zeros(hkv, dtype=np.int64)
    for h in range(hkv):
        c = min(int(head_budgets[h]), t_len)
        order = np.lexsort((np.arange(t_len), -s[h]))
        kept = np.sort(order[:c])
        idx[:c, h] = kept
        counts[h] = c
    return idx, counts


_orig_scores = O.scores
_orig_select_request = O.select_request


def _scores_mass_votes(mode, abar, alpha, tau, lam):
    return _orig_scores(O.SCORE_VOTE, abar, alpha, tau, lam)


def _scores_mass_with_anchor(mode, abar, alpha, tau, lam):
    s = _orig_scores(mode, abar, alpha, tau, lam)
    return s + lam * alpha if mode == O.SCORE_MASS else s


def _select_request_stream_zero(keys, values, qwin, budget, **kw):
    kw["b"] = 0
    return _orig_select_request(keys, values, qwin, budget, **kw)


def _select_first_budget(keys, values, qwin, cu_seqlens, budgets, proxies=None, **kw):
    res = []
    for b in range(len(budgets)):
        lo, hi = int(cu_seqlens[b]), int(cu_seqlens[b + 1])
        res.append(O.select_request(keys[lo:hi], values[lo:hi], qwin[b], int(budgets[0]), b=b,
                                    proxies=None if proxies is None else proxies[b], **kw))
    return res


MUTANTS = {
    "std_ddof0": ("window_stats", _window_stats_ddof0),
    "prefill_std_ddof0": ("prefill_stats", _prefill_stats_ddof0),
    "proxies_variance_not_std": ("build_proxies_from_stats", _proxies_from_stats_sigma_squared),
    "no_gamma": ("build_proxies", _build_proxies_no_gamma),
    "gqa_modulo_mapping": ("group_masses", _group_masses_wrong_gqa),
    "no_softmax_scale": ("group_masses", _group_masses_no_scale),
    "anchor_sum_not_mean": ("anchor_attention", _anchor_sum),
    "anchor_wrong_query": ("anchor_attention", _anchor_first_query),
    "cover_strict_inequality": ("cover_sets", _cover_strict),
    "topk_forgets_last_token": ("select_topk", _topk_forgets_last),
    "topk_ties_high_t": ("select_topk", _topk_high_t_ties),
    "box_muller_variance": ("proxy_normals", _normals_no_two),
    "rope_sign": ("rope_rotate", _rope_wrong_sign),
    "bf16_truncation": ("round_to", _round_truncate),
    "philox_9_rounds": ("philox4x64_10", _philox_9_rounds),
    "hidden_projection_transposed": ("hidden_proxies", _hidden_proxies_transposed),
    "hidden_projection_no_bias": ("hidden_proxies", _hidden_proxies_no_bias),
    "hidden_states_not_rounded": ("hidden_proxies", _hidden_proxies_unrounded_hidden),
    "hidden_normals_query_stream": ("hidden_normals", _hidden_normals_query_stream),
    "coverage_modulo_heads": ("attention_coverage", _coverage_modulo_heads),
    "coverage_no_scale": ("attention_coverage", _coverage_no_scale),
    "coverage_renormalised_on_kept": ("attention_coverage", _coverage_renormalised_on_kept),
    "head_budgets_ignored": ("select_topk_heads", _topk_heads_capacity_everywhere),
    "head_budgets_drop_last_token": ("select_topk_heads", _topk_heads_drops_last_token),
    "mass_mode_votes": ("scores", _scores_mass_votes),
    "mass_mode_with_anchor": ("scores", _scores_mass_with_anchor),
    "request_stream_always_zero": ("select_request", _select_request_stream_zero),
    "batch_uses_first_budget": ("select", _select_first_budget),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_mutant_is_caught(name, monkeypatch):
    attr, fn = MUTANTS[name]
    monkeypatch.setattr(O, attr, fn)
    caught = []
    for pin in P.ALL_PINS:
        try:
            pin(O)
        except Exception:
            caught.append(pin.__name__)
    assert caught, f"mutant {name} passed every pin"
