"""Pins of the CPU oracle against facts the paper and mathematics fix.

None of these compare the oracle with itself: each check uses an independent
library routine (numpy's Philox, scipy's softmax / distributions, Python's
statistics module, torch's bf16 rounding), a closed form (Appendix A.2), an
invariant (softmax rows sum to one, shift invariance, permutation
equivariance) or exhaustive brute force on tiny inputs. ``test_oracle_mutants``
plants plausible mistakes in the oracle and checks that these pins catch them.
"""
import itertools
import json
import math
import os
import statistics

import numpy as np
import pytest
import scipy.special
import scipy.stats

from oracle import mmshift_oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# ---------------------------------------------------------------------------
# pin functions (shared with the mutant tests)
# ---------------------------------------------------------------------------
def pin_philox_vs_numpy(orc=O):
    rng = np.random.default_rng(1)
    for _ in range(20):
        key = [int(x) for x in rng.integers(0, 2**63, size=2, dtype=np.uint64)]
        ctr = [int(x) for x in rng.integers(0, 2**63, size=4, dtype=np.uint64)]
        bg = np.random.Philox(key=key, counter=ctr)
        ref = bg.random_raw(8)
        # numpy advances the counter (low word first) before each block
        c1 = np.array([[ctr[0] + 1, ctr[1], ctr[2], ctr[3]],
                       [ctr[0] + 2, ctr[1], ctr[2], ctr[3]]], dtype=np.uint64)
        got = orc.philox4x64_10(c1, key).reshape(-1)
        np.testing.assert_array_equal(got, ref)


def pin_normals_distribution(orc=O):
    z = orc.proxy_normals(seed=7, layer_id=3, b=1, n_q_heads=4, n_proxies=4096, head_dim=64)
    flat = z.reshape(-1)
    n = flat.size
    assert abs(flat.mean()) < 5.0 / math.sqrt(n)
    assert abs(flat.var() - 1.0) < 5.0 * math.sqrt(2.0 / n)
    ks = scipy.stats.kstest(flat[:200000], "norm")
    assert ks.pvalue > 1e-4, ks
    # the two normals of one Box-Muller pair are uncorrelated
    pair = z.reshape(-1, 2)
    corr = np.corrcoef(pair[:, 0], pair[:, 1])[0, 1]
    assert abs(corr) < 5.0 / math.sqrt(pair.shape[0])
    # distinct counters (heads, requests, layers, seeds) give distinct streams
    z2 = orc.proxy_normals(seed=7, layer_id=4, b=1, n_q_heads=4, n_proxies=64, head_dim=64)
    assert not np.allclose(z[:, :64], z2)


def pin_window_stats(orc=O):
    rng = np.random.default_rng(2)
    q = rng.normal(size=(9, 3, 5)) * 3.0 + 1.0
    mu, sigma = orc.window_stats(q)
    for h in range(3):
        for j in range(5):
            col = [float(v) for v in q[:, h, j]]
            assert math.isclose(mu[h, j], statistics.fmean(col), rel_tol=1e-12, abs_tol=1e-12)
            assert math.isclose(sigma[h, j], statistics.stdev(col), rel_tol=1e-12)


def pin_prefill_stats(orc=O):
    """§3.2.1 statistics across all prompt tokens: against a second
    implementation (the statistics module), the closed form of an arithmetic
    progression, the single-token case, and the window path as the special
    case of a prompt that is its own window."""
    rng = np.random.default_rng(21)
    q = rng.normal(size=(37, 2, 4)) * 2.0 - 0.5
    mu, sigma = orc.prefill_stats(q)
    for h in range(2):
        for j in range(4):
            col = [float(v) for v in q[:, h, j]]
            assert math.isclose(mu[h, j], statistics.fmean(col), rel_tol=1e-12, abs_tol=1e-12)
            assert math.isclose(sigma[h, j], statistics.stdev(col), rel_tol=1e-12)
    # x_t = a + c t, t < T: mean a + c (T - 1) / 2, unbiased variance c^2 T (T + 1) / 12
    t_len, a, c = 1000, 0.25, -0.003
    ap = (a + c * np.arange(t_len))[:, None, None] * np.ones((1, 1, 3))
    mu, sigma = orc.prefill_stats(ap)
    assert np.allclose(mu, a + c * (t_len - 1) / 2, rtol=1e-12, atol=1e-15)
    assert np.allclose(sigma ** 2, c * c * t_len * (t_len + 1) / 12, rtol=1e-10)
    mu, sigma = orc.prefill_stats(q[:1])
    assert np.array_equal(mu, q[0]) and np.all(sigma == 0)
    qwin = rng.normal(size=(16, 2, 8))
    z = orc.proxy_normals(seed=5, layer_id=1, b=0, n_q_heads=2, n_proxies=32, head_dim=8)
    w = orc.build_proxies(qwin, z, 3.0, 50, orc.BF16)
    m, sg = orc.prefill_stats(qwin)
    assert np.array_equal(w, orc.build_proxies_from_stats(m, sg, z, 3.0, 50, orc.BF16))


def pin_hidden_proxies(orc=O):
    """§3.2.1 hidden-space proxies q~ = W_Q (mu + gamma sigma z) (+ bias):
    an identity projection reduces them to the query-space expansion; the
    proxies' mean and covariance follow W_Q mu + b and
    gamma^2 W_Q diag(sigma^2) W_Q^T (a non-symmetric W_Q, so a transposed
    operand fails); a difference of two hidden dims below half a bf16 ulp
    survives only if the hidden proxies are rounded before the projection;
    the hidden stream is Philox with key (seed, 1)."""
    rng = np.random.default_rng(31)
    hq, d, n = 3, 8, 40
    dm = hq * d
    mu = rng.normal(size=dm)
    sig = rng.uniform(0.2, 1.5, size=dm)
    z = orc.hidden_normals(seed=9, layer_id=2, b=1, n_proxies=n, d_model=dm)
    got = orc.hidden_proxies(mu, sig, z, np.eye(dm), None, 4.0, hq, 0.0, orc.BF16)
    ref = orc.build_proxies_from_stats(mu.reshape(hq, d), sig.reshape(hq, d),
                                       z.reshape(n, hq, d).transpose(1, 0, 2), 4.0, 100, orc.BF16)
    assert np.array_equal(got, ref)
    # moments over many proxies (float32: rounding far below the CLT band)
    dm, n, gamma = 8, 1 << 15, 2.0
    mu = np.array([0.3, -1.0, 2.0, 0.0, 0.5, -0.25, 1.5, -0.75])
    sig = np.array([0.5, 1.0, 0.25, 2.0, 0.75, 1.25, 0.1, 0.6])
    w = rng.normal(size=(dm, dm))
    bias = rng.normal(size=dm)
    z = orc.hidden_normals(seed=4, layer_id=0, b=0, n_proxies=n, d_model=dm)
    q = orc.hidden_proxies(mu, sig, z, w, bias, gamma, 1, 0.0, orc.F32)[0]   # [N, dm]
    mean_ref = w @ mu + bias
    cov_ref = gamma ** 2 * w @ np.diag(sig ** 2) @ w.T
    sd = np.sqrt(np.diag(cov_ref))
    assert np.all(np.abs(q.mean(axis=0) - mean_ref) < 6.0 * sd / math.sqrt(n))
    cov = np.cov(q.T)
    assert np.all(np.abs(cov - cov_ref) < 8.0 * np.outer(sd, sd) / math.sqrt(n))
    # rounding of H~ before the projection
    mu = np.zeros(8)
    mu[:2] = [1.0 + 0.49 * 2.0 ** -7, 1.0]
    w = np.zeros((8, 8))
    w[0, :2] = [1.0, -1.0]
    q = orc.hidden_proxies(mu, np.zeros(8), np.zeros((1, 8)), w, None, 1.0, 1, 0.0, orc.BF16)
    assert q.shape == (1, 1, 8) and np.all(q == 0.0)
    # the hidden stream is Philox with key (seed, 1)
    # numpy advances the counter before a block: counter (2, 0, 3, 7) is proxy 0, quad 2
    x = np.random.Philox(key=[5, 1], counter=[1, 0, 3, 7]).random_raw(4)
    w32 = np.stack([x & 0xFFFFFFFF, x >> 32], axis=-1).reshape(-1)
    u = orc.uniforms_from_bits(w32)
    zz = np.sqrt(-2.0 * np.log(u[0::2])) * np.cos(2.0 * np.pi * u[1::2])
    z = orc.hidden_normals(seed=5, layer_id=7, b=3, n_proxies=1, d_model=64)
    assert math.isclose(z[0, 4 * 2], zz[0], rel_tol=1e-12)


def pin_attention_coverage(orc=O):
    """Fig. 1b's attention mass coverage: every key kept gives 1; a set and
    its complement sum to 1; two keys give the logistic of their scaled logit
    gap; a query's own top-C keys cover more than any other C-subset (brute
    force); query heads 0-1 read KV head 0 (uniform keys: coverage C/T), heads
    2-3 KV head 1 (one dominant key)."""
    rng = np.random.default_rng(41)
    t_len, hkv, hq, d = 9, 2, 4, 8
    keys = rng.normal(size=(t_len, hkv, d))
    dq = rng.normal(size=(5, hq, d))
    every = np.repeat(np.arange(t_len)[:, None], hkv, axis=1)
    assert np.allclose(orc.attention_coverage(keys, dq, every, 0.3), 1.0, rtol=0, atol=1e-12)
    kept = np.array([[0, 1], [3, 4], [7, 8]])
    rest = np.array([[t for t in range(t_len) if t not in kept[:, h]] for h in range(hkv)]).T
    tot = orc.attention_coverage(keys, dq, kept, 0.3) + orc.attention_coverage(keys, dq, rest, 0.3)
    assert np.allclose(tot, 1.0, rtol=0, atol=1e-12)
    # two keys: coverage of key 0 = 1 / (1 + exp(-scale * (q.k0 - q.k1)))
    k2 = rng.normal(size=(2, 1, d))
    q2 = rng.normal(size=(3, 1, d))
    scale = 1.0 / math.sqrt(d)
    gap = (q2[:, 0, :] @ k2[0, 0]) - (q2[:, 0, :] @ k2[1, 0])
    got = orc.attention_coverage(k2, q2, np.array([[0]]), scale)[0]
    assert np.allclose(got, 1.0 / (1.0 + np.exp(-scale * gap)), rtol=1e-12)
    # brute force: the query's own top-C keys are the best C-subset
    q1 = dq[:1, :1, :]
    k1 = keys[:, :1, :]
    logits = (q1[0, 0] @ k1[:, 0, :].T) * 0.3
    best = np.sort(np.argsort(-logits)[:3])
    cov_best = orc.attention_coverage(k1, q1, best[:, None], 0.3)[0, 0]
    for sub in itertools.combinations(range(t_len), 3):
        c = orc.attention_coverage(k1, q1, np.array(sub)[:, None], 0.3)[0, 0]
        assert c <= cov_best + 1e-12
    # GQA: heads 0-1 -> KV head 0 (uniform), heads 2-3 -> KV head 1 (dominant key 5)
    kk = np.zeros((t_len, hkv, d))
    kk[:, 1, :] = rng.normal(size=(t_len, d)) * 0.01
    qq = np.ones((2, hq, d))
    kk[5, 1, :] = 50.0
    sel = np.array([[0, 5], [1, 6], [2, 7]])
    cov = orc.attention_coverage(kk, qq, sel, 1.0)
    assert np.allclose(cov[:2], 3.0 / t_len, rtol=0, atol=1e-12)
    assert np.all(cov[2:] > 1.0 - 1e-12)


def pin_head_budgets(orc=O):
    """Per-head budgets (§3.1's C_{l,h}): equal budgets reproduce the uniform
    selection; each head keeps exactly min(C_h, T) tokens, its own top ones
    (brute force over subsets: no other set of that size containing T-1 has
    a larger score sum), the rest of its rows -1; a smaller budget keeps a
    subset of a larger one's tokens; padded rows gather zeros."""
    rng = np.random.default_rng(53)
    hkv, t_len = 3, 10
    s = rng.integers(0, 4, size=(hkv, t_len)).astype(np.float64) + rng.random((hkv, t_len)) * 0.5
    idx_u = np.stack([orc.select_topk(s[h], 4) for h in range(hkv)], axis=1)
    idx_e, cnt_e = orc.select_topk_heads(s, [4, 4, 4], 4)
    assert np.array_equal(idx_u, idx_e) and np.array_equal(cnt_e, [4, 4, 4])
    idx, cnt = orc.select_topk_heads(s, [1, 3, 6], 6)
    assert idx.shape == (6, hkv) and np.array_equal(cnt, [1, 3, 6])
    for h, c in enumerate([1, 3, 6]):
        kept = idx[:c, h]
        assert np.all(idx[c:, h] == -1) and kept[-1] == t_len - 1 and np.all(np.diff(kept) > 0)
        best = max(sum(s[h][list(sub)]) for sub in itertools.combinations(range(t_len - 1), c - 1))
        assert math.isclose(s[h][kept[:-1]].sum(), best, rel_tol=0, abs_tol=1e-12)
    small, _ = orc.select_topk_heads(s, [2, 2, 2], 6)
    assert set(idx[:1, 0]) <= set(small[:2, 0])
    for h in (1, 2):
        assert set(small[:2, h]) <= set(idx[:cnt[h], h])
    keys = rng.normal(size=(t_len, hkv, 4))
    ok, ov = orc.gather(keys, keys, idx)
    assert np.all(ok[1:, 0] == 0.0) and np.array_equal(ok[:3, 1], keys[idx[:3, 1], 1])


def pin_sampler_closed_form(orc=O):
    """Appendix A.2: for q ~ N(mu, Sigma), E[exp(q.k/sqrt d)] =
    exp(mu.k/sqrt d + k^T Sigma k / (2d)). With Sigma = diag((gamma*sigma)^2)
    the proxies' Monte-Carlo mean must match within its CLT band."""
    rng = np.random.default_rng(3)
    d, w, n_p = 16, 8, 1 << 16
    qwin = rng.normal(size=(w, 1, d)) * 0.3 + 0.2
    z = orc.proxy_normals(seed=11, layer_id=0, b=0, n_q_heads=1, n_proxies=n_p, head_dim=d)
    gamma = 2.0
    prox = orc.build_proxies(qwin, z, gamma, t_len=100, dtype=orc.F32)[0]   # [Np, d]
    mu = qwin[:, 0, :].mean(axis=0)
    sig = qwin[:, 0, :].std(axis=0, ddof=1)
    # per-dimension moments of the proxies: mean mu, std gamma*sigma
    np.testing.assert_allclose(prox.mean(axis=0), mu, atol=6.0 * gamma * sig.max() / math.sqrt(n_p))
    np.testing.assert_allclose(prox.std(axis=0), gamma * sig, rtol=6.0 / math.sqrt(2 * n_p))
    for _ in range(4):
        k = rng.normal(size=d) * 0.5
        e = np.exp(prox @ k / math.sqrt(d))
        closed = math.exp(mu @ k / math.sqrt(d) + np.sum((gamma * sig) ** 2 * k ** 2) / (2 * d))
        se = e.std() / math.sqrt(n_p)
        assert abs(e.mean() - closed) < 6.0 * se, (e.mean(), closed, se)


def pin_rope(orc=O):
    rng = np.random.default_rng(4)
    d, theta = 16, 10000.0
    x = rng.normal(size=(3, d))
    pos = 37.0
    got = orc.rope_rotate(x, pos, theta)
    half = d // 2
    zc = (x[:, :half] + 1j * x[:, half:]) * np.exp(1j * pos * theta ** (-2.0 * np.arange(half) / d))
    np.testing.assert_allclose(got, np.concatenate([zc.real, zc.imag], axis=1), atol=1e-12)
    np.testing.assert_allclose(np.linalg.norm(got, axis=1), np.linalg.norm(x, axis=1), rtol=1e-12)
    # relative-position property: <R_m q, R_n k> depends on m - n only
    q, k = x[0], x[1]
    a = orc.rope_rotate(q, 50.0, theta) @ orc.rope_rotate(k, 20.0, theta)
    b = orc.rope_rotate(q, 130.0, theta) @ orc.rope_rotate(k, 100.0, theta)
    assert math.isclose(a, b, rel_tol=1e-9, abs_tol=1e-12)


def pin_round_bf16(orc=O):
    import torch
    rng = np.random.default_rng(5)
    x = (rng.normal(size=20000) * 10.0 ** rng.uniform(-6, 6, size=20000)).astype(np.float32)
    ref = torch.from_numpy(x).to(torch.bfloat16).to(torch.float64).numpy()
    np.testing.assert_array_equal(orc.round_to(x.astype(np.float64), orc.BF16), ref)
    # exact halfway cases go to the even neighbour
    one = 1.0
    ulp = 2.0 ** -7
    halfway = np.array([one + ulp / 2, one + 3 * ulp / 2, -(one + ulp / 2)])
    np.testing.assert_array_equal(orc.round_to(halfway, orc.BF16),
                                  np.array([one, one + 2 * ulp, -one]))


def _tiny_problem(seed, t_len=40, hq=4, hkv=2, d=8, n_p=8, scale_k=1.0):
    rng = np.random.default_rng(seed)
    keys = rng.normal(size=(t_len, hkv, d)) * scale_k
    proxies = rng.normal(size=(hq, n_p, d)) * 2.0
    q_last = rng.normal(size=(hq, d))
    return keys, proxies, q_last


def pin_mass_totals(orc=O):
    keys, proxies, q_last = _tiny_problem(6)
    hq, n_p, d = proxies.shape
    hkv = keys.shape[1]
    r = hq // hkv
    scale = 1.0 / math.sqrt(d)
    a = orc.softmax_rows(rng_logits := np.random.default_rng(6).normal(size=(5, 30)) * 20)
    np.testing.assert_allclose(a.sum(axis=1), 1.0, atol=1e-12)
    np.testing.assert_allclose(a, scipy.special.softmax(rng_logits, axis=1), rtol=1e-12, atol=1e-300)
    for n_groups in (1, 2, 4, 8):
        abar = orc.group_masses(proxies, keys, n_groups, scale)
        gs = n_p // n_groups
        np.testing.assert_allclose(abar.sum(axis=2), gs * r, rtol=1e-12)
        np.testing.assert_allclose(abar.sum(axis=(1, 2)), n_p * r, rtol=1e-12)
    alpha = orc.anchor_attention(q_last, keys, scale)
    np.testing.assert_allclose(alpha.sum(axis=1), 1.0, rtol=1e-12)


def pin_sigma_zero_single_query(orc=O):
    """Identical window queries: sigma = 0, every proxy equals mu, and each
    group mass is gs * (sum over the r heads of) one softmax row."""
    rng = np.random.default_rng(7)
    t_len, hq, hkv, d, w, n_p, n_groups = 50, 6, 2, 8, 5, 8, 2
    r = hq // hkv
    keys = rng.normal(size=(t_len, hkv, d))
    qrow = rng.normal(size=(hq, d))
    qwin = np.repeat(qrow[None], w, axis=0)
    z = rng.normal(size=(hq, n_p, d))
    prox = orc.build_proxies(qwin, z, 10.0, t_len, orc.F32)
    np.testing.assert_allclose(prox, np.broadcast_to(orc.round_to(qrow, orc.F32)[:, None, :], prox.shape))
    abar = orc.group_masses(prox, keys, n_groups, 1.0 / math.sqrt(d))
    gs = n_p // n_groups
    for h in range(hkv):
        heads = [hh for hh in range(hq) if hh // r == h]
        expect = sum(scipy.special.softmax(prox[hh, 0] @ keys[:, h, :].T / math.sqrt(d)) for hh in heads) * gs
        for g in range(n_groups):
            np.testing.assert_allclose(abar[h, g], expect, rtol=1e-10)


def pin_shift_and_permutation(orc=O):
    keys, proxies, q_last = _tiny_problem(8, t_len=30)
    t_len, hkv, d = keys.shape
    hq = proxies.shape[0]
    qwin = np.concatenate([np.random.default_rng(9).normal(size=(3, hq, d)), q_last[None]], axis=0)
    kw = dict(n_proxies=proxies.shape[1], n_groups=2, proxies=proxies, dtype=orc.F32, tau=0.9)
    base = orc.select_request(keys, keys, qwin, 12, **kw)
    # same vector added to every key of a head: every softmax row is unchanged
    u = np.random.default_rng(10).normal(size=(1, hkv, d)) * 3.0
    sh = orc.select_request(keys + u, keys, qwin, 12, **kw)
    np.testing.assert_allclose(sh["group_mass"], base["group_mass"], rtol=1e-9, atol=1e-300)
    np.testing.assert_allclose(sh["anchor"], base["anchor"], rtol=1e-9, atol=1e-300)
    np.testing.assert_array_equal(sh["idx"], base["idx"])
    # permuting the keys permutes masses and scores
    perm = np.random.default_rng(11).permutation(t_len - 1)
    perm = np.concatenate([perm, [t_len - 1]])
    pm = orc.select_request(keys[perm], keys[perm], qwin, 12, **kw)
    np.testing.assert_allclose(pm["group_mass"], base["group_mass"][:, :, perm], rtol=1e-9, atol=1e-300)
    np.testing.assert_allclose(pm["scores"], base["scores"][:, perm], rtol=1e-9, atol=1e-300)
    for h in range(hkv):
        assert set(perm[pm["idx"][:, h]]) == set(base["idx"][:, h])


def pin_budget_ge_t(orc=O):
    keys, proxies, q_last = _tiny_problem(12, t_len=17)
    qwin = np.stack([q_last, q_last * 0.5, q_last], axis=0)
    for budget in (17, 18, 1000):
        res = orc.select_request(keys, keys, qwin, budget, n_proxies=8, n_groups=4,
                                 proxies=proxies, dtype=orc.F32)
        for h in range(keys.shape[1]):
            np.testing.assert_array_equal(res["idx"][:, h], np.arange(17))
    res = orc.select_request(keys, keys, qwin, 1, n_proxies=8, n_groups=4, proxies=proxies,
                             dtype=orc.F32)
    np.testing.assert_array_equal(res["idx"], np.full((1, keys.shape[1]), 16))


def pin_lastattn(orc=O):
    """tau = 1 puts every key with positive mass in every cover set, so all
    votes tie at G and the ranking is the last query's attention alone (the
    'LastAttn' row of Table 5)."""
    rng = np.random.default_rng(13)
    t_len, hq, hkv, d = 60, 4, 2, 8
    r = hq // hkv
    keys = rng.normal(size=(t_len, hkv, d))
    qwin = rng.normal(size=(4, hq, d))
    proxies = rng.normal(size=(hq, 8, d))
    budget = 20
    res = orc.select_request(keys, keys, qwin, budget, n_proxies=8, n_groups=4, tau=1.0,
                             proxies=proxies, dtype=orc.F32)
    assert np.all(res["scores"] >= 4.0)
    for h in range(hkv):
        heads = [hh for hh in range(hq) if hh // r == h]
        att = np.mean([scipy.special.softmax(qwin[-1, hh] @ keys[:, h].T / math.sqrt(d)) for hh in heads], axis=0)
        np.testing.assert_allclose(res["anchor"][h], att, rtol=1e-12)
        top = np.argsort(-att[:t_len - 1], kind="stable")[:budget - 1]
        np.testing.assert_array_equal(res["idx"][:, h], np.sort(np.concatenate([top, [t_len - 1]])))


def pin_uniform_keys(orc=O):
    t_len, d = 100, 8
    keys = np.ones((t_len, 1, d))
    proxies = np.random.default_rng(14).normal(size=(2, 8, d))
    abar = orc.group_masses(proxies, keys, 2, 1.0 / math.sqrt(d))
    assert np.all(abar == abar[:, :, :1])
    member = orc.cover_sets(abar[0], 0.955)
    for g in range(2):
        np.testing.assert_array_equal(np.nonzero(member[g])[0], np.arange(96))


def _brute_cover(mass, tau):
    t_len = mass.size
    total = mass.sum()
    for size in range(0, t_len + 1):
        ok = [set(c) for c in itertools.combinations(range(t_len), size)
              if mass[list(c)].sum() >= tau * total - 1e-12]
        if ok:
            return size, ok
    raise AssertionError


def pin_cover_bruteforce(orc=O):
    rng = np.random.default_rng(15)
    for trial in range(60):
        t_len = int(rng.integers(1, 10))
        mass = rng.integers(0, 5, size=(2, t_len)).astype(np.float64)
        mass[:, 0] += 1.0                         # no all-zero group
        tau = float(rng.choice([0.3, 0.5, 0.7, 0.9, 1.0]))
        member = orc.cover_sets(mass, tau)
        for g in range(2):
            chosen = set(np.nonzero(member[g])[0].tolist())
            size, ok = _brute_cover(mass[g], tau)
            assert len(chosen) == size, (mass[g], tau, chosen, size)
            assert chosen in ok
            # prefix of the (mass desc, t asc) ranking
            for t in chosen:
                for u in set(range(t_len)) - chosen:
                    assert mass[g, t] > mass[g, u] or (mass[g, t] == mass[g, u] and t < u)


def pin_cover_last_member_bound(orc=O):
    """At realistic sizes: the tau-cover set is a prefix of the (mass desc, t
    asc) order whose mass reaches tau * total while the same prefix without
    its last member does not, and that last member's mass exceeds
    (1 - tau) * total / n (the members before it hold less than tau * total,
    the at most n - 1 keys after it at most its mass each)."""
    rng = np.random.default_rng(23)
    for n in (50, 700, 3000):
        for tau in (0.5, 0.9, 0.95, 0.99):
            mass = np.exp(rng.normal(0.0, 3.0, size=(3, n)))
            mass[1, rng.random(n) < 0.5] = 0.0              # many zero keys
            mass[2] = np.round(mass[2] * 4.0) / 4.0         # many ties
            mass[2, 0] += 1.0
            member = orc.cover_sets(mass, tau)
            for g in range(3):
                m, c = mass[g], member[g]
                order = np.lexsort((np.arange(n), -m))
                k = int(c.sum())
                assert c[order[:k]].all() and not c[order[k:]].any()
                total = m.sum()
                assert m[order[:k]].sum() >= tau * total * (1 - 1e-12)
                assert m[order[:k - 1]].sum() < tau * total
                assert m[order[k - 1]] > (1.0 - tau) * total / n


def pin_topk_bruteforce(orc=O):
    rng = np.random.default_rng(16)
    for trial in range(80):
        t_len = int(rng.integers(1, 10))
        s = rng.integers(0, 4, size=t_len).astype(np.float64) + 0.25 * rng.integers(0, 2, size=t_len)
        for budget in range(1, t_len + 2):
            got = orc.select_topk(s, budget)
            if budget >= t_len:
                np.testing.assert_array_equal(got, np.arange(t_len))
                continue
            assert got[-1] == t_len - 1 and np.all(np.diff(got) > 0)
            cand = [int(t) for t in got[:-1]]
            best = max(sum(s[list(c)]) for c in itertools.combinations(range(t_len - 1), budget - 1))
            assert math.isclose(sum(s[cand]), best)
            # among the best sets the lowest indices win ties
            bests = sorted(sorted(c) for c in itertools.combinations(range(t_len - 1), budget - 1)
                           if math.isclose(sum(s[list(c)]), best))
            assert cand == list(bests[0])


def pin_mass_scores_bruteforce(orc=O):
    """MASS scoring (Table 5's "+ Var. Exp." row): S_t is the attention mass
    of all proxies of the r grouped heads, summed. Against a brute loop over
    heads, proxies and keys with math.exp (no softmax routine, no grouping);
    the grouping must not matter, nor the order of the groups, nor the anchor."""
    keys, proxies, q_last = _tiny_problem(31, t_len=12, hq=4, hkv=2, d=4, n_p=6)
    t_len, hkv, d = keys.shape
    hq, n_p, _ = proxies.shape
    r = hq // hkv
    scale = 0.7
    brute = np.zeros((hkv, t_len))
    for hh in range(hq):
        for i in range(n_p):
            lg = [scale * sum(proxies[hh, i, j] * keys[t, hh // r, j] for j in range(d))
                  for t in range(t_len)]
            mx = max(lg)
            ex = [math.exp(x - mx) for x in lg]
            z = math.fsum(ex)
            for t in range(t_len):
                brute[hh // r, t] += ex[t] / z
    alpha = orc.anchor_attention(q_last, keys, scale)
    for n_groups in (1, 2, 3, 6):
        abar = orc.group_masses(proxies, keys, n_groups, scale)
        for h in range(hkv):
            s = orc.scores(orc.SCORE_MASS, abar[h], alpha[h], 0.9, 1.0)
            np.testing.assert_allclose(s, brute[h], rtol=1e-12)
            rev = orc.scores(orc.SCORE_MASS, abar[h][::-1], alpha[h] * 7.0, 0.5, 3.0)
            np.testing.assert_allclose(rev, brute[h], rtol=1e-12)
    # the whole method in MASS mode keeps T-1 and the top C-1 of that mass
    qwin = np.stack([q_last * 0.3, q_last], axis=0)
    res = orc.select_request(keys, keys, qwin, 5, n_proxies=n_p, n_groups=3, proxies=proxies,
                             dtype=orc.F32, softmax_scale=scale, score_mode=orc.SCORE_MASS)
    np.testing.assert_allclose(res["scores"], brute, rtol=1e-12)
    for h in range(hkv):
        top = sorted(range(t_len - 1), key=lambda t: (-brute[h, t], t))[:4]
        assert res["idx"][:, h].tolist() == sorted(top + [t_len - 1])


def pin_request_streams_and_slicing(orc=O):
    """A packed batch (Algorithm 1 runs per request): request b draws its
    proxies from Philox counter (i*d/8 + q, hq, b, layer) -- pinned against
    numpy's independent Philox and a Box-Muller written out with math.log /
    math.cos -- and each request's result depends only on its own slice of
    keys, queries and budget."""
    seed, layer, hq_n, n_p, d = 5, 3, 2, 3, 16
    nq = d // 8
    for b in (0, 1, 4):
        z = orc.proxy_normals(seed, layer, b, hq_n, n_p, d)
        for hq in range(hq_n):
            for i in range(n_p):
                for q in range(nq):
                    c0 = i * nq + q
                    if c0 == 0:
                        continue   # numpy would carry c0 - 1 into the next word
                    # numpy's Philox advances the counter before its first block
                    bg = np.random.Philox(key=[seed, 0], counter=[c0 - 1, hq, b, layer])
                    raw = bg.random_raw(4)
                    words = []
                    for v in raw.tolist():
                        words += [v & 0xFFFFFFFF, v >> 32]
                    u = [((w >> 9) + 0.5) * 2.0 ** -23 for w in words]
                    want = []
                    for m in range(4):
                        rad = math.sqrt(-2.0 * math.log(u[2 * m]))
                        ang = 2.0 * math.pi * u[2 * m + 1]
                        want += [rad * math.cos(ang), rad * math.sin(ang)]
                    got = [z[hq, i, 4 * q + k] for k in range(4)] + \
                          [z[hq, i, d // 2 + 4 * q + k] for k in range(4)]
                    np.testing.assert_allclose(got, want, rtol=1e-12, atol=1e-13)
    # slicing: three requests packed; request results depend on their own slice
    rng = np.random.default_rng(33)
    hq, hkv, d, w = 4, 2, 8, 3
    lens, budgets = (9, 14, 6), (4, 20, 2)
    cu = np.concatenate([[0], np.cumsum(lens)])
    keys = rng.normal(size=(cu[-1], hkv, d))
    vals = rng.normal(size=(cu[-1], hkv, d))
    qwin = rng.normal(size=(3, w, hq, d))
    kw = dict(n_proxies=8, n_groups=2, seed=2, layer_id=1, dtype=orc.F32, tau=0.9)
    res = orc.select(keys, vals, qwin, cu, budgets, **kw)
    keys2 = keys.copy()
    keys2[cu[0]:cu[1]] = rng.normal(size=(lens[0], hkv, d))   # change request 0 only
    qwin2 = qwin.copy()
    qwin2[0] = rng.normal(size=(w, hq, d))
    res2 = orc.select(keys2, vals, qwin2, cu, budgets, **kw)
    for b in (1, 2):
        for k in ("proxies", "group_mass", "scores", "idx", "out_k", "out_v"):
            np.testing.assert_array_equal(res2[b][k], res[b][k])
    assert not np.array_equal(res2[0]["group_mass"], res[0]["group_mass"])
    for b in range(3):
        assert res[b]["idx"].shape == (min(budgets[b], lens[b]), hkv)
        assert res[b]["idx"].max() == lens[b] - 1 and res[b]["idx"].min() >= 0
        # kept rows are the request's own rows
        lo = cu[b]
        h = np.arange(hkv)[None]
        np.testing.assert_array_equal(res[b]["out_v"], vals[lo + res[b]["idx"], h])
    # the same request content at another batch position draws other proxies
    alone = orc.select_request(keys[cu[1]:cu[2]], vals[cu[1]:cu[2]], qwin[1], budgets[1], b=0, **kw)
    assert not np.array_equal(alone["proxies"], res[1]["proxies"])
    alone1 = orc.select_request(keys[cu[1]:cu[2]], vals[cu[1]:cu[2]], qwin[1], budgets[1], b=1, **kw)
    np.testing.assert_array_equal(alone1["proxies"], res[1]["proxies"])


ALL_PINS = [pin_philox_vs_numpy, pin_normals_distribution, pin_window_stats, pin_prefill_stats,
            pin_hidden_proxies, pin_attention_coverage, pin_head_budgets,
            pin_sampler_closed_form, pin_rope, pin_round_bf16, pin_mass_totals,
            pin_sigma_zero_single_query, pin_shift_and_permutation, pin_budget_ge_t,
            pin_lastattn, pin_uniform_keys, pin_cover_bruteforce, pin_cover_last_member_bound,
            pin_topk_bruteforce,
            pin_mass_scores_bruteforce, pin_request_streams_and_slicing]


@pytest.mark.parametrize("pin", ALL_PINS, ids=[p.__name__ for p in ALL_PINS])
def test_pin(pin):
    pin()


def test_defaults_match_paper():
    with open(os.path.join(GOLDEN, "hyperparams.json")) as f:
        g = json.load(f)
    assert O.DEFAULTS["n_proxies"] == g["n_proxies"]
    assert O.DEFAULTS["n_groups"] == g["n_groups"]
    assert g["n_proxies"] // g["n_groups"] == g["group_size"]
    assert O.DEFAULTS["gamma"] == g["gamma"]
    assert O.DEFAULTS["tau"] == g["tau"]
    assert O.DEFAULTS["lam"] == g["lambda"]
