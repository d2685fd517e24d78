"""The per-key selection rule of tests/parity.py, exercised on the CPU.

The oracle's own selection must pass it; a kept set that swaps a key far
from the cutoff for another must fail it, even when the swap is consistent
with the swapped scores; a swap of two keys whose tolerance bands overlap at
the cutoff must pass; keys whose coverage votes are uncertain may move by
their uncertain votes, and no further. Mistakes are planted in the scores fed
to the rule, never in a GPU run.
"""
import numpy as np
import pytest

from paper_2607_22586_gb300 import synth as S
from oracle import mmshift_oracle as O
from tests import parity as PT

WL = S.WORKLOADS["qwen7b-1layer"].replace(seq_lens=(600,), n_visual=(560,), budgets=(64,),
                                          n_q_heads=4, n_kv_heads=1, n_centres=24)


@pytest.fixture(scope="module", params=[O.SCORE_VOTE, O.SCORE_MASS])
def case(request):
    li = S.make_layer(WL, 0)
    h = PT.hyper(n_proxies=64, n_groups=4, score_mode=request.param)
    prox = S.make_proxies(WL, h["n_proxies"], 0)
    ref = PT.oracle_layer(WL, li, h, 0, proxies=prox)[0]
    u = PT.score_bands(ref, h, 0)
    return h, ref, u


@pytest.fixture(autouse=True)
def _keep_log_for_gpu_runs():
    """The planted cases here stay out of the run's selection summary."""
    n = len(PT.SELECTION_LOG)
    yield
    del PT.SELECTION_LOG[n:]


def _own_topk(s, budget):
    T = s.shape[0]
    order = np.lexsort((np.arange(T - 1), -s[:T - 1]))
    return np.sort(np.concatenate([order[:budget - 1], [T - 1]]))


def test_oracle_selection_passes(case):
    h, ref, u = case
    s = ref["scores"][0]
    PT.check_selection(ref["idx"][:, 0], s.astype(np.float32), s, u, 64, "oracle itself")
    assert PT.SELECTION_LOG[-1][1] == 0 and PT.SELECTION_LOG[-1][2] >= 1


def test_far_swap_fails_even_when_self_consistent(case):
    """Drop the best candidate, keep the worst one instead; the GPU-side
    scores are swapped too, so only the band check can catch it."""
    h, ref, u = case
    s = ref["scores"][0].copy()
    T = s.shape[0]
    kept = set(ref["idx"][:, 0].tolist()) - {T - 1}
    best = max(kept, key=lambda t: s[t])
    worst = min(set(range(T - 1)) - kept, key=lambda t: s[t])
    assert s[best] - u[best] > s[worst] + u[worst]
    g = s.copy()
    g[best], g[worst] = s[worst], s[best]
    with pytest.raises(AssertionError, match="not a top-63 of any scores within tolerance"):
        PT.check_selection(_own_topk(g, 64), g, s, u, 64, "planted far swap")


def test_swap_inside_overlapping_bands_passes(case):
    """The oracle's last kept candidate and first dropped one, swapped: allowed
    when (and only when) their bands overlap."""
    h, ref, u = case
    s = ref["scores"][0]
    T = s.shape[0]
    order = np.lexsort((np.arange(T - 1), -s[:T - 1]))
    a, b = order[62], order[63]          # the (C-1)-th kept and the first dropped
    g = s.copy()
    g[a], g[b] = s[b], s[a]
    kept = _own_topk(g, 64)
    if s[a] - u[a] <= s[b] + u[b]:
        PT.check_selection(kept, g, s, u, 64, "swap at the cutoff")
        assert PT.SELECTION_LOG[-1][1] == 2
    else:
        with pytest.raises(AssertionError):
            PT.check_selection(kept, g, s, u, 64, "swap at the cutoff")


def test_band_is_per_key():
    """A key with no uncertain vote cannot move by a vote just because another
    key's vote is uncertain (a band shared by all keys would allow that)."""
    T = 40
    s = np.zeros(T)
    s[:10] = 2.0 + np.linspace(0.01, 0.02, 10)     # vote 2 + anchor
    s[10:30] = 1.0 + np.linspace(0.001, 0.004, 20)  # vote 1 + anchor
    s[30:T - 1] = np.linspace(1e-3, 9e-3, T - 31)   # vote 0 + anchor
    u = PT.RTOL * 0.01 + np.zeros(T)
    u[38] = 1.0 + u[38]                             # one uncertain vote, on a dropped key
    budget = 31                                     # keeps the 30 keys with votes >= 1
    PT.check_selection(_own_topk(s, budget), s.astype(np.float32), s, u, budget, "unperturbed")
    # key 38 may gain its uncertain vote; its anchor then beats key 10's
    g = s.copy()
    g[38] += 1.0
    kept = _own_topk(g, budget)
    assert 38 in kept and 10 not in kept
    PT.check_selection(kept, g, s, u, budget, "uncertain key moves")
    assert PT.SELECTION_LOG[-1][1] == 2
    # key 37 (certain vote 0) in place of key 12 (certain vote 1): outside its band
    g = s.copy()
    g[12], g[37] = s[37], s[12]
    with pytest.raises(AssertionError):
        PT.check_selection(_own_topk(g, budget), g, s, u, budget, "certain key moves")


def test_budget_at_least_length_keeps_all():
    s = np.linspace(1.0, 0.0, 9)
    u = np.full(9, 1e-6)
    PT.check_selection(np.arange(9), s, s, u, 9, "C = T")
    with pytest.raises(AssertionError):
        PT.check_selection(np.arange(1, 9), s, s, u, 9, "C = T, one missing")
