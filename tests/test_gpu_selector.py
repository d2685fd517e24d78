"""The torch-facing KVSelector: each of its paths gives exactly what the C
ABI entry it wraps gives (the entries themselves are checked against the
oracle in the other GPU tests)."""
import numpy as np
import pytest
import torch

import paper_2607_22586_gb300 as M
from paper_2607_22586_gb300 import synth as S
from paper_2607_22586_gb300.selector import KVSelector
from tests import parity as PT

pytestmark = pytest.mark.gpu

WL = S.WORKLOADS["72b-80l-ragged"].replace(
    name="selector", n_layers=2, seq_lens=(700, 1029), n_visual=(650, 1000), budgets=(64, 100),
    n_centres=32)


def _inputs():
    lis = [S.make_layer(WL, l) for l in range(2)]
    K = PT.dev(np.stack([li.K for li in lis]), WL.dtype)
    V = PT.dev(np.stack([li.V for li in lis]), WL.dtype)
    Q = PT.dev(np.stack([li.Qwin for li in lis]), WL.dtype)
    return lis, K, V, Q


def _selector(h):
    return KVSelector(WL.n_q_heads, WL.n_kv_heads, WL.head_dim, WL.window, torch.bfloat16,
                      WL.cu_seqlens(), WL.budgets, n_layers=2, params=PT.abi_params(h))


def test_selector_paths_match_the_entries():
    h = PT.hyper(n_proxies=64, n_groups=4, seed=8)
    lis, K, V, Q = _inputs()
    sel = _selector(h)
    idx, ok, _ = sel(K, V, Q)
    ref = PT.gpu_select(WL, lis, h)
    np.testing.assert_array_equal(PT.host(idx), ref["idx"])
    np.testing.assert_array_equal(PT.host(ok), ref["out_k"])
    sel.poll()

    # prompt-wide statistics
    qf = [S.make_prompt_queries(WL, l, lis[l]) for l in range(2)]
    stats = sel.prefill_stats(PT.dev(np.stack(qf), WL.dtype))
    idx_s = PT.host(sel(K, V, Q, stats=stats)[0]).copy()
    ref_s = PT.gpu_select(WL, lis, h, stats=stats)
    np.testing.assert_array_equal(idx_s, ref_s["idx"])

    # per-head budgets: uniform budgets reproduce the plain selection
    hb = torch.tensor(np.broadcast_to(np.array(WL.budgets, dtype=np.int32)[None, :, None],
                                      (2, WL.batch, WL.n_kv_heads)).copy(), device="cuda")
    idx_b = PT.host(sel(K, V, Q, head_budgets=hb)[0])
    np.testing.assert_array_equal(idx_b, ref["idx"])
    assert np.all(PT.host(sel.out_count) == np.minimum(WL.budgets, WL.seq_lens)[None, :, None])

    # coverage of the last selection
    dec = np.stack([S.make_decode_queries(WL, l, lis[l], 8) for l in range(2)])
    D = PT.dev(np.ascontiguousarray(dec.transpose(0, 1, 3, 2, 4)), WL.dtype)
    cov = PT.host(sel.coverage(K, Q, D))
    assert cov.shape == (2, WL.batch, WL.n_kv_heads, 8)
    assert np.all(cov >= 0.0) and np.all(cov <= 1.0 + 1e-6)
    with pytest.raises(ValueError):
        sel(K, V, Q, stats=stats, head_budgets=hb)
