"""GPU parity of per-layer, per-KV-head budgets (§3.1's C_{l,h}): the budgeted
top-k bit-exact against the oracle on generated scores, the whole selection
against the oracle with given proxies, uniform head budgets equal to the
plain selection, and out-of-range budgets reported."""
import numpy as np
import pytest
import torch

import paper_2607_22586_gb300 as M
from paper_2607_22586_gb300 import synth as S
from paper_2607_22586_gb300 import _lib as LB
from oracle import mmshift_oracle as O
from tests import parity as PT

pytestmark = pytest.mark.gpu

RAGGED = S.WORKLOADS["72b-80l-ragged"].replace(
    name="ragged-small", n_layers=1, seq_lens=(300, 1000, 77, 2), n_visual=(285, 950, 73, 0),
    budgets=(64, 2000, 16, 1), n_centres=32)


def _requests(wl):
    cu = wl.cu_seqlens()
    outs = np.concatenate([[0], np.cumsum(np.minimum(wl.budgets, wl.seq_lens))])
    return [(b, int(cu[b]), int(cu[b + 1]), int(outs[b])) for b in range(wl.batch)]


def _head_budgets(wl, L, seed):
    """Seeded budgets [L, B, Hkv] in [1, C_b], with the extremes present."""
    rng = np.random.default_rng(seed)
    hb = np.empty((L, wl.batch, wl.n_kv_heads), dtype=np.int32)
    for b, c in enumerate(wl.budgets):
        hb[:, b, :] = rng.integers(1, c + 1, size=(L, wl.n_kv_heads))
        hb[0, b, 0] = c
        hb[-1, b, -1] = 1
    return hb


@pytest.mark.parametrize("lens,budgets", [((5000,), (700,)), ((1, 2, 3, 64, 65), (1, 2, 2, 10, 64)),
                                          ((60000,), (4096,)), ((33, 4097), (40, 4097))])
def test_topk_head_budgets_exact(lens, budgets):
    wl = RAGGED.replace(seq_lens=lens, n_visual=tuple(0 for _ in lens), budgets=budgets, n_layers=2)
    T, hkv, L = wl.total_tokens, wl.n_kv_heads, 2
    s = np.stack([S.make_scores(hkv, T, 32, seed=len(lens) + l) for l in range(L)])
    hb = _head_budgets(wl, L, seed=7)
    shape = PT.shape_of(wl, L)
    ws_bytes = M.mmshift_workspace_size(shape, None)
    ws = torch.zeros(ws_bytes, dtype=torch.uint8, device="cuda")
    rows = M.mmshift_output_rows(shape)
    idx = torch.full((L, rows, hkv), -7, dtype=torch.int32, device="cuda")
    cnt = torch.full((L, wl.batch, hkv), -7, dtype=torch.int32, device="cuda")
    M.check(M.mmshift_topk_head_budgets(shape, torch.from_numpy(s).cuda(), torch.from_numpy(hb).cuda(),
                                        idx, cnt, ws, ws_bytes), "topk_head_budgets")
    assert M.mmshift_poll_status(ws) == 0
    idx, cnt = PT.host(idx), PT.host(cnt)
    for l in range(L):
        for b, lo, hi, olo in _requests(wl):
            cap = min(budgets[b], hi - lo)
            ref, rc = O.select_topk_heads(s[l][:, lo:hi].astype(np.float64), hb[l, b], budgets[b])
            np.testing.assert_array_equal(cnt[l, b], rc)
            np.testing.assert_array_equal(idx[l, olo:olo + cap], ref)


def test_select_head_budgets_given_proxies():
    wl = RAGGED
    li = S.make_layer(wl, 0)
    h = PT.hyper(n_proxies=64, n_groups=4)
    prox = S.make_proxies(wl, h["n_proxies"], 0)
    hb = _head_budgets(wl, 1, seed=3)
    shape = PT.shape_of(wl)
    params = PT.abi_params(h)
    rows = M.mmshift_output_rows(shape)
    hkv, d = wl.n_kv_heads, wl.head_dim
    ws_bytes = M.mmshift_workspace_size(shape, params)
    ws = torch.zeros(ws_bytes, dtype=torch.uint8, device="cuda")
    out_idx = torch.full((1, rows, hkv), -7, dtype=torch.int32, device="cuda")
    cnt = torch.full((1, wl.batch, hkv), -7, dtype=torch.int32, device="cuda")
    ok = torch.full((1, rows, hkv, d), 7.0, dtype=torch.bfloat16, device="cuda")
    ov = torch.full_like(ok, 7.0)
    sc = torch.empty((1, hkv, wl.total_tokens), device="cuda")
    dbg = M.make_debug(scores=sc)
    st = M.mmshift_select_head_budgets(shape, PT.dev(li.K[None], wl.dtype), PT.dev(li.V[None], wl.dtype),
                                       PT.dev(li.Qwin[None], wl.dtype), PT.dev(prox[None], wl.dtype),
                                       torch.from_numpy(hb).cuda(), params, out_idx, cnt, ok, ov, dbg,
                                       ws, ws_bytes)
    M.check(st, "select_head_budgets")
    assert M.mmshift_poll_status(ws) == 0
    idx, cnt, ok, sc = PT.host(out_idx)[0], PT.host(cnt)[0], PT.host(ok)[0], PT.host(sc)[0]
    refs = PT.oracle_layer(wl, li, h, 0, proxies=prox)
    for b, lo, hi, olo in _requests(wl):
        T = hi - lo
        cap = min(wl.budgets[b], T)
        ref = refs[b]
        s_ref = ref["scores"]
        for hh in range(hkv):
            c = min(int(hb[0, b, hh]), T)
            assert cnt[b, hh] == c
            got = idx[olo:olo + cap, hh]
            assert np.all(got[c:] == -1), "padding rows"
            kept = got[:c]
            # the head's own budget, checked per key like the uniform case
            u = PT.score_bands(ref, h, hh)
            assert np.all(np.abs(sc[hh, lo:hi] - s_ref[hh]) <= u), f"req {b} head {hh}: scores"
            PT.check_selection(kept, sc[hh, lo:hi], s_ref[hh], u, c, f"head budgets req {b} head {hh}")
            # gathered rows: bit-exact for kept rows, zero for padding
            np.testing.assert_array_equal(ok[olo:olo + c, hh], li.K[lo + kept, hh].astype(np.float32))
            assert np.all(ok[olo + c:olo + cap, hh] == 0.0)


def test_uniform_head_budgets_equal_plain_selection():
    wl = RAGGED.replace(seq_lens=(3000, 1333), n_visual=(2990, 1300), budgets=(256, 64), n_layers=2)
    lis = [S.make_layer(wl, l) for l in range(2)]
    h = PT.hyper(n_proxies=64, n_groups=4, seed=4)
    plain = PT.gpu_select(wl, lis, h)
    hb = np.empty((2, wl.batch, wl.n_kv_heads), dtype=np.int32)
    for b, c in enumerate(wl.budgets):
        hb[:, b, :] = c
    shape = PT.shape_of(wl, 2)
    params = PT.abi_params(h)
    rows = M.mmshift_output_rows(shape)
    ws_bytes = M.mmshift_workspace_size(shape, params)
    ws = torch.zeros(ws_bytes, dtype=torch.uint8, device="cuda")
    idx = torch.empty((2, rows, wl.n_kv_heads), dtype=torch.int32, device="cuda")
    ok = torch.empty((2, rows, wl.n_kv_heads, wl.head_dim), dtype=torch.bfloat16, device="cuda")
    ov = torch.empty_like(ok)
    M.check(M.mmshift_select_head_budgets(shape, PT.dev(np.stack([li.K for li in lis]), wl.dtype),
                                          PT.dev(np.stack([li.V for li in lis]), wl.dtype),
                                          PT.dev(np.stack([li.Qwin for li in lis]), wl.dtype), None,
                                          torch.from_numpy(hb).cuda(), params, idx, None, ok, ov, None,
                                          ws, ws_bytes), "select_head_budgets")
    assert M.mmshift_poll_status(ws) == 0
    np.testing.assert_array_equal(PT.host(idx), plain["idx"])
    np.testing.assert_array_equal(PT.host(ok), plain["out_k"])


def test_out_of_range_head_budget_is_reported_and_clamped():
    wl = RAGGED.replace(seq_lens=(500,), n_visual=(400,), budgets=(32,))
    s = S.make_scores(wl.n_kv_heads, 500, 32, seed=1)[None]
    hb = np.full((1, 1, wl.n_kv_heads), 16, dtype=np.int32)
    hb[0, 0, 1] = 0       # below 1: clamped to 1
    hb[0, 0, 2] = 99      # above the capacity 32: clamped to 32
    shape = PT.shape_of(wl)
    ws_bytes = M.mmshift_workspace_size(shape, None)
    ws = torch.zeros(ws_bytes, dtype=torch.uint8, device="cuda")
    idx = torch.empty((1, 32, wl.n_kv_heads), dtype=torch.int32, device="cuda")
    cnt = torch.empty((1, 1, wl.n_kv_heads), dtype=torch.int32, device="cuda")
    M.check(M.mmshift_topk_head_budgets(shape, torch.from_numpy(s).cuda(), torch.from_numpy(hb).cuda(),
                                        idx, cnt, ws, ws_bytes), "topk_head_budgets")
    assert M.mmshift_poll_status(ws) == LB.MMSHIFT_ERR_DEVICE
    cnt = PT.host(cnt)[0, 0]
    assert cnt[0] == 16 and cnt[1] == 1 and cnt[2] == 32
