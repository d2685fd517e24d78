"""GPU parity of the hidden-space proxies (§3.2.1, the paper's own
construction: proxy hidden states from the prefill hidden-state statistics,
projected by W_Q, placed by RoPE) against the oracle, through the C ABI:
mmshift_hidden_stats, mmshift_build_hidden_proxies, and selection with the
proxies they make.

Tolerance of the projected proxies. Both sides draw the same normals; the
GPU forms mu + gamma*sigma*z in fp32 and rounds it to bf16, the oracle in
fp64, so a hidden-state element whose fp64 value lies within the fp32
sampling error (2e-6 of |mu| + gamma*sigma*(1+|z|)) of a bf16 rounding
boundary may round the other way; the oracle marks those elements U from its
own values. The projection accumulates d_model products in fp32 (order
unspecified): off by at most ~d_model * 2^-24 of sum_k |h_k w_jk|, bounded
here by 2^-17 of it. So before RoPE the error of feature j is at most
  e_j = sum_{k in U} |w_jk| ulp(h_k) + 2^-17 sum_k |h_k w_jk|,
RoPE mixes the two features of a pair (|cos|, |sin| <= 1): e_x + e_y, and
the final bf16 rounding adds one ulp. Every proxy must lie within that
bound, and at most 2% may differ at all.
"""
import numpy as np
import pytest
import torch

import paper_2607_22586_gb300 as M
from paper_2607_22586_gb300 import synth as S
from oracle import mmshift_oracle as O
from tests import parity as PT

pytestmark = pytest.mark.gpu

QWEN1 = S.WORKLOADS["qwen7b-1layer"]


def _bf16_ulp(x):
    _, e = np.frexp(np.abs(x))
    return np.ldexp(1.0, e - 8)


def _stats(wl, h, layers=1):
    """Oracle hidden-state statistics per (layer, request): [L, B, 2, d_model]."""
    cu = wl.cu_seqlens()
    st = np.zeros((layers, wl.batch, 2, h[0].shape[1]), dtype=np.float32)
    for l in range(layers):
        for b in range(wl.batch):
            mu, sg = O.prefill_stats(h[l][cu[b]:cu[b + 1]])
            st[l, b, 0], st[l, b, 1] = mu, sg
    return st


def _gpu_hidden_proxies(wl, d_model, stats, ws_list, bias_list, h, rope_pos=None, wq_stride=0):
    L = len(ws_list)
    shape = PT.shape_of(wl, L)
    F = wl.n_q_heads * wl.head_dim
    stride = wq_stride or F * d_model
    wflat = np.zeros((L, stride), dtype=np.float32)
    for l, w in enumerate(ws_list):
        wflat[l, :F * d_model] = w.reshape(-1)
    W = PT.dev(wflat, wl.dtype)
    bias = None
    if bias_list[0] is not None:
        bias = PT.dev(np.stack(bias_list), wl.dtype)
    params = PT.abi_params(h)
    ws_bytes = M.mmshift_hidden_proxies_workspace_size(shape, d_model, params)
    ws = torch.zeros(ws_bytes, dtype=torch.uint8, device="cuda")
    out = torch.full((L, wl.batch, wl.n_q_heads, h["n_proxies"], wl.head_dim), float("nan"),
                     dtype=torch.bfloat16, device="cuda")
    st = torch.from_numpy(np.ascontiguousarray(stats)).cuda()
    M.check(M.mmshift_build_hidden_proxies(shape, d_model, st, W, wq_stride, bias, rope_pos, params,
                                           out, ws, ws_bytes), "build_hidden_proxies")
    M.check(M.mmshift_poll_status(ws), "status")
    torch.cuda.synchronize()
    return PT.host(out).astype(np.float64)


def _check_projection(got, stats, w, bias, h, b, pos, hq, layer_id):
    """One (layer, request): got [Hq, N, d] against the oracle's."""
    mu, sg = stats[0].astype(np.float64), stats[1].astype(np.float64)
    dm = mu.shape[0]
    z = O.hidden_normals(h["seed"], layer_id, b, h["n_proxies"], dm)
    ref = O.hidden_proxies(mu, sg, z, w, bias, h["gamma"], hq, pos, O.BF16, h["rope_theta"])
    # oracle-side uncertainty of the bf16 hidden states
    x64 = mu[None, :] + h["gamma"] * sg[None, :] * z
    hs = O.round_to(x64, O.BF16)
    eps = 2e-6 * (np.abs(mu)[None, :] + h["gamma"] * sg[None, :] * (1.0 + np.abs(z)))
    other = O.round_to(x64 + np.sign(x64 - hs) * eps, O.BF16)   # the value across a near boundary
    unc = other != hs
    wa = np.abs(np.asarray(w, dtype=np.float64))
    e = (unc * _bf16_ulp(np.maximum(np.abs(hs), 1e-30))) @ wa.T + 2.0 ** -17 * (np.abs(hs) @ wa.T)
    if bias is not None:
        e = e + 2.0 ** -20 * np.abs(np.asarray(bias, dtype=np.float64))[None, :]
    d = ref.shape[-1]
    e = e.reshape(e.shape[0], hq, d).transpose(1, 0, 2)
    if h["rope_theta"] > 0.0:
        # rotation mixes the pair; fp32 cos / sin add about 2^-22 of the pair's size
        pair = np.abs(ref[..., :d // 2]) + np.abs(ref[..., d // 2:])
        e = np.concatenate([e[..., :d // 2] + e[..., d // 2:] + 2.0 ** -19 * pair] * 2, axis=-1)
    bound = e + _bf16_ulp(np.maximum(np.abs(ref), np.abs(got))) * 1.0001
    diff = np.abs(got - ref)
    assert np.all(np.isfinite(got)), "unwritten proxies"
    assert np.all(diff <= bound), f"proxy off by {np.max(diff / bound):.3g} x bound"
    frac = np.mean(diff > 0)
    assert frac <= 2e-2, f"{frac:.3g} of proxies differ"
    return frac


CASES = [
    # (name, workload, d_model, n_proxies, bias, rope_theta)
    ("qwen7b-d3584-bias", QWEN1, 3584, 512, True, 0.0),
    ("qwen7b-d3584-rope", QWEN1, 3584, 512, True, 1e6),
    ("d64-heads-ragged-N", S.WORKLOADS["tiny-f32"].replace(dtype=S.BF16, n_q_heads=6, n_kv_heads=2,
                                                            seq_lens=(700, 33), n_visual=(650, 0),
                                                            budgets=(64, 8)), 512, 100, False, 1e4),
    ("d128-8heads", QWEN1.replace(n_q_heads=8, n_kv_heads=2, seq_lens=(1500,), n_visual=(1400,),
                                  budgets=(200,)), 1024, 256, True, 0.0),
]


@pytest.mark.parametrize("name,wl,dm,n_p,with_bias,rope", CASES, ids=[c[0] for c in CASES])
def test_hidden_proxies_match_oracle(name, wl, dm, n_p, with_bias, rope):
    h = PT.hyper(n_proxies=n_p, n_groups=max(1, n_p // 16) if n_p % 16 == 0 else 1, seed=17,
                 layer_id=3, rope_theta=rope, rope_pos_offset=2)
    hid = S.make_hidden_states(wl, 0, dm)
    w, bias = S.make_query_projection(wl, 0, dm, with_bias)
    st = _stats(wl, [hid])
    got = _gpu_hidden_proxies(wl, dm, st, [w], [bias], h)
    for b in range(wl.batch):
        _check_projection(got[0, b], st[0, b], w, bias, h, b, wl.seq_lens[b] + 2, wl.n_q_heads, 3)


def test_hidden_proxies_layers_stride_and_positions():
    """Two layers in one call (padded W_Q stride), explicit RoPE positions
    per request (M-RoPE text positions); each layer against the oracle."""
    wl = QWEN1.replace(n_q_heads=4, n_kv_heads=1, seq_lens=(900, 300), n_visual=(800, 250),
                       budgets=(64, 64), n_layers=2)
    dm = 512
    h = PT.hyper(n_proxies=128, n_groups=8, seed=23, layer_id=10, rope_theta=1e6)
    hid = [S.make_hidden_states(wl, l, dm) for l in range(2)]
    wb = [S.make_query_projection(wl, l, dm, True) for l in range(2)]
    st = _stats(wl, hid, 2)
    pos = [5000, 17]
    got = _gpu_hidden_proxies(wl, dm, st, [x[0] for x in wb], [x[1] for x in wb], h, rope_pos=pos,
                              wq_stride=wl.n_q_heads * wl.head_dim * dm + 64)
    for l in range(2):
        for b in range(wl.batch):
            _check_projection(got[l, b], st[l, b], wb[l][0], wb[l][1], h, b, pos[b], wl.n_q_heads,
                              10 + l)


def test_hidden_stats_match_oracle():
    wl = QWEN1.replace(seq_lens=(2000, 513, 1), n_visual=(1900, 500, 0), budgets=(64, 64, 1))
    dm = 3584
    hid = S.make_hidden_states(wl, 0, dm)
    shape = PT.shape_of(wl)
    stats = torch.full((1, wl.batch, 2, dm), -1.0, device="cuda")
    nb = M.mmshift_hidden_stats_workspace_size(shape, dm)
    ws = torch.zeros(nb, dtype=torch.uint8, device="cuda")
    M.check(M.mmshift_hidden_stats(shape, dm, PT.dev(hid, wl.dtype), 0, stats, ws, nb), "hidden_stats")
    torch.cuda.synchronize()
    got = PT.host(stats)[0]
    cu = wl.cu_seqlens()
    for b in range(wl.batch):
        mu, sg = O.prefill_stats(hid[cu[b]:cu[b + 1]])
        assert np.all(np.abs(got[b, 0] - mu) <= 5e-5 * (np.abs(mu) + sg) + 1e-30)
        assert np.all(np.abs(got[b, 1] - sg) <= 2e-4 * sg + 1e-6 * np.abs(mu) + 1e-30)


def test_select_with_hidden_proxies_agreement():
    """The whole chain on the GPU (hidden statistics, hidden proxies,
    selection with them) against the oracle's selection with its own hidden
    proxies: one-ulp proxy differences move single logits, so the selection
    must agree on almost every key."""
    wl = QWEN1
    dm = 3584
    h = PT.hyper(seed=29, layer_id=0)
    hid = S.make_hidden_states(wl, 0, dm)
    w, bias = S.make_query_projection(wl, 0, dm, True)
    li = S.make_layer(wl, 0)
    shape = PT.shape_of(wl)
    stats = torch.empty((1, wl.batch, 2, dm), device="cuda")
    nb = M.mmshift_hidden_stats_workspace_size(shape, dm)
    ws = torch.zeros(nb, dtype=torch.uint8, device="cuda")
    M.check(M.mmshift_hidden_stats(shape, dm, PT.dev(hid, wl.dtype), 0, stats, ws, nb), "hidden_stats")
    params = PT.abi_params(h)
    hb = M.mmshift_hidden_proxies_workspace_size(shape, dm, params)
    hws = torch.zeros(hb, dtype=torch.uint8, device="cuda")
    px = torch.empty((1, wl.batch, wl.n_q_heads, h["n_proxies"], wl.head_dim), dtype=torch.bfloat16,
                     device="cuda")
    M.check(M.mmshift_build_hidden_proxies(shape, dm, stats, PT.dev(w, wl.dtype), 0,
                                           PT.dev(bias, wl.dtype), None, params, px, hws, hb),
            "build_hidden_proxies")
    gpu = PT.gpu_select(wl, [li], h, proxies=px)
    mu, sg = O.prefill_stats(hid)
    z = O.hidden_normals(h["seed"], 0, 0, h["n_proxies"], dm)
    prox = O.hidden_proxies(mu, sg, z, w, bias, h["gamma"], wl.n_q_heads, wl.seq_lens[0], O.BF16)
    ref = PT.oracle_layer(wl, li, h, 0, proxies=prox[None])[0]
    err = np.abs(gpu["group_mass"][0].astype(np.float64) - ref["group_mass"])
    bad = err > PT.RTOL * np.abs(ref["group_mass"]) + PT.ATOL
    assert bad.mean() < 1e-2, f"{bad.mean():.2e} of group masses outside tolerance"
    for hh in range(wl.n_kv_heads):
        a, b = set(gpu["idx"][0][:, hh].tolist()), set(ref["idx"][:, hh].tolist())
        assert len(a & b) >= 0.98 * len(b), f"head {hh}: overlap {len(a & b)}/{len(b)}"
