"""GPU parity of the attention-mass coverage metric (§1, Fig. 1b) against the
oracle, through mmshift_coverage.

Tolerance: the GPU's kept and total masses are sums of masses each within
RTOL = 2e-3 of the oracle's (tests/parity.py), so their ratio is within
about 2 * RTOL of the oracle's coverage relative to it:
|gpu - ref| <= 4.02e-3 * ref + 1e-6. Kept sets come from the seeded input
generator (never from the CUDA path); at full size the oracle checks sampled
(layer, request, KV head, decode query) entries.
"""
import numpy as np
import pytest
import torch

import paper_2607_22586_gb300 as M
from paper_2607_22586_gb300 import synth as S
from oracle import mmshift_oracle as O
from tests import parity as PT

pytestmark = pytest.mark.gpu

COV_RTOL = 2.01 * 2 * PT.RTOL
COV_ATOL = 1e-6

QWEN1 = S.WORKLOADS["qwen7b-1layer"]
RAGGED = S.WORKLOADS["72b-80l-ragged"].replace(
    name="ragged-small", n_layers=1, seq_lens=(300, 1000, 77, 2), n_visual=(285, 950, 73, 0),
    budgets=(64, 2000, 16, 1), n_centres=32)
D64 = S.WORKLOADS["qwen7b-1layer"].replace(
    name="d64-bf16", n_q_heads=8, n_kv_heads=2, head_dim=64, seq_lens=(3000, 1500),
    n_visual=(2900, 1400), window=16, budgets=(256, 2000), n_centres=64, n_outlier=2)


def _gpu_coverage(wl, lis, dec, idx, n_dec, scale=0.0):
    L = len(lis)
    shape = PT.shape_of(wl, L)
    K = PT.dev(np.stack([li.K for li in lis]), wl.dtype)
    Q = PT.dev(np.stack([li.Qwin for li in lis]), wl.dtype)
    # decode queries in the proxies layout [L, B, Hq, n_dec, d]
    D = PT.dev(np.ascontiguousarray(np.stack(dec).transpose(0, 1, 3, 2, 4)), wl.dtype)
    I = torch.from_numpy(np.ascontiguousarray(np.stack(idx))).cuda()
    cov = torch.full((L, wl.batch, wl.n_kv_heads, n_dec), -1.0, device="cuda")
    nb = M.mmshift_coverage_workspace_size(shape, n_dec)
    ws = torch.zeros(nb, dtype=torch.uint8, device="cuda")
    M.check(M.mmshift_coverage(shape, K, Q, D, n_dec, scale, I, cov, ws, nb), "coverage")
    M.check(M.mmshift_poll_status(ws), "status")
    torch.cuda.synchronize()
    return PT.host(cov)


def _oracle_cov(wl, li, dec_b, idx, b, scale):
    """Oracle coverage of request b averaged over the r query heads: [Hkv, n_dec]."""
    cu = wl.cu_seqlens()
    outs = np.concatenate([[0], np.cumsum(np.minimum(wl.budgets, wl.seq_lens))])
    keys = li.K[cu[b]:cu[b + 1]]
    kept = idx[outs[b]:outs[b + 1]]
    c = O.attention_coverage(keys, dec_b, kept, scale)          # [Hq, n]
    r = wl.n_q_heads // wl.n_kv_heads
    return c.reshape(wl.n_kv_heads, r, -1).mean(axis=1)


def _close(got, ref, what):
    bound = COV_RTOL * ref + COV_ATOL
    err = np.abs(got - ref)
    assert np.all(err <= bound), f"{what}: coverage off by {np.max(err / bound):.3g} x bound"


@pytest.mark.parametrize("name", ["qwen7b-1layer", "ragged-small", "d64-bf16", "tiny-f32"])
def test_coverage_matches_oracle(name):
    """bf16 cases run the tensor-core scoring kernels, the fp32 case the
    CUDA-core ones."""
    wl = {"qwen7b-1layer": QWEN1, "ragged-small": RAGGED, "d64-bf16": D64,
          "tiny-f32": S.WORKLOADS["tiny-f32"]}[name]
    n_dec = 16
    li = S.make_layer(wl, 0)
    dec = S.make_decode_queries(wl, 0, li, n_dec)
    idx = S.make_kept_indices(wl, seed=5)
    got = _gpu_coverage(wl, [li], [dec], [idx], n_dec)[0]
    scale = 1.0 / np.sqrt(wl.head_dim)
    for b in range(wl.batch):
        ref = _oracle_cov(wl, li, dec[b], idx, b, scale)
        _close(got[b], ref, f"{name} req {b}")
        if wl.budgets[b] >= wl.seq_lens[b]:
            np.testing.assert_allclose(got[b], 1.0, rtol=0, atol=1e-6)


def test_coverage_complement_and_scale():
    """A kept set and its complement cover everything; an explicit softmax
    scale is the one applied."""
    wl = QWEN1.replace(seq_lens=(2000,), n_visual=(1900,), budgets=(500,))
    n_dec = 8
    li = S.make_layer(wl, 2)
    dec = S.make_decode_queries(wl, 2, li, n_dec)
    idx = S.make_kept_indices(wl, seed=9)
    rest = np.stack([np.setdiff1d(np.arange(2000), idx[:, h]) for h in range(wl.n_kv_heads)], axis=1)
    wl_rest = wl.replace(budgets=(rest.shape[0],))
    a = _gpu_coverage(wl, [li], [dec], [idx], n_dec, scale=0.05)[0]
    b = _gpu_coverage(wl_rest, [li], [dec], [rest.astype(np.int32)], n_dec, scale=0.05)[0]
    np.testing.assert_allclose(a + b, 1.0, rtol=0, atol=1e-5)
    _close(a[0], _oracle_cov(wl, li, dec[0], idx, 0, 0.05), "explicit scale")


def test_coverage_full_size_sampled():
    """Two layers of the 32K Qwen2.5-VL-7B-shaped stack: sampled (layer, KV
    head, decode query) entries against the oracle, the call repeated is
    bitwise identical."""
    wl = S.WORKLOADS["qwen7b-28l-32k"].replace(n_layers=2)
    n_dec = 32
    lis = [S.make_layer(wl, l) for l in range(2)]
    decs = [S.make_decode_queries(wl, l, lis[l], n_dec) for l in range(2)]
    idxs = [S.make_kept_indices(wl, seed=l) for l in range(2)]
    got = _gpu_coverage(wl, lis, decs, idxs, n_dec)
    again = _gpu_coverage(wl, lis, decs, idxs, n_dec)
    np.testing.assert_array_equal(got, again)
    scale = 1.0 / np.sqrt(wl.head_dim)
    r = wl.n_q_heads // wl.n_kv_heads
    rng = np.random.default_rng(0)
    for _ in range(4):
        l, h, g = int(rng.integers(2)), int(rng.integers(wl.n_kv_heads)), int(rng.integers(n_dec))
        heads = slice(h * r, (h + 1) * r)
        c = O.attention_coverage(lis[l].K[:, h:h + 1, :], decs[l][0][g:g + 1, heads, :],
                                 idxs[l][:, h:h + 1], scale)
        _close(got[l, 0, h, g:g + 1], np.array([c.mean()]), f"layer {l} head {h} query {g}")
