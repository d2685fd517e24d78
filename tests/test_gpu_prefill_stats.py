"""GPU parity of the full-prefill statistics path (§3.2.1: proxy statistics
over every prompt token) against the oracle, through the C ABI:
mmshift_prefill_stats, mmshift_build_proxies_from_stats, and selection with
the proxies they make.

Tolerance of the statistics. The GPU sums x - x0 and (x - x0)^2 in fp32 over
chunks of 512 queries (x0 the chunk's first query), then merges chunks with
the pairwise update. A sum of m fp32 terms is off by at most ~m*u times the
sum of magnitudes (u = 2^-24), so a chunk mean is off by at most
512 * 6e-8 = 3.1e-5 of the mean |x - x0|, typically ~sqrt(512) * u = 1.3e-6.
The second moment cancels against s1^2/n by the factor
1 + (mean - x0)^2 / sigma^2 (~10 when x0 lies 3 sigma out), so the std is off
by at most ~1.5e-4 of sigma. The bounds used: |d mu| <= 5e-5 (|mu| + sigma)
and |d sigma| <= 2e-4 sigma + 1e-6 |mu|. A dropped or repeated query, a
wrong chunk offset or the T divisor instead of T - 1 moves one of them by
more than 5e-4 at the sizes tested below (T <= 4096), and by more than
6e-3 at T = 77.
"""
import numpy as np
import pytest
import torch

import paper_2607_22586_gb300 as M
from paper_2607_22586_gb300 import synth as S
from oracle import mmshift_oracle as O
from tests import parity as PT

pytestmark = pytest.mark.gpu

MU_TOL = 5e-5
SIG_RTOL = 2e-4
SIG_MU_TOL = 1e-6

TINY = S.WORKLOADS["tiny-f32"]
QWEN1 = S.WORKLOADS["qwen7b-1layer"]
# ragged requests: chunk tails, a request shorter than one chunk, T = 2 and T = 1
RAGGED = S.WORKLOADS["72b-80l-ragged"].replace(
    name="ragged-small", n_layers=1, seq_lens=(300, 1000, 77, 2, 1537, 1),
    n_visual=(285, 950, 73, 0, 1500, 0), budgets=(64, 2000, 16, 1, 300, 1), n_centres=32)


def _gpu_stats(wl, qfull_layers, layer_stride=0):
    """Run mmshift_prefill_stats over the stacked layers; [L, B, 2, Hq, d]."""
    L = len(qfull_layers)
    shape = PT.shape_of(wl, L)
    ncol = wl.n_q_heads * wl.head_dim
    dense = wl.total_tokens * ncol
    stride = layer_stride or dense
    flat = np.zeros((L, stride), dtype=np.float32)
    for l, q in enumerate(qfull_layers):
        flat[l, :dense] = q.reshape(-1)
    Q = PT.dev(flat, wl.dtype)
    stats = torch.full((L, wl.batch, 2, ncol), -1.0, device="cuda")
    ws_bytes = M.mmshift_prefill_stats_workspace_size(shape)
    ws = torch.zeros(max(ws_bytes, 1), dtype=torch.uint8, device="cuda")
    M.check(M.mmshift_prefill_stats(shape, Q, layer_stride, stats, ws, ws_bytes), "prefill_stats")
    torch.cuda.synchronize()
    return PT.host(stats).reshape(L, wl.batch, 2, wl.n_q_heads, wl.head_dim), stats


def _check_stats(got_mu, got_sg, qreq, what):
    mu, sg = O.prefill_stats(qreq)
    dmu = np.abs(got_mu - mu)
    dsg = np.abs(got_sg - sg)
    mu_bound = MU_TOL * (np.abs(mu) + sg) + 1e-30
    sg_bound = SIG_RTOL * sg + SIG_MU_TOL * np.abs(mu) + 1e-30
    assert np.all(dmu <= mu_bound), f"{what}: mean off by {np.max(dmu / mu_bound):.3g} x bound"
    assert np.all(dsg <= sg_bound), f"{what}: std off by {np.max(dsg / sg_bound):.3g} x bound"
    if qreq.shape[0] == 1:
        np.testing.assert_array_equal(got_sg, 0.0)
        np.testing.assert_array_equal(got_mu, qreq[0])


@pytest.mark.parametrize("name", ["tiny-f32", "qwen7b-1layer", "ragged-small"])
def test_prefill_stats_match_oracle(name):
    wl = RAGGED if name == "ragged-small" else S.WORKLOADS[name]
    li = S.make_layer(wl, 0)
    qf = S.make_prompt_queries(wl, 0, li)
    got, _ = _gpu_stats(wl, [qf])
    cu = wl.cu_seqlens()
    for b in range(wl.batch):
        _check_stats(got[0, b, 0], got[0, b, 1], qf[cu[b]:cu[b + 1]], f"{name} req {b}")


def test_prefill_stats_layers_with_padded_stride():
    """Three layers in one call, layers spaced by a padded stride: each layer's
    statistics come from its own queries only, and equal a one-layer call bit
    for bit."""
    wl = RAGGED.replace(seq_lens=(700, 1029), n_visual=(650, 1000), budgets=(64, 100))
    lis = [S.make_layer(wl, l) for l in range(3)]
    qfs = [S.make_prompt_queries(wl, l, lis[l]) for l in range(3)]
    stride = wl.total_tokens * wl.n_q_heads * wl.head_dim + 8 * 37
    got, _ = _gpu_stats(wl, qfs, layer_stride=stride)
    cu = wl.cu_seqlens()
    for l in range(3):
        one, _ = _gpu_stats(wl, [qfs[l]])
        np.testing.assert_array_equal(got[l], one[0], err_msg=f"layer {l}")
        for b in range(wl.batch):
            _check_stats(got[l, b, 0], got[l, b, 1], qfs[l][cu[b]:cu[b + 1]], f"layer {l} req {b}")


def test_prefill_stats_shift_keeps_offset_columns_exact():
    """Columns with a large common offset (a bias of 3000 on unit noise): the
    shifted sums keep the std; an unshifted fp32 sum of squares would lose it."""
    wl = TINY.replace(seq_lens=(2000,), n_visual=(0,), budgets=(64,))
    rng = np.random.default_rng(11)
    q = rng.standard_normal((wl.total_tokens, wl.n_q_heads, wl.head_dim)).astype(np.float32)
    q[:, :, ::5] += np.float32(3000.0)
    got, _ = _gpu_stats(wl, [q])
    _check_stats(got[0, 0, 0], got[0, 0, 1], q, "offset columns")


@pytest.mark.parametrize("name,rope", [("tiny-f32", 0.0), ("qwen7b-1layer", 0.0),
                                       ("qwen7b-1layer", 1e6), ("ragged-small", 0.0)])
def test_proxies_from_stats_match_oracle(name, rope):
    """Same statistics on both sides (the oracle's, in fp32): the expansion,
    RoPE and rounding of mmshift_build_proxies_from_stats against the oracle's
    build_proxies_from_stats."""
    wl = RAGGED if name == "ragged-small" else S.WORKLOADS[name]
    li = S.make_layer(wl, 0)
    qf = S.make_prompt_queries(wl, 0, li)
    h = PT.hyper(seed=77, layer_id=4, rope_theta=rope, rope_pos_offset=1)
    cu = wl.cu_seqlens()
    st = np.zeros((1, wl.batch, 2, wl.n_q_heads, wl.head_dim), dtype=np.float32)
    for b in range(wl.batch):
        mu, sg = O.prefill_stats(qf[cu[b]:cu[b + 1]])
        st[0, b, 0], st[0, b, 1] = mu, sg
    shape = PT.shape_of(wl)
    out = torch.empty((1, wl.batch, wl.n_q_heads, h["n_proxies"], wl.head_dim),
                      dtype=PT.TORCH_DT[wl.dtype], device="cuda")
    stats = torch.from_numpy(st).cuda()
    M.check(M.mmshift_build_proxies_from_stats(shape, stats, PT.abi_params(h), out),
            "build_proxies_from_stats")
    got = PT.host(out)[0].astype(np.float64)
    for b in range(wl.batch):
        z = O.proxy_normals(h["seed"], h["layer_id"], b, wl.n_q_heads, h["n_proxies"], wl.head_dim)
        mu, sg = st[0, b, 0].astype(np.float64), st[0, b, 1].astype(np.float64)
        ref = O.build_proxies_from_stats(mu, sg, z, h["gamma"], wl.seq_lens[b], wl.dtype, rope,
                                         h["rope_pos_offset"])
        scale = np.abs(mu)[:, None, :] + h["gamma"] * sg[:, None, :] * (1.0 + np.abs(z))
        diff = np.abs(got[b] - ref)
        if wl.dtype == S.BF16:
            _, e = np.frexp(np.maximum(np.abs(ref), np.abs(got[b])))
            ulp = np.ldexp(1.0, e - 8)
            assert np.all(diff <= ulp + 2e-6 * scale), "bf16 proxies off by more than one ulp"
            assert np.mean(diff > 0) <= 1e-3, f"{np.mean(diff > 0):.2e} of proxies differ"
        else:
            assert np.all(diff <= 2e-6 * scale), f"max scaled error {np.max(diff / scale):.3g}"


def _gpu_prefill_select(wl, li, qf, h):
    """The full-prefill chain on the GPU: statistics, then the selection with
    them (mmshift_select_with_stats)."""
    _, stats = _gpu_stats(wl, [qf])
    return PT.gpu_select(wl, [li], h, stats=stats)


def _oracle_prefill(wl, li, qf, h):
    cu = wl.cu_seqlens()
    kw = PT.oracle_kw(h, wl.dtype)
    return [O.select_request(li.K[cu[b]:cu[b + 1]], li.V[cu[b]:cu[b + 1]], li.Qwin[b],
                             int(wl.budgets[b]), b=b, qfull=qf[cu[b]:cu[b + 1]], **kw)
            for b in range(wl.batch)]


def test_select_with_prefill_proxies_f32():
    wl = TINY
    li = S.make_layer(wl, 0)
    qf = S.make_prompt_queries(wl, 0, li)
    h = PT.hyper(seed=5)
    gpu = _gpu_prefill_select(wl, li, qf, h)
    refs = _oracle_prefill(wl, li, qf, h)
    cu = wl.cu_seqlens()
    outs = np.concatenate([[0], np.cumsum(np.minimum(wl.budgets, wl.seq_lens))])
    for b in range(wl.batch):
        PT.check_request(gpu, refs[b], h, int(cu[b]), int(cu[b + 1]), 0, f"prefill req {b}",
                         out_lo=int(outs[b]))


def test_select_with_prefill_proxies_bf16():
    """bf16: the statistics over all prompt queries are float32 sums (their
    error bound is derived above), which moves the rounding of a few proxy
    elements (at most 1e-2 of them; an element whose value nearly cancels can
    move by more than one ulp); the selection must then follow the per-key
    rule against the oracle re-run on the GPU's proxies."""
    wl = QWEN1
    li = S.make_layer(wl, 0)
    qf = S.make_prompt_queries(wl, 0, li)
    h = PT.hyper(seed=5)
    gpu = _gpu_prefill_select(wl, li, qf, h)
    own = _oracle_prefill(wl, li, qf, h)[0]["proxies"]
    got = gpu["proxies"][0, 0].astype(np.float64)
    pdiff = np.mean(got != own)
    assert pdiff <= 1e-2, f"{pdiff:.2e} of proxies differ from the oracle's"
    refs = PT.oracle_layer(wl, li, h, 0, proxies=gpu["proxies"][0])
    cu = wl.cu_seqlens()
    PT.check_request(gpu, refs[0], h, int(cu[0]), int(cu[1]), 0, "prefill bf16 req 0")


def test_prefill_stats_full_size_layer_sampled():
    """A Qwen2.5-VL-7B-shaped layer at 32K prompt tokens inside a 4-layer
    stack (padded stride): the sampled last layer against the oracle, and the
    call repeated is bitwise identical."""
    wl = S.WORKLOADS["qwen7b-28l-32k"].replace(n_layers=4)
    ncol = wl.n_q_heads * wl.head_dim
    stride = wl.total_tokens * ncol + 64
    L = wl.n_layers
    shape = PT.shape_of(wl, L)
    li = S.make_layer(wl, L - 1)
    qf = S.make_prompt_queries(wl, L - 1, li)
    Q = torch.empty((L, stride), dtype=PT.TORCH_DT[wl.dtype], device="cuda")
    g = torch.Generator(device="cuda").manual_seed(3)
    Q.normal_(generator=g)
    Q[L - 1, :wl.total_tokens * ncol] = PT.dev(qf.reshape(-1), wl.dtype)
    ws_bytes = M.mmshift_prefill_stats_workspace_size(shape)
    ws = torch.zeros(ws_bytes, dtype=torch.uint8, device="cuda")
    outs = []
    for _ in range(2):
        stats = torch.full((L, wl.batch, 2, ncol), -1.0, device="cuda")
        M.check(M.mmshift_prefill_stats(shape, Q, stride, stats, ws, ws_bytes), "prefill_stats")
        torch.cuda.synchronize()
        outs.append(PT.host(stats))
    np.testing.assert_array_equal(outs[0], outs[1])
    got = outs[0].reshape(L, wl.batch, 2, wl.n_q_heads, wl.head_dim)
    _check_stats(got[L - 1, 0, 0], got[L - 1, 0, 1], qf, "32K layer")
    # the other layers hold N(0, 1) draws: mean near 0, std near 1
    assert np.all(np.abs(got[:L - 1, 0, 0]) < 0.05) and np.all(np.abs(got[:L - 1, 0, 1] - 1) < 0.05)


def test_select_with_stats_equals_proxies_from_stats():
    """mmshift_select_with_stats is bitwise the selection with the proxies of
    mmshift_build_proxies_from_stats passed in; two layers, ragged requests."""
    wl = RAGGED.replace(seq_lens=(700, 1029, 5), n_visual=(650, 1000, 0), budgets=(64, 100, 8),
                        n_layers=2)
    lis = [S.make_layer(wl, l) for l in range(2)]
    qfs = [S.make_prompt_queries(wl, l, lis[l]) for l in range(2)]
    h = PT.hyper(n_proxies=64, n_groups=4, seed=21, layer_id=3)
    _, stats = _gpu_stats(wl, qfs)
    a = PT.gpu_select(wl, lis, h, stats=stats)
    shape = PT.shape_of(wl, 2)
    px = torch.empty((2, wl.batch, wl.n_q_heads, h["n_proxies"], wl.head_dim),
                     dtype=PT.TORCH_DT[wl.dtype], device="cuda")
    M.check(M.mmshift_build_proxies_from_stats(shape, stats, PT.abi_params(h), px),
            "build_proxies_from_stats")
    b = PT.gpu_select(wl, lis, h, proxies=px)
    for key in ("idx", "out_k", "out_v", "group_mass", "anchor", "scores", "proxies"):
        np.testing.assert_array_equal(a[key], b[key], err_msg=key)
