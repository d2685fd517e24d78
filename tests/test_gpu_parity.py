"""GPU parity: the CUDA path (through the C ABI) against the CPU oracle on the
same seeded inputs, element by element, with the tolerances of tests/parity.py.
"""
import numpy as np
import pytest
import torch

import paper_2607_22586_gb300 as M
from paper_2607_22586_gb300 import _lib as LB
from paper_2607_22586_gb300 import synth as S
from oracle import mmshift_oracle as O
from tests import parity as PT

pytestmark = pytest.mark.gpu

TINY = S.WORKLOADS["tiny-f32"]
QWEN1 = S.WORKLOADS["qwen7b-1layer"]
# ragged, 72B-head-shaped, small enough for the oracle: several key tiles and tails
RAGGED = S.WORKLOADS["72b-80l-ragged"].replace(
    name="ragged-small", n_layers=1, seq_lens=(300, 1000, 77, 2), n_visual=(285, 950, 73, 0),
    budgets=(64, 2000, 16, 1), n_centres=32)


def _requests(wl):
    cu = wl.cu_seqlens()
    outs = np.concatenate([[0], np.cumsum(np.minimum(wl.budgets, wl.seq_lens))])
    return [(b, int(cu[b]), int(cu[b + 1]), int(outs[b])) for b in range(wl.batch)]


def _check_all(wl, gpu, refs, h, layer=0, what=""):
    for b, lo, hi, olo in _requests(wl):
        if refs[b] is None:
            continue
        PT.check_request(gpu, refs[b], h, lo, hi, layer, f"{what} req {b}", out_lo=olo)
        PT.check_gather(gpu, wl, layer, lo, olo, min(wl.budgets[b], hi - lo), hi - lo, wl.n_kv_heads)


# ---------------------------------------------------------------------------
# step 1: proxies
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("name,rope", [("tiny-f32", 0.0), ("qwen7b-1layer", 0.0),
                                       ("qwen7b-1layer", 1e6), ("ragged-small", 0.0)])
def test_proxies_match_oracle(name, rope):
    wl = RAGGED if name == "ragged-small" else S.WORKLOADS[name]
    li = S.make_layer(wl, 0)
    h = PT.hyper(seed=1234, layer_id=5, rope_theta=rope, rope_pos_offset=3)
    shape = PT.shape_of(wl)
    Q = PT.dev(li.Qwin, wl.dtype)
    out = torch.empty((1, wl.batch, wl.n_q_heads, h["n_proxies"], wl.head_dim),
                      dtype=PT.TORCH_DT[wl.dtype], device="cuda")
    M.check(M.mmshift_build_proxies(shape, Q, PT.abi_params(h), out), "build_proxies")
    got = PT.host(out)[0].astype(np.float64)
    for b in range(wl.batch):
        z = O.proxy_normals(h["seed"], h["layer_id"], b, wl.n_q_heads, h["n_proxies"], wl.head_dim)
        ref = O.build_proxies(li.Qwin[b], z, h["gamma"], wl.seq_lens[b], wl.dtype, rope,
                              h["rope_pos_offset"])
        # fp32 sampling vs fp64: the pre-rounding error is bounded relative to
        # the magnitude of the two terms mu and gamma*sigma*z, not to their
        # (possibly cancelling) sum; rounding to bf16 adds at most one ulp
        mu, sig = O.window_stats(li.Qwin[b])
        scale = np.abs(mu)[:, None, :] + h["gamma"] * sig[:, None, :] * (1.0 + np.abs(z))
        if wl.dtype == S.BF16:
            PT.check_proxies(got[b], ref, f"{name} rope {rope} req {b}")
        else:
            diff = np.abs(got[b] - ref)
            assert np.all(diff <= 2e-6 * scale), f"max scaled error {np.max(diff / scale):.3g}"


@pytest.mark.parametrize("rope", [0.0, 1e6])
def test_sampled_proxies_same_with_and_without_refinement_list(rope):
    """Elements whose float32 value is too close to a bf16 rounding boundary
    are recomputed in float64: from a workspace list by a second kernel
    (mmshift_select), or in place by the sampler when the call has no
    workspace (mmshift_build_proxies). Both give the same bits."""
    wl = RAGGED.replace(seq_lens=(900, 333), n_visual=(850, 300), budgets=(64, 32), n_layers=2)
    lis = [S.make_layer(wl, l) for l in range(2)]
    h = PT.hyper(seed=77, layer_id=4, rope_theta=rope, rope_pos_offset=1)
    sel = PT.gpu_select(wl, lis, h)
    shape = PT.shape_of(wl, 2)
    Q = PT.dev(np.stack([li.Qwin for li in lis]), wl.dtype)
    out = torch.empty((2, wl.batch, wl.n_q_heads, h["n_proxies"], wl.head_dim),
                      dtype=torch.bfloat16, device="cuda")
    M.check(M.mmshift_build_proxies(shape, Q, PT.abi_params(h), out), "build_proxies")
    np.testing.assert_array_equal(PT.host(out), sel["proxies"])
    assert sel["launches"] >= 2


# ---------------------------------------------------------------------------
# steps 2-6 with identical (given) proxies
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("name", ["tiny-f32", "qwen7b-1layer", "ragged-small"])
@pytest.mark.parametrize("mode", [O.SCORE_VOTE, O.SCORE_MASS])
def test_select_given_proxies(name, mode):
    wl = RAGGED if name == "ragged-small" else S.WORKLOADS[name]
    li = S.make_layer(wl, 0)
    h = PT.hyper(score_mode=mode)
    prox = S.make_proxies(wl, h["n_proxies"], 0)
    gpu = PT.gpu_select(wl, [li], h, proxies=prox[None])
    # bf16 scoring runs on the tensor cores, fp32 on the CUDA cores
    assert gpu["score_path"] == (1 if wl.dtype == S.BF16 else 0)
    refs = PT.oracle_layer(wl, li, h, 0, proxies=prox)
    _check_all(wl, gpu, refs, h, what=name)


@pytest.mark.parametrize("kw", [dict(n_proxies=64, n_groups=4), dict(n_proxies=128, n_groups=32),
                                dict(tau=1.0), dict(tau=0.5, lam=0.0), dict(n_proxies=0, n_groups=0),
                                dict(n_proxies=32, n_groups=2, softmax_scale=0.05)])
def test_select_hyperparameters(kw):
    wl = QWEN1.replace(seq_lens=(1500,), n_visual=(1400,), budgets=(200,))
    li = S.make_layer(wl, 3)
    h = PT.hyper(**kw)
    prox = S.make_proxies(wl, max(h["n_proxies"], 1), 3)[:, :, :h["n_proxies"]]
    pin = prox if h["n_proxies"] else None
    gpu = PT.gpu_select(wl, [li], h, proxies=None if pin is None else pin[None])
    refs = PT.oracle_layer(wl, li, h, 0, proxies=pin)
    _check_all(wl, gpu, refs, h, what=str(kw))


@pytest.mark.parametrize("kw", [dict(n_proxies=32, n_groups=2), dict(n_proxies=128, n_groups=32),
                                dict(n_proxies=64, n_groups=4, tau=0.5)])
def test_votes_exact_on_the_calls_own_masses(kw):
    """The coverage vote of a full selection call (where the group totals
    are known in advance, so its candidates come from the first pass) equals
    the oracle's cover sets on the group masses the call itself computed,
    key for key: the votes recovered from the scores (vote = S - lambda *
    anchor, an integer) match O.votes(O.cover_sets(masses)) exactly."""
    wl = QWEN1.replace(seq_lens=(6000, 900), n_visual=(5800, 850), budgets=(512, 100))
    li = S.make_layer(wl, 1)
    h = PT.hyper(**kw)
    gpu = PT.gpu_select(wl, [li], h)
    G, lam = h["n_groups"], np.float32(h["lam"])
    for b, lo, hi, olo in _requests(wl):
        for hh in range(wl.n_kv_heads):
            gm = gpu["group_mass"][0][hh, :G, lo:hi].astype(np.float64)
            v_own = O.votes(O.cover_sets(gm, h["tau"]))
            an = gpu["anchor"][0][hh, lo:hi]
            v_gpu = np.rint(gpu["scores"][0][hh, lo:hi].astype(np.float64) -
                            (lam * an).astype(np.float32).astype(np.float64))
            np.testing.assert_array_equal(v_gpu, v_own, err_msg=f"{kw} req {b} head {hh}")


@pytest.mark.parametrize("lens", [(200, 333), (3000, 1333)])
def test_multi_layer_call_matches_single_layer_calls(lens):
    """Bitwise equal whether the layers run in one call or one by one; the
    longer requests span several key splits (one with an odd tile count), so
    the CTAs' split ranges start at different places in the two calls."""
    wl = RAGGED.replace(seq_lens=lens, n_visual=(lens[0] - 10, lens[1] - 33), budgets=(50, 64))
    lis = [S.make_layer(wl, l) for l in range(3)]
    h = PT.hyper(n_proxies=64, n_groups=4, seed=9, layer_id=2)
    multi = PT.gpu_select(wl, lis, h)
    for l in range(3):
        single = PT.gpu_select(wl, [lis[l]], dict(h, layer_id=2 + l))
        for key in ("idx", "out_k", "group_mass", "anchor", "scores", "proxies"):
            np.testing.assert_array_equal(multi[key][l], single[key][0], err_msg=key)


# head_dim 64 in bf16 takes the tensor-core path too (softmax pass on CTA
# pairs, mass pass with a separate anchor block and four groups per block)
D64 = S.WORKLOADS["qwen7b-1layer"].replace(
    name="d64-bf16", n_q_heads=8, n_kv_heads=2, head_dim=64, seq_lens=(3000, 1500),
    n_visual=(2900, 1400), window=16, budgets=(256, 2000), n_centres=64, n_outlier=2)


@pytest.mark.parametrize("kw", [dict(n_proxies=64, n_groups=4, score_mode=O.SCORE_VOTE),
                                dict(n_proxies=64, n_groups=4, score_mode=O.SCORE_MASS),
                                dict(n_proxies=512, n_groups=32)])
def test_select_head_dim_64_tensor_cores(kw):
    wl = D64
    li = S.make_layer(wl, 0)
    h = PT.hyper(**kw)
    prox = S.make_proxies(wl, h["n_proxies"], 0)
    gpu = PT.gpu_select(wl, [li], h, proxies=prox[None])
    assert gpu["score_path"] == 1
    refs = PT.oracle_layer(wl, li, h, 0, proxies=prox)
    _check_all(wl, gpu, refs, h, what=f"d64 {kw}")


# ---------------------------------------------------------------------------
# end to end with the sampled proxies
# ---------------------------------------------------------------------------
def test_end_to_end_sampled_f32():
    wl = TINY
    li = S.make_layer(wl, 0)
    h = PT.hyper(seed=3)
    gpu = PT.gpu_select(wl, [li], h)
    refs = PT.oracle_layer(wl, li, h, 0)
    _check_all(wl, gpu, refs, h, what="tiny sampled")


def test_end_to_end_sampled_bf16():
    """The proxies sampled on the GPU against the oracle's (level A), then the
    whole selection against the oracle re-run on the GPU's proxies (level B,
    the per-key rule). Where the proxies are identical this is the oracle's
    own end-to-end result (level C)."""
    wl = QWEN1
    li = S.make_layer(wl, 0)
    h = PT.hyper(seed=3)
    gpu = PT.gpu_select(wl, [li], h)
    z = O.proxy_normals(h["seed"], 0, 0, wl.n_q_heads, h["n_proxies"], wl.head_dim)
    own = O.build_proxies(li.Qwin[0], z, h["gamma"], wl.total_tokens, wl.dtype)
    PT.check_proxies(gpu["proxies"][0, 0], own, "qwen7b-1layer sampled")
    refs = PT.oracle_layer(wl, li, h, 0, proxies=gpu["proxies"][0])
    _check_all(wl, gpu, refs, h, what="qwen7b-1layer sampled")


# ---------------------------------------------------------------------------
# selection steps alone, on generated masses / scores (exact)
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("tau", [0.95, 0.5, 1.0])
def test_scores_topk_exact_on_generated_masses(tau, lens=(700, 2500, 40)):
    # (only the lengths and budgets matter here: masses and anchors are generated)
    wl = RAGGED.replace(seq_lens=lens, n_visual=tuple(0 for _ in lens), budgets=(100, 300, 8))
    h = PT.hyper(n_proxies=64, n_groups=8, tau=tau)
    T, hkv, G = wl.total_tokens, wl.n_kv_heads, h["n_groups"]
    gm = S.make_group_masses(hkv, G, T, 112.0, seed=5)
    # masses per request must be each request's own distribution
    anchor = S.make_scores(hkv, T, 0, seed=6) * np.float32(0.5)
    shape = PT.shape_of(wl)
    params = PT.abi_params(h)
    ws_bytes = M.mmshift_workspace_size(shape, params)
    ws = torch.zeros(ws_bytes, dtype=torch.uint8, device="cuda")
    rows = M.mmshift_output_rows(shape)
    idx = torch.full((1, rows, hkv), -1, dtype=torch.int32, device="cuda")
    sc = torch.empty((1, hkv, T), device="cuda")
    st = M.mmshift_scores_topk(shape, params, torch.from_numpy(gm).cuda(),
                               torch.from_numpy(anchor).cuda(), sc, idx, ws, ws_bytes)
    M.check(st, "scores_topk")
    torch.cuda.synchronize()
    sc, idx = PT.host(sc)[0], PT.host(idx)[0]
    for b, lo, hi, olo in _requests(wl):
        keep = min(wl.budgets[b], hi - lo)
        for hh in range(hkv):
            v = O.votes(O.cover_sets(gm[hh, :, lo:hi].astype(np.float64), tau))
            s_exp = (v.astype(np.float32) + np.float32(h["lam"]) * anchor[hh, lo:hi]).astype(np.float32)
            np.testing.assert_array_equal(sc[hh, lo:hi], s_exp)
            np.testing.assert_array_equal(idx[olo:olo + keep, hh],
                                          O.select_topk(s_exp.astype(np.float64), wl.budgets[b]))


@pytest.mark.parametrize("lens", [(701, 2498, 43), (3, 5, 1)])
def test_scores_topk_exact_with_unaligned_requests(lens):
    """Request offsets and lengths that are not multiples of four keys, so
    the coverage vote's 16-byte passes start and end with scalar keys."""
    test_scores_topk_exact_on_generated_masses(0.95, lens)


@pytest.mark.parametrize("tau", [0.95, 0.5])
@pytest.mark.parametrize("kind", ["flat", "two_level"])
def test_cover_exact_when_many_keys_are_heavy(tau, kind):
    """Group 0's masses make the coverage vote leave its usual path (a few
    keys above the bound on the last cover key's weight, ranked one per
    thread). flat: all masses share one float exponent ([0.5, 1), on a grid
    of 2^-8 so that many are equal), so every key is above the bound and
    9,000 share the threshold's first digit, more than the shared-memory
    candidate list holds: the digit passes, the tie scan and the bitmap pass
    read the masses. two_level: 2,000 such keys among light ones (2^-20),
    more than one per thread but few enough for the list: the digit passes
    and the tie ranking run among them. Group 1 takes the usual path. Votes
    and kept sets equal the oracle's."""
    wl = RAGGED.replace(seq_lens=(9000, 300), n_visual=(8000, 280), budgets=(900, 64))
    h = PT.hyper(n_proxies=32, n_groups=2, tau=tau)
    T, hkv, G = wl.total_tokens, wl.n_kv_heads, h["n_groups"]
    gm = S.make_group_masses(hkv, G, T, 112.0, seed=7)
    rng = np.random.default_rng(9)
    flat = (np.floor(rng.uniform(0.5, 1.0, size=(hkv, T)) * 256.0) / 256.0).astype(np.float32)
    if kind == "two_level":
        light = rng.random(size=(hkv, T)) >= 2000.0 / 9000.0
        flat[light] = np.float32(2.0 ** -20)
    gm[:, 0, :] = flat
    anchor = S.make_scores(hkv, T, 0, seed=8) * np.float32(0.5)
    shape = PT.shape_of(wl)
    params = PT.abi_params(h)
    ws_bytes = M.mmshift_workspace_size(shape, params)
    ws = torch.zeros(ws_bytes, dtype=torch.uint8, device="cuda")
    rows = M.mmshift_output_rows(shape)
    idx = torch.full((1, rows, hkv), -1, dtype=torch.int32, device="cuda")
    sc = torch.empty((1, hkv, T), device="cuda")
    st = M.mmshift_scores_topk(shape, params, torch.from_numpy(gm).cuda(),
                               torch.from_numpy(anchor).cuda(), sc, idx, ws, ws_bytes)
    M.check(st, "scores_topk")
    torch.cuda.synchronize()
    sc, idx = PT.host(sc)[0], PT.host(idx)[0]
    for b, lo, hi, olo in _requests(wl):
        keep = min(wl.budgets[b], hi - lo)
        for hh in range(hkv):
            v = O.votes(O.cover_sets(gm[hh, :, lo:hi].astype(np.float64), tau))
            s_exp = (v.astype(np.float32) + np.float32(h["lam"]) * anchor[hh, lo:hi]).astype(np.float32)
            np.testing.assert_array_equal(sc[hh, lo:hi], s_exp)
            np.testing.assert_array_equal(idx[olo:olo + keep, hh],
                                          O.select_topk(s_exp.astype(np.float64), wl.budgets[b]))


@pytest.mark.parametrize("lens,budgets", [((5000,), (700,)), ((1, 2, 3, 64, 65), (1, 1, 2, 10, 64)),
                                          ((60000,), (4096,)), ((33, 4097), (32, 4097))])
def test_topk_exact_on_generated_scores(lens, budgets):
    wl = RAGGED.replace(seq_lens=lens, n_visual=tuple(0 for _ in lens), budgets=budgets)
    T, hkv = wl.total_tokens, wl.n_kv_heads
    s = S.make_scores(hkv, T, 32, seed=len(lens))
    shape = PT.shape_of(wl)
    ws_bytes = M.mmshift_workspace_size(shape, None)
    ws = torch.zeros(ws_bytes, dtype=torch.uint8, device="cuda")
    rows = M.mmshift_output_rows(shape)
    idx = torch.full((1, rows, hkv), -1, dtype=torch.int32, device="cuda")
    M.check(M.mmshift_topk(shape, torch.from_numpy(s).cuda(), idx, ws, ws_bytes), "topk")
    torch.cuda.synchronize()
    idx = PT.host(idx)[0]
    for b, lo, hi, olo in _requests(wl):
        keep = min(budgets[b], hi - lo)
        for hh in range(hkv):
            np.testing.assert_array_equal(idx[olo:olo + keep, hh],
                                          O.select_topk(s[hh, lo:hi].astype(np.float64), budgets[b]))


@pytest.mark.parametrize("tiny", ["all", "most"])
def test_topk_exact_with_tiny_scores(tiny):
    """Scores scaled by 2^-50 (every key, or 80% of them), so that the radix
    digits fall in the float's low exponents: the kept sets still equal the
    oracle's."""
    wl = RAGGED.replace(seq_lens=(5000, 700), n_visual=(0, 0), budgets=(700, 64))
    T, hkv = wl.total_tokens, wl.n_kv_heads
    s = S.make_scores(hkv, T, 32, seed=11)
    rng = np.random.default_rng(3)
    small = np.ones(s.shape, dtype=bool) if tiny == "all" else rng.random(s.shape) < 0.8
    s = np.where(small, s * np.float32(2.0 ** -50), s).astype(np.float32)
    shape = PT.shape_of(wl)
    ws_bytes = M.mmshift_workspace_size(shape, None)
    ws = torch.zeros(ws_bytes, dtype=torch.uint8, device="cuda")
    rows = M.mmshift_output_rows(shape)
    idx = torch.full((1, rows, hkv), -1, dtype=torch.int32, device="cuda")
    M.check(M.mmshift_topk(shape, torch.from_numpy(s).cuda(), idx, ws, ws_bytes), "topk")
    torch.cuda.synchronize()
    idx = PT.host(idx)[0]
    for b, lo, hi, olo in _requests(wl):
        keep = min(wl.budgets[b], hi - lo)
        for hh in range(hkv):
            np.testing.assert_array_equal(idx[olo:olo + keep, hh],
                                          O.select_topk(s[hh, lo:hi].astype(np.float64), wl.budgets[b]))


def test_topk_exact_when_the_fine_bin_holds_many_keys():
    """48 layers x 4 heads, more units than SMs (512-thread CTAs), and per
    head 20% of 4,000 keys in one 12-bit first-digit bin (scores on a 2^-12
    grid in [1, 1.0625), so many tie) above keys in [0.25, 0.5): the bin's
    kept keys are found by the later digit passes and, among equal keys, by
    index. Kept sets equal the oracle's."""
    L = 48
    wl = RAGGED.replace(seq_lens=(4000,), n_visual=(0,), budgets=(300,))
    T, hkv = wl.total_tokens, wl.n_kv_heads
    rng = np.random.default_rng(21)
    s = rng.uniform(0.25, 0.5, size=(L, hkv, T)).astype(np.float32)
    grid = (1.0 + np.floor(rng.uniform(0.0, 1.0, size=(L, hkv, T)) * 256.0) / 4096.0)
    s = np.where(rng.random(size=(L, hkv, T)) < 0.2, grid, s).astype(np.float32)
    shape = PT.shape_of(wl, L)
    ws_bytes = M.mmshift_workspace_size(shape, None)
    ws = torch.zeros(ws_bytes, dtype=torch.uint8, device="cuda")
    rows = M.mmshift_output_rows(shape)
    idx = torch.full((L, rows, hkv), -1, dtype=torch.int32, device="cuda")
    M.check(M.mmshift_topk(shape, torch.from_numpy(s).cuda(), idx, ws, ws_bytes), "topk")
    torch.cuda.synchronize()
    idx = PT.host(idx)
    for l in range(L):
        for hh in range(hkv):
            np.testing.assert_array_equal(idx[l, :300, hh],
                                          O.select_topk(s[l, hh].astype(np.float64), 300))


def test_gather_bit_exact_and_bad_index_reported():
    wl = RAGGED
    li = S.make_layer(wl, 1)
    shape = PT.shape_of(wl)
    rows = M.mmshift_output_rows(shape)
    rng = np.random.default_rng(0)
    idx = np.zeros((rows, wl.n_kv_heads), dtype=np.int32)
    for b, lo, hi, olo in _requests(wl):
        keep = min(wl.budgets[b], hi - lo)
        idx[olo:olo + keep] = rng.integers(0, hi - lo, size=(keep, wl.n_kv_heads))
    K, V = PT.dev(li.K, wl.dtype), PT.dev(li.V, wl.dtype)
    ok, ov = (torch.empty((1, rows, wl.n_kv_heads, wl.head_dim), dtype=torch.bfloat16, device="cuda")
              for _ in range(2))
    ws_bytes = M.mmshift_workspace_size(shape, None)
    ws = torch.zeros(ws_bytes, dtype=torch.uint8, device="cuda")
    M.check(M.mmshift_gather(shape, K, V, torch.from_numpy(idx).cuda(), ok, ov, ws, ws_bytes), "gather")
    assert M.mmshift_poll_status(ws) == 0
    ok, ov = PT.host(ok)[0], PT.host(ov)[0]
    hh = np.arange(wl.n_kv_heads)[None]
    for b, lo, hi, olo in _requests(wl):
        keep = min(wl.budgets[b], hi - lo)
        np.testing.assert_array_equal(ok[olo:olo + keep], li.K[lo + idx[olo:olo + keep], hh])
        np.testing.assert_array_equal(ov[olo:olo + keep], li.V[lo + idx[olo:olo + keep], hh])
    # an out-of-range index: row zero-filled, status reported, context intact
    idx[0, 0] = 10 ** 6
    M.check(M.mmshift_gather(shape, K, V, torch.from_numpy(idx).cuda(), ok_t := torch.empty(
        (1, rows, wl.n_kv_heads, wl.head_dim), dtype=torch.bfloat16, device="cuda"),
        torch.empty_like(ok_t), ws, ws_bytes), "gather")
    assert M.mmshift_poll_status(ws) == M._lib.MMSHIFT_ERR_DEVICE
    assert torch.all(ok_t[0, 0, 0] == 0)
    assert M.mmshift_poll_status(ws) == 0


def test_values_in_mapped_host_memory():
    """V may live in page-locked host memory (only the kept rows are read):
    the results equal those with V on the device; pageable host memory for V,
    and host memory for K, are refused before anything is launched."""
    wl = RAGGED
    li = S.make_layer(wl, 0)
    h = PT.hyper(n_proxies=64, n_groups=4, seed=12)
    ref = PT.gpu_select(wl, [li], h)
    shape = PT.shape_of(wl)
    params = PT.abi_params(h)
    rows = M.mmshift_output_rows(shape)
    ws_bytes = M.mmshift_workspace_size(shape, params)
    ws = torch.zeros(ws_bytes, dtype=torch.uint8, device="cuda")
    K, Q = PT.dev(li.K[None], wl.dtype), PT.dev(li.Qwin[None], wl.dtype)
    V_dev = PT.dev(li.V[None], wl.dtype)
    V_pin = V_dev.cpu().pin_memory()
    idx = torch.full((1, rows, wl.n_kv_heads), -7, dtype=torch.int32, device="cuda")
    ok = torch.empty((1, rows, wl.n_kv_heads, wl.head_dim), dtype=torch.bfloat16, device="cuda")
    ov = torch.empty_like(ok)
    M.check(M.mmshift_select(shape, K, V_pin, Q, None, params, idx, ok, ov, None, ws, ws_bytes),
            "select with pinned V")
    assert M.mmshift_poll_status(ws) == 0
    np.testing.assert_array_equal(PT.host(idx), ref["idx"])
    np.testing.assert_array_equal(PT.host(ok), ref["out_k"])
    np.testing.assert_array_equal(PT.host(ov), ref["out_v"])
    V_pageable = V_dev.cpu()
    assert M.mmshift_select(shape, K, V_pageable, Q, None, params, idx, ok, ov, None, ws,
                            ws_bytes) == LB.MMSHIFT_ERR_INVALID_ARG
    assert M.mmshift_select(shape, K.cpu().pin_memory(), V_dev, Q, None, params, idx, ok, ov, None,
                            ws, ws_bytes) == LB.MMSHIFT_ERR_INVALID_ARG


def test_select_captured_in_a_cuda_graph():
    """mmshift_select enqueues only stream work (tensor maps are encoded on
    the host), so a serving loop can capture it once in a CUDA graph and
    replay it: the replay gives the same results as a direct call."""
    wl = RAGGED.replace(seq_lens=(3000, 1333), n_visual=(2990, 1300), budgets=(256, 64), n_layers=2)
    lis = [S.make_layer(wl, l) for l in range(2)]
    h = PT.hyper(n_proxies=64, n_groups=4, seed=6)
    ref = PT.gpu_select(wl, lis, h)
    shape = PT.shape_of(wl, 2)
    params = PT.abi_params(h)
    rows = M.mmshift_output_rows(shape)
    ws_bytes = M.mmshift_workspace_size(shape, params)
    ws = torch.zeros(ws_bytes, dtype=torch.uint8, device="cuda")
    K = PT.dev(np.stack([li.K for li in lis]), wl.dtype)
    V = PT.dev(np.stack([li.V for li in lis]), wl.dtype)
    Q = PT.dev(np.stack([li.Qwin for li in lis]), wl.dtype)
    idx = torch.full((2, rows, wl.n_kv_heads), -7, dtype=torch.int32, device="cuda")
    ok = torch.zeros((2, rows, wl.n_kv_heads, wl.head_dim), dtype=torch.bfloat16, device="cuda")
    ov = torch.zeros_like(ok)
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):      # one call outside the capture (module loading, attributes)
        M.check(M.mmshift_select(shape, K, V, Q, None, params, idx, ok, ov, None, ws, ws_bytes, side),
                "warm-up")
    torch.cuda.current_stream().wait_stream(side)
    torch.cuda.synchronize()
    idx.fill_(-7)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        st = torch.cuda.current_stream()
        M.check(M.mmshift_select(shape, K, V, Q, None, params, idx, ok, ov, None, ws, ws_bytes, st),
                "captured select")
    for _ in range(2):
        idx.fill_(-7)
        g.replay()
    torch.cuda.synchronize()
    assert M.mmshift_poll_status(ws) == 0
    np.testing.assert_array_equal(PT.host(idx), ref["idx"])
    np.testing.assert_array_equal(PT.host(ok), ref["out_k"])
