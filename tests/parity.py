"""Helpers shared by the parity tests: run the CUDA path through the C ABI and
the oracle on the same seeded inputs, and compare them under the tolerances
the parity contract fixes.

Tolerances (written here once, used by every GPU test):
  * masses (group masses, anchor, summed mass): |gpu - ref| <= RTOL * |ref| + ATOL
    with RTOL = 2e-3 (bf16 inputs, fp32 accumulation) and ATOL = 1e-9 for
    masses that fp32 cannot resolve (the GPU flushes exp2 results below
    2^-126 to zero);
  * proxies (level A): bf16 equal to the oracle's except one ulp on at most
    1e-5 of the elements (check_proxies); float32 within 2e-6 of the
    magnitude of mu and gamma*sigma*z (the GPU samples in fp32, the oracle in
    fp64);
  * votes: may differ only where the oracle's own decision is within the mass
    tolerance of the tau-coverage boundary;
  * selection, per key: every key t gets the band S_t +- u_t in which the
    contract's tolerances leave the oracle's score (score_bands). The GPU's
    kept set must be exactly the top-(C-1) of the GPU's own scores (plus T-1),
    and it must be the top-(C-1) of SOME scores inside those bands: the
    lowest upper end among the kept candidates is at least the highest lower
    end among the dropped ones (check_selection). A key on which GPU and
    oracle disagree is therefore admitted only when its own band reaches the
    cutoff that the other keys' bands allow;
  * gathered K/V: bit-exact given the GPU's indices.
"""
from __future__ import annotations

import numpy as np
import torch

import paper_2607_22586_gb300 as M
from paper_2607_22586_gb300 import synth as S
from oracle import mmshift_oracle as O

RTOL = 2e-3
ATOL = 1e-9
SUM_RTOL = 1e-5
# The GPU holds S_t = vote + lambda * alpha_t in float32: two roundings, each
# at most half an ulp, so |fl(S) - S| <= 2^-23 |S| (S >= lambda * alpha >= 0).
SCORE_F32_REL = 2.0 ** -23

# Level A: at most this fraction of bf16 proxy elements may differ from the
# oracle's, by one ulp.
PROXY_ULP_FRAC = 1e-5

# One entry per checked (unit, KV head): (what, mismatched keys, keys in the
# cutoff band). tests/conftest.py prints a summary at the end of the run.
SELECTION_LOG: list = []
# One entry per level-A comparison: (what, differing elements, elements).
PROXY_LOG: list = []

TORCH_DT = {S.BF16: torch.bfloat16, S.F32: torch.float32}
ABI_DT = {S.BF16: 0, S.F32: 1}


def f32(x: float) -> float:
    return float(np.float32(x))


def hyper(**kw):
    """Hyper-parameters as the C ABI sees them (float32) for both sides."""
    h = dict(n_proxies=512, n_groups=32, gamma=10.0, tau=0.95, lam=1.0, seed=0, layer_id=0,
             score_mode=0, softmax_scale=0.0, rope_theta=0.0, rope_pos_offset=0)
    h.update(kw)
    for k in ("gamma", "tau", "lam", "softmax_scale", "rope_theta"):
        h[k] = f32(h[k])
    return h


def abi_params(h):
    return M.default_params(n_proxies=h["n_proxies"], n_groups=h["n_groups"], gamma=h["gamma"],
                            tau=h["tau"], lam=h["lam"], seed=h["seed"], layer_id=h["layer_id"],
                            score_mode=h["score_mode"], softmax_scale=h["softmax_scale"],
                            rope_theta=h["rope_theta"], rope_pos_offset=h["rope_pos_offset"])


def oracle_kw(h, dtype):
    kw = dict(h)
    kw["dtype"] = dtype
    if kw["softmax_scale"] == 0.0:
        kw["softmax_scale"] = 0.0
    return kw


def dev(a: np.ndarray, dtype: str) -> torch.Tensor:
    t = torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32))
    return t.to(TORCH_DT[dtype]).cuda().contiguous()


def host(t: torch.Tensor) -> np.ndarray:
    return t.float().cpu().numpy() if t.dtype != torch.int32 else t.cpu().numpy()


def shape_of(wl: S.Workload, n_layers: int = 1, window=None):
    w = wl.window if window is None else window
    return M.make_shape(wl.n_q_heads, wl.n_kv_heads, wl.head_dim, w, ABI_DT[wl.dtype],
                        wl.cu_seqlens(), wl.budgets, n_layers=n_layers,
                        layer_stride_kv=wl.total_tokens * wl.n_kv_heads * wl.head_dim,
                        layer_stride_q=wl.batch * w * wl.n_q_heads * wl.head_dim)


def gpu_select(wl: S.Workload, layers, h, proxies=None, stats=None, ws=None):
    """Run mmshift_select over ``layers`` (list of LayerInputs) in one call
    with every debug output (mmshift_select_with_stats when ``stats``, a
    device tensor [L, B, 2, Hq*d], is given; ``ws`` reuses a workspace
    tensor); returns numpy arrays [L, ...]."""
    L = len(layers)
    shape = shape_of(wl, L)
    params = abi_params(h)
    K = dev(np.stack([li.K for li in layers]), wl.dtype)
    V = dev(np.stack([li.V for li in layers]), wl.dtype)
    Q = dev(np.stack([li.Qwin for li in layers]), wl.dtype)
    if proxies is None or isinstance(proxies, torch.Tensor):
        pin = proxies
    else:
        pin = dev(proxies, wl.dtype)
    rows = M.mmshift_output_rows(shape)
    ws_bytes = M.mmshift_workspace_size(shape, params)
    if ws is None:
        ws = torch.zeros(ws_bytes, dtype=torch.uint8, device="cuda")
    assert ws.numel() >= ws_bytes
    hkv, hq, d, T = wl.n_kv_heads, wl.n_q_heads, wl.head_dim, wl.total_tokens
    G = h["n_groups"]
    out_idx = torch.full((L, rows, hkv), -7, dtype=torch.int32, device="cuda")
    out_k = torch.empty((L, rows, hkv, d), dtype=TORCH_DT[wl.dtype], device="cuda")
    out_v = torch.empty_like(out_k)
    gm = torch.full((L, hkv, max(G, 1), T), -1.0, device="cuda")
    an = torch.full((L, hkv, T), -1.0, device="cuda")
    ms = torch.full((L, hkv, T), -1.0, device="cuda")
    sc = torch.full((L, hkv, T), -1.0, device="cuda")
    px = torch.empty((L, wl.batch, hq, max(h["n_proxies"], 1), d), dtype=TORCH_DT[wl.dtype], device="cuda")
    dbg = M.make_debug(proxies=px, group_mass=gm, anchor=an, mass=ms, scores=sc)
    if stats is None:
        st = M.mmshift_select(shape, K, V, Q, pin, params, out_idx, out_k, out_v, dbg, ws, ws_bytes)
    else:
        st = M.mmshift_select_with_stats(shape, K, V, Q, stats, params, out_idx, out_k, out_v, dbg,
                                         ws, ws_bytes)
    M.check(st, "mmshift_select")
    M.check(M.mmshift_poll_status(ws), "mmshift_poll_status")
    torch.cuda.synchronize()
    return dict(score_path=dbg.score_path, launches=dbg.launches,
                idx=host(out_idx), out_k=host(out_k), out_v=host(out_v), group_mass=host(gm),
                anchor=host(an), mass=host(ms), scores=host(sc), proxies=host(px),
                K=np.stack([li.K for li in layers]), V=np.stack([li.V for li in layers]))


def oracle_layer(wl: S.Workload, li: S.LayerInputs, h, layer_id: int, proxies=None, requests=None):
    """Oracle results for one layer: list over requests (None where skipped)."""
    cu = wl.cu_seqlens()
    out = []
    kw = oracle_kw(h, wl.dtype)
    kw["layer_id"] = layer_id
    for b in range(wl.batch):
        if requests is not None and b not in requests:
            out.append(None)
            continue
        lo, hi = int(cu[b]), int(cu[b + 1])
        out.append(O.select_request(li.K[lo:hi], li.V[lo:hi], li.Qwin[b], int(wl.budgets[b]), b=b,
                                    proxies=None if proxies is None else proxies[b], **kw))
    return out


def check_proxies(got: np.ndarray, ref: np.ndarray, what: str):
    """Level A for bf16 proxies: every element within one bf16 ulp of the
    oracle's (8 significant bits: ulp = 2^(e-8) for |x| in [2^(e-1), 2^e)),
    and at most PROXY_ULP_FRAC of them different at all."""
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    diff = np.abs(got - ref)
    _, e = np.frexp(np.maximum(np.abs(ref), np.abs(got)))
    ulp = np.ldexp(1.0, e - 8)
    n = int(np.count_nonzero(diff))
    PROXY_LOG.append((what, n, diff.size))
    assert np.all(diff <= ulp), f"{what}: proxies off by more than one bf16 ulp"
    assert n <= PROXY_ULP_FRAC * diff.size, (
        f"{what}: {n} of {diff.size} proxy elements ({n / diff.size:.2e}) differ from the oracle's")


def mass_close(gpu: np.ndarray, ref: np.ndarray, what: str):
    err = np.abs(gpu.astype(np.float64) - ref)
    bound = RTOL * np.abs(ref) + ATOL
    bad = err > bound
    assert not bad.any(), (f"{what}: {bad.sum()} of {bad.size} outside tolerance; "
                           f"worst rel {np.max(err / (np.abs(ref) + 1e-30)):.3g}")


def uncertain_votes(abar: np.ndarray, tau: float) -> np.ndarray:
    """[G, T] bool: where the oracle's coverage decision is within tolerance."""
    G, T = abar.shape
    unc = np.zeros((G, T), dtype=bool)
    for g in range(G):
        order = np.lexsort((np.arange(T), -abar[g]))
        csum = np.cumsum(abar[g][order])
        total = csum[-1]
        target = tau * total
        eps = SUM_RTOL * total + ATOL
        k = int(np.argmax(csum >= target))
        theta = abar[g][order[k]]
        before = np.concatenate([[0.0], csum[:-1]])
        near_sum = (before <= target + eps) & (csum >= target - eps)
        near_val = np.abs(abar[g][order] - theta) <= RTOL * theta + ATOL
        unc[g, order] = near_sum | near_val
    return unc


def score_bands(ref, h, hh):
    """[T] half-widths u_t of the band around the oracle's score S_t of KV head
    hh that the contract's tolerances leave open.

    VOTE (§3.2.2-3.2.3, S = vote + lambda * alpha): one vote per group whose
    coverage decision at t is within tolerance of the group's cutoff
    (uncertain_votes), lambda times the anchor's tolerance, and the float32
    holding of S on the GPU. MASS (S = sum_g abar_g): the summed mass's
    tolerance, G absolute floors.
    """
    G, tau, lam, mode = h["n_groups"], h["tau"], h["lam"], h["score_mode"]
    s = np.asarray(ref["scores"][hh], dtype=np.float64)
    if mode == O.SCORE_MASS:
        return RTOL * np.abs(s) + max(G, 1) * ATOL
    u = lam * (RTOL * np.asarray(ref["anchor"][hh], dtype=np.float64) + ATOL)
    if G:
        u = u + uncertain_votes(ref["group_mass"][hh], tau).sum(axis=0)
    return u + SCORE_F32_REL * np.abs(s)


def check_selection(kept, s_gpu, s_ref, u, budget, what):
    """One KV head's kept indices (ascending, no padding) against the oracle.

    The budgeted rule of §3.2.3 / Algorithm 1: T-1 always, plus the top C-1 of
    t < T-1 (ties: lower t). Checks (1) the set is exactly that rule applied
    to the GPU's own scores s_gpu, and (2) it is that rule applied to scores
    inside the oracle's bands s_ref +- u: min over kept candidates of
    (s_ref + u) >= max over dropped candidates of (s_ref - u). Records the
    number of keys that differ from the oracle's set and the number of keys
    whose band reaches the oracle's cutoff.
    """
    kept = np.asarray(kept, dtype=np.int64)
    T = s_ref.shape[0]
    if budget >= T:
        np.testing.assert_array_equal(kept, np.arange(T), err_msg=f"{what}: budget >= T keeps all")
        SELECTION_LOG.append((what, 0, 0))
        return
    assert kept.shape[0] == budget, f"{what}: {kept.shape[0]} kept rows, budget {budget}"
    assert np.all(np.diff(kept) > 0) and kept[-1] == T - 1 and kept[0] >= 0, f"{what}: malformed idx"
    cand = np.arange(T - 1)
    order = np.lexsort((cand, -np.asarray(s_gpu[:T - 1], dtype=np.float64)))
    expect = np.sort(np.concatenate([order[:budget - 1], [T - 1]]))
    np.testing.assert_array_equal(kept, expect, err_msg=f"{what}: not the top-k of its own scores")
    ref_kept = O.select_topk(s_ref, budget)
    mism = sorted(set(kept.tolist()) ^ set(ref_kept.tolist()))
    n_band = 0
    if budget >= 2:
        lo, hi = s_ref[:T - 1] - u[:T - 1], s_ref[:T - 1] + u[:T - 1]
        inside = np.zeros(T - 1, dtype=bool)
        inside[kept[:-1]] = True
        top = lo[~inside].max() if (~inside).any() else -np.inf
        bot = hi[inside].min() if inside.any() else np.inf
        cpos = np.lexsort((cand, -s_ref[:T - 1]))[budget - 2]   # the oracle's (C-1)-th key
        cut, ucut = s_ref[cpos], u[cpos]
        n_band = int(np.sum(np.abs(s_ref[:T - 1] - cut) <= u[:T - 1] + ucut))
        if bot < top:
            far_in = [int(t) for t in np.nonzero(inside & (hi < top))[0]]
            far_out = [int(t) for t in np.nonzero(~inside & (lo > bot))[0]]
            raise AssertionError(
                f"{what}: kept set is not a top-{budget - 1} of any scores within tolerance: "
                f"{len(mism)} keys differ from the oracle ({n_band} keys in the cutoff band); "
                f"kept below the band: {far_in[:8]}, dropped above it: {far_out[:8]}; "
                f"cutoff {cut:.9g} +- {ucut:.3g}")
    SELECTION_LOG.append((what, len(mism), n_band))


def check_request(gpu, ref, h, lo, hi, layer, what="", out_lo=0):
    """Compare one request of one layer: masses, anchor, votes, scores, selection, gather."""
    G, tau, lam, mode = h["n_groups"], h["tau"], h["lam"], h["score_mode"]
    hkv = ref["anchor"].shape[0]
    T = hi - lo
    if G:
        mass_close(gpu["group_mass"][layer][:, :G, lo:hi], ref["group_mass"], what + " group_mass")
    mass_close(gpu["anchor"][layer][:, lo:hi], ref["anchor"], what + " anchor")
    mass_close(gpu["mass"][layer][:, lo:hi], ref["mass"], what + " mass")
    s_gpu = gpu["scores"][layer][:, lo:hi].astype(np.float64)
    s_ref = ref["scores"]
    if mode == O.SCORE_VOTE and G:
        for hh in range(hkv):
            unc = uncertain_votes(ref["group_mass"][hh], tau)
            v_ref = O.votes(O.cover_sets(ref["group_mass"][hh], tau))
            anc_gpu = gpu["anchor"][layer][hh, lo:hi].astype(np.float64)
            v_gpu = np.rint(s_gpu[hh] - np.float32(lam) * anc_gpu)
            dv = np.abs(v_gpu - v_ref)
            assert np.all(dv <= unc.sum(axis=0)), f"{what} head {hh}: vote mismatch outside band"
    keep_rows = ref["idx"].shape[0]
    idx_gpu = gpu["idx"][layer][out_lo:out_lo + keep_rows]
    budget = keep_rows if keep_rows < T else T
    for hh in range(hkv):
        got = idx_gpu[:, hh]
        assert got.shape[0] == keep_rows
        u = score_bands(ref, h, hh)
        assert np.all(np.abs(s_gpu[hh] - s_ref[hh]) <= u), f"{what} head {hh}: score outside its band"
        check_selection(got, s_gpu[hh], s_ref[hh], u, budget, f"{what} head {hh}")
    return float(np.max(np.abs(s_gpu - s_ref))) if T else 0.0


def check_gather(gpu, wl, layer, lo_tok, out_lo, keep, T, hkv):
    idx = gpu["idx"][layer][out_lo:out_lo + keep]
    h = np.arange(hkv)[None, :]
    kref = gpu["K"][layer][lo_tok + idx, h]
    vref = gpu["V"][layer][lo_tok + idx, h]
    np.testing.assert_array_equal(gpu["out_k"][layer][out_lo:out_lo + keep], kref)
    np.testing.assert_array_equal(gpu["out_v"][layer][out_lo:out_lo + keep], vref)
