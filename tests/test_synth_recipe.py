"""The seeded input generator follows the stated recipe and workload shapes.

The parity tests and the benchmark stand these inputs in for the paper's
multimodal workloads, so their structure is part of what the numbers mean:
visual keys in tight per-head clusters, a few critical visual keys scaled x3,
text keys spread out, outlier channels x8, window queries at half the mean
key plus unit noise, and the prompt lengths and budgets of each workload.
"""
import numpy as np

from paper_2607_22586_gb300 import synth as S


def test_workload_shapes():
    W = S.WORKLOADS
    t = W["tiny-f32"]
    assert (t.n_q_heads, t.n_kv_heads, t.head_dim, t.dtype) == (4, 1, 64, S.F32)
    assert (t.seq_lens, t.n_visual, t.window, t.budgets, t.n_crit) == ((1024,), (960,), 16, (128,), 16)
    q = W["qwen7b-1layer"]
    assert (q.n_q_heads, q.n_kv_heads, q.head_dim, q.dtype) == (28, 4, 128, S.BF16)
    assert (q.seq_lens, q.n_visual, q.window, q.budgets, q.n_outlier) == ((4096,), (3840,), 32, (512,), 4)
    s = W["qwen7b-28l-32k"]
    assert (s.n_layers, s.seq_lens, s.n_images, s.n_centres, s.budgets) == (28, (32768,), 4, 512, (2048,))
    assert s.n_visual[0] == 4 * 8064 and s.seq_lens[0] - s.n_visual[0] == 512
    e = W["qwen7b-28l-8k"]
    assert (e.n_layers, e.seq_lens, e.n_visual) == (28, (8192,), (7936,))
    assert S.SWEEP_8K_WINDOWS == (16, 32, 64) and S.SWEEP_8K_BUDGETS == (256, 1024, 2048)
    g = W["72b-80l-ragged"]
    assert (g.n_q_heads, g.n_kv_heads, g.head_dim, g.n_layers) == (64, 8, 128, 80)
    assert g.seq_lens == (2048, 3000, 4096, 6000, 8192, 12000, 16384, 24576)
    assert g.n_visual == tuple(round(0.95 * n) for n in g.seq_lens)
    # 10% of each length, to the nearest multiple of 64
    assert g.budgets == (192, 320, 384, 576, 832, 1216, 1664, 2432)


def test_deterministic_per_seed_and_layer():
    wl = S.WORKLOADS["tiny-f32"]
    a, b, c = S.make_layer(wl, 0), S.make_layer(wl, 0), S.make_layer(wl, 1)
    for x, y in ((a.K, b.K), (a.V, b.V), (a.Qwin, b.Qwin)):
        np.testing.assert_array_equal(x, y)
    assert not np.array_equal(a.K, c.K)


def test_key_structure_tiny():
    wl = S.WORKLOADS["tiny-f32"]
    K = S.make_layer(wl, 0).K[:, 0].astype(np.float64)       # [T, d]
    nv = wl.n_visual[0]
    norms = np.linalg.norm(K, axis=1)
    vis_med = np.median(norms[:nv])
    crit = np.flatnonzero(norms[:nv] > 2.0 * vis_med)
    assert crit.size == wl.n_crit                                 # the x3 critical keys
    assert np.allclose(np.median(norms[crit]) / vis_med, 3.0, rtol=0.15)
    d2 = ((K[:, None, :] - K[None, :, :]) ** 2).sum(-1)
    np.fill_diagonal(d2, np.inf)
    nn = np.sqrt(d2.min(axis=1))
    plain = np.setdiff1d(np.arange(nv), crit)
    # same-cluster neighbours: key - key' ~ N(0, 2 * 0.1^2) per dim -> ~1.1 at d = 64
    assert np.mean(nn[plain] < 2.0) > 0.97
    # text keys are i.i.d. N(0, I): no neighbour closer than a few units
    assert np.all(nn[nv:] > 4.0)


def test_outlier_channels_and_window_queries():
    wl = S.WORKLOADS["qwen7b-1layer"]
    li = S.make_layer(wl, 0)
    K = li.K.astype(np.float64)                                   # [T, Hkv, d]
    text = K[wl.n_visual[0]:]                                     # unclustered keys
    ch_std = text.std(axis=(0, 1))
    top = np.sort(np.argsort(ch_std)[-wl.n_outlier:])
    rest = np.setdiff1d(np.arange(wl.head_dim), top)
    assert np.allclose(ch_std[top] / ch_std[rest].mean(), wl.outlier_scale, rtol=0.15)
    # window queries: 0.5 * mean_t K[:, h] + N(0, 1) for the r query heads of h
    r = wl.n_q_heads // wl.n_kv_heads
    kmean = K.mean(axis=0)                                        # [Hkv, d]
    resid = li.Qwin[0].astype(np.float64) - 0.5 * np.repeat(kmean, r, axis=0)[None]
    assert abs(resid.mean()) < 0.02 and abs(resid.std() - 1.0) < 0.02
    # values: N(0, 1)
    V = li.V.astype(np.float64)
    assert abs(V.mean()) < 0.01 and abs(V.std() - 1.0) < 0.01


def test_multi_image_clusters_are_per_image():
    # the 32K stack: four images with their own 512 centres each; a (not
    # critical) visual key's nearest neighbour among all visual keys lies in
    # its own cluster, hence in its own image
    wl = S.WORKLOADS["qwen7b-28l-32k"].replace(n_layers=1)
    nv = wl.n_visual[0]
    K = S.make_layer(wl, 0).K[:nv, 0].astype(np.float32)         # KV head 0, visual keys
    per = nv // wl.n_images
    norms = np.linalg.norm(K, axis=1)
    rng = np.random.default_rng(0)
    idx = rng.choice(np.flatnonzero(norms < 2.0 * np.median(norms)), size=400, replace=False)
    q = K[idx]
    d2 = (q ** 2).sum(1)[:, None] + (K ** 2).sum(1)[None, :] - 2.0 * q @ K.T
    d2[np.arange(idx.size), idx] = np.inf
    nn = np.argmin(d2, axis=1)
    assert np.mean(nn // per == idx // per) > 0.99
    # and that neighbour is close: same-cluster keys differ by ~0.1 * sqrt(2 d)
    assert np.median(np.sqrt(np.maximum(d2.min(axis=1), 0.0))) < 2.5
