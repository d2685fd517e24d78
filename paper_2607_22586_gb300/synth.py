"""Seeded synthetic MLLM-shaped inputs for prefill-only KV selection.

This module only draws inputs; it holds none of the selection method's
arithmetic. Both the CPU oracle (through the tests) and the CUDA path (through
the tests and the benchmark) consume exactly the arrays it returns.

The workloads stand in for the paper's multimodal benchmarks (OCRBench, DocVQA,
ChartQA, TextVQA, TextCaps, MMMU), whose prompts are dominated by visual tokens
(Table 4 lists 642-4830 input tokens on average, mostly visual). No dataset
item is reproduced: every key, value and query is a seeded random draw with
the structure below.

Recipe (per layer, per request):
  * visual keys: every KV head has its own cluster centres ~ N(0, I); each
    visual token is assigned to one cluster uniformly at random (the assignment
    is shared by all KV heads of the request, as the same image patch feeds
    every head); key = centre + N(0, noise^2 I);
  * a uniform random subset of the visual tokens ("critical" patches, shared by
    all heads) is scaled by ``crit_scale``;
  * text keys (the tail of the prompt) are i.i.d. N(0, I);
  * optional outlier channels: a fixed set of channels, chosen once per seed
    and shared by all tokens, heads and layers, is scaled by ``outlier_scale``
    on every key;
  * window queries (the last W query positions): 0.5 * mean_t(K[:, h]) + N(0, I)
    for every query head of KV head h;
  * values are i.i.d. N(0, I).
Floating-point draws are float32 from ``numpy.random.Generator(Philox)`` keyed
by (seed, layer); bf16 workloads are rounded to bf16 (round-to-nearest-even).
"""
from __future__ import annotations

import dataclasses
from typing import List, Optional, Sequence

import numpy as np

BF16 = "bf16"
F32 = "f32"


@dataclasses.dataclass(frozen=True)
class Workload:
    """Shape and generation recipe of one synthetic workload."""

    name: str
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    dtype: str
    n_layers: int
    seq_lens: Sequence[int]          # prompt length T_b of each request
    n_visual: Sequence[int]          # visual tokens of each request (prefix)
    window: int                      # observation window W
    budgets: Sequence[int]           # per-KV-head budget C_b of each request
    n_images: int = 1                # visual part split in equal images
    n_centres: int = 60              # clusters per image and KV head
    noise: float = 0.1               # std of a visual key around its centre
    crit_frac: Optional[float] = None  # fraction of visual tokens scaled
    n_crit: Optional[int] = None     # or an absolute number of them
    crit_scale: float = 3.0
    n_outlier: int = 0
    outlier_scale: float = 8.0
    seed: int = 0

    @property
    def batch(self) -> int:
        return len(self.seq_lens)

    @property
    def total_tokens(self) -> int:
        return int(sum(self.seq_lens))

    def cu_seqlens(self) -> np.ndarray:
        return np.concatenate([[0], np.cumsum(self.seq_lens)]).astype(np.int32)

    def replace(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)


def _round_nearest_64(x: float) -> int:
    """Nearest multiple of 64, halves rounded up."""
    return int(np.floor(x / 64.0 + 0.5)) * 64


_CFG4_LENS = (2048, 3000, 4096, 6000, 8192, 12000, 16384, 24576)

WORKLOADS = {
    # Tiny single layer in fp32.
    "tiny-f32": Workload(
        name="tiny-f32", n_q_heads=4, n_kv_heads=1, head_dim=64, dtype=F32,
        n_layers=1, seq_lens=(1024,), n_visual=(960,), window=16,
        budgets=(128,), n_centres=60, n_crit=16),
    # Qwen2.5-VL-7B-shaped single layer.
    "qwen7b-1layer": Workload(
        name="qwen7b-1layer", n_q_heads=28, n_kv_heads=4, head_dim=128,
        dtype=BF16, n_layers=1, seq_lens=(4096,), n_visual=(3840,), window=32,
        budgets=(512,), n_centres=256, crit_frac=0.01, n_outlier=4),
    # Full 28-layer stack, 8K prompt; window and budget are swept.
    "qwen7b-28l-8k": Workload(
        name="qwen7b-28l-8k", n_q_heads=28, n_kv_heads=4, head_dim=128,
        dtype=BF16, n_layers=28, seq_lens=(8192,), n_visual=(7936,), window=32,
        budgets=(1024,), n_centres=256, crit_frac=0.01, n_outlier=4),
    # High-resolution multi-image long context: 4 images x 8064 + 512 text.
    "qwen7b-28l-32k": Workload(
        name="qwen7b-28l-32k", n_q_heads=28, n_kv_heads=4, head_dim=128,
        dtype=BF16, n_layers=28, seq_lens=(32768,), n_visual=(32256,),
        window=32, budgets=(2048,), n_images=4, n_centres=512, crit_frac=0.01,
        n_outlier=4),
    # 72B-class ragged batch of 8 requests, 80 layers.
    "72b-80l-ragged": Workload(
        name="72b-80l-ragged", n_q_heads=64, n_kv_heads=8, head_dim=128,
        dtype=BF16, n_layers=80, seq_lens=_CFG4_LENS,
        n_visual=tuple(int(round(0.95 * t)) for t in _CFG4_LENS), window=32,
        budgets=tuple(_round_nearest_64(0.1 * t) for t in _CFG4_LENS),
        n_centres=256, crit_frac=0.01, n_outlier=4),
}

# Sweep of the 28-layer 8K stack.
SWEEP_8K_WINDOWS = (16, 32, 64)
SWEEP_8K_BUDGETS = (256, 1024, 2048)


def bf16_round_bits(x: np.ndarray) -> np.ndarray:
    """float32 -> bf16 bit patterns (uint16), round to nearest even."""
    u = np.array(x, dtype=np.float32, copy=True).view(np.uint32)
    lsb = u >> np.uint32(16)
    lsb &= np.uint32(1)
    u += np.uint32(0x7FFF)
    u += lsb
    u >>= np.uint32(16)
    return u.astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (b.astype(np.uint32) << np.uint32(16)).view(np.float32)


def round_to_dtype(x: np.ndarray, dtype: str) -> np.ndarray:
    """float32 copy of x holding values exactly representable in dtype."""
    if dtype == BF16:
        return bf16_bits_to_f32(bf16_round_bits(x))
    return np.ascontiguousarray(x, dtype=np.float32)


def _outlier_channels(wl: Workload) -> np.ndarray:
    if wl.n_outlier == 0:
        return np.zeros(0, dtype=np.int64)
    rng = np.random.Generator(np.random.Philox(key=[wl.seed, 0xFFFFFFFF]))
    return np.sort(rng.choice(wl.head_dim, size=wl.n_outlier, replace=False))


def _request_keys(rng: np.random.Generator, wl: Workload, t_len: int,
                  n_vis: int, outliers: np.ndarray) -> np.ndarray:
    """Keys of one request, [T, Hkv, d] float32 (before dtype rounding)."""
    hkv, d = wl.n_kv_heads, wl.head_dim
    keys = np.empty((t_len, hkv, d), dtype=np.float32)
    per_img = [n_vis // wl.n_images + (1 if i < n_vis % wl.n_images else 0)
               for i in range(wl.n_images)]
    start = 0
    for n_img in per_img:
        centres = rng.standard_normal((hkv, wl.n_centres, d), dtype=np.float32)
        assign = rng.integers(0, wl.n_centres, size=n_img)
        noise = rng.standard_normal((n_img, hkv, d), dtype=np.float32)
        keys[start:start + n_img] = (
            centres[:, assign, :].transpose(1, 0, 2) + np.float32(wl.noise) * noise)
        start += n_img
    keys[n_vis:] = rng.standard_normal((t_len - n_vis, hkv, d), dtype=np.float32)
    if wl.n_crit is not None:
        n_crit = wl.n_crit
    else:
        n_crit = int(round((wl.crit_frac or 0.0) * n_vis))
    if n_crit:
        crit = rng.choice(n_vis, size=n_crit, replace=False)
        keys[crit] *= np.float32(wl.crit_scale)
    if outliers.size:
        keys[:, :, outliers] *= np.float32(wl.outlier_scale)
    return keys


@dataclasses.dataclass
class LayerInputs:
    """One layer of a workload. Arrays are float32 holding dtype-exact values;
    ``*_bits`` are the same data as bf16 bit patterns (bf16 workloads only)."""

    K: np.ndarray      # [total_T, Hkv, d]
    V: np.ndarray      # [total_T, Hkv, d]
    Qwin: np.ndarray   # [B, W, Hq, d]

    def native(self, dtype: str):
        """(K, V, Qwin) in the storage dtype: uint16 bf16 bits or float32."""
        if dtype == BF16:
            # values are already bf16-exact: the high half of the float32 is it
            return tuple((np.ascontiguousarray(a).view(np.uint32) >> np.uint32(16)).astype(np.uint16)
                         for a in (self.K, self.V, self.Qwin))
        return self.K, self.V, self.Qwin


def make_layer(wl: Workload, layer: int) -> LayerInputs:
    """Draw one layer of ``wl``; deterministic in (wl.seed, layer)."""
    rng = np.random.Generator(np.random.Philox(key=[wl.seed, layer]))
    outliers = _outlier_channels(wl)
    hq, hkv, d, w = wl.n_q_heads, wl.n_kv_heads, wl.head_dim, wl.window
    r = hq // hkv
    ks, vs, qs = [], [], []
    for t_len, n_vis in zip(wl.seq_lens, wl.n_visual):
        k = round_to_dtype(_request_keys(rng, wl, t_len, n_vis, outliers), wl.dtype)
        v = round_to_dtype(rng.standard_normal((t_len, hkv, d), dtype=np.float32), wl.dtype)
        kmean = k.mean(axis=0, dtype=np.float64).astype(np.float32)  # [Hkv, d]
        q = (np.float32(0.5) * np.repeat(kmean, r, axis=0)[None, :, :]
             + rng.standard_normal((w, hq, d), dtype=np.float32))
        ks.append(k)
        vs.append(v)
        qs.append(round_to_dtype(q, wl.dtype))
    return LayerInputs(K=np.concatenate(ks), V=np.concatenate(vs), Qwin=np.stack(qs))


def make_prompt_queries(wl: Workload, layer: int, li: LayerInputs,
                        seed_tag: int = 0x51465550) -> np.ndarray:
    """All prompt queries of one layer, [total_T, Hq, d] (dtype-exact float32),
    consistent with ``li`` (the layer drawn by make_layer).

    Text positions follow the window recipe (half the request's per-head key
    mean plus unit normal noise); visual positions add a seeded per-(head,
    dimension) modality offset drawn N(0, 1) per request, so that prompt-wide
    and window statistics differ the way text and image tokens do. The last
    min(W, T) rows of each request are its window queries ``li.Qwin``.
    """
    rng = np.random.Generator(np.random.Philox(key=[wl.seed ^ seed_tag, layer]))
    hq, hkv, d, w = wl.n_q_heads, wl.n_kv_heads, wl.head_dim, wl.window
    r = hq // hkv
    cu = wl.cu_seqlens()
    out = np.empty((wl.total_tokens, hq, d), dtype=np.float32)
    for b, (t_len, n_vis) in enumerate(zip(wl.seq_lens, wl.n_visual)):
        k = li.K[cu[b]:cu[b + 1]]
        kmean = k.mean(axis=0, dtype=np.float64).astype(np.float32)
        q = (np.float32(0.5) * np.repeat(kmean, r, axis=0)[None, :, :]
             + rng.standard_normal((t_len, hq, d), dtype=np.float32))
        q[:n_vis] += rng.standard_normal((hq, d), dtype=np.float32)[None]
        q = round_to_dtype(q, wl.dtype)
        nw = min(w, t_len)
        q[t_len - nw:] = li.Qwin[b, w - nw:]
        out[cu[b]:cu[b + 1]] = q
    return out


def make_hidden_states(wl: Workload, layer: int, d_model: int,
                       seed_tag: int = 0x48494444) -> np.ndarray:
    """Prefill hidden states of one layer, [total_T, d_model] (dtype-exact
    float32): per feature a mean N(0, 0.5^2) and a scale U(0.5, 1.5) shared by
    the requests, four massive-activation features with mean +-20 (large,
    nearly constant features of LLM residual streams), a per-request
    N(0, 0.5^2) modality offset on visual positions, unit normal noise."""
    rng = np.random.Generator(np.random.Philox(key=[wl.seed ^ seed_tag, layer]))
    mean = rng.normal(0.0, 0.5, size=d_model).astype(np.float32)
    scale = rng.uniform(0.5, 1.5, size=d_model).astype(np.float32)
    massive = rng.choice(d_model, size=min(4, d_model), replace=False)
    mean[massive] = np.float32(20.0) * np.sign(rng.standard_normal(massive.size)).astype(np.float32)
    out = np.empty((wl.total_tokens, d_model), dtype=np.float32)
    cu = wl.cu_seqlens()
    for b, (t_len, n_vis) in enumerate(zip(wl.seq_lens, wl.n_visual)):
        h = mean[None, :] + scale[None, :] * rng.standard_normal((t_len, d_model), dtype=np.float32)
        h[:n_vis] += np.float32(0.5) * rng.standard_normal(d_model, dtype=np.float32)[None]
        out[cu[b]:cu[b + 1]] = round_to_dtype(h, wl.dtype)
    return out


def make_query_projection(wl: Workload, layer: int, d_model: int, with_bias: bool = True,
                          seed_tag: int = 0x57515052):
    """Query projection of one layer: W_Q [Hq*d, d_model] with entries
    N(0, 1/d_model) (so projected proxies have O(1) features) and a bias
    [Hq*d] N(0, 0.5^2) or None; dtype-exact float32."""
    rng = np.random.Generator(np.random.Philox(key=[wl.seed ^ seed_tag, layer]))
    f = wl.n_q_heads * wl.head_dim
    w = rng.standard_normal((f, d_model), dtype=np.float32) * np.float32(1.0 / np.sqrt(d_model))
    bias = (rng.standard_normal(f, dtype=np.float32) * np.float32(0.5)) if with_bias else None
    return (round_to_dtype(w, wl.dtype),
            None if bias is None else round_to_dtype(bias, wl.dtype))


def make_decode_queries(wl: Workload, layer: int, li: LayerInputs, n_dec: int,
                        spread: float = 1.5, seed_tag: int = 0x44454351) -> np.ndarray:
    """Synthetic decode-time queries of one layer, [B, n_dec, Hq, d]
    (dtype-exact float32): the window recipe (half the request's per-head
    key mean) with noise of std ``spread`` > 1, since decode-time queries
    spread wider than prefill ones (§1, Fig. 1a)."""
    rng = np.random.Generator(np.random.Philox(key=[wl.seed ^ seed_tag, layer]))
    hq, hkv, d = wl.n_q_heads, wl.n_kv_heads, wl.head_dim
    cu = wl.cu_seqlens()
    out = np.empty((wl.batch, n_dec, hq, d), dtype=np.float32)
    for b in range(wl.batch):
        kmean = li.K[cu[b]:cu[b + 1]].mean(axis=0, dtype=np.float64).astype(np.float32)
        q = (np.float32(0.5) * np.repeat(kmean, hq // hkv, axis=0)[None]
             + np.float32(spread) * rng.standard_normal((n_dec, hq, d), dtype=np.float32))
        out[b] = round_to_dtype(q, wl.dtype)
    return out


def make_kept_indices(wl: Workload, seed: int) -> np.ndarray:
    """A seeded kept set in the output layout [R, Hkv] int32: per request
    and KV head min(C_b, T_b) distinct ascending indices, always T_b - 1 (the
    shape a selection produces, for tests that need one the oracle can take)."""
    rng = np.random.Generator(np.random.Philox(key=[seed, 0x4B455054]))
    rows = []
    for t_len, c in zip(wl.seq_lens, wl.budgets):
        keep = min(c, t_len)
        blk = np.empty((keep, wl.n_kv_heads), dtype=np.int32)
        for h in range(wl.n_kv_heads):
            rest = rng.choice(t_len - 1, size=keep - 1, replace=False) if keep > 1 else np.zeros(0, int)
            blk[:, h] = np.sort(np.concatenate([rest, [t_len - 1]]))
        rows.append(blk)
    return np.concatenate(rows)


def make_proxies(wl: Workload, n_proxies: int, layer: int, scale: float = 8.0,
                 seed_tag: int = 0x50524F58) -> np.ndarray:
    """Seeded stand-alone proxy set [B, Hq, N_p, d] (dtype-exact float32).

    Used where a test feeds both implementations the same proxies: draws are
    N(0, scale^2), the magnitude variance-expanded proxies reach at gamma=10.
    """
    rng = np.random.Generator(np.random.Philox(key=[wl.seed ^ seed_tag, layer]))
    p = rng.standard_normal((wl.batch, wl.n_q_heads, n_proxies, wl.head_dim),
                            dtype=np.float32) * np.float32(scale)
    return round_to_dtype(p, wl.dtype)


def make_group_masses(n_heads: int, n_groups: int, t_len: int, mass_per_group: float,
                      seed: int, zero_frac: float = 0.05,
                      dup_frac: float = 0.2) -> np.ndarray:
    """Seeded non-negative group masses [H, G, T] for the vote/selection step.

    Log-normally spread like attention mass, with planted exact duplicates and
    zeros so that ties are exercised. Every value is a float32 that is also a
    multiple of 2**-40, so sums of them are exact both in float64 and in 64-bit
    fixed point with 40 fractional bits.
    """
    rng = np.random.Generator(np.random.Philox(key=[seed, 0x4D415353]))
    x = np.exp(rng.normal(0.0, 3.0, size=(n_heads, n_groups, t_len)))
    x[rng.random(x.shape) < zero_frac] = 0.0
    dup = rng.random(x.shape) < dup_frac
    src = rng.integers(0, t_len, size=x.shape)
    x = np.where(dup, np.take_along_axis(x, src, axis=2), x)
    x = x / x.sum(axis=2, keepdims=True) * mass_per_group
    x32 = x.astype(np.float32).astype(np.float64)
    small = x32 < 2.0 ** -17          # below this a float32 ulp is < 2**-40
    x32[small] = np.round(x32[small] * 2.0 ** 40) * 2.0 ** -40
    return x32.astype(np.float32)


def make_scores(n_heads: int, t_len: int, n_groups: int, seed: int,
                anchor_zero_frac: float = 0.3) -> np.ndarray:
    """Seeded scores [H, T] shaped like vote + anchor: integer votes in
    [0, G] plus an anchor in [0, 1) that is exactly zero for a fraction of keys
    (so equal scores occur), float32."""
    rng = np.random.Generator(np.random.Philox(key=[seed, 0x53434F52]))
    votes = rng.integers(0, n_groups + 1, size=(n_heads, t_len)).astype(np.float32)
    anchor = rng.random((n_heads, t_len), dtype=np.float32) * np.float32(0.999)
    anchor[rng.random((n_heads, t_len)) < anchor_zero_frac] = 0.0
    return (votes + anchor).astype(np.float32)


def layers(wl: Workload, which: Optional[Sequence[int]] = None) -> List[LayerInputs]:
    idx = range(wl.n_layers) if which is None else which
    return [make_layer(wl, l) for l in idx]
