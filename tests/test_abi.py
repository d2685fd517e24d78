"""Host-side checks of the C ABI that need no GPU: the library builds and
loads, exports every entry point declared in include/mmshift.h, and rejects
bad arguments before touching the device."""
import ctypes
import os
import re

import pytest

import paper_2607_22586_gb300 as M
from paper_2607_22586_gb300 import _lib as L

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_entry_points():
    with open(os.path.join(ROOT, "include", "mmshift.h")) as f:
        text = f.read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(mmshift_[a-z_0-9]+)\s*\(", text)))


def test_library_exports_every_declared_symbol():
    lib = M.load_library()
    names = declared_entry_points()
    assert len(names) >= 12
    for n in names:
        assert hasattr(lib, n), n
    assert sorted(L.EXPORTED) == names


def test_default_params_are_the_papers():
    p = M.default_params()
    assert (p.n_proxies, p.n_groups) == (512, 32)
    assert p.gamma == 10.0 and p.lambda_ == 1.0
    assert abs(p.tau - 0.95) < 1e-7
    assert p.score_mode == L.MMSHIFT_SCORE_VOTE


def _shape(**kw):
    base = dict(n_q_heads=8, n_kv_heads=2, head_dim=128, window=8, dtype=0,
                cu_seqlens=[0, 100, 250], budgets=[16, 300])
    base.update(kw)
    return M.make_shape(**base)


def test_output_rows_and_workspace():
    s = _shape()
    assert M.mmshift_output_rows(s) == 16 + 150
    n = M.mmshift_workspace_size(s, M.default_params())
    assert n > 0 and n % 256 == 0


@pytest.mark.parametrize("bad,code", [
    (dict(n_q_heads=7), L.MMSHIFT_ERR_INVALID_ARG),      # Hq not a multiple of Hkv
    (dict(window=1), L.MMSHIFT_ERR_INVALID_ARG),         # std needs W >= 2
    (dict(head_dim=96), L.MMSHIFT_ERR_UNSUPPORTED),
    (dict(dtype=5), L.MMSHIFT_ERR_UNSUPPORTED),
    (dict(cu_seqlens=[0, 100, 100]), L.MMSHIFT_ERR_INVALID_ARG),   # empty request
    (dict(cu_seqlens=[1, 100, 200]), L.MMSHIFT_ERR_INVALID_ARG),
    (dict(budgets=[16, 0]), L.MMSHIFT_ERR_INVALID_ARG),
])
def test_bad_shapes_rejected(bad, code):
    s = _shape(**bad)
    with pytest.raises(L.MMShiftError) as ei:
        M.mmshift_workspace_size(s, M.default_params())
    assert ei.value.code == code


@pytest.mark.parametrize("bad", [
    dict(n_proxies=500), dict(n_groups=0), dict(gamma=0.0), dict(tau=0.0), dict(tau=1.5),
    dict(lam=-1.0), dict(score_mode=7), dict(layer_id=-1), dict(softmax_scale=-1.0),
])
def test_bad_params_rejected(bad):
    p = M.default_params(**bad)
    with pytest.raises(L.MMShiftError) as ei:
        M.mmshift_workspace_size(_shape(), p)
    assert ei.value.code == L.MMSHIFT_ERR_INVALID_ARG


def test_null_and_workspace_errors_return_before_any_launch():
    s = _shape()
    p = M.default_params()
    n = M.mmshift_workspace_size(s, p)
    fake = 1 << 40  # never dereferenced: validation fails first
    assert M.mmshift_select(s, None, fake, fake, None, p, fake, fake, fake, None, fake, n) == \
        L.MMSHIFT_ERR_INVALID_ARG
    assert M.mmshift_select(s, fake, fake, fake, None, p, fake, fake, fake, None, fake, n - 256) == \
        L.MMSHIFT_ERR_WORKSPACE
    assert M.mmshift_select(s, fake, fake, fake, None, p, fake, fake, fake, None, fake + 8, n) == \
        L.MMSHIFT_ERR_WORKSPACE
    assert M.mmshift_topk(s, None, fake, fake, n) == L.MMSHIFT_ERR_INVALID_ARG
    assert M.mmshift_gather(s, fake, fake, None, fake, fake, fake, n) == L.MMSHIFT_ERR_INVALID_ARG
    lib = M.load_library()
    assert lib.mmshift_status_string(L.MMSHIFT_ERR_TIMEOUT) == b"device-side wait timed out"


def test_prefill_stats_validation_before_any_launch():
    s = _shape()
    n = M.mmshift_prefill_stats_workspace_size(s)
    # per layer and request: ceil(T / 512) chunks x 3 partial sums x Hq * d floats
    assert n == ((1 * 2 * 1 * 3 * 8 * 128 * 4 + 255) // 256) * 256
    fake = 1 << 40
    assert M.mmshift_prefill_stats(s, None, 0, fake, fake, n) == L.MMSHIFT_ERR_INVALID_ARG
    assert M.mmshift_prefill_stats(s, fake + 4, 0, fake, fake, n) == L.MMSHIFT_ERR_INVALID_ARG  # unaligned
    assert M.mmshift_prefill_stats(s, fake, 0, fake, fake, n - 256) == L.MMSHIFT_ERR_WORKSPACE
    assert M.mmshift_prefill_stats(s, fake, 12, fake, fake, n) == L.MMSHIFT_ERR_INVALID_ARG  # stride
    s2 = _shape(n_layers=2, layer_stride_kv=250 * 2 * 128, layer_stride_q=2 * 8 * 8 * 128)
    assert M.mmshift_prefill_stats(s2, fake, 100, fake, fake, n) == L.MMSHIFT_ERR_INVALID_ARG  # too small
    p = M.default_params()
    assert M.mmshift_build_proxies_from_stats(s, None, p, fake) == L.MMSHIFT_ERR_INVALID_ARG
    assert M.mmshift_build_proxies_from_stats(s, fake, p, None) == L.MMSHIFT_ERR_INVALID_ARG


def test_hidden_entries_validation_before_any_launch():
    s = _shape()
    p = M.default_params()
    dm = 1024
    n = M.mmshift_hidden_stats_workspace_size(s, dm)
    assert n == ((1 * 2 * 1 * 3 * dm * 4 + 255) // 256) * 256
    fake = 1 << 40
    assert M.mmshift_hidden_stats(s, dm, None, 0, fake, fake, n) == L.MMSHIFT_ERR_INVALID_ARG
    assert M.mmshift_hidden_stats(s, dm, fake + 8, 0, fake, fake, n) == L.MMSHIFT_ERR_INVALID_ARG
    assert M.mmshift_hidden_stats(s, dm, fake, 0, fake, fake, n - 256) == L.MMSHIFT_ERR_WORKSPACE
    assert M.mmshift_hidden_stats(s, 1020, fake, 0, fake, fake, n) == L.MMSHIFT_ERR_INVALID_ARG
    # hidden proxies: N = 512 proxies -> 4 tiles of 128 rows, sampled states in the workspace
    w = M.mmshift_hidden_proxies_workspace_size(s, dm, p)
    assert w >= 256 + 2 * 512 * dm * 2
    args = dict(hstats=fake, W_Q=fake, wq_layer_stride=0, bias_q=None, rope_pos=None, params=p,
                proxies=fake, workspace=fake, workspace_bytes=w)

    def call(shape=s, d_model=dm, **kw):
        a = dict(args)
        a.update(kw)
        return M.mmshift_build_hidden_proxies(shape, d_model, a["hstats"], a["W_Q"], a["wq_layer_stride"],
                                              a["bias_q"], a["rope_pos"], a["params"], a["proxies"],
                                              a["workspace"], a["workspace_bytes"])

    assert call(W_Q=None) == L.MMSHIFT_ERR_INVALID_ARG
    assert call(hstats=None) == L.MMSHIFT_ERR_INVALID_ARG
    assert call(W_Q=fake + 4) == L.MMSHIFT_ERR_INVALID_ARG            # unaligned weights
    assert call(workspace=fake + 16) == L.MMSHIFT_ERR_INVALID_ARG      # unaligned workspace
    assert call(wq_layer_stride=12) == L.MMSHIFT_ERR_INVALID_ARG       # stride not a multiple of 8
    assert call(workspace_bytes=w - 256) == L.MMSHIFT_ERR_WORKSPACE
    assert call(d_model=1000) == L.MMSHIFT_ERR_UNSUPPORTED             # not a multiple of 64
    assert call(shape=_shape(dtype=1)) == L.MMSHIFT_ERR_UNSUPPORTED     # bf16 only
    assert call(shape=_shape(n_q_heads=3, n_kv_heads=1, head_dim=64)) == L.MMSHIFT_ERR_UNSUPPORTED
    s2 = _shape(n_layers=2, layer_stride_kv=250 * 2 * 128, layer_stride_q=2 * 8 * 8 * 128)
    w2 = M.mmshift_hidden_proxies_workspace_size(s2, dm, p)
    assert call(shape=s2, wq_layer_stride=8 * 128 * dm - 8, workspace_bytes=w2) == L.MMSHIFT_ERR_INVALID_ARG
    assert call(params=M.default_params(n_proxies=0, n_groups=0)) == L.MMSHIFT_OK   # nothing to do


def test_coverage_validation_before_any_launch():
    s = _shape()
    n = M.mmshift_coverage_workspace_size(s, 16)
    assert n > 0 and n % 256 == 0
    fake = 1 << 40
    args = [fake, fake, fake, 16, 0.0, fake, fake, fake, n]
    bad = list(args)
    bad[3] = 0
    assert M.mmshift_coverage(s, *bad) == L.MMSHIFT_ERR_INVALID_ARG          # no decode queries
    bad = list(args)
    bad[3] = 1025
    assert M.mmshift_coverage(s, *bad) == L.MMSHIFT_ERR_INVALID_ARG          # more than 1024
    bad = list(args)
    bad[4] = -1.0
    assert M.mmshift_coverage(s, *bad) == L.MMSHIFT_ERR_INVALID_ARG          # negative scale
    for i in (0, 1, 2, 5, 6):
        bad = list(args)
        bad[i] = None
        assert M.mmshift_coverage(s, *bad) == L.MMSHIFT_ERR_INVALID_ARG, i
    bad = list(args)
    bad[8] = n - 256
    assert M.mmshift_coverage(s, *bad) == L.MMSHIFT_ERR_WORKSPACE
    with pytest.raises(L.MMShiftError):
        M.mmshift_coverage_workspace_size(s, 0)
