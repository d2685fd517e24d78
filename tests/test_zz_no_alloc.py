"""The allocation-free vote + top-k entry point.

Some callers cannot allocate device memory at all -- a runtime or plugin host
that owns every device allocation and grants the library no workspace, or a
serving loop whose memory plan is frozen after start-up. For them the library
offers mmshift_scores_topk_noalloc, whose scratch is a static device array
compiled into the library. These tests check, through the C ABI, that it
returns exactly what the workspace-based mmshift_scores_topk returns, on two
different calls in a row (the shared array keeps the previous call's bytes),
and that a problem too large for the array is refused up front.

This file is named to be collected last.
"""
import numpy as np
import pytest
import torch

import paper_2607_22586_gb300 as M
from paper_2607_22586_gb300 import _lib as L
from paper_2607_22586_gb300 import synth as S
from tests import parity as PT

BASE = S.WORKLOADS["72b-80l-ragged"]


def _case(seed, lens, budgets, n_groups, tau):
    wl = BASE.replace(n_layers=1, seq_lens=lens, n_visual=tuple(0 for _ in lens), budgets=budgets)
    h = PT.hyper(n_proxies=16 * n_groups, n_groups=n_groups, tau=tau)
    gm = S.make_group_masses(wl.n_kv_heads, n_groups, wl.total_tokens, 128.0, seed=seed)
    anchor = S.make_scores(wl.n_kv_heads, wl.total_tokens, 0, seed=seed + 1) * np.float32(0.5)
    return wl, h, gm, anchor


@pytest.mark.gpu
def test_noalloc_matches_workspace_entry_point_on_two_calls():
    cases = [_case(11, (3000, 700, 5), (256, 64, 2), 32, 0.95),
             _case(12, (9000, 128), (1024, 200), 8, 0.5)]
    for wl, h, gm, anchor in cases:
        shape = PT.shape_of(wl)
        params = PT.abi_params(h)
        rows = M.mmshift_output_rows(shape)
        hkv, T = wl.n_kv_heads, wl.total_tokens
        gm_d = torch.from_numpy(gm).cuda()
        an_d = torch.from_numpy(anchor).cuda()
        # reference: the workspace entry point
        ws_bytes = M.mmshift_workspace_size(shape, params)
        ws = torch.zeros(ws_bytes, dtype=torch.uint8, device="cuda")
        idx_ref = torch.full((1, rows, hkv), -1, dtype=torch.int32, device="cuda")
        sc_ref = torch.empty((1, hkv, T), device="cuda")
        M.check(M.mmshift_scores_topk(shape, params, gm_d, an_d, sc_ref, idx_ref, ws, ws_bytes),
                "scores_topk")
        # allocation-free: scores kept in the static scratch, then in a caller buffer
        idx_a = torch.full((1, rows, hkv), -1, dtype=torch.int32, device="cuda")
        M.check(M.mmshift_scores_topk_noalloc(shape, params, gm_d, an_d, None, idx_a), "noalloc")
        idx_b = torch.full((1, rows, hkv), -1, dtype=torch.int32, device="cuda")
        sc_b = torch.empty((1, hkv, T), device="cuda")
        M.check(M.mmshift_scores_topk_noalloc(shape, params, gm_d, an_d, sc_b, idx_b), "noalloc")
        torch.cuda.synchronize()
        assert torch.equal(idx_a, idx_ref)
        assert torch.equal(idx_b, idx_ref)
        assert torch.equal(sc_b, sc_ref)


@pytest.mark.gpu
def test_noalloc_mass_mode_scores_in_scratch():
    """MASS scoring (no vote, no anchor): the scores live in the static array
    where the vote's bitmaps would start; twice in a row, equal to the
    workspace entry point."""
    wl, h, gm, _ = _case(13, (2500, 900, 3), (300, 128, 1), 8, 0.95)
    h = dict(h, score_mode=L.MMSHIFT_SCORE_MASS)
    shape = PT.shape_of(wl)
    params = PT.abi_params(h)
    rows = M.mmshift_output_rows(shape)
    hkv, T = wl.n_kv_heads, wl.total_tokens
    gm_d = torch.from_numpy(gm).cuda()
    ws_bytes = M.mmshift_workspace_size(shape, params)
    ws = torch.zeros(ws_bytes, dtype=torch.uint8, device="cuda")
    idx_ref = torch.full((1, rows, hkv), -1, dtype=torch.int32, device="cuda")
    sc_ref = torch.empty((1, hkv, T), device="cuda")
    M.check(M.mmshift_scores_topk(shape, params, gm_d, None, sc_ref, idx_ref, ws, ws_bytes),
            "scores_topk mass")
    for _ in range(2):
        idx = torch.full((1, rows, hkv), -1, dtype=torch.int32, device="cuda")
        M.check(M.mmshift_scores_topk_noalloc(shape, params, gm_d, None, None, idx), "noalloc mass")
        torch.cuda.synchronize()
        assert torch.equal(idx, idx_ref)


def test_noalloc_rejects_problem_larger_than_its_scratch():
    # 8 KV heads x 32 groups x 300K tokens of bitmaps + scores exceed 8 MiB;
    # refused by host-side validation before any device work
    wl, h, _, _ = _case(1, (300000,), (1024,), 32, 0.95)
    shape = PT.shape_of(wl)
    fake = 1 << 40
    st = M.mmshift_scores_topk_noalloc(shape, PT.abi_params(h), fake, fake, None, fake)
    assert st == L.MMSHIFT_ERR_WORKSPACE
    assert L.MMSHIFT_NOALLOC_SCRATCH_BYTES == 8 << 20
