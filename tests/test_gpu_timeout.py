"""Failure detection of the bounded device-side waits, without a GPU fault.

Every mbarrier wait in the tensor-core kernels is bounded: a CTA whose wait
gives up raises the timeout bit in the workspace status word, stops issuing
work, waits (bounded) for the TMA loads and MMAs it already issued, frees its
tensor memory and exits. Here one wait is made to run out on purpose (the
test-only mmshift_debug.test_stuck_wait: a wait on a barrier that nothing
arrives on, bounded at 64 polls); the host must read MMSHIFT_ERR_TIMEOUT,
and the very next normal call on the same workspace must match the oracle.
"""
import numpy as np
import pytest
import torch

import paper_2607_22586_gb300 as M
from paper_2607_22586_gb300 import _lib as LB
from paper_2607_22586_gb300 import synth as S
from tests import parity as PT

pytestmark = pytest.mark.gpu

WL = S.WORKLOADS["qwen7b-1layer"].replace(seq_lens=(1500, 700), n_visual=(1400, 650),
                                          budgets=(200, 64))


def _requests(wl):
    cu = wl.cu_seqlens()
    outs = np.concatenate([[0], np.cumsum(np.minimum(wl.budgets, wl.seq_lens))])
    return [(b, int(cu[b]), int(cu[b + 1]), int(outs[b])) for b in range(wl.batch)]


def test_stuck_wait_reports_timeout_and_next_call_is_clean():
    li = S.make_layer(WL, 0)
    h = PT.hyper(n_proxies=64, n_groups=4, seed=2)
    prox = S.make_proxies(WL, h["n_proxies"], 0)
    shape = PT.shape_of(WL)
    params = PT.abi_params(h)
    ws_bytes = M.mmshift_workspace_size(shape, params)
    ws = torch.zeros(ws_bytes, dtype=torch.uint8, device="cuda")
    rows = M.mmshift_output_rows(shape)
    K, V, Q = PT.dev(li.K, WL.dtype), PT.dev(li.V, WL.dtype), PT.dev(li.Qwin, WL.dtype)
    P = PT.dev(prox[None], WL.dtype)
    idx = torch.full((1, rows, WL.n_kv_heads), -7, dtype=torch.int32, device="cuda")
    ok = torch.empty((1, rows, WL.n_kv_heads, WL.head_dim), dtype=torch.bfloat16, device="cuda")
    ov = torch.empty_like(ok)
    for _ in range(2):
        dbg = M.make_debug(test_stuck_wait=1)
        M.check(M.mmshift_select(shape, K, V, Q, P, params, idx, ok, ov, dbg, ws, ws_bytes),
                "select with a stuck wait")
        assert dbg.score_path == 1, "the bounded waits live on the tensor-core path"
        assert M.mmshift_poll_status(ws) == LB.MMSHIFT_ERR_TIMEOUT
    # the status word is cleared by the poll; the context and the workspace
    # serve the next, normal call, which matches the oracle
    gpu = PT.gpu_select(WL, [li], h, proxies=prox[None], ws=ws)
    refs = PT.oracle_layer(WL, li, h, 0, proxies=prox)
    for b, lo, hi, olo in _requests(WL):
        PT.check_request(gpu, refs[b], h, lo, hi, 0, f"after timeout req {b}", out_lo=olo)
        PT.check_gather(gpu, WL, 0, lo, olo, min(WL.budgets[b], hi - lo), hi - lo, WL.n_kv_heads)
    assert M.mmshift_poll_status(ws) == LB.MMSHIFT_OK
