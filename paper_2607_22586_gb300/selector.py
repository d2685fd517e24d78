"""Torch-facing convenience around the C ABI: owns the workspace and outputs
of one workload shape and calls ``mmshift_select`` on the current stream.
PyTorch only provides device memory and streams here."""
from __future__ import annotations

from typing import Optional, Sequence

import torch

from . import _lib as L

_DT = {torch.bfloat16: L.MMSHIFT_BF16, torch.float32: L.MMSHIFT_F32}


class KVSelector:
    def __init__(self, n_q_heads: int, n_kv_heads: int, head_dim: int, window: int,
                 dtype: torch.dtype, cu_seqlens: Sequence[int], budgets: Sequence[int],
                 n_layers: int = 1, params: Optional[L.Params] = None, device="cuda"):
        if dtype not in _DT:
            raise ValueError(f"unsupported dtype {dtype}")
        self.dtype = dtype
        self.device = torch.device(device)
        if self.device.type == "cuda" and self.device.index is None:
            self.device = torch.device("cuda", torch.cuda.current_device())
        total = int(cu_seqlens[-1])
        self.total_tokens = total
        self.n_layers = n_layers
        self.n_kv_heads, self.head_dim = n_kv_heads, head_dim
        self.n_q_heads = n_q_heads
        self.budgets = list(budgets)
        self.out_count = None
        self.shape = L.make_shape(n_q_heads, n_kv_heads, head_dim, window, _DT[dtype], cu_seqlens,
                                  budgets, n_layers=n_layers,
                                  layer_stride_kv=total * n_kv_heads * head_dim,
                                  layer_stride_q=len(budgets) * window * n_q_heads * head_dim)
        self.params = params if params is not None else L.default_params()
        self.rows = L.mmshift_output_rows(self.shape)
        self.ws_bytes = L.mmshift_workspace_size(self.shape, self.params)
        # zeroed once: the first 256 bytes hold the device status word
        self.workspace = torch.zeros(self.ws_bytes, dtype=torch.uint8, device=self.device)
        self.out_idx = torch.empty((n_layers, self.rows, n_kv_heads), dtype=torch.int32, device=self.device)
        self.out_k = torch.empty((n_layers, self.rows, n_kv_heads, head_dim), dtype=dtype, device=self.device)
        self.out_v = torch.empty_like(self.out_k)

    def _stream(self, stream):
        return torch.cuda.current_stream(self.device) if stream is None else stream

    def _check(self, *ts):
        for t in ts:
            if t.dtype != self.dtype or not t.is_contiguous() or t.device != self.device:
                raise ValueError("inputs must be contiguous tensors of the selector's dtype/device")

    def __call__(self, K: torch.Tensor, V: torch.Tensor, qwin: torch.Tensor,
                 proxies_in: Optional[torch.Tensor] = None, debug: Optional[L.Debug] = None,
                 stream=None, stats: Optional[torch.Tensor] = None,
                 head_budgets: Optional[torch.Tensor] = None):
        """Select for every layer. ``stats`` ([L, B, 2, Hq*d] float32, e.g.
        from prefill_stats) replaces the window statistics of the proxies;
        ``head_budgets`` ([L, B, Hkv] int32 on the device, each in [1, C_b])
        gives every (layer, KV head) its own budget, the per-request budgets
        being the capacity (padding rows -1, counts in ``self.out_count``)."""
        self._check(K, V, qwin)
        stream = self._stream(stream)
        if stats is not None and (proxies_in is not None or head_budgets is not None):
            raise ValueError("stats cannot be combined with proxies_in or head_budgets")
        if stats is not None:
            L.check(L.mmshift_select_with_stats(self.shape, K, V, qwin, stats, self.params, self.out_idx,
                                                self.out_k, self.out_v, debug, self.workspace,
                                                self.ws_bytes, stream), "mmshift_select_with_stats")
        elif head_budgets is not None:
            if head_budgets.dtype != torch.int32 or head_budgets.device != self.device:
                raise ValueError("head_budgets must be an int32 tensor on the selector's device")
            if self.out_count is None:
                self.out_count = torch.empty((self.n_layers, len(self.budgets), self.n_kv_heads),
                                             dtype=torch.int32, device=self.device)
            L.check(L.mmshift_select_head_budgets(self.shape, K, V, qwin, proxies_in,
                                                  head_budgets.contiguous(), self.params, self.out_idx,
                                                  self.out_count, self.out_k, self.out_v, debug,
                                                  self.workspace, self.ws_bytes, stream),
                    "mmshift_select_head_budgets")
        else:
            L.check(L.mmshift_select(self.shape, K, V, qwin, proxies_in, self.params, self.out_idx,
                                     self.out_k, self.out_v, debug, self.workspace, self.ws_bytes,
                                     stream), "mmshift_select")
        return self.out_idx, self.out_k, self.out_v

    def prefill_stats(self, qfull: torch.Tensor, layer_stride: int = 0, stream=None) -> torch.Tensor:
        """Proxy statistics over every prompt query (Section 3.2.1): qfull
        [L, T_total, Hq, d] -> [L, B, 2, Hq*d] float32 (mean, std)."""
        self._check(qfull)
        n = L.mmshift_prefill_stats_workspace_size(self.shape)
        ws = torch.empty(max(n, 1), dtype=torch.uint8, device=self.device)
        out = torch.empty((self.n_layers, len(self.budgets), 2, self.n_q_heads * self.head_dim),
                          dtype=torch.float32, device=self.device)
        L.check(L.mmshift_prefill_stats(self.shape, qfull, layer_stride, out, ws, n, self._stream(stream)),
                "mmshift_prefill_stats")
        return out

    def coverage(self, K: torch.Tensor, qwin: torch.Tensor, dec_q: torch.Tensor,
                 idx: Optional[torch.Tensor] = None, softmax_scale: float = 0.0,
                 stream=None) -> torch.Tensor:
        """Attention-mass coverage (Section 1, Fig. 1b) of ``idx`` (default:
        the last selection) for decode queries dec_q [L, B, Hq, n_dec, d]:
        [L, B, Hkv, n_dec] float32, averaged over each KV head's query heads."""
        self._check(K, qwin, dec_q)
        n_dec = dec_q.shape[3]
        n = L.mmshift_coverage_workspace_size(self.shape, n_dec)
        ws = torch.zeros(n, dtype=torch.uint8, device=self.device)
        out = torch.empty((self.n_layers, len(self.budgets), self.n_kv_heads, n_dec),
                          dtype=torch.float32, device=self.device)
        L.check(L.mmshift_coverage(self.shape, K, qwin, dec_q, n_dec, softmax_scale,
                                   self.out_idx if idx is None else idx, out, ws, n,
                                   self._stream(stream)), "mmshift_coverage")
        L.check(L.mmshift_poll_status(ws, self._stream(stream)), "mmshift_coverage status")
        return out

    def poll(self, stream=None) -> None:
        if stream is None:
            stream = torch.cuda.current_stream(self.device)
        L.check(L.mmshift_poll_status(self.workspace, stream), "mmshift_poll_status")
