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
        total = int(cu_seqlens[-1])
        self.total_tokens = total
        self.n_layers = n_layers
        self.n_kv_heads, self.head_dim = n_kv_heads, head_dim
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

    def __call__(self, K: torch.Tensor, V: torch.Tensor, qwin: torch.Tensor,
                 proxies_in: Optional[torch.Tensor] = None, debug: Optional[L.Debug] = None,
                 stream=None):
        for t in (K, V, qwin):
            if t.dtype != self.dtype or not t.is_contiguous() or t.device != self.device:
                raise ValueError("K, V and Qwin must be contiguous tensors of the selector's dtype/device")
        if stream is None:
            stream = torch.cuda.current_stream(self.device)
        L.check(L.mmshift_select(self.shape, K, V, qwin, proxies_in, self.params, self.out_idx,
                                 self.out_k, self.out_v, debug, self.workspace, self.ws_bytes, stream),
                "mmshift_select")
        return self.out_idx, self.out_k, self.out_v

    def poll(self, stream=None) -> None:
        if stream is None:
            stream = torch.cuda.current_stream(self.device)
        L.check(L.mmshift_poll_status(self.workspace, stream), "mmshift_poll_status")
