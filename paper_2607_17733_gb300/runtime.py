"""Small runtime around the C ABI: quantized linear layers and CUDA-graph steps.

MxLinear packs a bf16 weight once (step A2) and runs the hot path per call:
quantize the activations (A1) and multiply (A3/A4), all in libmxs kernels on
the current stream.  GraphStep captures any sequence of such calls into one
CUDA graph, so a decode step of many small launches replays with one host call.
"""
from __future__ import annotations

import numpy as np
import torch

from . import mxs


class MxLinear:
    """y = x W^T with x, W quantized to MXINT under one per-layer width map."""

    def __init__(self, w: torch.Tensor, bits, with_planes: bool = False, rounding: int = mxs.RNE):
        assert w.dtype == torch.bfloat16 and w.is_cuda and w.dim() == 2
        self.N, self.K = w.shape
        self.bits = np.ascontiguousarray(np.asarray(bits, np.uint8))
        assert self.bits.size * 32 == self.K
        self.rounding = rounding
        self.layout = mxs.W_COMPACT_AND_PLANES if with_planes else mxs.W_COMPACT
        self.packed = mxs.pack_weight(w, self.bits, layout=self.layout, rounding=rounding)
        torch.cuda.current_stream().synchronize()  # static from here on (fused() streams it early)
        n4 = int(np.sum(self.bits == 4))
        n68 = self.bits.size - n4
        # bytes a GEMM must read of this weight: codes + one scale byte per block
        self.weight_bytes = self.N * (16 * n4 + 32 * n68 + self.bits.size)

    def buffers(self, M: int, device=None) -> dict:
        """Activation codes / scales / output buffers for M tokens."""
        device = device or self.packed.device
        rb = mxs.act_row_bytes(self.K, self.bits)
        return {
            "codes": torch.empty((M, rb), dtype=torch.uint8, device=device),
            "scales": torch.empty((M, self.K // 32), dtype=torch.uint8, device=device),
            "y": torch.empty((M, self.N), dtype=torch.float32, device=device),
            "ws": None,
            # the workspace of fused(): the activations' MMA planes (M > 1), the
            # CUDA-core path's arrival counters and partial sums (M = 1)
            "planes": torch.empty(max(mxs.linear_decode_workspace_bytes(M, self.K, self.N, self.bits), 16),
                                  dtype=torch.uint8, device=device) if M <= 16 else None,
        }

    def quantize(self, x: torch.Tensor, bufs: dict):
        mxs.quantize_act(x, self.bits, rounding=self.rounding, codes=bufs["codes"], scales=bufs["scales"])

    def matmul(self, bufs: dict) -> torch.Tensor:
        return mxs.gemm(bufs["codes"], bufs["scales"], None, self.bits, self.packed, self.N,
                        w_layout=self.layout, y=bufs["y"], workspace=bufs["ws"])

    def fused(self, x: torch.Tensor, y: torch.Tensor, planes: torch.Tensor | None = None) -> torch.Tensor:
        """M <= 16: quantize to MMA planes and run the decode GEMM in one call
        (two kernels, the GEMM a programmatic dependent of the quantizer)."""
        return mxs.linear_decode(x, self.bits, self.packed, self.N, rounding=self.rounding, y=y, workspace=planes)

    def __call__(self, x: torch.Tensor, bufs: dict | None = None) -> torch.Tensor:
        bufs = bufs or self.buffers(x.shape[0], x.device)
        if x.shape[0] <= 16:
            return self.fused(x, bufs["y"], bufs["planes"])
        self.quantize(x, bufs)
        return self.matmul(bufs)


class GraphStep:
    """Capture `fn()` (a sequence of libmxs calls on the current stream) once and
    replay it.  fn is run once eagerly on the capture stream first."""

    def __init__(self, fn, stream: torch.cuda.Stream | None = None):
        self.stream = stream or torch.cuda.Stream()
        self.stream.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(self.stream):
            fn()
        self.stream.synchronize()
        self.graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(self.graph, stream=self.stream):
            fn()
        torch.cuda.synchronize()

    def replay(self):
        self.graph.replay()
