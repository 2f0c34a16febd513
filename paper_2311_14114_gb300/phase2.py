"""Quantized fine-tuning forward (Algorithm 1, Phase II): every step
quantizes the fp32 master weights and the activations with per-group scales
computed on the fly, then evaluates the layers under integer MAC execution.

A layer here is the library's hot path end to end: soniq_pack_weights on the
current master weights (Sec. 3 step 3), soniq_quantize_act on the layer input
(steps 1-2; the unsigned quantizer clips negative inputs, which plays the role
of the ReLU between layers), soniq_mp_gemm (the exact integer products and the
scale epilogue).  This module only sequences the calls and owns the buffers;
every arithmetic step runs in the library's kernels.  The backward pass
(straight-through estimator) and the optimizer update of Phase II act on the
fp32 master weights outside this path."""
from __future__ import annotations

from typing import List, Sequence

import torch

from . import soniq as sq


class FakeQuantMLP:
    """A stack of linear layers whose master weights stay fp32 on the GPU.

    layers: per layer a dict with W (fp32 [N][K], numpy or torch), perm,
    count, bits (as the workloads module makes them); sub_k: scale runs along
    K (the GroupSize of Algorithm 1) for every layer, 0 for one scale per
    group."""

    def __init__(self, layers: Sequence[dict], M: int, sub_k: int = 0, device="cuda"):
        self.M = int(M)
        self.layouts: List[sq.Layout] = []
        self.W: List[torch.Tensor] = []
        self.Wp, self.s_w, self.Ap, self.s_a, self.Y = [], [], [], [], []
        for lay in layers:
            W = torch.as_tensor(lay["W"], dtype=torch.float32).to(device).contiguous()
            layout = sq.Layout(lay["perm"], lay["count"], lay["bits"], sub_k=sub_k, device=device)
            N = W.shape[0]
            self.layouts.append(layout)
            self.W.append(W)
            self.Wp.append(torch.empty((N, layout.row_bytes(True)), dtype=torch.uint8, device=device))
            self.s_w.append(torch.empty(layout.scale_shape(N), dtype=torch.float32, device=device))
            self.Ap.append(torch.empty((self.M, layout.row_bytes(False)), dtype=torch.uint8, device=device))
            self.s_a.append(torch.empty(layout.scale_shape(None), dtype=torch.float32, device=device))
            self.Y.append(torch.empty((self.M, N), dtype=torch.float16, device=device))

    def forward(self, X: torch.Tensor, stream=None) -> torch.Tensor:
        """One Phase II forward over X (fp16 [M][K0]); returns the last layer's
        fp16 outputs (the intermediate ones stay in self.Y)."""
        x = X
        for i, layout in enumerate(self.layouts):
            sq.pack_weights(layout, self.W[i], Wp=self.Wp[i], s_w=self.s_w[i], stream=stream)
            sq.quantize_act(layout, x, "tensor", s_a=self.s_a[i], Ap=self.Ap[i], stream=stream)
            sq.mp_gemm(layout, self.Ap[i], self.s_a[i], self.Wp[i], self.s_w[i], Y=self.Y[i], stream=stream)
            x = self.Y[i]
        return x
