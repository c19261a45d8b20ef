"""A stack of W4A4 linears run back to back on one stream: the layer sequence of the backbone
or of the DiT action head, each layer reading its own input buffer.

Host-side plumbing only: every layer is one ``qvla_w4a4_linear`` call (the fused rotate +
quantise kernel, then the GEMM with its dequantisation epilogue), or ``qvla_w4a8_linear`` for
8-bit activation codes, so a stack of L linears is 2L kernel launches.  The kernels are launched with programmatic stream serialization, so
consecutive launches overlap their set-up with the previous kernel's tail; ``capture`` records
a whole pass as a CUDA graph, which removes the host launch cost as well.  The per-step scale
of a DiT layer is fixed at launch, so a DiT stack has one graph per denoising step.

A stack may hold several input sets (one per denoising step, say): a pass at step t reads set
t when there are as many sets as steps.  One workspace (the largest any layer needs) serves all
layers: the linears run in stream order and each kernel waits for its predecessor before
touching the workspace.
"""

from __future__ import annotations

import numpy as np
import torch

from . import qvla as Q

_DT = {"f16": (Q.F16, torch.float16), "bf16": (Q.BF16, torch.bfloat16)}


class LinearStack:
    """Layers built from ``workloads.StackWeights``-like records (fields name, k, n,
    had_block, packed, wscale, bias, gated), all with m rows of input."""

    def __init__(self, weights, m: int, xdtype: str = "f16", ydtype: str = "f16", device=None, input_sets: int = 1,
                 act_bits: int = 4):
        if act_bits not in (4, 8):
            raise ValueError("act_bits must be 4 or 8")
        self.m = m
        self.act_bits = act_bits
        self._linear = Q.qvla_w4a4_linear if act_bits == 4 else Q.qvla_w4a8_linear
        ws_bytes = Q.qvla_linear_workspace_bytes if act_bits == 4 else Q.qvla_w4a8_workspace_bytes
        self.device = torch.device("cuda") if device is None else device
        xdt, self.xtorch = _DT[xdtype]
        ydt, self.ytorch = _DT[ydtype]
        self.layers, self.names, self.y = [], [], []
        self.sets = [[] for _ in range(input_sets)]
        for w in weights:
            if w.gated:
                h = w.n
                layer = Q.qvla_layer_create_gated(h, w.k, w.had_block, xdt, ydt, w.packed[:h], w.wscale[:h],
                                                  w.packed[h:], w.wscale[h:],
                                                  None if w.bias is None else w.bias[:h],
                                                  None if w.bias is None else w.bias[h:])
            else:
                layer = Q.qvla_layer_create(w.n, w.k, w.had_block, xdt, ydt, w.packed, w.wscale, w.bias)
            self.layers.append(layer)
            self.names.append(w.name)
            for xs in self.sets:
                xs.append(torch.zeros(m, w.k, dtype=self.xtorch, device=self.device))
            self.y.append(torch.empty(m, w.n, dtype=self.ytorch, device=self.device))
        self.ws_bytes = max(ws_bytes(layer, m) for layer in self.layers)
        self.ws = torch.empty(self.ws_bytes, dtype=torch.uint8, device=self.device)
        self.weight_bytes = sum(int(w.packed.nbytes) for w in weights)
        self.ops = sum(2 * m * w.k * (2 * w.n if w.gated else w.n) for w in weights)

    def set_step_tables(self, tables) -> None:
        """One per-step scale table per layer: float32 [T], or [T, G] for per-group scales."""
        for layer, t in zip(self.layers, tables):
            t = np.asarray(t, dtype=np.float32)
            if t.ndim == 2:
                Q.qvla_set_step_group_scales(layer, t)
            else:
                Q.qvla_set_step_scales(layer, t)

    @property
    def x(self):
        """The inputs of the first set."""
        return self.sets[0]

    def inputs(self, step: int):
        return self.sets[step] if len(self.sets) > 1 and step >= 0 else self.sets[0]

    def set_input(self, i: int, x, input_set: int = 0) -> None:
        self.sets[input_set][i].copy_(torch.as_tensor(x).to(self.xtorch))

    def run(self, step: int = -1, stream=None) -> None:
        """One pass over every layer; step -1 quantises per token, step t >= 0 with the tables."""
        stream = torch.cuda.current_stream() if stream is None else stream
        for layer, x, y in zip(self.layers, self.inputs(step), self.y):
            self._linear(layer, x, self.m, step, y, self.ws, self.ws_bytes, stream)

    def capture(self, step: int = -1) -> torch.cuda.CUDAGraph:
        """A CUDA graph of one pass (2 kernels per layer), replayed with ``graph.replay()``."""
        self.run(step)  # outside capture: first-call set-up (function attributes, occupancy queries)
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            self.run(step, torch.cuda.current_stream())
        return g

    def close(self) -> None:
        for layer in self.layers:
            layer.close()
        self.layers = []
