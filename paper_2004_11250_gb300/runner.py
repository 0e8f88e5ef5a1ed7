"""Turn a network description (``synth.Net``) into library handles and run it.

Thin glue over the C-ABI binding: every conv is packed by ``pp_pack_layer``,
uploaded by ``pp_layer_create`` / ``pp_dense_create`` and chained by the
``pp_net_*`` executor.  Device memory and streams come from torch.
"""
from __future__ import annotations

from typing import List

import torch

from . import ppconv as pp
from . import synth


def op_flags(op: synth.Op) -> int:
    f = 0
    if op.skip_from >= 0:
        f |= pp.PP_ADD_SKIP
    if op.relu:
        f |= pp.PP_RELU
    if op.pool:
        f |= pp.PP_POOL2
    return f


class DeviceLayer:
    """One conv op on the device (pruned or dense) with its packed form kept for inspection."""

    def __init__(self, layer, stream=None):
        self.spec = layer
        self.packed = None
        self.dense = isinstance(layer, synth.DenseLayer)
        if self.dense:
            self.handle = pp.pp_dense_create(layer.w, layer.bias, stream)
        else:
            self.packed = pp.pp_pack_layer(layer.w, layer.mask, layer.taps)
            self.handle = pp.pp_layer_create(self.packed, layer.bias, stream)

    def forward(self, x, y, skip, N, H, W, flags, stream=None):
        fn = pp.pp_dense_forward if self.dense else pp.pp_conv_forward
        fn(self.handle, x, y, skip, N, H, W, flags, stream)

    def close(self):
        if self.handle:
            (pp.pp_dense_destroy if self.dense else pp.pp_layer_destroy)(self.handle)
            self.handle = None
        if self.packed:
            pp.pp_packed_destroy(self.packed)
            self.packed = None


class DeviceNet:
    """A whole network: its layers plus a finalized ``pp_net`` executor."""

    def __init__(self, spec: synth.Net, use_graph: bool = True, stream=None):
        self.spec = spec
        N, C, H, W = spec.x.shape
        self.layers: List[DeviceLayer] = [DeviceLayer(op.layer, stream) for op in spec.ops]
        self.net = pp.pp_net_create(N, C, H, W)
        for op, L in zip(spec.ops, self.layers):
            add = pp.pp_net_add_dense if L.dense else pp.pp_net_add_conv
            add(self.net, L.handle, op_flags(op), op.skip_from)
        pp.pp_net_finalize(self.net)
        pp.pp_net_use_graph(self.net, use_graph)
        self.out_shape = pp.pp_net_output_shape(self.net)

    def run(self, x: torch.Tensor, y: torch.Tensor, stream=None):
        pp.pp_net_run(self.net, x, y, stream if stream is not None else torch.cuda.current_stream())

    def run_host(self, x_host, y_host, stream=None):
        pp.pp_net_run_host(self.net, x_host, y_host, stream if stream is not None else torch.cuda.current_stream())

    def run_layerwise(self, x: torch.Tensor, stream=None) -> List[torch.Tensor]:
        """Run op by op with one fresh output tensor per op; returns all activations (index 0 = x)."""
        acts = [x]
        N = x.shape[0]
        for op, L in zip(self.spec.ops, self.layers):
            xin = acts[-1]
            _, _, H, W = xin.shape
            Ho, Wo = (H // 2, W // 2) if op.pool else (H, W)
            y = torch.empty((N, L.spec.Co, Ho, Wo), device=x.device, dtype=torch.float32)
            skip = acts[op.skip_from] if op.skip_from >= 0 else None
            L.forward(xin, y, skip, N, H, W, op_flags(op),
                      stream if stream is not None else torch.cuda.current_stream())
            acts.append(y)
        return acts

    def close(self):
        if self.net:
            pp.pp_net_destroy(self.net)
            self.net = None
        for L in self.layers:
            L.close()
