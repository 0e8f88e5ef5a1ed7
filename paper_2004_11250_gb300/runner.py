"""Turn a network description (``synth.Net``) into library handles and run it.

Thin glue over the C-ABI binding: every conv is packed by ``pp_pack_layer``,
uploaded by ``pp_layer_create`` / ``pp_dense_create`` and chained by the
``pp_net_*`` executor.  Device memory and streams come from torch.
"""
from __future__ import annotations

from typing import List, Optional

import numpy as np
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
    """One conv op on the device (pruned or dense) with its packed form kept for inspection.

    in_layout: the channel order of the op's input activation (position c holds original channel
    in_layout[c]); the weights' input channels are permuted to match before packing.  None = original order.
    """

    def __init__(self, layer, stream=None, in_layout: Optional[np.ndarray] = None, precision: int = 0,
                 input_bound: float = 0.0):
        self.spec = layer
        self.packed = None
        self.dense = isinstance(layer, synth.DenseLayer)
        w = layer.w
        mask = np.ones((layer.Co, layer.Ci), np.uint8) if self.dense else layer.mask
        if in_layout is not None:
            w, mask, _ = pp.pp_permute_input_channels(w, mask, in_layout)
        if self.dense:
            self.handle = pp.pp_dense_create(w, layer.bias, stream)
        else:
            self.packed = pp.pp_pack_layer(w, mask, layer.taps)
            self.handle = pp.pp_layer_create(self.packed, layer.bias, stream)
            if precision != pp.PP_PRECISION_TF32X3:
                pp.pp_layer_set_precision(self.handle, precision, input_bound, stream)

    def perm(self) -> np.ndarray:
        return pp.pp_packed_arrays(self.packed)["perm"].copy()

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


def fold_groups(spec: synth.Net):
    """Activations that must share one channel order (a skip tensor and the output it is added to), and
    whether each group must keep the original order (it holds the network input or output, or a dense
    layer's output)."""
    n = len(spec.ops)
    root = list(range(n + 1))

    def find(a):
        while root[a] != a:
            root[a] = root[root[a]]
            a = root[a]
        return a

    for k, op in enumerate(spec.ops):
        if op.skip_from >= 0:
            root[find(op.skip_from)] = find(k + 1)
    fixed = {find(0), find(n)}
    for k, op in enumerate(spec.ops):
        if isinstance(op.layer, synth.DenseLayer):
            fixed.add(find(k + 1))
    return [find(a) in fixed for a in range(n + 1)]


class DeviceNet:
    """A whole network: its layers plus a finalized ``pp_net`` executor.

    fold_perm: fold each pruned layer's filter reorder (Section 3 "Matrix reorder") into the next layer:
    the layer stores reordered filter j at channel j and the next layer's weights are packed with their
    input channels permuted to match, so activations between layers stay in reordered order.  Activations
    tied to the network input or output, to a dense layer, or to such a group through a skip keep the
    original order; an op adding a skip stores its output in the skip's order.

    precision / input_bound: the tensor-core arithmetic of every pruned layer that has a tensor-core
    layout (pp_layer_set_precision).
    """

    def __init__(self, spec: synth.Net, use_graph: bool = True, stream=None, fold_perm: bool = False,
                 precision: int = 0, input_bound: float = 0.0):
        self.spec = spec
        N, C, H, W = spec.x.shape
        self.layers: List[DeviceLayer] = []
        self.layouts: List[np.ndarray] = [np.arange(C, dtype=np.int32)]  # per activation: original channel at each position
        keep_orig = fold_groups(spec) if fold_perm else [True] * (len(spec.ops) + 1)
        for k, op in enumerate(spec.ops):
            lay_in = self.layouts[k]
            ident = bool((lay_in == np.arange(len(lay_in))).all())
            L = DeviceLayer(op.layer, stream, None if ident else lay_in, precision, input_bound)
            Co = op.layer.Co
            if keep_orig[k + 1]:
                lay_out = np.arange(Co, dtype=np.int32)
            elif op.skip_from >= 0:
                lay_out = self.layouts[op.skip_from]
            else:
                lay_out = L.perm().astype(np.int32)  # filter j (original perm[j]) at channel j
            if not L.dense and fold_perm:
                order = np.empty(Co, np.int32)
                order[lay_out] = np.arange(Co, dtype=np.int32)  # original filter o -> its channel
                pp.pp_layer_set_output_order(L.handle, order, stream)
            self.layers.append(L)
            self.layouts.append(lay_out)
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
