"""ResNet-18-style quaternion backbone forward through the libquan C ABI.

Layer list (inputs.backbone_layers): 7x7/2 quaternion stem (4 -> 64 real channels) with
IQBN + ReLU, 3x3/2 max pooling applied to every real channel on its own, then four
stages of two basic blocks (64/128/256/512 real channels, 3x3 quaternion convolutions
with IQBN, 1x1/2 quaternion shortcut where the shape changes, the block's second
convolution adding the block input before its ReLU).  Every operation runs in libquan
kernels on one CUDA stream; torch only allocates device memory.
"""
from __future__ import annotations

import numpy as np

from . import inputs as _inputs


class BackboneRunner:
    """Weights, activations and the per-step launch sequence of the backbone."""

    def __init__(self, torch, quan, inputs=_inputs, N: int = 256, H: int = 224, seed: int = 4,
                 x_bits=None, act: int = _inputs.ACT_RELU, fuse_stem_pool: bool = False,
                 rgb: bool = False, rgb_host=None, overlap_shortcuts: bool = False,
                 split_k: bool = False):
        self.torch, self.quan, self.N, self.H = torch, quan, N, H
        dev = torch.device("cuda")
        self.act = act
        self.layers = inputs.backbone_layers(N=N, H=H, seed=seed, act=act)
        # stem + 3x3/2 max pool as one call (quan_qconv2d_maxpool_fwd): the stem's full
        # output is never written, one kernel writes the pooled tensor
        L0, L1 = self.layers[0], self.layers[1]
        self.fused = (fuse_stem_pool and L0.kind == "conv" and L1.kind == "maxpool" and
                      L1.src == 0 and (L1.k, L1.stride, L1.pad) == (3, 2, 1))
        # rgb: the input is fp32 RGB, mapped by Eq. 4 inside the fused stem's loader
        self.rgb = rgb
        if rgb and not self.fused:
            raise ValueError("RGB input needs the fused stem (fuse_stem_pool=True)")

        def up(bits):
            return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(
                torch.bfloat16).to(dev)

        self.params = []
        self.outs = []
        for L in self.layers:
            if L.kind == "conv":
                prm = inputs.backbone_params(L)
                self.params.append({
                    "w": [up(prm[k]) for k in ("wr", "wi", "wj", "wk")],
                    "scale": torch.from_numpy(prm["scale"]).to(dev),
                    "shift": torch.from_numpy(prm["shift"]).to(dev),
                    "host": prm})
                s = L.spec
                if self.fused and len(self.outs) == 0:
                    # the fused call's workspace (none: 0 bytes) stands in for the stem's
                    # output
                    self.ws_bytes = quan.quan_qconv2d_maxpool_workspace_size(
                        N, s.H, s.W, s.Cout, s.kh, s.kw, s.stride, s.pad)
                    self.outs.append(torch.empty(self.ws_bytes // 2, dtype=torch.bfloat16,
                                                 device=dev))
                    self.stem_shape = (N, s.Ho, s.Wo, s.Cout)
                    continue
                self.outs.append(torch.empty((N, s.Ho, s.Wo, s.Cout), dtype=torch.bfloat16,
                                             device=dev))
            else:
                src = self.outs[L.src]
                _, Hs, Ws, C = self.stem_shape if (self.fused and L.src == 0) else src.shape
                Ho = (Hs + 2 * L.pad - L.k) // L.stride + 1
                Wo = (Ws + 2 * L.pad - L.k) // L.stride + 1
                self.params.append(None)
                self.outs.append(torch.empty((N, Ho, Wo, C), dtype=torch.bfloat16, device=dev))
        if rgb:
            self.x_host = inputs.backbone_rgb(N=N, H=H, seed=seed) if rgb_host is None \
                else rgb_host
            self.x = torch.from_numpy(np.ascontiguousarray(self.x_host)).to(dev)
        else:
            if x_bits is None:
                x_bits = inputs.backbone_input(N=N, H=H, seed=seed)
            self.x_host = x_bits
            self.x = up(x_bits)
        # one launch per layer; the fused stem + max pool is one launch for two layers
        self.launches_per_step = len(self.layers) - (1 if self.fused else 0)
        # split_k: the convolutions run through quan_qconv2d_fwd_ex with one workspace (the
        # layers run one after another on the main stream; the shortcuts on the side stream
        # run without one), so layers whose tiles leave a partial last wave of CTAs spread
        # their work evenly over the SMs
        self.workspace = quan.fwd_workspace() if split_k else None
        # overlap_shortcuts: a downsampling block's 1x1/2 shortcut (the layer after the
        # block's 3x3/2 convolution, reading the same input) runs on a second stream, forked
        # before the 3x3/2 convolution and joined before the block's second convolution,
        # so its CTAs can take the SMs the convolution's last wave leaves idle
        self.side = {}
        if overlap_shortcuts:
            for i, L in enumerate(self.layers):
                P = self.layers[i - 1] if i > 0 else None
                if (L.kind == "conv" and P is not None and P.kind == "conv" and L.src == P.src
                        and L.spec.kh == 1 and P.spec.kh > 1):
                    self.side[i] = (torch.cuda.Event(), torch.cuda.Event())
            self.side_stream = torch.cuda.Stream() if self.side else None
        self.footprint = (sum(t.numel() * 2 for t in self.outs) +
                          self.x.numel() * self.x.element_size())

    # ---------------------------------------------------------------- execution
    def layer_input(self, idx: int):
        src = self.layers[idx].src
        return self.x if src == -1 else self.outs[src]

    def run_layer(self, idx: int, stream, x=None, out=None, workspace=None):
        L = self.layers[idx]
        q = self.quan
        x = self.layer_input(idx) if x is None else x
        out = self.outs[idx] if out is None else out
        if L.kind == "maxpool":
            if self.fused and L.src == 0:
                return out  # produced by the stem's fused call
            N, H, W, C = x.shape
            q.quan_maxpool2d_fwd(x, N, H, W, C, L.k, L.stride, L.pad, out, stream)
            return out
        s, prm = L.spec, self.params[idx]
        N, H, W, C = x.shape
        if self.rgb and idx == 0:
            pooled = self.outs[1] if out is self.outs[0] else out
            q.quan_qconv2d_maxpool_rgb_fwd(x, *prm["w"], None, prm["scale"], prm["shift"], N, H,
                                           W, s.Cout, s.kh, s.kw, s.stride, s.pad, s.act,
                                           pooled, stream)
            return pooled
        if self.fused and idx == 0:
            pooled = self.outs[1] if out is self.outs[0] else out
            q.quan_qconv2d_maxpool_fwd(x, *prm["w"], None, prm["scale"], prm["shift"], N, H, W,
                                       s.Cin, s.Cout, s.kh, s.kw, s.stride, s.pad, s.act,
                                       self.outs[0], self.ws_bytes, pooled, stream)
            return pooled
        if workspace is not None:
            q.quan_qconv2d_fwd_ex(x, *prm["w"], None, prm["scale"], prm["shift"], N, H, W,
                                  s.Cin, s.Cout, s.kh, s.kw, s.stride, s.pad, s.act,
                                  self.outs[L.res] if L.res is not None else None, workspace,
                                  workspace.numel(), out, stream)
        elif L.res is not None:
            q.quan_qconv2d_fwd_res(x, *prm["w"], None, prm["scale"], prm["shift"], N, H, W,
                                   s.Cin, s.Cout, s.kh, s.kw, s.stride, s.pad, s.act,
                                   self.outs[L.res], out, stream)
        else:
            q.quan_qconv2d_fwd(x, *prm["w"], None, prm["scale"], prm["shift"], N, H, W,
                               s.Cin, s.Cout, s.kh, s.kw, s.stride, s.pad, s.act, out, stream)
        return out

    def step(self, stream):
        ws = self.workspace
        if not self.side:
            for i in range(len(self.layers)):
                self.run_layer(i, stream, workspace=ws)
            return
        torch = self.torch
        main = torch.cuda.ExternalStream(stream)
        side = self.side_stream
        pending = None  # the join of a shortcut whose output the next main-stream layer reads
        for i in range(len(self.layers)):
            if i + 1 in self.side:  # fork just before the block's 3x3/2 convolution
                self.side[i + 1][0].record(main)
            if i in self.side:
                fork, join = self.side[i]
                side.wait_event(fork)
                self.run_layer(i, side.cuda_stream)
                join.record(side)
                pending = join
                continue
            if pending is not None:
                main.wait_event(pending)
                pending = None
            self.run_layer(i, stream, workspace=ws)
        if pending is not None:
            main.wait_event(pending)

    @property
    def output(self):
        return self.outs[-1]

    # ---------------------------------------------------------------- accounting
    @property
    def flops(self) -> float:
        return sum(L.spec.flops for L in self.layers if L.kind == "conv")

    def layer_table(self):
        rows = []
        for i, L in enumerate(self.layers):
            if L.kind == "conv":
                s = L.spec
                rows.append((i, "conv", s.H, s.Cin, s.Cout, s.kh, s.stride, s.flops))
            else:
                rows.append((i, "maxpool", None, None, None, L.k, L.stride, 0.0))
        return rows

    # ---------------------------------------------------------------- e2e (host buffers)
    # Buffer set b of the end-to-end pipeline is an input image batch and a copy of the
    # last layer's output; the intermediate activations are shared, which is safe because
    # every step's kernels run in order on one stream.
    def e2e_setup(self, nbuf: int = 2):
        torch = self.torch
        self.h_x = torch.from_numpy(
            np.ascontiguousarray(self.x_host).reshape(-1).view(np.uint8)).pin_memory()
        # (the device copy target below has the input's dtype: bf16 pixels or fp32 RGB)
        out = self.outs[-1]
        self.h_out = [torch.empty(out.numel() * 2, dtype=torch.uint8).pin_memory()
                      for _ in range(nbuf)]
        self.e_x = [torch.empty_like(self.x) for _ in range(nbuf)]
        self.e_out = [torch.empty_like(out) for _ in range(nbuf)]
        self.h2d = self.h_x.numel()
        self.d2h = self.h_out[0].numel()

    def e2e_in(self, b):
        return [(self.e_x[b].view(-1).view(self.torch.uint8), self.h_x)]

    def e2e_out(self, b):
        return [(self.h_out[b], self.e_out[b].view(-1).view(self.torch.uint8))]

    def e2e_compute(self, b, stream):
        last = len(self.layers) - 1
        for i in range(len(self.layers)):
            x = self.e_x[b] if self.layers[i].src == -1 else None
            self.run_layer(i, stream, x=x, out=self.e_out[b] if i == last else None,
                           workspace=self.workspace)
