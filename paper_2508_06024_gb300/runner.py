"""Device buffers and calls for one MoE layer through the C ABI.

PyTorch provides the device memory and the stream; every step runs in
libec2moe.so.  Used by the tests, ``bench.py`` and ``__graft_entry__``.
"""

from __future__ import annotations

from typing import Dict, Optional

import torch

from . import ec2moe as C
from .synth import LayerConfig


def desc_for(cfg: LayerConfig, T: Optional[int] = None) -> C.LayerDesc:
    return C.make_desc(T=cfg.T if T is None else T, d=cfg.d, E=cfg.E, d_ff=cfg.d_ff, k=cfg.k,
                       n_groups=cfg.n_groups, act=cfg.act, dtype=cfg.dtype, r=cfg.r, n_shared=cfg.n_shared,
                       d_ff_shared=cfg.d_ff_shared, renorm_topk=cfg.renorm_topk, top_groups=cfg.top_groups)


def weights_for(inp: Dict[str, Optional[torch.Tensor]]) -> C.LayerWeights:
    return C.make_weights(W_local=inp["W_local"], b_local=inp["b_local"], W_global=inp.get("W_global"),
                          b_global=inp.get("b_global"), W1=inp.get("W1"), W3=inp.get("W3"), W2=inp.get("W2"),
                          W1s=inp.get("W1s"), W3s=inp.get("W3s"), W2s=inp.get("W2s"), V_enc=inp.get("V_enc"),
                          V_dec=inp.get("V_dec"))


class LayerRun:
    """Output and workspace buffers of one layer shape on one device."""

    def __init__(self, cfg: LayerConfig, inp: Dict[str, Optional[torch.Tensor]], device="cuda"):
        self.cfg = cfg
        self.inp = inp
        self.desc = desc_for(cfg)
        self.weights = weights_for(inp)
        self.mask = C.host_mask(inp["mask"].to("cpu"))
        dt = cfg.torch_dtype
        T = cfg.T
        self.Y = torch.empty(T, cfg.d, dtype=dt, device=device)
        self.topk_idx = torch.empty(T, cfg.k, dtype=torch.int32, device=device)
        self.topk_w = torch.empty(T, cfg.k, dtype=torch.float32, device=device)
        self.counts = torch.empty(cfg.E, dtype=torch.int32, device=device)
        self.Z = torch.empty(T, cfg.r, dtype=dt, device=device) if cfg.r > 0 else None
        self.ws_bytes = C.ec2moe_workspace_size(self.desc)
        self.workspace = torch.empty(max(self.ws_bytes, 16), dtype=torch.uint8, device=device)

    def forward_pipelined(self, n_micro: int, stream_end=None, stream_cloud=None,
                          X: Optional[torch.Tensor] = None) -> torch.Tensor:
        """The end/cloud pipelined layer call (two streams, n_micro micro-batches)."""
        need = C.ec2moe_pipelined_workspace_size(self.desc, n_micro)
        if getattr(self, "pws", None) is None or self.pws.numel() < need:
            self.pws = torch.empty(max(need, 16), dtype=torch.uint8, device=self.Y.device)
        C.ec2moe_layer_forward_pipelined(self.desc, self.weights, self.inp["X"] if X is None else X, self.mask,
                                         self.Y, self.topk_idx, self.topk_w, self.counts, self.Z, self.pws,
                                         self.pws.numel(), n_micro, stream_end, stream_cloud)
        return self.Y

    def forward(self, X: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
        C.ec2moe_layer_forward(self.desc, self.weights, self.inp["X"] if X is None else X, self.mask, self.Y,
                               self.topk_idx, self.topk_w, self.counts, self.Z, self.workspace, self.ws_bytes,
                               stream)
        return self.Y


def main(argv=None) -> int:
    """Runs `--calls` eager layer calls of a preset shape (for profilers such as
    ncu, which want a short program with a known launch sequence)."""
    import argparse

    from . import build as B
    from . import synth as S

    ap = argparse.ArgumentParser(description="run a preset MoE layer shape through the C ABI")
    ap.add_argument("--workload", default="mixtral_bf16")
    ap.add_argument("--calls", type=int, default=2)
    for key in ("T", "E", "n_allowed", "k", "r", "d_ff", "n_groups", "seed"):
        ap.add_argument(f"--{key}", type=int, default=None)
    args = ap.parse_args(argv)
    over = {k: getattr(args, k) for k in ("T", "E", "n_allowed", "k", "r", "d_ff", "n_groups", "seed")
            if getattr(args, k) is not None}
    cfg = S.preset(args.workload, **over)
    B.build()
    C.load()
    run = LayerRun(cfg, S.make_inputs(cfg, device="cuda"), device="cuda")
    for _ in range(args.calls):
        run.forward()
    status = C.ec2moe_last_device_error()
    torch.cuda.synchronize()
    print(f"{cfg}: {args.calls} calls, {C.ec2moe_last_launch_count()} launches per call, "
          f"status {C.status_string(status)}")
    return 0 if status == C.OK else 1


if __name__ == "__main__":
    raise SystemExit(main())
