"""Streamed execution of the W8A8 layer over batches that live in host memory.

Three CUDA streams and `depth` device buffer sets: the upload stream copies
batch i + 1 into its buffer while the compute stream runs a3 + a4/a5 on batch
i and the download stream copies batch i - 1's output back, so the host links
and the GPU work overlap.  Events order the three streams per buffer set (an
upload waits until the compute of the batch that used its buffer `depth`
batches ago is done; a computation waits for its upload and for the download
that last used its output buffer).  Host buffers must be pinned for the
copies to be asynchronous.  Every step of the layer runs in the library's
kernels through the binding; this module only moves data and orders streams.
"""

from __future__ import annotations

import torch

from . import w8a8


class StreamedLinear:
    """One quantized linear layer (lambda, Wq, w_scale, bias on the device)
    applied to a stream of [M, K] bf16 host batches, writing [M, N] bf16 host
    outputs."""

    def __init__(self, M: int, K: int, N: int, smooth, Wq, w_scale, bias=None, depth: int = 2,
                 device=None, plan=None, codes: str = "f16"):
        """codes: "f16" (a3 writes the codes as fp16 values and the GEMM takes
        them unconverted) or "int8" (the int8 container; the GEMM call gets a
        workspace and expands the codes first).  plan: ``w8a8.chunk_plan(Wq)``
        or None.  One workspace serves every buffer set: the GEMMs run in
        order on one stream."""
        if codes not in ("f16", "int8"):
            raise ValueError("codes must be 'f16' or 'int8'")
        self.M, self.K, self.N = M, K, N
        self.smooth, self.Wq, self.w_scale, self.bias = smooth, Wq, w_scale, bias
        self.plan, self.f16 = plan, codes == "f16"
        dev = device if device is not None else Wq.device
        self.depth = depth
        self.X = [torch.empty(M, K, dtype=torch.bfloat16, device=dev) for _ in range(depth)]
        self.Xq = [torch.empty(M, K, dtype=torch.float16 if self.f16 else torch.int8, device=dev)
                   for _ in range(depth)]
        self.sx = [torch.empty(M, dtype=torch.float32, device=dev) for _ in range(depth)]
        self.ss = [torch.empty(M, dtype=torch.int32, device=dev) for _ in range(depth)] if self.f16 else None
        self.ws = None if self.f16 else w8a8.linear_workspace(M, K, device=dev)
        self.Y = [torch.empty(M, N, dtype=torch.bfloat16, device=dev) for _ in range(depth)]
        self.up = torch.cuda.Stream(device=dev)
        self.comp = torch.cuda.Stream(device=dev)
        self.down = torch.cuda.Stream(device=dev)
        self.x_ready = [torch.cuda.Event() for _ in range(depth)]
        self.x_free = [torch.cuda.Event() for _ in range(depth)]
        self.y_ready = [torch.cuda.Event() for _ in range(depth)]
        self.y_free = [torch.cuda.Event() for _ in range(depth)]
        self.started = [False] * depth

    def run(self, X_host, Y_host):
        """Process the batches X_host[i] -> Y_host[i] (lists of pinned host
        tensors, the same length).  Returns when all work is enqueued; the
        outputs are ready after `synchronize()` (or after `done_event` on the
        download stream)."""
        if len(X_host) != len(Y_host):
            raise ValueError("one output buffer per input batch")
        for i, (xh, yh) in enumerate(zip(X_host, Y_host)):
            s = i % self.depth
            with torch.cuda.stream(self.up):
                if self.started[s]:
                    self.up.wait_event(self.x_free[s])
                self.X[s].copy_(xh, non_blocking=True)
                self.x_ready[s].record(self.up)
            with torch.cuda.stream(self.comp):
                self.comp.wait_event(self.x_ready[s])
                if self.started[s]:
                    self.comp.wait_event(self.y_free[s])
                if self.f16:
                    w8a8.quant_act_f16codes(self.X[s], self.smooth, Xq16=self.Xq[s], x_scale=self.sx[s],
                                            sumsq=self.ss[s], stream=self.comp)
                else:
                    w8a8.quant_act(self.X[s], self.smooth, Xq=self.Xq[s], x_scale=self.sx[s],
                                   stream=self.comp)
                self.x_free[s].record(self.comp)
                if self.f16:
                    w8a8.linear_f16codes(self.Xq[s], self.sx[s], self.Wq, self.w_scale, self.bias,
                                         Y=self.Y[s], plan=self.plan,
                                         x_sumsq=self.ss[s] if self.plan is not None else None,
                                         stream=self.comp)
                else:
                    w8a8.linear(self.Xq[s], self.sx[s], self.Wq, self.w_scale, self.bias, Y=self.Y[s],
                                plan=self.plan, workspace=self.ws, stream=self.comp)
                self.y_ready[s].record(self.comp)
            with torch.cuda.stream(self.down):
                self.down.wait_event(self.y_ready[s])
                yh.copy_(self.Y[s], non_blocking=True)
                self.y_free[s].record(self.down)
            self.started[s] = True

    def synchronize(self):
        for st in (self.up, self.comp, self.down):
            st.synchronize()
