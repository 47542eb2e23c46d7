"""The streamed runner (three streams, double-buffered device tensors) gives
bitwise the same outputs as calling the layer batch by batch, with either code
container, with and without a drain plan and a workspace."""

import numpy as np
import pytest
import torch

from paper_2606_12280_gb300 import workloads as wl

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("codes,with_plan", [("f16", True), ("int8", True), ("int8", False)])
def test_streamed_matches_direct(codes, with_plan):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2606_12280_gb300 import w8a8
    from paper_2606_12280_gb300.streamed import StreamedLinear
    M, K, N = 300, 512, 264
    c = wl.make_case(M, K, N, seed=7)
    dev = "cuda"
    W = torch.from_numpy(c.W[0]).to(dev)
    lam = w8a8.smooth_scales(w8a8.channel_absmax(torch.from_numpy(c.X_cal.view(np.int16))
                                                  .view(torch.bfloat16).to(dev)), W, 0.5)
    Wq, sw = w8a8.quantize_weights(W, lam)
    bias = torch.from_numpy(c.bias[0]).to(dev)
    batches = [torch.from_numpy(wl.random_bf16((M, K), seed=100 + i, scale=1.0 + i).view(np.int16))
               .view(torch.bfloat16).pin_memory() for i in range(5)]
    outs = [torch.empty(M, N, dtype=torch.bfloat16).pin_memory() for _ in range(5)]
    plan = w8a8.chunk_plan(Wq) if with_plan else None
    r = StreamedLinear(M, K, N, lam, Wq, sw, bias, depth=2, plan=plan, codes=codes)
    r.run(batches, outs)
    r.synchronize()
    for xh, yh in zip(batches, outs):
        want = w8a8.quantized_linear_forward(xh.to(dev), lam, Wq, sw, bias, plan=plan, codes=codes)
        other = w8a8.quantized_linear_forward(xh.to(dev), lam, Wq, sw, bias,
                                              codes="int8" if codes == "f16" else "f16")
        with_ws = w8a8.quantized_linear_forward(xh.to(dev), lam, Wq, sw, bias, plan=plan, codes=codes,
                                                workspace=w8a8.linear_workspace(M, K))
        torch.cuda.synchronize()
        assert torch.equal(yh, want.cpu())
        assert torch.equal(want, other)
        assert torch.equal(want, with_ws)
