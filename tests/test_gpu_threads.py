"""Two host threads launch through the C ABI at the same time.

The library looks kernel attributes, occupancy and device addresses up once
per device and keeps no other state, so concurrent callers on their own
streams must get exactly what serial calls give.  The check runs in a fresh
process, so that the threads' calls are the first ones of every launcher (the
one-time set-up happens under contention), with different shapes per thread.
"""

import os
import subprocess
import sys
import textwrap

import pytest
import torch

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

SCRIPT = textwrap.dedent(r"""
    import sys, threading
    sys.path.insert(0, sys.argv[1])
    import torch
    from paper_2606_12280_gb300 import w8a8
    from paper_2606_12280_gb300 import workloads as wl

    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    w8a8.lib()

    def inputs(M, K, N, seed):
        c = wl.make_case(M, K, N, seed=seed)
        bf = lambda a: torch.from_numpy(a.view("int16")).view(torch.bfloat16).to(dev)
        W = torch.from_numpy(c.W[0]).to(dev)
        return bf(c.X_cal), bf(c.X[0]), W, torch.from_numpy(c.bias[0]).to(dev)

    def layer(args, stream):
        Xc, X, W, b = args
        with torch.cuda.stream(stream):
            lam = w8a8.smooth_scales(w8a8.channel_absmax(Xc, stream=stream), W, 0.5, stream=stream)
            Wq, sw = w8a8.quantize_weights(W, lam, stream=stream)
            Xq, sx = w8a8.quant_act(X, lam, stream=stream)
            Y8 = w8a8.linear(Xq, sx, Wq, sw, b, stream=stream)
            ss = torch.empty(X.shape[0], dtype=torch.int32, device=dev)
            q16, sx16 = w8a8.quant_act_f16codes(X, lam, sumsq=ss, stream=stream)
            Y16 = w8a8.linear_f16codes(q16, sx16, Wq, sw, b, plan=w8a8.chunk_plan(Wq, stream=stream),
                                       x_sumsq=ss, stream=stream)
            sums = torch.zeros(4, X.shape[1], dtype=torch.float64, device=dev)
            amax = torch.zeros(X.shape[1], dtype=torch.float32, device=dev)
            w8a8.act_stats_update(X, sums, amax, stream=stream)
            Yb = w8a8.linear_bf16(X, W.to(torch.bfloat16), b, stream=stream)
        stream.synchronize()
        return [t.clone() for t in (lam, Wq, sw, Xq, sx, Y8, q16, Y16, sums, amax, Yb)]

    shapes = [(300, 528, 264, 1), (517, 1040, 520, 2)]
    data = [inputs(*s) for s in shapes]
    torch.cuda.synchronize()
    streams = [torch.cuda.Stream(device=dev) for _ in shapes]
    results = [None, None]
    start = threading.Barrier(2)

    def worker(i):
        torch.cuda.set_device(dev)
        start.wait()
        results[i] = layer(data[i], streams[i])

    threads = [threading.Thread(target=worker, args=(i,)) for i in range(2)]
    for t in threads:
        t.start()
    for t in threads:
        t.join()
    names = ["lambda", "Wq", "w_scale", "Xq", "x_scale", "Y_int8_codes", "Xq16", "Y_f16_codes",
             "stats_sums", "stats_absmax", "Y_bf16"]
    for i in range(2):
        again = layer(data[i], streams[0])
        for name, a, b in zip(names, results[i], again):
            if name == "stats_sums":
                # fp64 block sums added with atomics: the order, hence the
                # last bits, may differ from run to run
                assert torch.allclose(a, b, rtol=1e-12, atol=1e-9), f"{name} differs"
            else:
                assert torch.equal(a, b), f"{name}: a concurrent call differs from the serial one"
        # the two containers agree as they must
        assert torch.equal(results[i][5], results[i][7])
    assert w8a8.device_status() == 0
    print("threads ok")
""")


def test_two_threads_first_calls_concurrent(tmp_path):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    script = tmp_path / "threads.py"
    script.write_text(SCRIPT)
    r = subprocess.run([sys.executable, str(script), ROOT], capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stdout[-2000:] + r.stderr[-2000:]
    assert "threads ok" in r.stdout
