"""The routed block and the routed FFN captured in a CUDA graph (a serving
loop's way to launch them): every replay reproduces the eager call bit for
bit -- per-launch state (stream-K flags, the launch token baked into the
captured kernels) must not leak from one replay into the next."""
import numpy as np
import pytest
import torch

from paper_2608_29291_gb300 import cer
from paper_2608_29291_gb300 import inputs as gen
from tests.gpu_helpers import bf16_dev, f32_dev, scorers

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _device():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    cer.load()
    yield
    cer.cer_sync_status()


def _capture(fn, stream):
    """Run fn once eagerly (the library's per-context setup), then capture it."""
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        fn()
    return g


@pytest.mark.parametrize("task", [0, 1], ids=["und", "gen"])
def test_routed_block_replays_bit_identical(task):
    kw = dict(B=3, N=700, d=1024, I=2048, C=1024, r0=50, r1=700, K=200, Hc=256, He=256 if task else 0,
              E=64 if task else 0, task=task)
    w = gen.Workload(name="graph_block", **kw)
    inp = gen.make_inputs(w)
    core, exp = scorers(inp)
    h0 = bf16_dev(inp["h"])
    h = h0.clone()
    t = f32_dev(inp["t"])
    Wg, Wu, WdT = (bf16_dev(inp[k]) for k in ("Wg", "Wu", "WdT"))
    Wg, Wu, WdT = cer.pack_ffn_weights(Wg, Wu, WdT, torch.from_numpy(inp["chan"]).cuda())
    ws = cer.workspace(cer.cer_routed_block_workspace_size(w.B, w.N, w.d, w.Hc, w.He, task, w.r0, w.r1, w.K, w.C,
                                                           False), h.device)
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        def step():
            cer.cer_routed_block(h, core, exp, t, task, w.r0, w.r1, w.K, Wg, Wu, WdT, None, ws=ws, stream=s)
        step()
        cer.cer_sync_status(s)
        ref = h.clone()
        h.copy_(h0)
        g = _capture(step, s)
        for _ in range(3):
            h.copy_(h0)
            g.replay()
            s.synchronize()
            assert torch.equal(h.view(torch.int16), ref.view(torch.int16))
        cer.cer_sync_status(s)


def test_routed_ffn_with_stream_k_replays_bit_identical():
    """(2000, 2560, 4096): the down GEMM splits its last wave by K block, so
    every replay publishes and consumes the stream-K flags again."""
    M, d, I = 2000, 2560, 4096
    rng = np.random.default_rng(7)
    X = bf16_dev(gen.f32_to_bf16_bits(rng.normal(0, 1, (M, d)).astype(np.float32)))
    Wg, Wu = (bf16_dev(gen.bf16_normal(M, n, (I, d), d ** -.5)) for n in ("g", "u"))
    WdT = bf16_dev(gen.bf16_normal(M, "dn", (I, d), I ** -.5))
    Y = torch.empty((M, d), dtype=torch.bfloat16, device="cuda")
    ws = cer.workspace(cer.cer_routed_ffn_workspace_size(M, d, I, False), X.device)
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        def ffn():
            cer.cer_routed_ffn(X, Wg, Wu, WdT, None, Y, ws=ws, stream=s)
        ffn()
        cer.cer_sync_status(s)
        ref = Y.clone()
        g = _capture(ffn, s)
        for _ in range(3):
            Y.fill_(0)
            g.replay()
            s.synchronize()
            assert torch.equal(Y.view(torch.int16), ref.view(torch.int16))
        cer.cer_sync_status(s)
