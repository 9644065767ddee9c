"""GPU edge cases of the routed-block path through the C ABI: empty inputs
(every entry point returns OK and records no error) and the scorer at the
largest shapes the ABI accepts (d = 16384; core and expansion hidden widths
of 4096 with a 1024-wide time embedding), against the oracle."""
import zlib

import numpy as np
import pytest
import torch

from oracle import cer_oracle as ora
from paper_2608_29291_gb300 import cer
from paper_2608_29291_gb300 import inputs as gen
from tests.gpu_helpers import bf16_dev, f32_dev, score_err, scorers

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _device():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    cer.load()
    yield
    cer.cer_sync_status()


def _und_scorer(d, Hc, seed):
    rng = np.random.default_rng(seed)
    W1 = gen.f32_to_bf16_bits(rng.normal(0, d ** -.5, (Hc, d)).astype(np.float32))
    return dict(W1=W1, w2=rng.normal(0, Hc ** -.5, Hc).astype(np.float32), b1=rng.normal(0, .1, Hc).astype(np.float32))


@pytest.mark.parametrize("B,N", [(0, 300), (2, 0)], ids=["B0", "N0"])
def test_empty_inputs_are_no_ops(B, N):
    d, Hc, I = 256, 128, 512
    core, _ = scorers(_und_scorer(d, Hc, 1))
    h = torch.empty((B, N, d), dtype=torch.bfloat16, device="cuda")
    logits = torch.empty((B, N), dtype=torch.float32, device="cuda")
    cer.cer_score(h, core, None, None, 0, logits)
    idx = torch.empty((B, 0), dtype=torch.int32, device="cuda")
    cer.cer_select_topk(logits, 0, N, 0, idx)
    X = torch.empty((0, d), dtype=torch.bfloat16, device="cuda")
    cer.cer_gather(h, idx, X)
    cer.cer_scatter_add(h, idx, X)
    rng = np.random.default_rng(2)
    W = [bf16_dev(gen.f32_to_bf16_bits(rng.normal(0, .05, (I, d)).astype(np.float32))) for _ in range(3)]
    cer.cer_routed_ffn(X, W[0], W[1], W[2], None, torch.empty((0, d), dtype=torch.bfloat16, device="cuda"))
    # the block, in place and out of place (K = 0 of an empty routable range)
    cer.cer_routed_block(h, core, None, None, 0, 0, N, 0, W[0], W[1], W[2], None)
    cer.cer_routed_block(h, core, None, None, 0, 0, N, 0, W[0], W[1], W[2], None, out=torch.empty_like(h))
    # every call above returned OK (the wrappers raise otherwise) and no
    # kernel recorded an error
    cer.cer_sync_status()


def test_empty_keep_set_leaves_h_and_writes_empty_lists():
    """K = 0 over the whole sequence: no row is kept, so the FFN has M = 0
    rows and h is returned untouched (in place)."""
    B, N, d, Hc, I = 2, 257, 256, 128, 512
    rng = np.random.default_rng(3)
    core, _ = scorers(_und_scorer(d, Hc, 4))
    hb = gen.f32_to_bf16_bits(rng.normal(0, 1, (B, N, d)).astype(np.float32))
    h = bf16_dev(hb)
    W = [bf16_dev(gen.f32_to_bf16_bits(rng.normal(0, .05, (I, d)).astype(np.float32))) for _ in range(3)]
    mask = torch.full((B, N), 7, dtype=torch.uint8, device="cuda")
    cer.cer_routed_block(h, core, None, None, 0, 0, N, 0, W[0], W[1], W[2], None, mask=mask)
    cer.cer_sync_status()
    assert np.array_equal(h.view(torch.int16).cpu().numpy().view(np.uint16), hb)
    assert not mask.cpu().numpy().any()


def _max_case(name):
    rng = np.random.default_rng(zlib.crc32(name.encode()))

    def bf(shape, s):
        return gen.f32_to_bf16_bits(rng.normal(0, s, shape).astype(np.float32))
    if name == "d16384":
        # the widest hidden state: 256 K blocks per tile, 64-wide chunks
        B, N, d, Hc = 1, 300, 16384, 256
        inp = dict(h=bf((B, N, d), 1), **_und_scorer(d, Hc, 5), t=np.zeros(B, np.float32))
        return inp, 0
    if name == "hidden4096_emb1024":
        # the widest scorers: 8192 hidden units (32 chunks of the pair scorer),
        # ragged rows (520 = 2 x 256 + 8), the widest time embedding
        B, N, d, Hc, He, E = 2, 260, 256, 4096, 4096, 1024
        inp = dict(h=bf((B, N, d), 1), W1=bf((Hc, d), d ** -.5), w2=rng.normal(0, Hc ** -.5, Hc).astype(np.float32),
                   b1=rng.normal(0, .1, Hc).astype(np.float32), W1e=bf((1, He, d), d ** -.5),
                   w2e=rng.normal(0, He ** -.5, (1, He)).astype(np.float32), Ue=bf((1, He, E), E ** -.5),
                   b1e=rng.normal(0, .1, (1, He)).astype(np.float32), t=np.array([0.2, 0.85], np.float32))
        return inp, 1
    raise KeyError(name)


@pytest.mark.parametrize("name", ["d16384", "hidden4096_emb1024"])
def test_score_at_the_largest_shapes(name):
    inp, task = _max_case(name)
    B, N, d = inp["h"].shape
    core, exp = scorers(inp)
    logits = torch.empty((B, N), dtype=torch.float32, device="cuda")
    cer.cer_score(bf16_dev(inp["h"]), core, exp, f32_dev(inp["t"]), task, logits)
    cer.cer_sync_status()
    want = ora.score(inp["h"], inp["W1"], inp["w2"], inp.get("b1"), inp["t"], task, inp.get("W1e"), inp.get("w2e"),
                     inp.get("Ue"), inp.get("b1e"))
    assert score_err(logits.cpu().numpy(), want, d) <= 1.0
