"""GPU parity of the UCS statistics (Sec. 3.4) against the oracle: drop-set
counts exact and J / J_rand / RDA bit-exact (both sides form them in fp64 from
the same integers); the redundancy gap within 2e-5 absolute (fp32 cosines and
means), its skip decision equal away from the threshold."""
import numpy as np
import pytest
import torch

from oracle import cer_oracle as ora
from paper_2608_29291_gb300 import cer
from paper_2608_29291_gb300 import inputs as gen
from tests.gpu_helpers import bf16_dev, bits_host

pytestmark = pytest.mark.gpu
GAP_TOL = 2e-5


@pytest.fixture(scope="module", autouse=True)
def _device():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    cer.load()


def _u8(a):
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.uint8)).cuda()


@pytest.mark.parametrize("B,N,r0,r1,p_t,p_r", [(1, 6, 1, 5, .5, .5), (4, 1024, 0, 729, .6, .6),
                                               (8, 1088, 64, 1088, .5, .3), (2, 4096, 0, 3840, .7, .7),
                                               (3, 300, 10, 10, .5, .5), (2, 500, 0, 500, 1.0, 1.0),
                                               (2, 500, 0, 500, 0.0, 0.0), (1, 49152, 0, 49152, .1, .9)])
def test_drop_set_stats_bit_exact(B, N, r0, r1, p_t, p_r):
    rng = np.random.default_rng(N + B)
    m_t = (rng.random((B, N)) < p_t).astype(np.uint8)
    m_r = np.where(rng.random((B, N)) < 0.8, m_t, (rng.random((B, N)) < p_r)).astype(np.uint8)
    J = torch.empty(B, dtype=torch.float32, device="cuda")
    Jr, R = torch.empty_like(J), torch.empty_like(J)
    counts = torch.empty((B, 3), dtype=torch.int32, device="cuda")
    cer.cer_drop_set_stats(_u8(m_t), _u8(m_r), r0, r1, J, Jr, R, counts)
    cer.cer_sync_status()
    wJ, wJr, wR, wc = ora.drop_set_stats(m_t, m_r, r0, r1)
    assert np.array_equal(counts.cpu().numpy(), wc)
    assert np.array_equal(J.cpu().numpy(), wJ.astype(np.float32))
    assert np.array_equal(Jr.cpu().numpy(), wJr.astype(np.float32))
    assert np.array_equal(R.cpu().numpy(), wR.astype(np.float32))


def test_drop_set_stats_on_block_keep_masks_across_timesteps():
    """The intended use: keep masks of two routing decisions (t and t_ref)."""
    w = gen.Workload("gen_small", B=3, N=300, d=256, I=64, C=64, r0=20, r1=300, K=140, Hc=128, He=64, E=64,
                     task=1, seed=4)
    inp = gen.make_inputs(w)
    rng = np.random.default_rng(5)
    lg_t = rng.normal(size=(w.B, w.N)).astype(np.float32)
    lg_r = (lg_t + 0.3 * rng.normal(size=(w.B, w.N))).astype(np.float32)
    _, m_t = ora.select_topk(lg_t, w.r0, w.r1, w.K)
    _, m_r = ora.select_topk(lg_r, w.r0, w.r1, w.K)
    J = torch.empty(w.B, dtype=torch.float32, device="cuda")
    R = torch.empty_like(J)
    cer.cer_drop_set_stats(_u8(m_t), _u8(m_r), w.r0, w.r1, J, None, R)
    cer.cer_sync_status()
    wJ, _, wR, _ = ora.drop_set_stats(m_t, m_r, w.r0, w.r1)
    assert np.array_equal(J.cpu().numpy(), wJ.astype(np.float32))
    assert np.array_equal(R.cpu().numpy(), wR.astype(np.float32))
    del inp


@pytest.mark.parametrize("B,N,d", [(1, 3, 8), (4, 1024, 1536), (2, 4096, 3584), (3, 257, 264)])
def test_redundancy_gap_matches_oracle(B, N, d):
    rng = np.random.default_rng(B * N + d)
    h_in = gen.f32_to_bf16_bits(rng.normal(0, 1, (B, N, d)).astype(np.float32))
    mask = (rng.random((B, N)) < 0.5).astype(np.uint8)
    upd = gen.f32_to_bf16_bits(rng.normal(0, 0.3, (B, N, d)).astype(np.float32))
    h_out = np.where(mask[:, :, None] == 1, gen.f32_to_bf16_bits((ora.bf16_to_f64(h_in) + ora.bf16_to_f64(upd))
                                                                 .astype(np.float32)), h_in).astype(np.uint16)
    if N >= 3:
        h_in[0, 1] = 0                      # zero rows: equal -> cos 1, different -> cos 0
        h_out[0, 1] = 0
        h_in[0, 2] = 0
    gap = torch.empty(B, dtype=torch.float32, device="cuda")
    skip = torch.empty(B, dtype=torch.uint8, device="cuda")
    delta = 0.004
    cer.cer_redundancy_gap(bf16_dev(h_in), bf16_dev(h_out), _u8(mask), delta, gap, skip)
    cer.cer_sync_status()
    want = ora.redundancy_gap(h_in, h_out, mask)
    got = gap.cpu().numpy().astype(np.float64)
    assert np.max(np.abs(got - want)) <= GAP_TOL
    sk = skip.cpu().numpy()
    for b in range(B):
        if abs(want[b] - delta) > GAP_TOL:
            assert sk[b] == (1 if want[b] <= delta else 0)


def test_redundancy_gap_of_the_routed_block():
    """g of the routed block itself: dropped rows are unchanged (cos 1)."""
    w = gen.Workload("und_small", B=2, N=500, d=512, I=1024, C=512, r0=0, r1=400, K=150, Hc=256, He=0, E=0,
                     task=0, seed=6)
    inp = gen.make_inputs(w)
    core, _ = __import__("tests.gpu_helpers", fromlist=["scorers"]).scorers(inp)
    h = bf16_dev(inp["h"])
    h0 = h.clone()
    mask = torch.empty((w.B, w.N), dtype=torch.uint8, device="cuda")
    Wg, Wu, WdT = cer.pack_ffn_weights(bf16_dev(inp["Wg"]), bf16_dev(inp["Wu"]), bf16_dev(inp["WdT"]),
                                       torch.from_numpy(inp["chan"]).cuda())
    cer.cer_routed_block(h, core, None, torch.zeros(w.B, device="cuda"), 0, w.r0, w.r1, w.K, Wg, Wu, WdT, None,
                         mask=mask)
    gap = torch.empty(w.B, dtype=torch.float32, device="cuda")
    cer.cer_redundancy_gap(h0, h, mask, 0.004, gap)
    cer.cer_sync_status()
    want = ora.redundancy_gap(bits_host(h0), bits_host(h), mask.cpu().numpy())
    assert np.max(np.abs(gap.cpu().numpy() - want)) <= GAP_TOL
    assert np.all(want > 0)      # kept rows change (cos < 1), dropped rows do not (cos 1): the gap is positive
