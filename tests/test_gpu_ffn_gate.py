"""GPU parity of the UCS FFN gate (Sec. 3.4 (2), Eq. 8 / Eq. 9) against the
oracle: saliency within 4e-3 relative (the GPU reads the bf16-rounded
activation) plus 1e-6 of the largest saliency, leakage within 2e-3
absolute, the decision equal away from the threshold, and the FFN output
of the branch taken within the block tolerance."""
import numpy as np
import pytest
import torch

from oracle import cer_oracle as ora
from paper_2608_29291_gb300 import cer
from paper_2608_29291_gb300 import inputs as gen
from tests.gpu_helpers import bf16_dev, bits_host, f32_dev, ffn_out_ok, out_err_ok, scorers

pytestmark = pytest.mark.gpu
OUT_TOL = 2e-2
LEAK_TOL = 2e-3


@pytest.fixture(scope="module", autouse=True)
def _device():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    cer.load()


def _weights(I, d, seed, zero_pruned_down=False, C=None):
    Wg, Wu = (gen.bf16_normal(seed, n, (I, d), d ** -.5) for n in ("g", "u"))
    WdT = gen.bf16_normal(seed, "dn", (I, d), I ** -.5)
    chan = gen.channel_keep_set(seed, "c", I, C)
    if zero_pruned_down:
        pruned = np.setdiff1d(np.arange(I), chan)
        WdT = WdT.copy()
        WdT[pruned] = 0
    return Wg, Wu, WdT, chan


def _check_gate(X, Wg, Wu, WdT, chan, delta, got_sal_perm, got_leak, got_flag, perm, Y_bits):
    sal = ora.ffn_saliency(X, Wg, Wu, WdT)
    pruned = np.setdiff1d(np.arange(Wg.shape[0]), chan)
    lam = ora.ffn_leakage(sal, pruned)
    got_sal = np.empty_like(sal)
    got_sal[perm] = got_sal_perm
    assert np.all(np.abs(got_sal - sal) <= 4e-3 * sal + 1e-6 * sal.max())
    assert abs(got_leak - lam) <= LEAK_TOL
    if abs(lam - delta) > LEAK_TOL:
        assert got_flag == (1 if lam <= delta else 0)
    use = chan if got_flag == 1 else np.arange(Wg.shape[0])
    want = ora.routed_ffn(X, Wg, Wu, WdT, use, act_bf16=True)
    ok, excess = ffn_out_ok(ora.bf16_to_f64(Y_bits), want)
    assert ok, excess
    return lam


@pytest.mark.parametrize("M,d,I,C,delta,zero", [(300, 256, 1024, 768, 0.15, False), (300, 256, 1024, 768, 0.99, False),
                                                (300, 320, 1024, 576, 0.99, False),
                                                (129, 512, 2048, 1024, 0.15, True), (1, 256, 512, 256, 0.5, False),
                                                (2348, 1536, 8960, 6720, 0.15, False)])
def test_gated_ffn_matches_oracle(M, d, I, C, delta, zero):
    Wg, Wu, WdT, chan = _weights(I, d, M + I, zero, C)
    X = gen.bf16_normal(M, "x", (M, d), 1.0)
    Wg_p, Wu_p, WdT_p, norms, perm = cer.gate_weights(bf16_dev(Wg), bf16_dev(Wu), bf16_dev(WdT),
                                                     torch.from_numpy(chan).cuda())
    Y = torch.empty((M, d), dtype=torch.bfloat16, device="cuda")
    sal = torch.empty(I, dtype=torch.float32, device="cuda")
    leak = torch.empty(1, dtype=torch.float32, device="cuda")
    flag = torch.empty(1, dtype=torch.uint8, device="cuda")
    cer.cer_routed_ffn_gated(bf16_dev(X), Wg_p, Wu_p, WdT_p, C, norms, delta, Y, sal, leak, flag)
    cer.cer_sync_status()
    lam = _check_gate(X, Wg, Wu, WdT, chan, delta, sal.cpu().numpy(), float(leak.item()), int(flag.item()),
                      perm.cpu().numpy(), bits_host(Y))
    if zero:
        assert lam == 0.0 and int(flag.item()) == 1      # pruned channels carry nothing: the pruned FFN runs
    if delta == 0.99:
        assert int(flag.item()) == 1


def test_channel_norms_match_oracle():
    WdT = gen.bf16_normal(3, "w", (640, 264), 0.1)
    norms = torch.empty(640, dtype=torch.float32, device="cuda")
    cer.cer_ffn_channel_norms(bf16_dev(WdT), norms)
    cer.cer_sync_status()
    want = np.sqrt(np.sum(ora.bf16_to_f64(WdT) ** 2, axis=1))
    assert np.allclose(norms.cpu().numpy(), want, rtol=2e-6)


@pytest.mark.parametrize("delta", [0.15, 0.0])
def test_gated_block_matches_oracle(delta):
    w = gen.Workload("gated", B=2, N=400, d=512, I=1024, C=768, r0=0, r1=350, K=120, Hc=128, He=64, E=64,
                     task=1, seed=8)
    inp = gen.make_inputs(w)
    core, exp = scorers(inp)
    h = bf16_dev(inp["h"])
    Wg_p, Wu_p, WdT_p, norms, perm = cer.gate_weights(bf16_dev(inp["Wg"]), bf16_dev(inp["Wu"]),
                                                     bf16_dev(inp["WdT"]), torch.from_numpy(inp["chan"]).cuda())
    idx = torch.empty((w.B, w.k_tot), dtype=torch.int32, device="cuda")
    sal = torch.empty(w.I, dtype=torch.float32, device="cuda")
    leak = torch.empty(1, dtype=torch.float32, device="cuda")
    flag = torch.empty(1, dtype=torch.uint8, device="cuda")
    cer.cer_routed_block_gated(h, core, exp, f32_dev(inp["t"]), w.task, w.r0, w.r1, w.K, Wg_p, Wu_p, WdT_p, w.C,
                               norms, delta, sal, leak, flag, idx=idx)
    cer.cer_sync_status()
    gi = idx.cpu().numpy()
    X = ora.gather(inp["h"], gi)
    out = bits_host(h)
    sal_np = sal.cpu().numpy()
    lam = float(leak.item())
    f = int(flag.item())
    want_sal = ora.ffn_saliency(X, inp["Wg"], inp["Wu"], inp["WdT"])
    got = np.empty_like(want_sal)
    got[perm.cpu().numpy()] = sal_np
    assert np.all(np.abs(got - want_sal) <= 4e-3 * want_sal + 1e-6 * want_sal.max())
    want_lam = ora.ffn_leakage(want_sal, np.setdiff1d(np.arange(w.I), inp["chan"]))
    assert abs(lam - want_lam) <= LEAK_TOL
    if delta == 0.0:
        assert f == 0                                    # leakage > 0: the full FFN runs
    use = inp["chan"] if f == 1 else np.arange(w.I)
    exact = ora.bf16_to_f64(inp["h"]).copy()
    for b in range(w.B):
        exact[b, gi[b]] += ora.routed_ffn(ora.gather(inp["h"][b:b + 1], gi[b:b + 1]), inp["Wg"], inp["Wu"],
                                          inp["WdT"], use, act_bf16=True)
    ok, excess = ffn_out_ok(ora.bf16_to_f64(out), exact)
    assert ok, excess
