"""Pins of the CPU oracle against things other than itself.

Each test checks the oracle against a hand-derived value (tests/golden/), a
brute-force enumeration, a closed form, a textbook constant, an invariant of the
paper's definitions, or an independent library routine (torch CPU).  The
mutation test at the end plants plausible mistakes in the oracle and checks that
these pins catch every one of them.
"""
import itertools
import json
import math
import os

import numpy as np
import pytest
import torch
import torch.nn.functional as F

from oracle import cer_oracle as ora
from paper_2608_29291_gb300 import inputs as gen

GOLD = os.path.join(os.path.dirname(__file__), "golden")


def _bits(x):
    """Exact bf16 bit patterns of small dyadic test values (via torch's conversion)."""
    t = torch.tensor(np.asarray(x, dtype=np.float32)).to(torch.bfloat16)
    assert torch.equal(t.float(), torch.tensor(np.asarray(x, dtype=np.float32))), "value not bf16-exact"
    return t.view(torch.int16).numpy().view(np.uint16)


def _load(name):
    with open(os.path.join(GOLD, name)) as f:
        return json.load(f)


def _hand_inputs(g):
    return dict(
        h=_bits(g["h"])[None],
        W1=_bits(g["W1"]), w2=np.array(g["w2"], np.float32), b1=None,
        W1e=_bits(g["W1e"]), w2e=np.array(g["w2e"], np.float32), Ue=_bits(g["Ue"]), b1e=None,
        t=np.array(g["t"], np.float32),
        Wg=_bits(g["Wg"]), Wu=_bits(g["Wu"]), WdT=_bits(g["WdT"]),
        chan=np.array(g["chan"], np.int32))


# ------------------------------------------------------------------ hand example

def _hand_checks():
    """All hand-example checks; returns a list of failure strings (empty = pass)."""
    g = _load("hand_4tok.json")
    x = _hand_inputs(g)
    fails = []
    for task, key in ((ora.TASK_UND, "und"), (ora.TASK_GEN, "gen")):
        lg = ora.score(x["h"], x["W1"], x["w2"], None, x["t"], task, x["W1e"], x["w2e"], x["Ue"], None)
        if not np.allclose(lg[0], np.float32(g["logits_" + key]), rtol=0, atol=0):
            # stored fp32: compare to the fp32 rounding of the hand value
            if not np.allclose(lg[0], g["logits_" + key], rtol=2e-7, atol=0):
                fails.append(f"logits_{key}: {lg[0]} vs {g['logits_' + key]}")
        res = ora.routed_block(x["h"], x["W1"], x["w2"], None, x["t"], task, 0, 4, g["K"],
                               x["Wg"], x["Wu"], x["WdT"], x["chan"], x["W1e"], x["w2e"], x["Ue"], None)
        if res["idx"][0].tolist() != g["idx_" + key]:
            fails.append(f"idx_{key}: {res['idx'][0].tolist()}")
        if not np.allclose(res["Y"], g["Y_" + key], rtol=0, atol=1e-12):
            fails.append(f"Y_{key}: {res['Y']}")
        out = ora.bf16_to_f64(res["out"][0])
        if not np.array_equal(out, np.array(g["out_" + key], dtype=np.float64)):
            fails.append(f"out_{key}: {out}")
    emb = ora.sinusoidal_embedding(0.0, 2)
    if emb.tolist() != g["emb_at_t0"]:
        fails.append(f"emb: {emb}")
    return fails


def test_hand_example():
    assert _hand_checks() == []


# ------------------------------------------------------------------ selection

def _select_golden_checks():
    g = _load("select_ties.json")
    vals = np.array([float(v) for v in g["logits"]], dtype=np.float32)[None]
    fails = []
    for c in g["cases"]:
        idx, mask = ora.select_topk(vals, c["r0"], c["r1"], c["K"])
        if idx[0].tolist() != c["idx"]:
            fails.append(f"{c}: got {idx[0].tolist()}")
        if sorted(np.nonzero(mask[0])[0].tolist()) != c["idx"]:
            fails.append(f"mask {c}")
    return fails


def test_select_golden_ties_signed_zero_inf():
    assert _select_golden_checks() == []


def _brute_force_set(vals, r0, r1, K):
    """The unique K-subset S of [r0, r1) with every member ranked above every
    non-member (larger value, or equal value and lower index); found by trying all."""
    routable = list(range(r0, r1))
    found = []
    for S in itertools.combinations(routable, K):
        inside = set(S)
        ok = all(vals[i] > vals[j] or (vals[i] == vals[j] and i < j)
                 for i in inside for j in routable if j not in inside)
        if ok:
            found.append(S)
    assert len(found) == 1, f"brute force found {len(found)} valid sets"
    return sorted(set(found[0]) | set(range(0, r0)) | set(range(r1, len(vals))))


def _brute_force_checks(n_cases=400, seed=1):
    rng = np.random.default_rng(seed)
    alphabet = np.array([-1.0, -0.0, 0.0, 1.0, 2.0, -np.inf, np.inf, 1e-30], dtype=np.float32)
    fails = []
    for _ in range(n_cases):
        N = int(rng.integers(1, 9))
        sub = alphabet[rng.choice(len(alphabet), size=int(rng.integers(1, 4)), replace=False)]
        vals = sub[rng.integers(0, len(sub), size=N)]
        r0 = int(rng.integers(0, N + 1))
        r1 = int(rng.integers(r0, N + 1))
        K = int(rng.integers(0, r1 - r0 + 1))
        want = _brute_force_set([float(v) for v in vals], r0, r1, K)
        idx, mask = ora.select_topk(vals[None], r0, r1, K)
        if idx[0].tolist() != want or np.nonzero(mask[0])[0].tolist() != want:
            fails.append((vals.tolist(), r0, r1, K, idx[0].tolist(), want))
    return fails


def test_topk_brute_force_exhaustive_small():
    assert _brute_force_checks() == []


def test_topk_nan_is_error():
    v = np.array([[0.5, np.nan, 1.0]], dtype=np.float32)
    with pytest.raises(ora.OracleNaN):
        ora.select_topk(v, 0, 3, 1)
    # a NaN outside the routable range does not take part in the ranking
    idx, _ = ora.select_topk(v, 2, 3, 1)
    assert idx[0].tolist() == [0, 1, 2]


def test_sigmoid_ranking_equals_logit_ranking():
    """App. B.2: the sigmoid is monotonic, so TopK on p and on l agree (where the
    fp64 sigmoid keeps the values distinct)."""
    rng = np.random.default_rng(3)
    for _ in range(20):
        lg = rng.normal(0, 3, size=(1, 64)).astype(np.float32)
        p = ora.sigmoid(lg)
        assert len(np.unique(p)) == 64
        K = int(rng.integers(0, 65))
        idx, _ = ora.select_topk(lg, 0, 64, K)
        want = np.sort(np.argsort(-p[0], kind="stable")[:K])
        assert idx[0].tolist() == want.tolist()


def test_sigmoid_values():
    """p = sigmoid(l) of Eq. 6 by value: sigma(0) = 1/2; sigma(ln 3) = 3/4 and
    sigma(-ln 3) = 1/4 (1 / (1 + 1/3) and 1 / (1 + 3)); sigma(ln 9) = 9/10;
    the symmetry sigma(x) + sigma(-x) = 1; the limits; and torch's sigmoid in
    fp64 as an independent library routine."""
    assert ora.sigmoid(np.array([0.0]))[0] == 0.5
    assert abs(ora.sigmoid(np.array([math.log(3.0)]))[0] - 0.75) < 1e-15
    assert abs(ora.sigmoid(np.array([-math.log(3.0)]))[0] - 0.25) < 1e-15
    assert abs(ora.sigmoid(np.array([math.log(9.0)]))[0] - 0.9) < 1e-15
    x = np.random.default_rng(4).normal(0, 4, 1000)
    assert np.max(np.abs(ora.sigmoid(x) + ora.sigmoid(-x) - 1.0)) < 1e-15
    with np.errstate(over="ignore"):
        assert ora.sigmoid(np.array([-800.0]))[0] == 0.0 and ora.sigmoid(np.array([800.0]))[0] == 1.0
    want = torch.sigmoid(torch.from_numpy(x)).numpy()
    assert np.max(np.abs(ora.sigmoid(x) - want)) < 1e-15


# ------------------------------------------------------------------ scalar pieces

def test_bf16_widening_exact():
    bits = np.array([0x3F80, 0xC000, 0x0001, 0x8000, 0x7F80, 0x4049], dtype=np.uint16)
    want = [1.0, -2.0, 2.0 ** -133, -0.0, math.inf, 3.140625]
    got = ora.bf16_to_f64(bits)
    assert got.tolist() == want
    assert math.copysign(1, got[3]) == -1


def test_round_to_bf16_matches_torch_rne():
    rng = np.random.default_rng(0)
    f = rng.normal(0, 10, 20000).astype(np.float32)
    # exact halfway cases and their neighbours
    base = rng.integers(0, 0x7F00, 2000).astype(np.uint32) << np.uint32(16)   # finite, both signs below
    half = np.concatenate([base | 0x8000, base | 0x7FFF, base | 0x8001, (base + (1 << 16)) | 0x8000])
    half = np.concatenate([half, half | np.uint32(0x80000000)])
    f = np.concatenate([f, half.view(np.float32)])
    want = torch.tensor(f).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    got = ora.round_to_bf16(f.astype(np.float64))
    assert np.array_equal(got, want)


def test_gelu_textbook_and_library():
    assert ora.gelu(np.array([0.0]))[0] == 0.0
    assert abs(ora.gelu(np.array([1.0]))[0] - 0.8413447460685429) < 1e-15      # Phi(1)
    assert abs(ora.gelu(np.array([2.0]))[0] - 2 * 0.9772498680518208) < 1e-14  # 2 Phi(2)
    x = np.linspace(-6, 6, 1001)
    assert np.allclose(ora.gelu(x) - ora.gelu(-x), x, rtol=0, atol=1e-14)
    ref = F.gelu(torch.tensor(x, dtype=torch.float64), approximate="none").numpy()
    assert np.allclose(ora.gelu(x), ref, rtol=1e-14, atol=1e-15)


def test_sinusoid_invariants():
    E = 16
    assert ora.sinusoidal_embedding(0.0, E).tolist() == [1.0] * 8 + [0.0] * 8
    for t in (0.1, 0.37, 0.9):
        e = ora.sinusoidal_embedding(t, E).astype(np.float64)
        assert np.allclose(e[:8] ** 2 + e[8:] ** 2, 1.0, atol=1e-6)
        # lowest-frequency pair: f = 10000^(-7/8)
        a = 1000 * t * 10000 ** (-7 / 8)
        assert abs(e[7] - math.cos(a)) < 1e-6 and abs(e[15] - math.sin(a)) < 1e-6


def test_segment_index():
    assert [ora.segment_index(t, 4) for t in (0.0, 0.2499, 0.25, 0.5, 0.999, 1.0)] == [0, 0, 1, 2, 3, 3]
    assert ora.segment_index(0.7, 1) == 0


# ------------------------------------------------------------------ scorer

def _random_scorer(rng, d=32, Hc=16, He=8, E=8, S=3, B=3, N=10):
    def bf(shape, s):
        return gen.f32_to_bf16_bits((rng.normal(0, s, shape)).astype(np.float32))
    return dict(h=bf((B, N, d), 1.0), W1=bf((Hc, d), d ** -0.5),
                w2=rng.normal(0, 1, Hc).astype(np.float32),
                b1=rng.normal(0, .1, Hc).astype(np.float32),
                W1e=bf((S, He, d), d ** -0.5), w2e=rng.normal(0, 1, (S, He)).astype(np.float32),
                Ue=bf((S, He, E), E ** -0.5), b1e=rng.normal(0, .1, (S, He)).astype(np.float32),
                t=rng.uniform(0, 1, B).astype(np.float32))


def test_score_matches_torch_library():
    rng = np.random.default_rng(5)
    p = _random_scorer(rng)
    got = ora.score(p["h"], p["W1"], p["w2"], p["b1"], p["t"], ora.TASK_GEN,
                    p["W1e"], p["w2e"], p["Ue"], p["b1e"])

    def T(bits):
        return torch.tensor(bits.astype(np.int16)).view(torch.bfloat16).double()
    h = T(p["h"])
    core = F.linear(F.gelu(F.linear(h, T(p["W1"]), torch.tensor(p["b1"]).double())),
                    torch.tensor(p["w2"]).double()[None])[..., 0]
    for b in range(h.shape[0]):
        t = float(p["t"][b])
        m = min(2, int(math.floor(t * 3)))
        half = 4
        f = torch.tensor([10000.0 ** (-j / half) for j in range(half)], dtype=torch.float64)
        emb = torch.cat([torch.cos(1000 * t * f), torch.sin(1000 * t * f)]).float().double()
        bias = T(p["Ue"][m]) @ emb + torch.tensor(p["b1e"][m]).double()
        e = F.linear(F.gelu(F.linear(h[b], T(p["W1e"][m]), bias)), torch.tensor(p["w2e"][m]).double()[None])[..., 0]
        want = (core[b] + e).float().numpy()
        assert np.allclose(got[b], want, rtol=1e-6, atol=1e-7)


def test_understanding_ignores_expansion_and_t():
    rng = np.random.default_rng(6)
    p = _random_scorer(rng)
    a = ora.score(p["h"], p["W1"], p["w2"], p["b1"], p["t"], ora.TASK_UND, p["W1e"], p["w2e"], p["Ue"], p["b1e"])
    b = ora.score(p["h"], p["W1"], p["w2"], p["b1"], p["t"] * 0 + 0.9, ora.TASK_UND)
    assert np.array_equal(a, b)


def test_zero_U_makes_expansion_time_invariant():
    rng = np.random.default_rng(7)
    p = _random_scorer(rng, S=1)
    Z = np.zeros_like(p["Ue"])
    a = ora.score(p["h"], p["W1"], p["w2"], p["b1"], p["t"], ora.TASK_GEN, p["W1e"], p["w2e"], Z, p["b1e"])
    b = ora.score(p["h"], p["W1"], p["w2"], p["b1"], 1 - p["t"], ora.TASK_GEN, p["W1e"], p["w2e"], Z, p["b1e"])
    assert np.array_equal(a, b)
    # and differs once U is non-zero (t enters)
    c = ora.score(p["h"], p["W1"], p["w2"], p["b1"], 1 - p["t"], ora.TASK_GEN, p["W1e"], p["w2e"], p["Ue"], p["b1e"])
    assert not np.array_equal(a, c)


def test_single_hidden_unit_closed_form():
    """Hc = 1, w2 = 1: the logit is GELU(w . h) exactly (w . h = 0.5 -> 0.5 Phi(0.5))."""
    h = _bits([[[0.5, 0.0], [-0.5, 1.0]]])
    W1 = _bits([[1.0, 0.0]])
    lg = ora.score(h, W1, np.array([1.0], np.float32), None, np.zeros(1, np.float32), ora.TASK_UND)
    phi_half = 0.6914624612740131       # standard normal CDF at 0.5 (normal table)
    assert abs(lg[0, 0] - 0.5 * phi_half) < 1e-7
    assert abs(lg[0, 1] + 0.5 * (1 - phi_half)) < 1e-7


# ------------------------------------------------------------------ FFN and block

def _T(bits):
    return torch.tensor(bits.astype(np.int16)).view(torch.bfloat16).double()


def test_ffn_dense_matches_torch_swiglu():
    rng = np.random.default_rng(8)
    M, d, I = 7, 24, 40
    X = gen.f32_to_bf16_bits(rng.normal(0, 1, (M, d)).astype(np.float32))
    Wg, Wu, WdT = (gen.f32_to_bf16_bits(rng.normal(0, s, (I, d)).astype(np.float32)) for s in (0.3, 0.3, 0.2))
    Y = ora.routed_ffn(X, Wg, Wu, WdT, np.arange(I, dtype=np.int32))
    x = _T(X)
    want = (F.silu(x @ _T(Wg).T) * (x @ _T(Wu).T)) @ _T(WdT)
    assert np.allclose(Y, want.numpy(), rtol=1e-12, atol=1e-12)


def test_ffn_bf16_activation_matches_torch():
    """The bf16-operand activation: torch's SiLU in fp64, its fp32 -> bf16
    conversions (round to nearest even), then an fp64 contraction, agree with
    the oracle's act_bf16 path to fp64 rounding; and the rounding changes the
    result (so the flag is not ignored)."""
    rng = np.random.default_rng(12)
    M, d, I = 9, 32, 40
    X = gen.f32_to_bf16_bits(rng.normal(0, 2, (M, d)).astype(np.float32))
    Wg, Wu, WdT = (gen.f32_to_bf16_bits(rng.normal(0, 0.3, (I, d)).astype(np.float32)) for _ in range(3))
    chan = np.arange(0, I, 2)
    x = _T(X)
    g = x @ _T(Wg[chan]).T
    u = x @ _T(Wu[chan]).T
    a = (F.silu(g) * u).float().bfloat16().double()
    want = (a @ _T(WdT[chan])).numpy()
    got = ora.routed_ffn(X, Wg, Wu, WdT, chan, act_bf16=True)
    assert np.max(np.abs(got - want)) < 1e-12 * max(1.0, np.max(np.abs(want)))
    exact = ora.routed_ffn(X, Wg, Wu, WdT, chan)
    assert np.max(np.abs(got - exact)) > 1e-6


def test_ffn_pruned_equals_dense_with_removed_channels_zeroed():
    rng = np.random.default_rng(9)
    M, d, I = 9, 16, 32
    X = gen.f32_to_bf16_bits(rng.normal(0, 1, (M, d)).astype(np.float32))
    Wg, Wu, WdT = (gen.f32_to_bf16_bits(rng.normal(0, s, (I, d)).astype(np.float32)) for s in (0.3, 0.3, 0.2))
    chan = np.sort(rng.choice(I, 11, replace=False)).astype(np.int32)
    Y = ora.routed_ffn(X, Wg, Wu, WdT, chan)
    drop = np.setdiff1d(np.arange(I), chan)
    Wg0, WdT0 = Wg.copy(), WdT.copy()
    Wg0[drop] = 0
    WdT0[drop] = 0
    Yd = ora.routed_ffn(X, Wg0, Wu, WdT0, np.arange(I, dtype=np.int32))
    assert np.allclose(Y, Yd, rtol=1e-12, atol=1e-12)


def _small_block(seed=10, B=2, N=12, d=16, I=24, C=10, r0=2, r1=11, K=4, task=ora.TASK_GEN):
    rng = np.random.default_rng(seed)
    p = _random_scorer(rng, d=d, B=B, N=N)
    p.update(Wg=gen.f32_to_bf16_bits(rng.normal(0, .3, (I, d)).astype(np.float32)),
             Wu=gen.f32_to_bf16_bits(rng.normal(0, .3, (I, d)).astype(np.float32)),
             WdT=gen.f32_to_bf16_bits(rng.normal(0, .2, (I, d)).astype(np.float32)),
             chan=np.sort(rng.choice(I, C, replace=False)).astype(np.int32))
    args = (p["h"], p["W1"], p["w2"], p["b1"], p["t"], task, r0, r1, K, p["Wg"], p["Wu"], p["WdT"], p["chan"],
            p["W1e"], p["w2e"], p["Ue"], p["b1e"])
    return p, args


def test_block_invariants():
    p, args = _small_block()
    res = ora.routed_block(*args)
    h, idx, out, mask = p["h"], res["idx"], res["out"], res["mask"]
    B, N, _ = h.shape
    assert idx.shape == (B, 4 + N - 9)
    for b in range(B):
        assert np.all(np.diff(idx[b]) > 0)                        # strictly ascending, no duplicates
        assert set(range(0, 2)) | set(range(11, N)) <= set(idx[b].tolist())
        dropped = np.setdiff1d(np.arange(N), idx[b])
        assert np.array_equal(out[b, dropped], h[b, dropped])     # bypass: bit-identical
        assert mask[b].sum() == idx.shape[1]
        assert np.array_equal(np.nonzero(mask[b])[0], idx[b])


def test_block_zero_k_keeps_h_when_everything_routable():
    p, args = _small_block(r0=0, r1=12, K=0)
    res = ora.routed_block(*args)
    assert res["idx"].shape[1] == 0
    assert np.array_equal(res["out"], p["h"])


def test_block_full_keep_equals_dense_block():
    """K = N_r and C = I: the routed block is the dense block h + SwiGLU(h)."""
    I = 24
    p, args = _small_block(r0=0, r1=12, K=12, C=I)
    args = list(args)
    args[12] = np.arange(I, dtype=np.int32)
    res = ora.routed_block(*args)
    h = _T(p["h"])
    dense = h + (F.silu(h @ _T(p["Wg"]).T) * (h @ _T(p["Wu"]).T)) @ _T(p["WdT"])
    want = dense.float().to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(res["out"], want)


# ------------------------------------------------------------------ the generator

def test_splitmix64_known_answers():
    """SplitMix64 seeded with 0: its first outputs are published test values."""
    w = gen.raw_u64(0, 0, 2)
    assert [int(v) for v in w] == [0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4]


def test_generator_reproducible_and_distinct():
    a = gen.bf16_normal(0, "h", (64, 64), 1.0)
    b = gen.bf16_normal(0, "h", (64, 64), 1.0)
    c = gen.bf16_normal(0, "W1", (64, 64), 1.0)
    assert np.array_equal(a, b) and not np.array_equal(a, c)
    z = ora.bf16_to_f64(gen.bf16_normal(1, "x", (200000,), 1.0))
    assert abs(z.mean()) < 0.01 and abs(z.std() - 1) < 0.01
    cs = gen.channel_keep_set(0, "chan", 100, 37)
    assert len(np.unique(cs)) == 37 and np.all(np.diff(cs) > 0) and cs.max() < 100
    assert gen.keep_count(0.4, 729) == 292 and gen.keep_count(0.3, 3840) == 1152
    assert gen.keep_count(0.75, 8960) == 6720


# ------------------------------------------------------------------ planted mistakes

def _all_pin_failures():
    f = _hand_checks() + _select_golden_checks() + _brute_force_checks(n_cases=150)
    try:
        test_score_matches_torch_library()
        test_ffn_dense_matches_torch_swiglu()
        test_block_full_keep_equals_dense_block()
        test_block_invariants()
        test_sigmoid_values()
        test_ffn_bf16_activation_matches_torch()
    except AssertionError as e:
        f.append(str(e))
    return f


def _tanh_gelu(x):
    return 0.5 * x * (1 + np.tanh(math.sqrt(2 / math.pi) * (x + 0.044715 * x ** 3)))


MUTATIONS = {
    "tanh_gelu": ("gelu", lambda orig: _tanh_gelu),
    "relu_for_gelu": ("gelu", lambda orig: (lambda x: np.maximum(x, 0))),
    "drop_expansion": ("score", lambda orig: (lambda h, W1, w2, b1, t, task, *a, **k: orig(h, W1, w2, b1, t, ora.TASK_UND))),
    "ties_to_higher_index": ("select_topk", lambda orig: (
        lambda lg, r0, r1, K: _reverse_ties(orig, lg, r0, r1, K))),
    "down_not_transposed": ("routed_ffn", lambda orig: (
        lambda X, Wg, Wu, WdT, chan, **kw: _ffn_wrong_down(X, Wg, Wu, WdT, chan))),
    "silu_without_gate": ("routed_ffn", lambda orig: (
        lambda X, Wg, Wu, WdT, chan, **kw: _ffn_no_silu(X, Wg, Wu, WdT, chan))),
    "bias_sign": ("mlp_score", lambda orig: (lambda x, W1, w2, bias: orig(x, W1, w2, -bias))),
    "sigmoid_tanh_scale": ("sigmoid", lambda orig: (lambda x: 0.5 * (1 + np.tanh(np.asarray(x, np.float64))))),
    "sigmoid_offset": ("sigmoid", lambda orig: (lambda x: orig(np.asarray(x, np.float64) + 0.01))),
    "act_bf16_truncated": ("round_to_bf16", lambda orig: (
        lambda x: (np.asarray(x, np.float64).astype(np.float32).view(np.uint32) >> np.uint32(16)).astype(np.uint16))),
}


def _reverse_ties(orig, lg, r0, r1, K):
    lg = np.asarray(lg, np.float32)
    idx, mask = orig(lg[:, ::-1].copy(), lg.shape[1] - r1, lg.shape[1] - r0, K)
    N = lg.shape[1]
    return np.sort(N - 1 - idx, axis=1).astype(np.int32), mask[:, ::-1].copy()


def _ffn_wrong_down(X, Wg, Wu, WdT, chan):
    cs = np.asarray(chan, np.int64)
    x = ora.bf16_to_f64(X)
    g = x @ ora.bf16_to_f64(Wg[cs]).T
    u = x @ ora.bf16_to_f64(Wu[cs]).T
    a = g / (1 + np.exp(-g)) * u
    Wd = ora.bf16_to_f64(WdT).T          # treats WdT as W_down [d, I]
    return a @ Wd[cs] if Wd.shape[0] == WdT.shape[0] else a @ Wd[:, cs].T


def _ffn_no_silu(X, Wg, Wu, WdT, chan):
    cs = np.asarray(chan, np.int64)
    x = ora.bf16_to_f64(X)
    return ((x @ ora.bf16_to_f64(Wg[cs]).T) * (x @ ora.bf16_to_f64(Wu[cs]).T)) @ ora.bf16_to_f64(WdT[cs])


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_pins_catch_planted_mistake(name, monkeypatch):
    attr, make = MUTATIONS[name]
    monkeypatch.setattr(ora, attr, make(getattr(ora, attr)))
    assert _all_pin_failures(), f"planted mistake {name} went unnoticed"


def test_pins_pass_unmutated():
    assert _all_pin_failures() == []



# ------------------------------------------------------------------ UCS statistics (Sec. 3.4)

def test_drop_jaccard_and_rda_hand_examples():
    """Eq. 10 / Eq. 11 by hand.  N = 6, routable [1, 5): tokens 0 and 5 are never dropped."""
    m_t = np.array([[1, 0, 0, 1, 1, 1]], np.uint8)     # D_t = {1, 2}
    m_ref = np.array([[0, 0, 1, 0, 1, 0]], np.uint8)   # D_ref = {1, 3} (0 and 5 not routable)
    J, Jr, R, counts = ora.drop_set_stats(m_t, m_ref, 1, 5)
    assert counts[0].tolist() == [2, 2, 1]
    assert J[0] == 1 / 3                      # |{1}| / |{1, 2, 3}|
    assert abs(Jr[0] - 1 / 3) < 1e-15         # E|A&B| = 2*2/4 = 1, E|A|B| = 4 - 1 = 3
    assert abs(R[0]) < 1e-15                  # exactly chance level
    J, Jr, R, _ = ora.drop_set_stats(m_t, m_t, 1, 5)
    assert J[0] == 1.0 and R[0] == 1.0        # identical drop sets
    m_dis = np.array([[1, 1, 1, 0, 0, 1]], np.uint8)   # D = {3, 4}, disjoint from D_t
    J, Jr, R, _ = ora.drop_set_stats(m_t, m_dis, 1, 5)
    assert J[0] == 0.0 and abs(R[0] + 0.5) < 1e-15     # (0 - 1/3) / (1 - 1/3)
    none = np.ones((1, 6), np.uint8)
    J, Jr, R, _ = ora.drop_set_stats(none, none, 1, 5)
    assert J[0] == 1.0 and R[0] == 1.0        # nothing dropped on either side


def test_random_jaccard_reading_pieces_by_brute_force():
    """The J_rand reading is E|A&B| / E|A|B|; both expectations are exact for
    uniformly random subsets of the given sizes (enumerated here)."""
    n = 6
    for a in range(n + 1):
        for b in range(n + 1):
            inter, union, cnt = 0, 0, 0
            for A in itertools.combinations(range(n), a):
                for B in itertools.combinations(range(n), b):
                    sa, sb = set(A), set(B)
                    inter += len(sa & sb)
                    union += len(sa | sb)
                    cnt += 1
            e_i, e_u = inter / cnt, union / cnt
            assert abs(e_i - a * b / n) < 1e-12
            assert abs(e_u - (a + b - a * b / n)) < 1e-12
            want = 1.0 if a + b == 0 else e_i / e_u
            assert abs(ora.expected_random_jaccard(a, b, n) - want) < 1e-12


def test_drop_jaccard_invariants():
    rng = np.random.default_rng(21)
    for _ in range(50):
        N = int(rng.integers(1, 40))
        r0 = int(rng.integers(0, N))
        r1 = int(rng.integers(r0, N + 1))
        a = rng.integers(0, 2, (2, N)).astype(np.uint8)
        b = rng.integers(0, 2, (2, N)).astype(np.uint8)
        J1, _, R1, _ = ora.drop_set_stats(a, b, r0, r1)
        J2, _, R2, _ = ora.drop_set_stats(b, a, r0, r1)
        assert np.array_equal(J1, J2) and np.allclose(R1, R2)      # symmetric
        assert np.all((J1 >= 0) & (J1 <= 1)) and np.all(R1 <= 1 + 1e-12)
        a2 = a.copy()
        a2[:, :r0] ^= 1
        a2[:, r1:] ^= 1
        assert np.array_equal(ora.drop_set_stats(a2, b, r0, r1)[0], J1)   # non-routable tokens ignored


def test_redundancy_gap_hand_example_and_identity():
    """Eq. 7 by hand: cos = [1, 0, 1], R = {1, 2}: g = 2/3 - 1/2 = 1/6."""
    h_in = _bits([[[1, 0], [0, 1], [1, 1]]])
    h_out = _bits([[[1, 0], [1, 0], [1, 1]]])
    g = ora.redundancy_gap(h_in, h_out, np.array([[0, 1, 1]], np.uint8))
    assert abs(g[0] - 1 / 6) < 1e-15
    g = ora.redundancy_gap(h_in, h_in, np.array([[1, 0, 1]], np.uint8))
    assert abs(g[0]) < 1e-15                               # unchanged layer: no gap (fp64 rounding of sqrt 2)
    g = ora.redundancy_gap(h_in, h_out, np.array([[0, 0, 0]], np.uint8))
    assert g[0] == 0.0                                     # empty retained set
    assert ora.cosine(np.zeros(3), np.zeros(3)) == 1.0 and ora.cosine(np.zeros(3), np.ones(3)) == 0.0


def test_cosine_matches_torch_library():
    rng = np.random.default_rng(22)
    a, b = rng.normal(size=(2, 50, 33))
    want = F.cosine_similarity(torch.tensor(a), torch.tensor(b), dim=1).numpy()
    got = np.array([ora.cosine(a[i], b[i]) for i in range(50)])
    assert np.allclose(got, want, rtol=1e-13, atol=1e-14)


def test_ffn_saliency_and_leakage_hand_example():
    """Eq. 8 / Eq. 9 by hand, SiLU arguments only 0 and +-1: rows x = e1, e2;
    z = [[2s, 0, 0], [0, 0, s]] (s = sigma(1)); mean |z| = [s, 0, s/2];
    ||W_down[:, c]|| = [5, 1, 2] -> saliency [5s, 0, s]."""
    s = 0.7310585786300049
    X = _bits([[1, 0], [0, 1]])
    Wg = _bits([[1, 0], [0, 0], [-1, 1]])
    Wu = _bits([[2, 0], [1, 1], [0, 1]])
    WdT = _bits([[3, 4], [1, 0], [0, 2]])
    sal = ora.ffn_saliency(X, Wg, Wu, WdT)
    assert np.allclose(sal, [5 * s, 0.0, s], rtol=0, atol=1e-15)
    assert abs(ora.ffn_leakage(sal, [2]) - 1 / 6) < 1e-15
    assert ora.ffn_leakage(sal, [1]) == 0.0
    assert abs(ora.ffn_leakage(sal, [0, 2]) - 1.0) < 1e-15
    assert ora.ffn_leakage(sal, []) == 0.0


def test_zero_leakage_means_pruned_ffn_equals_full_ffn():
    """If the channels proposed for removal carry no saliency (Eq. 9 gives 0),
    removing them leaves the FFN output on the retained rows unchanged."""
    rng = np.random.default_rng(23)
    M, d, I = 6, 16, 12
    X = gen.f32_to_bf16_bits(rng.normal(0, 1, (M, d)).astype(np.float32))
    Wg, Wu, WdT = (gen.f32_to_bf16_bits(rng.normal(0, .3, (I, d)).astype(np.float32)) for _ in range(3))
    P = np.array([1, 4, 7])
    WdT[P] = 0                                    # ||W_down[:, c]|| = 0 for c in P
    sal = ora.ffn_saliency(X, Wg, Wu, WdT)
    assert ora.ffn_leakage(sal, P) == 0.0
    keep = np.setdiff1d(np.arange(I), P).astype(np.int32)
    assert np.allclose(ora.routed_ffn(X, Wg, Wu, WdT, keep), ora.routed_ffn(X, Wg, Wu, WdT, np.arange(I)),
                       rtol=1e-13, atol=1e-13)
    # and scaling a down-projection row by 2 scales that channel's saliency by 2
    W2 = WdT.copy()
    W2[0] = gen.f32_to_bf16_bits(ora.bf16_to_f64(WdT[0]).astype(np.float32) * 2)
    assert abs(ora.ffn_saliency(X, Wg, Wu, W2)[0] - 2 * sal[0]) < 1e-12 * max(1, sal[0])


# ------------------------------------------------------------------ attention on the packed sequence (Sec. 3.4)

def _rope_checks():
    f = []
    # dh = 4: the rotate-half pairs are (0, 2) and (1, 3); theta_0 = 1, theta_1 = base^(-1/2).
    x = np.zeros((1, 1, 4))
    x[0, 0, 0] = 1.0
    y = ora.rope(x, np.array([1]), 1e6)
    if not np.allclose(y[0, 0], [math.cos(1), 0, math.sin(1), 0], atol=1e-15):
        f.append(f"rope pair (0, 2): {y[0, 0]}")
    x = np.zeros((1, 1, 4))
    x[0, 0, 1] = 1.0
    y = ora.rope(x, np.array([2]), 100.0)          # theta_1 = 0.1, angle 0.2
    if not np.allclose(y[0, 0], [0, math.cos(0.2), 0, math.sin(0.2)], atol=1e-15):
        f.append(f"rope pair (1, 3): {y[0, 0]}")
    rng = np.random.default_rng(3)
    z = rng.normal(size=(5, 3, 16))
    if not np.array_equal(ora.rope(z, np.zeros(5), 1e6), z):
        f.append("rope at position 0 is not the identity")
    r = ora.rope(z, np.array([0, 7, 300, 4095, 16383]), 1e6)
    n_in = np.hypot(z[..., :8], z[..., 8:])
    n_out = np.hypot(r[..., :8], r[..., 8:])
    if not np.allclose(n_in, n_out, rtol=1e-13):
        f.append("rope changes the norm of a rotated pair")
    # Relative position: <rope(q, p + s), rope(k, p' + s)> does not depend on s.
    q, k = rng.normal(size=(1, 1, 128)), rng.normal(size=(1, 1, 128))
    dots = [float(np.sum(ora.rope(q, [10 + s], 1e6) * ora.rope(k, [3 + s], 1e6))) for s in (0, 1, 977, 12000)]
    if max(dots) - min(dots) > 1e-9 * max(1.0, abs(dots[0])):
        f.append(f"rope dot products depend on the absolute position: {dots}")
    return f


def _attention_checks():
    f = []
    e = math.e
    Q = np.array([[[1.0, 0.0]], [[0.0, 1.0]]])     # L = 2, one head, dh = 2
    V = np.array([[[1.0, 2.0]], [[3.0, 4.0]]])
    O = ora.packed_attention(Q, Q.copy(), V, causal=False, scale=1.0)
    want = np.array([[(e + 3) / (e + 1), (2 * e + 4) / (e + 1)], [(1 + 3 * e) / (e + 1), (2 + 4 * e) / (e + 1)]])
    if not np.allclose(O[:, 0], want, atol=1e-15):
        f.append(f"attention hand example (full): {O[:, 0]}")
    Oc = ora.packed_attention(Q, Q.copy(), V, causal=True, scale=1.0)
    if not (np.array_equal(Oc[0, 0], [1.0, 2.0]) and np.allclose(Oc[1, 0], want[1], atol=1e-15)):
        f.append(f"attention hand example (causal): {Oc[:, 0]}")
    # Equal scores (Q = 0): prefix means of V (causal), the mean of V (full);
    # query head h reads key/value head h // 2 (4 query heads, 2 kv heads).
    rng = np.random.default_rng(4)
    V = rng.normal(size=(6, 2, 8))
    K = rng.normal(size=(6, 2, 8))
    Q0 = np.zeros((6, 4, 8))
    Oc = ora.packed_attention(Q0, K, V, causal=True)
    Of = ora.packed_attention(Q0, K, V, causal=False)
    for i in range(6):
        for h in range(4):
            if not np.allclose(Oc[i, h], V[: i + 1, h // 2].mean(axis=0), atol=1e-14):
                f.append(f"causal equal-score row {i} head {h}")
            if not np.allclose(Of[i, h], V[:, h // 2].mean(axis=0), atol=1e-14):
                f.append(f"full equal-score row {i} head {h}")
    O1 = ora.packed_attention(rng.normal(size=(1, 3, 8)), K[:1, :1], V[:1, :1], causal=True)
    if not np.allclose(O1, np.repeat(V[:1, :1], 3, axis=1), atol=1e-15):
        f.append("a single key does not return its value")
    # Independent library routine: torch's scaled_dot_product_attention in fp64.
    L, Hq, Hkv, dh = 37, 6, 2, 16
    Q, K, V = rng.normal(size=(L, Hq, dh)), rng.normal(size=(L, Hkv, dh)), rng.normal(size=(L, Hkv, dh))
    for causal in (False, True):
        q = torch.tensor(Q).permute(1, 0, 2)[None]
        k = torch.tensor(K).permute(1, 0, 2).repeat_interleave(Hq // Hkv, dim=0)[None]
        v = torch.tensor(V).permute(1, 0, 2).repeat_interleave(Hq // Hkv, dim=0)[None]
        ref = F.scaled_dot_product_attention(q, k, v, is_causal=causal)[0].permute(1, 0, 2).numpy()
        got = ora.packed_attention(Q, K, V, causal=causal)
        if not np.allclose(got, ref, atol=1e-12):
            f.append(f"attention differs from torch sdpa (causal={causal}): {np.abs(got - ref).max()}")
    return f


def test_rope_pins():
    assert _rope_checks() == []


def test_attention_pins():
    assert _attention_checks() == []


def _attention_strict_causal(orig):
    def f(Q, K, V, causal, scale=None):
        if not causal:
            return orig(Q, K, V, causal, scale)
        L, Hq, dh = Q.shape
        sc = 1.0 / math.sqrt(dh) if scale is None else scale
        O = np.zeros_like(Q)
        for h in range(Hq):
            kh = h // (Hq // K.shape[1])
            S = Q[:, h] @ K[:, kh].T * sc
            S = np.where(np.tril(np.ones((L, L), bool), -1), S, -1e300)   # j < i instead of j <= i
            P = np.exp(S - S.max(axis=1, keepdims=True))
            O[:, h] = (P / P.sum(axis=1, keepdims=True)) @ V[:, kh]
        return O
    return f


def _attention_gqa_modulo(orig):
    def f(Q, K, V, causal, scale=None):
        Hq, Hkv = Q.shape[1], K.shape[1]
        perm = [h % Hkv for h in range(Hq)]          # h % Hkv instead of h // (Hq / Hkv)
        Kx, Vx = K[:, perm], V[:, perm]
        return orig(Q, Kx, Vx, causal, scale)
    return f


def _rope_adjacent_pairs(orig):
    def f(x, pos, base):
        T, H, dh = x.shape
        ang = np.outer(np.asarray(pos, np.float64), ora.rope_frequencies(dh, base))
        c, s = np.cos(ang)[:, None, :], np.sin(ang)[:, None, :]
        ev, od = x[..., 0::2], x[..., 1::2]
        y = np.empty_like(x)
        y[..., 0::2] = ev * c - od * s
        y[..., 1::2] = od * c + ev * s
        return y
    return f


ATTENTION_MUTATIONS = {
    "causal_excludes_self": ("packed_attention", _attention_strict_causal),
    "gqa_modulo_heads": ("packed_attention", _attention_gqa_modulo),
    "no_score_scale": ("packed_attention", lambda orig: (lambda Q, K, V, causal, scale=None: orig(Q, K, V, causal, 1.0))),
    "rope_adjacent_pairs": ("rope", _rope_adjacent_pairs),
    "rope_sign": ("rope", lambda orig: (lambda x, pos, base: orig(x, -np.asarray(pos, np.float64), base))),
}


@pytest.mark.parametrize("name", sorted(ATTENTION_MUTATIONS))
def test_attention_pins_catch_planted_mistake(name, monkeypatch):
    attr, make = ATTENTION_MUTATIONS[name]
    monkeypatch.setattr(ora, attr, make(getattr(ora, attr)))
    assert _rope_checks() + _attention_checks(), f"planted mistake {name} went unnoticed"


def test_routed_attention_composition():
    """The sublayer against torch as a second opinion (projections, rotary
    embedding from its closed form, sdpa with grouped heads), a zero output
    projection leaving h bit-identical, and dropped rows bypassing."""
    rng = np.random.default_rng(8)
    B, N, d, Hq, Hkv = 2, 40, 64, 4, 2
    h = _bits(np.round(rng.normal(size=(B, N, d)) * 8) / 8 + 0.0)   # + 0.0: no negative zeros (-0 + 0 = +0)
    idx = np.stack([np.sort(rng.choice(N, 13, replace=False)) for _ in range(B)]).astype(np.int32)
    WqkvT = gen.bf16_normal(3, "wqkv", (d, (Hq + 2 * Hkv) * 128), d ** -.5)
    WoT = gen.bf16_normal(3, "wo", (Hq * 128, d), (Hq * 128) ** -.5)
    for causal in (True, False):
        res = ora.routed_attention(h, idx, WqkvT, WoT, Hq, Hkv, causal, 1e6)
        X = torch.tensor(ora.bf16_to_f64(ora.gather(h, idx)))
        qkv = X @ torch.tensor(ora.bf16_to_f64(WqkvT))
        T = qkv.shape[0]
        q = qkv[:, : Hq * 128].reshape(T, Hq, 128)
        k = qkv[:, Hq * 128: (Hq + Hkv) * 128].reshape(T, Hkv, 128)
        v = qkv[:, (Hq + Hkv) * 128:].reshape(T, Hkv, 128)
        pos = torch.tensor(idx.reshape(-1), dtype=torch.float64)
        inv = 1e6 ** (-torch.arange(0, 128, 2, dtype=torch.float64) / 128)
        ang = pos[:, None] * inv[None]
        cos, sin = torch.cos(ang).repeat(1, 2)[:, None], torch.sin(ang).repeat(1, 2)[:, None]

        def rot(x):
            return x * cos + torch.cat([-x[..., 64:], x[..., :64]], dim=-1) * sin
        q, k = rot(q), rot(k)
        outs = []
        for b in range(B):
            s = slice(b * 13, (b + 1) * 13)
            qq = q[s].permute(1, 0, 2)[None]
            kk = k[s].permute(1, 0, 2).repeat_interleave(Hq // Hkv, dim=0)[None]
            vv = v[s].permute(1, 0, 2).repeat_interleave(Hq // Hkv, dim=0)[None]
            outs.append(F.scaled_dot_product_attention(qq, kk, vv, is_causal=causal)[0].permute(1, 0, 2).reshape(13, -1))
        Y = torch.cat(outs) @ torch.tensor(ora.bf16_to_f64(WoT))
        assert np.allclose(res["Y"], Y.numpy(), atol=1e-10), np.abs(res["Y"] - Y.numpy()).max()
    zero = ora.routed_attention(h, idx, WqkvT, np.zeros_like(WoT), Hq, Hkv, True, 1e6)
    assert np.array_equal(zero["out"], h)
    kept = np.zeros((B, N), bool)
    for b in range(B):
        kept[b, idx[b]] = True
    assert np.array_equal(res["out"][~kept], h[~kept])
