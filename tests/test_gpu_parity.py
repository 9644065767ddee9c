"""GPU parity: every C-ABI entry point against the CPU oracle on the same seeded
inputs.  Bars: keep lists and masks bit-exact given the same fp32 logits;
gather and scatter bit-exact; logits within 1e-4 relative to max(|l|, RMS(l));
FFN and block outputs (bf16) within 2e-2 x RMS of the oracle's unrounded fp64
output plus half a bf16 ulp for the final rounding."""
import zlib

import numpy as np
import pytest
import torch

from oracle import cer_oracle as ora
from paper_2608_29291_gb300 import cer
from paper_2608_29291_gb300 import inputs as gen
from tests.gpu_helpers import (bf16_dev, bits_host, f32_dev, ffn_out_ok, i32_dev, out_err_ok, rms, score_bar,
                               score_err, scorers)

pytestmark = pytest.mark.gpu

OUT_TOL = 2e-2


@pytest.fixture(scope="module", autouse=True)
def _device():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    cer.load()
    yield
    cer.cer_sync_status()


def test_device_is_sm103():
    assert torch.cuda.get_device_capability() == (10, 3)


# ------------------------------------------------------------------ S2 select

def _logit_cases():
    rng = np.random.default_rng(11)
    cases = []
    ties = np.array([0.0, -0.0, 1.5, -2.0, -np.inf], np.float32)
    cases.append(("n1_k0", np.array([[0.3]], np.float32), 0, 1, 0))
    cases.append(("n1_k1", np.array([[0.3]], np.float32), 0, 1, 1))
    v = np.array([[0.0, -0.0, 0.0, -1.0, -np.inf, 3.0]], np.float32)
    for r0, r1, K in [(0, 6, 0), (0, 6, 1), (0, 6, 3), (0, 6, 5), (0, 6, 6), (1, 5, 2), (2, 4, 1), (3, 3, 0)]:
        cases.append((f"golden_{r0}_{r1}_{K}", v, r0, r1, K))
    cases.append(("heavy_ties", ties[rng.integers(0, 5, (3, 1000))], 17, 990, 411))
    cases.append(("all_equal", np.full((2, 1000), 0.25, np.float32), 0, 1000, 300))
    n16 = rng.normal(0, 1, (1, 16384)).astype(np.float32)
    for K in (0, 1, 1638, 8192, 16383, 16384):
        cases.append((f"n16384_k{K}", n16, 0, 16384, K))
    cases.append(("n49152_max", rng.normal(0, 2, (1, 49152)).astype(np.float32), 0, 49152, 12345))
    cases.append(("gen_layout", rng.normal(0, 1, (8, 1088)).astype(np.float32), 64, 1088, 512))
    cases.append(("und_layout", rng.normal(0, 1, (4, 1024)).astype(np.float32), 0, 729, 292))
    q = np.round(rng.normal(0, 1, (4, 3000)) * 4).astype(np.float32) / 4      # quantised: many ties
    cases.append(("quantised", q, 100, 2900, 1399))
    return cases


@pytest.mark.parametrize("case", _logit_cases(), ids=lambda c: c[0])
def test_select_topk_bit_exact(case):
    _, logits, r0, r1, K = case
    B, N = logits.shape
    k_tot = K + N - (r1 - r0)
    lg = f32_dev(logits)
    idx = torch.full((B, k_tot), -1, dtype=torch.int32, device="cuda")
    mask = torch.full((B, N), 7, dtype=torch.uint8, device="cuda")
    cer.cer_select_topk(lg, r0, r1, K, idx, mask)
    cer.cer_sync_status()
    want_idx, want_mask = ora.select_topk(logits, r0, r1, K)
    assert np.array_equal(idx.cpu().numpy(), want_idx)
    assert np.array_equal(mask.cpu().numpy(), want_mask)


def test_select_nan_reports_status_then_clears():
    lg = f32_dev(np.array([[0.1, np.nan, 0.3, 0.2]], np.float32))
    idx = torch.empty((1, 2), dtype=torch.int32, device="cuda")
    cer.cer_select_topk(lg, 0, 4, 2, idx)
    with pytest.raises(cer.CerError) as e:
        cer.cer_sync_status()
    assert e.value.status == 5
    cer.cer_sync_status()   # cleared
    # a NaN outside the routable range is not an error
    cer.cer_select_topk(lg, 2, 4, 1, torch.empty((1, 3), dtype=torch.int32, device="cuda"))
    cer.cer_sync_status()


# ------------------------------------------------------------------ S3 / S5 rows

def _rows_case(B, N, d, K, seed):
    rng = np.random.default_rng(seed)
    h = gen.f32_to_bf16_bits(rng.normal(0, 1, (B, N, d)).astype(np.float32))
    idx, _ = ora.select_topk(rng.normal(0, 1, (B, N)).astype(np.float32), 0, N, K)
    Y = gen.f32_to_bf16_bits(rng.normal(0, 1, (B * K, d)).astype(np.float32))
    return h, idx, Y


@pytest.mark.parametrize("B,N,d,K", [(1, 1, 8, 1), (3, 100, 264, 37), (2, 4096, 3584, 1229), (4, 1024, 1536, 0)])
def test_gather_bit_exact(B, N, d, K):
    h, idx, _ = _rows_case(B, N, d, K, 1)
    X = torch.zeros((B * K, d), dtype=torch.bfloat16, device="cuda")
    cer.cer_gather(bf16_dev(h), i32_dev(idx), X)
    cer.cer_sync_status()
    assert np.array_equal(bits_host(X), ora.gather(h, idx))


@pytest.mark.parametrize("B,N,d,K", [(1, 1, 8, 1), (3, 100, 264, 37), (2, 4096, 3584, 1229)])
def test_scatter_add_bit_exact(B, N, d, K):
    h, idx, Y = _rows_case(B, N, d, K, 2)
    hd = bf16_dev(h)
    cer.cer_scatter_add(hd, i32_dev(idx), bf16_dev(Y))
    cer.cer_sync_status()
    want = ora.scatter_add(h, idx, ora.bf16_to_f64(Y))
    assert np.array_equal(bits_host(hd), want)


def test_out_of_range_index_is_reported_not_followed():
    h, idx, _ = _rows_case(1, 50, 64, 10, 3)
    idx = idx.copy()
    idx[0, 4] = 50 + 7
    X = torch.zeros((10, 64), dtype=torch.bfloat16, device="cuda")
    cer.cer_gather(bf16_dev(h), i32_dev(idx), X)
    with pytest.raises(cer.CerError) as e:
        cer.cer_sync_status()
    assert e.value.status == 10
    got = bits_host(X)
    good = [j for j in range(10) if j != 4]
    assert np.array_equal(got[good], h[0, idx[0, good]])
    assert not got[4].any()


# ------------------------------------------------------------------ S1 score

def _score_case(name):
    rng = np.random.default_rng(zlib.crc32(name.encode()))

    def bf(shape, s):
        return gen.f32_to_bf16_bits(rng.normal(0, s, shape).astype(np.float32))
    if name == "tiny":
        w = gen.tiny()
        inp = gen.make_inputs(w)
        return inp, w.task
    if name == "und_ragged_bias":
        B, N, d, Hc = 3, 300, 512, 256
        inp = dict(h=bf((B, N, d), 1), W1=bf((Hc, d), d ** -.5), w2=rng.normal(0, Hc ** -.5, Hc).astype(np.float32),
                   b1=rng.normal(0, .1, Hc).astype(np.float32), t=np.zeros(B, np.float32))
        return inp, 0
    if name == "und_odd_d":
        # d / 64 odd: the last ring slot of two K blocks is half past the contraction
        B, N, d, Hc = 2, 200, 320, 128
        inp = dict(h=bf((B, N, d), 1), W1=bf((Hc, d), d ** -.5), w2=rng.normal(0, Hc ** -.5, Hc).astype(np.float32),
                   b1=rng.normal(0, .1, Hc).astype(np.float32), t=np.zeros(B, np.float32))
        return inp, 0
    if name in ("gen_segments", "gen_segments_noU"):
        B, N, d, Hc, He, E, S = 4, 130, 384, 192, 128, 32, 4
        inp = dict(h=bf((B, N, d), 1), W1=bf((Hc, d), d ** -.5), w2=rng.normal(0, Hc ** -.5, Hc).astype(np.float32),
                   b1=None, W1e=bf((S, He, d), d ** -.5), w2e=rng.normal(0, He ** -.5, (S, He)).astype(np.float32),
                   Ue=bf((S, He, E), E ** -.5) if name == "gen_segments" else None,
                   b1e=rng.normal(0, .1, (S, He)).astype(np.float32),
                   t=np.array([0.05, 0.3, 0.6, 0.999], np.float32))
        return inp, 1
    if name in ("gen_wide_ragged", "und_wide_ragged"):
        # 256-wide core and expansion scorers (Hc + He >= 512: the pair-MMA
        # scorer, 256 flattened rows per tile): 2100 rows end in a ragged tile
        # whose last warp straddles the end of h
        gen_ = name.startswith("gen")
        B, N, d, Hc, He, E = 3, 700, 1024, 512 if not gen_ else 256, 256, 64
        inp = dict(h=bf((B, N, d), 1), W1=bf((Hc, d), d ** -.5), w2=rng.normal(0, Hc ** -.5, Hc).astype(np.float32),
                   b1=rng.normal(0, .1, Hc).astype(np.float32), t=np.array([0.1, 0.5, 0.9], np.float32))
        if gen_:
            inp.update(W1e=bf((1, He, d), d ** -.5), w2e=rng.normal(0, He ** -.5, (1, He)).astype(np.float32),
                       Ue=bf((1, He, E), E ** -.5), b1e=None)
        return inp, 1 if gen_ else 0
    raise KeyError(name)


def _oracle_logits(inp, task):
    return ora.score(inp["h"], inp["W1"], inp["w2"], inp.get("b1"), inp["t"], task, inp.get("W1e"),
                     inp.get("w2e"), inp.get("Ue"), inp.get("b1e"))


@pytest.mark.parametrize("name", ["tiny", "und_ragged_bias", "und_odd_d", "gen_segments", "gen_segments_noU",
                                  "gen_wide_ragged", "und_wide_ragged"])
def test_score_matches_oracle(name):
    inp, task = _score_case(name)
    B, N, d = inp["h"].shape
    core, exp = scorers(inp)
    logits = torch.empty((B, N), dtype=torch.float32, device="cuda")
    probs = torch.empty((B, N), dtype=torch.float32, device="cuda")
    cer.cer_score(bf16_dev(inp["h"]), core, exp, f32_dev(inp["t"]), task, logits, probs)
    cer.cer_sync_status()
    want = _oracle_logits(inp, task)
    assert score_err(logits.cpu().numpy(), want, d) <= 1.0
    assert np.max(np.abs(probs.cpu().numpy() - ora.sigmoid(want))) <= 1e-5


# ------------------------------------------------------------------ S4 FFN

# Stream-K splits (tiles cut by K block across slots, the owner adding the
# others' partial sums): a last wave at most half full -- the down GEMM of
# (2000, 2560, ...), the gate/up GEMM of (200, 4096, ...); fewer tiles than
# half the slots, each tile over up to four slots -- the down GEMM of
# (129, 1536, ...) and (200, 4096, ...), the gate/up GEMM of (1000, 1792, ...),
# and both GEMMs of (100, 3584, ...) (one-CTA down tiles, ragged rows).
@pytest.mark.parametrize("M,d,I,C,pruned", [(1, 256, 1024, 512, True), (127, 256, 1024, 512, True),
                                            (65, 320, 640, 576, True),
                                            (300, 512, 640, 640, False), (129, 1536, 8960, 6720, True),
                                            (1000, 1792, 1536, 960, True), (2000, 2560, 4096, 4096, False),
                                            (200, 4096, 10240, 10240, False), (100, 3584, 18944, 4736, True)])
def test_routed_ffn_matches_oracle(M, d, I, C, pruned):
    rng = np.random.default_rng(M + d)
    X = gen.f32_to_bf16_bits(rng.normal(0, 1, (M, d)).astype(np.float32))
    Wg, Wu = (gen.bf16_normal(M, n, (I, d), d ** -.5) for n in ("g", "u"))
    WdT = gen.bf16_normal(M, "dn", (I, d), I ** -.5)
    chan = gen.channel_keep_set(M, "c", I, C) if pruned else None
    Y = torch.empty((M, d), dtype=torch.bfloat16, device="cuda")
    cer.cer_routed_ffn(bf16_dev(X), bf16_dev(Wg), bf16_dev(Wu), bf16_dev(WdT), i32_dev(chan), Y)
    cer.cer_sync_status()
    want = ora.routed_ffn(X, Wg, Wu, WdT, chan if pruned else np.arange(I), act_bf16=True)
    ok, excess = ffn_out_ok(ora.bf16_to_f64(bits_host(Y)), want)
    assert ok, excess


# ------------------------------------------------------------------ fused block

_WEIGHTS = {}


def _inputs(w):
    """Inputs of a full-size workload; FFN weights drawn once per (seed, I, d)."""
    key = (w.seed, w.I, w.d)
    if key not in _WEIGHTS:
        _WEIGHTS.clear()
        inp = gen.make_inputs(w)
        _WEIGHTS[key] = (inp["Wg"], inp["Wu"], inp["WdT"])
        return inp
    return gen.make_inputs(w, ffn_weights=_WEIGHTS[key])


def _run_block(w, inp, out_of_place=False, prepacked=True):
    """The fused block on the GPU.  prepacked: kept-channel weight slices made
    once by cer_pack_ffn_weights (chan=None in the block); else the block gets
    the full weights and the channel list."""
    core, exp = scorers(inp)
    h = bf16_dev(inp["h"])
    out = torch.empty_like(h) if out_of_place else None
    logits = torch.empty((w.B, w.N), dtype=torch.float32, device="cuda")
    idx = torch.empty((w.B, w.k_tot), dtype=torch.int32, device="cuda")
    mask = torch.empty((w.B, w.N), dtype=torch.uint8, device="cuda")
    Wg, Wu, WdT = bf16_dev(inp["Wg"]), bf16_dev(inp["Wu"]), bf16_dev(inp["WdT"])
    chan = i32_dev(inp["chan"]) if w.C < w.I else None
    if prepacked and chan is not None:
        Wg, Wu, WdT = cer.pack_ffn_weights(Wg, Wu, WdT, chan)
        chan = None
    cer.cer_routed_block(h, core, exp if w.task == 1 else None, f32_dev(inp["t"]), w.task, w.r0, w.r1, w.K,
                         Wg, Wu, WdT, chan, out=out, logits=logits, idx=idx, mask=mask)
    cer.cer_sync_status()
    res = dict(out=bits_host(out if out_of_place else h), logits=logits.cpu().numpy(), idx=idx.cpu().numpy(),
               mask=mask.cpu().numpy())
    if out_of_place:
        res["h_after"] = bits_host(h)
    return res


def _tile_edge_rows(M, extra, seed):
    """The first and last row of every 128-row tile of the packed rows, plus
    `extra` random rows: a wrong tile of either GEMM shows in its edge rows."""
    edges = {r for t in range(0, M, 128) for r in (t, min(t + 127, M - 1))}
    rng = np.random.default_rng(seed)
    edges |= set(rng.choice(M, min(extra, M), replace=False).tolist())
    return np.array(sorted(edges), dtype=np.int64)


def _check_block(w, inp, res, rows=None):
    """Compare one fused-block run with the oracle; rows: the packed rows to
    check against the oracle FFN (default: every kept row)."""
    h = inp["h"]
    # S1: logits against the oracle's
    want_logits = _oracle_logits(inp, w.task)
    assert score_err(res["logits"], want_logits, w.d) <= 1.0
    # S2: the GPU keep list is exactly the oracle's selection on the GPU's logits ...
    idx_o, mask_o = ora.select_topk(res["logits"], w.r0, w.r1, w.K)
    assert np.array_equal(res["idx"], idx_o)
    assert np.array_equal(res["mask"], mask_o)
    # ... and any difference from the oracle's own selection is a near-tie at the K-th boundary
    idx_ref, _ = ora.select_topk(want_logits, w.r0, w.r1, w.K)
    for b in range(w.B):
        diff = set(idx_ref[b].tolist()) ^ set(res["idx"][b].tolist())
        if diff and w.K > 0:
            routable = want_logits[b, w.r0:w.r1].astype(np.float64)
            kth = np.sort(routable)[::-1][w.K - 1]
            # four times the score bar at the K-th logit (on the scale of the whole score array)
            allow = 4 * float(score_bar(np.append(want_logits.reshape(-1), kth), w.d)[-1])
            for i in diff:
                assert abs(float(want_logits[b, i]) - kth) <= allow
    # S5 bypass: dropped rows bit-identical
    dropped = res["mask"] == 0
    assert np.array_equal(res["out"][dropped], h[dropped])
    # S3-S5 kept rows against the oracle FFN evaluated on the GPU's keep list
    if rows is None:
        rows = np.arange(w.M)
    b_of = rows // w.k_tot
    tok = res["idx"].reshape(-1)[rows]
    X = h[b_of, tok]
    y = ora.routed_ffn(X, inp["Wg"], inp["Wu"], inp["WdT"], inp["chan"], act_bf16=True)
    exact = ora.bf16_to_f64(X) + y
    ok, excess = ffn_out_ok(ora.bf16_to_f64(res["out"][b_of, tok]), exact)
    assert ok, excess


def _small(name):
    base = dict(B=2, N=300, d=256, I=1024, C=512, r0=20, r1=290, K=100, Hc=128, He=64, E=64, task=1)
    variants = {
        "ragged_gen": {},
        "und_text_tail": dict(task=0, He=0, E=0, r0=0, r1=200, K=77, B=3),
        "k0": dict(K=0),
        "dense_all_kept": dict(r0=0, r1=300, K=300, C=1024),
        "segments": dict(n_segments=4, B=4, N=130, r0=0, r1=130, K=65),
        "one_token": dict(B=1, N=1, r0=0, r1=1, K=1),
        "d3584": dict(B=1, N=200, d=3584, I=2048, C=1024, r0=0, r1=200, K=60),
        # 256-wide scorers (whole 256-column hidden chunks) with ragged row tiles.
        "wide_scorer_gen": dict(B=3, N=700, d=1024, Hc=256, He=256, r0=50, r1=700, K=200),
        "wide_scorer_und": dict(task=0, He=0, E=0, Hc=256, B=2, N=1000, d=512, r0=0, r1=900, K=300),
    }
    kw = dict(base)
    kw.update(variants[name])
    return gen.Workload(name=name, **kw)


@pytest.mark.parametrize("name", ["ragged_gen", "und_text_tail", "k0", "dense_all_kept", "segments", "one_token",
                                  "d3584", "wide_scorer_gen", "wide_scorer_und"])
@pytest.mark.parametrize("prepacked", [True, False], ids=["packed", "chan"])
def test_routed_block_small(name, prepacked):
    w = _small(name)
    inp = gen.make_inputs(w)
    res = _run_block(w, inp, prepacked=prepacked)
    _check_block(w, inp, res)


def test_pack_ffn_weights_bit_exact():
    I, d, C = 1000, 264, 333
    Wg, Wu, WdT = (gen.bf16_normal(5, n, (I, d), 0.1) for n in ("g", "u", "d"))
    chan = gen.channel_keep_set(5, "c", I, C)
    outs = cer.pack_ffn_weights(bf16_dev(Wg), bf16_dev(Wu), bf16_dev(WdT), i32_dev(chan))
    cer.cer_sync_status()
    for W, o in zip((Wg, Wu, WdT), outs):
        assert np.array_equal(bits_host(o), W[chan])


def test_routed_block_tiny_config_full_compare():
    w = gen.tiny()
    inp = gen.make_inputs(w)
    res = _run_block(w, inp)
    _check_block(w, inp, res)
    full = ora.routed_block(inp["h"], inp["W1"], inp["w2"], None, inp["t"], w.task, w.r0, w.r1, w.K, inp["Wg"],
                            inp["Wu"], inp["WdT"], inp["chan"], inp["W1e"], inp["w2e"], inp["Ue"], None)
    if np.array_equal(full["idx"], res["idx"]):
        exact = ora.bf16_to_f64(inp["h"]).copy()
        kept = full["idx"][0]
        exact[0, kept] += full["Y"]
        ok, excess = out_err_ok(ora.bf16_to_f64(res["out"]), exact, OUT_TOL)
        assert ok, excess


def test_routed_block_out_of_place_leaves_h():
    w = _small("ragged_gen")
    inp = gen.make_inputs(w)
    res = _run_block(w, inp, out_of_place=True)
    assert np.array_equal(res["h_after"], inp["h"])
    _check_block(w, inp, res)


def test_stage_events_are_recorded():
    w = _small("ragged_gen")
    inp = gen.make_inputs(w)
    core, exp = scorers(inp)
    h = bf16_dev(inp["h"])
    evs = [torch.cuda.Event(enable_timing=True) for _ in range(6)]
    cer.cer_routed_block(h, core, exp, f32_dev(inp["t"]), 1, w.r0, w.r1, w.K, bf16_dev(inp["Wg"]),
                         bf16_dev(inp["Wu"]), bf16_dev(inp["WdT"]), i32_dev(inp["chan"]), stage_events=evs)
    cer.cer_sync_status()
    times = [evs[i].elapsed_time(evs[i + 1]) for i in range(5)]
    assert all(t >= 0 for t in times) and sum(times) > 0


@pytest.mark.parametrize("wname", ["und_1p5b", "gen_1p5b", "long_7b"])
def test_routed_block_full_size_every_row(wname):
    """The three full-size configs: every logit, the whole keep list and mask,
    every dropped row and every kept row of the output."""
    w = gen.WORKLOADS[wname]()
    inp = _inputs(w)
    res = _run_block(w, inp)
    _check_block(w, inp, res)


# Points of the 7B sweep (B = 1, d = 3584, I = 18944, generation): together
# they take every N, token keep ratio and FFN keep ratio of the grid at least
# once.  (1024, 0.1, 0.25) is M = 102, both GEMMs split over up to four SM
# pairs each (stream-K); (16384, 0.9, 1.0) is the largest point.
SWEEP_PARITY = [(1024, 0.1, 0.25), (2048, 0.3, 0.5), (4096, 0.5, 1.0), (8192, 0.7, 0.5), (16384, 0.9, 0.25),
                (16384, 0.9, 1.0)]


@pytest.mark.parametrize("n,tr,fr", SWEEP_PARITY)
def test_routed_block_sweep_points(n, tr, fr):
    """Every logit, keep-list entry and dropped row; the kept rows in full up
    to M * C = 6e7 (the oracle FFN in fp64 then takes seconds), beyond that
    every 128-row tile's first and last row plus 256 random rows."""
    w = gen.sweep(n, tr, fr)
    inp = _inputs(w)
    res = _run_block(w, inp)
    rows = None if w.M * w.C <= 60_000_000 else _tile_edge_rows(w.M, 256, seed=2)
    _check_block(w, inp, res, rows)
