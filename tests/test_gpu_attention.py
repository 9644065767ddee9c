"""GPU parity of attention on the packed sequence (Sec. 3.4; Qwen2.5 rotary
embedding and grouped key/value heads, App. A.5) against the oracle.

Rotary embedding: every rotated value within one bf16 ulp of the oracle's fp64
rotation of the same inputs (the GPU rounds an fp32 rotation to bf16), value
heads bit-identical.  Attention: the oracle runs in fp64 on the same bf16
Q, K, V.  The tolerance follows from the arithmetic: every softmax weight
w_ij is rounded to bf16 (relative error <= 2^-8) before its product with V,
the rest accumulates in fp32, and the output is rounded to bf16, so
|out - exact| <= (2^-8 + 2^-12) * sum_j w_ij |v_j| + half a bf16 ulp, where
sum_j w_ij |v_j| is the oracle's attention applied to |V|."""
import numpy as np
import pytest
import torch

from oracle import cer_oracle as ora
from paper_2608_29291_gb300 import cer
from paper_2608_29291_gb300 import inputs as gen
from tests.gpu_helpers import bf16_dev, bits_host, i32_dev, out_err_ok, ulp_bf16

pytestmark = pytest.mark.gpu
DH = 128
W_REL = 2.0 ** -8 + 2.0 ** -12     # bf16 rounding of a softmax weight, plus fp32 slack


@pytest.fixture(scope="module", autouse=True)
def _device():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    cer.load()


def _qkv(seed, B, L, Hq, Hkv, q_scale=1.0):
    """Seeded packed rows [B*L, (Hq + 2 Hkv) * 128]; the query heads scaled by
    q_scale so the softmax is neither flat nor one-hot."""
    W = (Hq + 2 * Hkv) * DH
    x = ora.bf16_to_f64(gen.bf16_normal(seed, "qkv", (B * L, W), 1.0))
    x[:, : Hq * DH] *= q_scale
    return ora.round_to_bf16(x)


def _split(x, Hq, Hkv):
    T = x.shape[0]
    q = x[:, : Hq * DH].reshape(T, Hq, DH)
    k = x[:, Hq * DH: (Hq + Hkv) * DH].reshape(T, Hkv, DH)
    v = x[:, (Hq + Hkv) * DH:].reshape(T, Hkv, DH)
    return q, k, v


def _positions(seed, B, L, N):
    """An ascending keep list of L tokens out of N per sequence (original positions)."""
    rng = np.random.default_rng(seed)
    return np.stack([np.sort(rng.choice(N, L, replace=False)) for _ in range(B)]).astype(np.int32)


@pytest.mark.parametrize("B,L,Hq,Hkv,N", [(2, 37, 4, 2, 100), (1, 1, 12, 2, 1), (3, 300, 12, 2, 16384),
                                          (2, 128, 28, 4, 4096)])
def test_rope_matches_oracle(B, L, Hq, Hkv, N):
    bits = _qkv(B * 1000 + L, B, L, Hq, Hkv)
    pos = _positions(L + N, B, L, N)
    qkv = bf16_dev(bits)
    cer.cer_rope_packed(qkv, B, L, Hq, Hkv, i32_dev(pos.reshape(-1)), 1e6)
    cer.cer_sync_status()
    got = ora.bf16_to_f64(bits_host(qkv))
    x = ora.bf16_to_f64(bits)
    q, k, v = _split(x, Hq, Hkv)
    p = pos.reshape(-1)
    want = np.concatenate([ora.rope(q, p, 1e6).reshape(B * L, -1), ora.rope(k, p, 1e6).reshape(B * L, -1)], axis=1)
    n_rot = (Hq + Hkv) * DH
    err = np.abs(got[:, :n_rot] - want)
    # One bf16 ulp, plus the fp32 rotation's own error (~2e-7 of the pair's
    # norm) where the rotated value cancels towards zero.
    xr = x[:, :n_rot].reshape(B * L, Hq + Hkv, 2, DH // 2)
    norm = np.sqrt(xr[:, :, 0] ** 2 + xr[:, :, 1] ** 2)
    bound = ulp_bf16(want) + 1e-6 * np.concatenate([norm, norm], axis=2).reshape(B * L, n_rot)
    assert np.all(err <= bound), float(np.max(err / bound))
    assert np.array_equal(bits_host(qkv)[:, n_rot:], bits[:, n_rot:])      # value heads untouched


def test_rope_at_large_positions():
    """Positions up to 2^31 - 1, where an fp32 product of position and
    frequency would have lost the angle entirely."""
    Hq, Hkv = 4, 2
    pos = np.array([[0, 1, 4095, (1 << 24) - 3, (1 << 24) - 1, 1 << 24, (1 << 24) + 5, 123456789, (1 << 30) + 7,
                     (1 << 31) - 1]], dtype=np.int32)
    B, L = pos.shape
    bits = _qkv(77, B, L, Hq, Hkv)
    qkv = bf16_dev(bits)
    cer.cer_rope_packed(qkv, B, L, Hq, Hkv, i32_dev(pos.reshape(-1)), 1e6)
    cer.cer_sync_status()
    got = ora.bf16_to_f64(bits_host(qkv))
    x = ora.bf16_to_f64(bits)
    q, k, v = _split(x, Hq, Hkv)
    p = pos.reshape(-1)
    want = np.concatenate([ora.rope(q, p, 1e6).reshape(B * L, -1), ora.rope(k, p, 1e6).reshape(B * L, -1)], axis=1)
    n_rot = (Hq + Hkv) * DH
    xr = x[:, :n_rot].reshape(B * L, Hq + Hkv, 2, DH // 2)
    norm = np.sqrt(xr[:, :, 0] ** 2 + xr[:, :, 1] ** 2)
    bound = ulp_bf16(want) + 1e-6 * np.concatenate([norm, norm], axis=2).reshape(B * L, n_rot)
    err = np.abs(got[:, :n_rot] - want)
    assert np.all(err <= bound), float(np.max(err / bound))


def test_rope_negative_position_reported():
    bits = _qkv(5, 1, 4, 2, 1)
    qkv = bf16_dev(bits)
    cer.cer_rope_packed(qkv, 1, 4, 2, 1, i32_dev(np.array([0, 3, -1, 7])), 1e6)
    with pytest.raises(cer.CerError) as e:
        cer.cer_sync_status()
    assert e.value.status == 10                                          # CER_ERR_INDEX
    assert np.array_equal(bits_host(qkv)[2], bits[2])                     # that row left as it was


def _attention_ok(got, q, k, v, causal):
    """got [L, Hq, dh] against the oracle on one sequence, within the derived bound."""
    want = ora.packed_attention(q, k, v, causal=causal)
    spread = ora.packed_attention(q, k, np.abs(v), causal=causal)    # sum_j w_ij |v_j|
    bound = W_REL * spread + 0.5 * ulp_bf16(np.maximum(np.abs(got), np.abs(want)))
    err = np.abs(got - want)
    return bool(np.all(err <= bound)), float(np.max(err / bound))


def _check_attention(B, L, Hq, Hkv, causal, seed, sample_heads=None):
    bits = _qkv(seed, B, L, Hq, Hkv, q_scale=2.0)
    qkv = bf16_dev(bits)
    out = cer.cer_packed_attention(qkv, B, L, Hq, Hkv, causal)
    cer.cer_sync_status()
    got = ora.bf16_to_f64(bits_host(out)).reshape(B, L, Hq, DH)
    q, k, v = _split(ora.bf16_to_f64(bits), Hq, Hkv)
    q, k, v = (a.reshape(B, L, -1, DH) for a in (q, k, v))
    heads = list(range(Hq)) if sample_heads is None else list(sample_heads)
    group = Hq // Hkv
    for b in range(B):
        kv = sorted({h // group for h in heads})
        qs = q[b][:, heads]
        ks, vs = k[b][:, kv], v[b][:, kv]
        # the sampled query heads keep their own key/value heads
        remap = [kv.index(h // group) for h in heads]
        ks, vs = ks[:, remap], vs[:, remap]
        ok, worst = _attention_ok(got[b][:, heads], qs, ks, vs, bool(causal))
        assert ok, (b, worst)


@pytest.mark.parametrize("causal", [1, 0], ids=["causal", "full"])
@pytest.mark.parametrize("B,L,Hq,Hkv", [(1, 1, 1, 1), (2, 77, 4, 2), (1, 128, 2, 1), (2, 129, 6, 1),
                                        (3, 300, 12, 2), (1, 587, 7, 1)])
def test_packed_attention_matches_oracle(B, L, Hq, Hkv, causal):
    _check_attention(B, L, Hq, Hkv, causal, seed=B * 7919 + L * 31 + Hq)


def test_packed_attention_full_size_und():
    """und_1p5b: 4 sequences of 587 packed tokens, Qwen2.5-1.5B heads (12 query,
    2 key/value), causal prefill."""
    _check_attention(4, 587, 12, 2, 1, seed=11, sample_heads=[0, 5, 6, 11])


def test_packed_attention_full_size_long_bidirectional():
    """long_7b: 2 sequences of 1408 packed tokens, Qwen2.5-7B heads (28 query,
    4 key/value), bidirectional."""
    _check_attention(2, 1408, 28, 4, 0, seed=12, sample_heads=[0, 13, 27])


def test_rope_then_attention_on_a_keep_list():
    """The composed path: the kept rows of a top-K selection, rotated at their
    original positions, then attention over the packed sequence."""
    B, N, K, Hq, Hkv = 2, 400, 150, 4, 2
    logits = gen.f32_normal(9, "lg", (B, N), 1.0)
    idx, _ = ora.select_topk(logits, 0, N, K)
    L = idx.shape[1]
    bits = _qkv(21, B, L, Hq, Hkv)
    qkv = bf16_dev(bits)
    cer.cer_rope_packed(qkv, B, L, Hq, Hkv, i32_dev(idx.reshape(-1)), 1e6)
    out = cer.cer_packed_attention(qkv, B, L, Hq, Hkv, 1)
    cer.cer_sync_status()
    rot = ora.bf16_to_f64(bits_host(qkv))      # the GPU's rotated (bf16) rows: checked above
    q, k, v = (a.reshape(B, L, -1, DH) for a in _split(rot, Hq, Hkv))
    got = ora.bf16_to_f64(bits_host(out)).reshape(B, L, Hq, DH)
    for b in range(B):
        ok, worst = _attention_ok(got[b], q[b], k[b], v[b], True)
        assert ok, worst


def test_empty_inputs_are_no_ops():
    cer.cer_rope_packed(torch.empty(0, device="cuda", dtype=torch.bfloat16), 0, 5, 2, 1, None, 1e6)
    cer.cer_packed_attention(torch.empty(0, device="cuda", dtype=torch.bfloat16), 3, 0, 2, 1, 1,
                             out=torch.empty(0, device="cuda", dtype=torch.bfloat16))
    cer.cer_sync_status()


# ------------------------------------------------------------------ the attention sublayer

BLOCK_TOL = 2e-2     # the routed block's output tolerance: 2e-2 * RMS + half a bf16 ulp


def _sublayer_inputs(seed, B, N, d, L, Hq, Hkv):
    h = gen.bf16_normal(seed, "h", (B, N, d), 1.0)
    rng = np.random.default_rng(seed)
    idx = np.stack([np.sort(rng.choice(N, L, replace=False)) for _ in range(B)]).astype(np.int32)
    WqkvT = gen.bf16_normal(seed, "wqkv", (d, (Hq + 2 * Hkv) * DH), d ** -0.5)
    WoT = gen.bf16_normal(seed, "wo", (Hq * DH, d), (Hq * DH) ** -0.5)
    return h, idx, WqkvT, WoT


@pytest.mark.parametrize("B,N,d,L,Hq,Hkv,causal,inplace", [
    (2, 300, 256, 100, 4, 2, 1, True), (1, 200, 512, 200, 2, 1, 0, False), (3, 130, 128, 1, 1, 1, 1, True),
    (2, 700, 768, 333, 6, 3, 0, True), (1, 1024, 1536, 587, 12, 2, 1, True)])
def test_routed_attention_matches_oracle(B, N, d, L, Hq, Hkv, causal, inplace):
    h, idx, WqkvT, WoT = _sublayer_inputs(B * 131 + L, B, N, d, L, Hq, Hkv)
    hd = bf16_dev(h)
    out = None if inplace else torch.empty_like(hd)
    qkv = torch.empty((B * L, (Hq + 2 * Hkv) * DH), dtype=torch.bfloat16, device="cuda")
    cer.cer_routed_attention(hd, i32_dev(idx), bf16_dev(WqkvT), bf16_dev(WoT), Hq, Hkv, causal, out=out, qkv=qkv)
    cer.cer_sync_status()
    got = bits_host(hd if inplace else out)
    if not inplace:
        assert np.array_equal(bits_host(hd), h)                           # h untouched
    res = ora.routed_attention(h, idx, WqkvT, WoT, Hq, Hkv, bool(causal), 1e6)
    kept = np.zeros((B, N), bool)
    for b in range(B):
        kept[b, idx[b]] = True
    assert np.array_equal(got[~kept], h[~kept])                           # dropped rows bypass
    exact = ora.bf16_to_f64(h).copy()
    for b in range(B):
        exact[b, idx[b]] += res["Y"][b * L:(b + 1) * L]
    ok, excess = out_err_ok(ora.bf16_to_f64(got[kept]), exact[kept], BLOCK_TOL)
    assert ok, excess
    # the compressed KV cache: the rotated key and value heads of the packed rows
    cache = ora.bf16_to_f64(bits_host(qkv))[:, Hq * DH:].reshape(B * L, 2 * Hkv, DH)
    want = np.concatenate([res["K"], res["V"]], axis=1)
    ok, excess = out_err_ok(cache, want, BLOCK_TOL)
    assert ok, excess
