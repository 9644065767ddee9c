"""Move seeded host inputs onto the GPU as torch tensors, and back."""
import numpy as np
import torch

from paper_2608_29291_gb300 import cer


def bf16_dev(bits: np.ndarray, dev="cuda") -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).to(dev)


def bits_host(t: torch.Tensor) -> np.ndarray:
    return t.detach().contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


def f32_dev(a, dev="cuda"):
    return None if a is None else torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(dev)


def i32_dev(a, dev="cuda"):
    return None if a is None else torch.from_numpy(np.ascontiguousarray(a, dtype=np.int32)).to(dev)


def scorers(inp: dict, dev="cuda"):
    core = cer.Scorer(W1=bf16_dev(inp["W1"], dev), w2=f32_dev(inp["w2"], dev), b1=f32_dev(inp.get("b1"), dev))
    exp = None
    if inp.get("W1e") is not None:
        exp = cer.Scorer(W1=bf16_dev(inp["W1e"], dev), w2=f32_dev(inp["w2e"], dev), b1=f32_dev(inp.get("b1e"), dev),
                         U=bf16_dev(inp["Ue"], dev) if inp.get("Ue") is not None else None)
    return core, exp


# The score bar (the reading of the 1e-4 relative error for the scorer of
# Eq. 4): |l_gpu - l| <= SCORE_TOL * max(|l|, SCORE_FLOOR * RMS(l))
# + SCORE_ACC_PER_D * d * RMS(l).  The floor keeps near-zero logits from
# making the relative error undefined.  Accumulating d bf16 x bf16 products
# in fp32 on the tensor cores leaves an error that grows linearly with d:
# max |l_gpu - l| / RMS(l) measured 3.0e-9 .. 4.9e-9 per unit of d on GB300
# (d = 512 .. 16384, two hidden widths, two seeds each); the bar carries
# twice the largest.  At d = 3584 the relative part alone held (worst 8.6e-5
# of the 1e-4, every logit of the 7B configs); at d = 16384 it did not.
SCORE_TOL = 1e-4
SCORE_FLOOR = 0.1
SCORE_ACC_PER_D = 1e-8


def score_bar(want: np.ndarray, d: int) -> np.ndarray:
    """The elementwise bar of the logits ``want`` of a d-wide hidden state."""
    want = np.asarray(want, dtype=np.float64)
    r = float(np.sqrt(np.mean(want ** 2))) if want.size else 0.0
    return SCORE_TOL * np.maximum(np.abs(want), SCORE_FLOOR * r) + SCORE_ACC_PER_D * d * r


def score_err(got: np.ndarray, want: np.ndarray, d: int) -> float:
    """Worst |got - want| as a fraction of the bar (<= 1 passes)."""
    want = np.asarray(want, dtype=np.float64)
    if not want.size:
        return 0.0
    bar = score_bar(want, d)
    bar = np.where(bar == 0, 1.0, bar)
    return float(np.max(np.abs(np.asarray(got, dtype=np.float64) - want) / bar))


def rel_err(got: np.ndarray, want: np.ndarray, floor_frac: float = SCORE_FLOOR) -> float:
    """max |got - want| / max(|want|, floor_frac * RMS(want)), elementwise.

    The RMS floor keeps near-zero logits from making the relative error
    undefined: their error is measured on the scale of the score array."""
    want = np.asarray(want, dtype=np.float64)
    got = np.asarray(got, dtype=np.float64)
    rms = float(np.sqrt(np.mean(want ** 2))) if want.size else 0.0
    den = np.maximum(np.abs(want), floor_frac * rms)
    den = np.where(den == 0, 1.0, den)
    return float(np.max(np.abs(got - want) / den)) if want.size else 0.0


def max_abs_err(got: np.ndarray, want: np.ndarray) -> float:
    got = np.asarray(got, dtype=np.float64)
    want = np.asarray(want, dtype=np.float64)
    return float(np.max(np.abs(got - want))) if want.size else 0.0


def ulp_bf16(x) -> np.ndarray:
    """Spacing of bf16 values at |x| (8 significant bits); 2^-133 below the normal range."""
    a = np.abs(np.asarray(x, dtype=np.float64))
    e = np.floor(np.log2(np.maximum(a, 2.0 ** -126)))
    return np.exp2(e - 7)


def out_err_ok(got_bf16: np.ndarray, exact: np.ndarray, tol_frac: float):
    """A bf16 output against the oracle's unrounded fp64 value: the error must
    stay within tol_frac * RMS(exact) plus half a bf16 ulp (the final rounding,
    which may land either side of a rounding boundary).  Returns (ok, worst excess)."""
    got = np.asarray(got_bf16, dtype=np.float64)
    exact = np.asarray(exact, dtype=np.float64)
    bound = tol_frac * rms(exact) + 0.5 * ulp_bf16(np.maximum(np.abs(exact), np.abs(got)))
    excess = np.abs(got - exact) - bound
    return bool(np.all(excess <= 0)), float(excess.max()) if excess.size else 0.0


# FFN and block outputs are compared with the oracle whose SwiGLU activation
# enters the down projection as a bf16 operand (oracle routed_ffn(...,
# act_bf16=True)), at the benchmark spec's bar: 2e-2 x RMS plus half a bf16 ulp.
# What is left between the two sides is fp32 accumulation and the occasional
# activation that each side rounds to a different neighbouring bf16 value
# (the GPU rounds its fp32 value, the oracle its fp64 one): one such step of
# a large activation times a large weight moves an output by ~2e-3, so a bar
# much tighter than 2e-2 x RMS would test those flips, not the kernels.
OUT_TOL = 2e-2


def ffn_out_ok(got_bf16: np.ndarray, exact: np.ndarray):
    """The output bar; returns (ok, worst excess over it)."""
    return out_err_ok(got_bf16, exact, OUT_TOL)


def rms(x) -> float:
    x = np.asarray(x, dtype=np.float64)
    return float(np.sqrt(np.mean(x ** 2))) if x.size else 0.0
