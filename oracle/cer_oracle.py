"""CPU oracle for CE-Router's token-routed compacted block.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import or run
anything under ``oracle/``.  The CUDA library never calls it and it calls nothing
of the CUDA library: the two share no code.

Plain, slow, obviously correct: numpy in fp64 (the paper fixes no precision),
one step per paper passage, no blocking, fusion or reordering.  Data arrive as
the same bf16 bit patterns (uint16) and fp32 arrays the GPU reads; they are
widened exactly to fp64.  Library primitives used as steps: numpy matmul,
numpy exp/cos/sin/floor, scipy.special.erf, Python's ``sorted``.

Paper passages followed (CE-Router, "Core-Expansion Routing and Unified
Computation Scheduling"):
  * Sec. 3.2, Eq. 4 (core_expansion_formulation): logits l^U = c_l(h),
    l^G = c_l(h) + e_{l,m(t)}(h); core and expansions are token-wise MLPs with a
    scalar output; M segments of the denoising timesteps.
  * Sec. 3.4, Eq. 6 (router_inference_outputs): p = sigmoid(l), R = TopK(p, K);
    App. B.2: the sigmoid is monotonic, so ranking logits gives the same set.
  * Sec. 3.4, task-adaptive token compaction: the kept set R is gathered into
    a compact sequence for the FFN, the dropped set D passes through unchanged.
  * Sec. 3.4 (2) FFN pruning and App. A.4: FFN restricted to the channels kept
    by the static mask; the backbone is Qwen2.5 (App. A.5), a SwiGLU FFN.

Readings where the paper is silent or leaves a choice open:
  * scorer MLP form w2 . GELU(W1 h + b1) with exact-erf GELU; expansion adds
    U . emb(t) before the GELU, emb a sinusoid [cos(1000 t f_j), sin(1000 t f_j)],
    f_j = 10000^(-j/(E/2)), computed in fp64 and rounded to fp32;
  * segment m(t) = min(M-1, floor(t*M)) in fp64 (equal-width progress segments);
  * ranking on fp32 logits, larger first, ties to the lower token index,
    -0.0 equal to +0.0, a NaN among the routable logits is an error;
  * tokens outside the routable range [r0, r1) are always kept; the kept list is
    in ascending token order;
  * FFN without biases or norm, y = W_down[:, Cs] (SiLU(W_gate[Cs] x) * (W_up[Cs] x));
    the update is not scaled by p;
  * block output bf16(h + y) for kept rows: the fp64 sum rounded to fp32, then
    to bf16 (round to nearest even at both steps); dropped rows bit-identical.

UCS statistics (Sec. 3.4, Unified Computation Scheduling):
  * Eq. 8 (ffn_saliency), Eq. 9 (ffn_leakage): channel saliency on the
    retained tokens and the leakage of the pruned channel set;
  * Eq. 7 (redundancy_gap): mean input-output cosine over all tokens minus
    the mean over the retained tokens;
  * Eq. 10 (drop_jaccard), Eq. 11 (rda): Jaccard similarity of two drop sets and
    its random-adjusted form.
  Readings: the drop set D is the routable tokens not kept (tokens outside
  the routable range are never dropped); the expected random Jaccard is the
  ratio of expectations E|A&B| / E|A|B| with E|A&B| = |A||B|/n for uniformly
  random drop sets of the same sizes among the n routable tokens; an empty
  union gives J = 1, J_rand = 1 gives RDA = 1 (identical patterns); the
  retained set R is every kept token; a zero-norm pair has cosine 1 when the
  vectors are equal, else 0; empty R gives g = 0.

Attention on the packed sequence (Sec. 3.4, token compaction: attention runs,
like the FFN, only over the kept tokens gathered into a compact sequence; in
understanding mode their keys and values are the reduced KV cache):
  * rope: rotary position embedding of the Qwen2.5 backbone (App. A.5),
    rotate-half pairing (j, j + dh/2), theta_j = base^(-2j/dh);
  * packed_attention: softmax(Q K^T / sqrt(dh)) V per head over one packed
    sequence, query head h reading key/value head h // (Hq / Hkv).
  Readings: a packed token keeps its original position (its index in the
  full sequence) for the rotary embedding; the keep list is ascending, so a
  causal mask by original position is the causal mask on the packed order;
  understanding (LLM prefill) is causal, generation attends bidirectionally
  among the packed tokens (a flag); a query with no admissible key is not
  possible (every token attends to itself).

Parity status: every function below is pinned by tests/test_oracle_pins.py
(hand-computed example, brute-force top-k, closed forms, library special cases,
invariants).  Agreement with what the paper's authors ran is unpinned: the paper
prints no numerical value of the router, the FFN or the block.
"""
from __future__ import annotations

import math

import numpy as np
from scipy.special import erf

TASK_UND = 0
TASK_GEN = 1


class OracleNaN(ValueError):
    """A routable logit is NaN: no top-K set is defined."""


# ---------------------------------------------------------------- bf16 <-> fp64

def bf16_to_f64(bits: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns (uint16) to fp64."""
    b = np.ascontiguousarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)
    return b.view(np.float32).astype(np.float64)


def round_to_bf16(x: np.ndarray) -> np.ndarray:
    """fp64 -> fp32 (nearest even) -> bf16 (nearest even); returns uint16 bits."""
    f = np.asarray(x, dtype=np.float64).astype(np.float32)
    u = f.view(np.uint32).astype(np.uint64)
    lsb = (u >> np.uint64(16)) & np.uint64(1)
    r = (u + np.uint64(0x7FFF) + lsb) >> np.uint64(16)
    out = r.astype(np.uint16)
    nan = np.isnan(f)
    out[nan] = 0x7FC0
    return out


# ---------------------------------------------------------------- scorer pieces

def gelu(x: np.ndarray) -> np.ndarray:
    """GELU with the exact Gaussian CDF: x * Phi(x) = 0.5 x (1 + erf(x / sqrt 2))."""
    return 0.5 * x * (1.0 + erf(x / math.sqrt(2.0)))


def sinusoidal_embedding(t: float, E: int) -> np.ndarray:
    """E-dim progress embedding of t (reading: cos half then sin half), fp32."""
    half = E // 2
    j = np.arange(half, dtype=np.float64)
    freq = np.power(10000.0, -j / half)
    arg = 1000.0 * float(t) * freq
    return np.concatenate([np.cos(arg), np.sin(arg)]).astype(np.float32)


def segment_index(t: float, n_segments: int) -> int:
    """m(t): the denoising segment holding progress t (Sec. 3.2; equal widths)."""
    return int(min(n_segments - 1, math.floor(float(t) * n_segments)))


def mlp_score(x: np.ndarray, W1: np.ndarray, w2: np.ndarray, bias: np.ndarray) -> np.ndarray:
    """Token-wise MLP with scalar output (Sec. 3.2): w2 . GELU(W1 x + bias), per row of x."""
    a = x @ W1.T + bias[None, :]
    return gelu(a) @ w2


def score(h, W1, w2, b1, t, task, W1e=None, w2e=None, Ue=None, b1e=None) -> np.ndarray:
    """Routing logits of Eq. 4 for every token; returns fp32 [B, N].

    h: bf16 bits [B, N, d].  Core: W1 bf16 [Hc, d], w2 fp32 [Hc], b1 fp32 [Hc] or None.
    Expansion (generation only): W1e bf16 [S, He, d], w2e fp32 [S, He],
    Ue bf16 [S, He, E] or None, b1e fp32 [S, He] or None; segment m(t_b) per sequence.
    """
    B, N, d = h.shape
    hf = bf16_to_f64(h)
    W1f = bf16_to_f64(W1)
    w2f = np.asarray(w2, dtype=np.float64)
    bc = np.zeros(W1.shape[0]) if b1 is None else np.asarray(b1, dtype=np.float64)
    out = np.empty((B, N), dtype=np.float32)
    for b in range(B):
        logit = mlp_score(hf[b], W1f, w2f, bc)                      # l^U = c_l(h)
        if task == TASK_GEN:
            S = W1e.shape[0]
            m = segment_index(t[b], S)
            bias = np.zeros(W1e.shape[1])
            if Ue is not None:
                emb = sinusoidal_embedding(t[b], Ue.shape[2]).astype(np.float64)
                bias = bias + bf16_to_f64(Ue[m]) @ emb
            if b1e is not None:
                bias = bias + np.asarray(b1e[m], dtype=np.float64)
            logit = logit + mlp_score(hf[b], bf16_to_f64(W1e[m]),
                                      np.asarray(w2e[m], dtype=np.float64), bias)
        out[b] = logit.astype(np.float32)                           # l^G = c_l + e_{l,m(t)}
    return out


def sigmoid(x: np.ndarray) -> np.ndarray:
    """Bounded importance p = sigmoid(l) of Eq. 6, in fp64."""
    return 1.0 / (1.0 + np.exp(-np.asarray(x, dtype=np.float64)))


# ---------------------------------------------------------------- selection

def select_topk(logits: np.ndarray, r0: int, r1: int, K: int):
    """Per-sequence keep set R (Eq. 6): the K routable tokens of largest logit
    (ties to the lower index, -0.0 == +0.0) plus every token outside [r0, r1).

    Returns idx int32 [B, k_tot] (ascending token order) and mask uint8 [B, N].
    """
    logits = np.asarray(logits, dtype=np.float32)
    B, N = logits.shape
    if not (0 <= r0 <= r1 <= N) or not (0 <= K <= r1 - r0):
        raise ValueError("bad routable range or K")
    k_tot = K + N - (r1 - r0)
    idx = np.empty((B, k_tot), dtype=np.int32)
    mask = np.zeros((B, N), dtype=np.uint8)
    for b in range(B):
        vals = [float(v) for v in logits[b]]
        if any(math.isnan(vals[i]) for i in range(r0, r1)):
            raise OracleNaN(f"NaN logit in sequence {b}")
        ranked = sorted(range(r0, r1), key=lambda i: (-vals[i], i))
        keep = set(ranked[:K]) | set(range(0, r0)) | set(range(r1, N))
        kept = sorted(keep)
        idx[b] = kept
        mask[b, kept] = 1
    return idx, mask


# ---------------------------------------------------------------- compaction

def gather(h: np.ndarray, idx: np.ndarray) -> np.ndarray:
    """Pack R (Sec. 3.4): X[b * k_tot + j] = h[b, idx[b, j]]; bf16 bits [B*k_tot, d]."""
    B, k_tot = idx.shape
    return np.concatenate([h[b, idx[b]] for b in range(B)], axis=0) if B else \
        np.empty((0, h.shape[2]), dtype=np.uint16)


def routed_ffn(X: np.ndarray, Wg: np.ndarray, Wu: np.ndarray, WdT: np.ndarray,
               chan: np.ndarray, act_bf16: bool = False) -> np.ndarray:
    """SwiGLU FFN on the packed rows restricted to the kept channels Cs; fp64 [M, d].

    y = sum_{c in Cs} WdT[c, :] * SiLU(Wg[c] . x) * (Wu[c] . x), with WdT the
    down projection stored channel-major (row c is W_down[:, c], the vector whose
    norm enters the saliency of Eq. 8).

    act_bf16: the activation a = SiLU(g) * u enters the down projection as a
    bf16 operand (the precision the comparison contract fixes: bf16 operands,
    fp32 accumulation), i.e. rounded to fp32 and then to bf16, both to nearest
    even, before its fp64 contraction with WdT.  Everything else stays fp64.
    """
    cs = np.asarray(chan, dtype=np.int64)
    x = bf16_to_f64(X)
    g = x @ bf16_to_f64(Wg[cs]).T
    u = x @ bf16_to_f64(Wu[cs]).T
    with np.errstate(over="ignore"):
        a = g / (1.0 + np.exp(-g)) * u          # SiLU(g) * u, SiLU(g) = g * sigmoid(g)
    if act_bf16:
        a = bf16_to_f64(round_to_bf16(a))
    return a @ bf16_to_f64(WdT[cs])


def scatter_add(h: np.ndarray, idx: np.ndarray, Y: np.ndarray) -> np.ndarray:
    """Unpack (Sec. 3.4): kept rows become bf16(h + y), dropped rows stay bit-identical."""
    out = h.copy()
    B, k_tot = idx.shape
    for b in range(B):
        rows = Y[b * k_tot:(b + 1) * k_tot]
        out[b, idx[b]] = round_to_bf16(bf16_to_f64(h[b, idx[b]]) + rows)
    return out


def routed_block(h, W1, w2, b1, t, task, r0, r1, K, Wg, Wu, WdT, chan,
                 W1e=None, w2e=None, Ue=None, b1e=None) -> dict:
    """Whole routed block: score -> TopK -> gather -> pruned FFN -> scatter-add."""
    logits = score(h, W1, w2, b1, t, task, W1e, w2e, Ue, b1e)
    idx, mask = select_topk(logits, r0, r1, K)
    X = gather(h, idx)
    Y = routed_ffn(X, Wg, Wu, WdT, chan)
    out = scatter_add(h, idx, Y)
    return {"logits": logits, "idx": idx, "mask": mask, "Y": Y, "out": out}


# ---------------------------------------------------------------- UCS statistics

def drop_set(mask_row: np.ndarray, r0: int, r1: int) -> np.ndarray:
    """D: the routable tokens [r0, r1) that are not kept (bool over [0, N))."""
    d = np.zeros(mask_row.shape[0], dtype=bool)
    d[r0:r1] = np.asarray(mask_row[r0:r1]) == 0
    return d


def drop_jaccard(mask_t, mask_ref, r0, r1):
    """Eq. 10 per sequence: |D_t & D_ref| / |D_t | D_ref|; also returns the counts
    (|D_t|, |D_ref|, |D_t & D_ref|)."""
    mask_t, mask_ref = np.atleast_2d(mask_t), np.atleast_2d(mask_ref)
    B = mask_t.shape[0]
    J = np.empty(B)
    counts = np.empty((B, 3), dtype=np.int64)
    for b in range(B):
        Dt, Dr = drop_set(mask_t[b], r0, r1), drop_set(mask_ref[b], r0, r1)
        inter, union = int(np.sum(Dt & Dr)), int(np.sum(Dt | Dr))
        J[b] = 1.0 if union == 0 else inter / union
        counts[b] = (int(Dt.sum()), int(Dr.sum()), inter)
    return J, counts


def expected_random_jaccard(a: int, b: int, n: int) -> float:
    """J_rand of Eq. 11 (reading): E|A&B| / E|A|B| for uniformly random drop sets
    of sizes a and b among n tokens, E|A&B| = a b / n."""
    if a + b == 0 or n == 0:
        return 1.0
    e = a * b / n
    return e / ((a + b) - e)


def rda(J: float, J_rand: float) -> float:
    """Eq. 11: (J - J_rand) / (1 - J_rand); J_rand = 1 gives 1 (identical patterns)."""
    if J_rand == 1.0:
        return 1.0
    return (J - J_rand) / (1.0 - J_rand)


def drop_set_stats(mask_t, mask_ref, r0, r1):
    """Per sequence (J, J_rand, RDA) in fp64."""
    J, counts = drop_jaccard(mask_t, mask_ref, r0, r1)
    n = r1 - r0
    Jr = np.array([expected_random_jaccard(int(c[0]), int(c[1]), n) for c in counts])
    R = np.array([rda(J[b], Jr[b]) for b in range(len(J))])
    return J, Jr, R, counts


def cosine(a: np.ndarray, b: np.ndarray) -> float:
    na, nb = float(np.sqrt(np.dot(a, a))), float(np.sqrt(np.dot(b, b)))
    if na == 0.0 or nb == 0.0:
        return 1.0 if np.array_equal(a, b) else 0.0
    return float(np.dot(a, b)) / (na * nb)


def redundancy_gap(h_in, h_out, mask):
    """Eq. 7 per sequence: g = mean_all cos(h_in_i, h_out_i) - mean_{i in R} cos(...).

    h_in, h_out: bf16 bits [B, N, d]; mask: uint8 [B, N] (1 = retained)."""
    a, o = bf16_to_f64(h_in), bf16_to_f64(h_out)
    B, N, _ = a.shape
    g = np.empty(B)
    for b in range(B):
        cos = np.array([cosine(a[b, i], o[b, i]) for i in range(N)])
        kept = np.asarray(mask[b]) != 0
        g[b] = 0.0 if not kept.any() else cos.mean() - cos[kept].mean()
    return g


def ffn_saliency(X, Wg, Wu, WdT):
    """Eq. 8 over all I channels: s_c = mean_{i in R} |z_{i,c}| * ||W_down[:, c]||_2,
    z the SwiGLU activation SiLU(Wg x) * (Wu x) of retained row x (rows of X)."""
    x = bf16_to_f64(X)
    g = x @ bf16_to_f64(Wg).T
    u = x @ bf16_to_f64(Wu).T
    with np.errstate(over="ignore"):
        z = g / (1.0 + np.exp(-g)) * u
    col_norm = np.sqrt(np.sum(bf16_to_f64(WdT) ** 2, axis=1))     # ||W_down[:, c]|| = ||WdT[c]||
    return np.abs(z).mean(axis=0) * col_norm


def ffn_leakage(saliency: np.ndarray, pruned) -> float:
    """Eq. 9: the share of the total saliency held by the channels the static
    mask proposes to remove."""
    total = float(np.sum(saliency))
    return float(np.sum(saliency[np.asarray(pruned, dtype=np.int64)])) / total if total > 0 else 0.0


# ---------------------------------------------------------------- attention on the packed sequence

def rope_frequencies(dh: int, base: float) -> np.ndarray:
    """theta_j = base^(-2j/dh), j < dh/2: the rotary frequencies of the Qwen2.5
    backbone (App. A.5)."""
    j = np.arange(dh // 2, dtype=np.float64)
    return float(base) ** (-2.0 * j / dh)


def rope(x: np.ndarray, pos: np.ndarray, base: float) -> np.ndarray:
    """Rotary embedding of x [T, heads, dh] (fp64) at positions pos [T], in the
    rotate-half pairing: for j < dh/2, with a = p theta_j,
    x'[j] = x[j] cos a - x[j + dh/2] sin a,  x'[j + dh/2] = x[j + dh/2] cos a + x[j] sin a.
    Packed tokens keep their original positions (Sec. 3.4 compaction; reading)."""
    T, H, dh = x.shape
    ang = np.outer(np.asarray(pos, dtype=np.float64), rope_frequencies(dh, base))
    c = np.cos(ang)[:, None, :]
    s = np.sin(ang)[:, None, :]
    lo, hi = x[..., : dh // 2], x[..., dh // 2:]
    return np.concatenate([lo * c - hi * s, hi * c + lo * s], axis=-1)


def packed_attention(Q: np.ndarray, K: np.ndarray, V: np.ndarray, causal: bool, scale: float | None = None):
    """Softmax attention over one packed sequence (Sec. 3.4: attention runs on
    the retained tokens only).  Q [L, Hq, dh], K and V [L, Hkv, dh] in fp64;
    query head h uses key/value head h // (Hq // Hkv).  causal: packed token i
    attends to packed tokens j <= i (the packed order is the original order).
    Returns O [L, Hq, dh]."""
    L, Hq, dh = Q.shape
    Hkv = K.shape[1]
    group = Hq // Hkv
    if scale is None:
        scale = 1.0 / math.sqrt(dh)
    O = np.empty((L, Hq, dh), dtype=np.float64)
    allowed = np.tril(np.ones((L, L), dtype=bool)) if causal else np.ones((L, L), dtype=bool)
    for h in range(Hq):
        kh = h // group
        S = (Q[:, h, :] @ K[:, kh, :].T) * scale
        S = np.where(allowed, S, -np.inf)
        S = S - S.max(axis=1, keepdims=True)
        P = np.exp(S)
        P = P / P.sum(axis=1, keepdims=True)
        O[:, h, :] = P @ V[:, kh, :]
    return O


def routed_attention(h, idx, WqkvT, WoT, Hq: int, Hkv: int, causal: bool, base: float) -> dict:
    """Attention sublayer on the packed sequence (Sec. 3.4): pack R, project to
    queries, keys and values (Q | K | V = X WqkvT, the projection stored
    input-major [d, (Hq + 2 Hkv) * 128]), rotate Q and K at the tokens'
    original positions idx, attend within each packed sequence, project back
    (Y = A WoT, WoT [Hq * 128, d]) and scatter-add: kept rows become
    bf16(h + Y), dropped rows bypass.  fp64 throughout, no intermediate
    rounding.  Returns the packed K and V too (the compressed KV cache)."""
    B, k_tot = idx.shape
    X = bf16_to_f64(gather(h, idx))
    QKV = X @ bf16_to_f64(WqkvT)
    T = X.shape[0]
    dh = 128
    Q = QKV[:, : Hq * dh].reshape(T, Hq, dh)
    K = QKV[:, Hq * dh: (Hq + Hkv) * dh].reshape(T, Hkv, dh)
    V = QKV[:, (Hq + Hkv) * dh:].reshape(T, Hkv, dh)
    pos = np.asarray(idx, dtype=np.int64).reshape(-1)
    Q = rope(Q, pos, base)
    K = rope(K, pos, base)
    A = np.empty((T, Hq * dh), dtype=np.float64)
    for b in range(B):
        s = slice(b * k_tot, (b + 1) * k_tot)
        A[s] = packed_attention(Q[s], K[s], V[s], causal).reshape(k_tot, Hq * dh)
    Y = A @ bf16_to_f64(WoT)
    return {"Y": Y, "out": scatter_add(h, idx, Y), "K": K, "V": V, "A": A}
