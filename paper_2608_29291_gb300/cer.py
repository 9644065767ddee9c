"""Python binding of libcer.so (include/cer_api.h): argument marshalling only.

Every function named ``cer_*`` here calls the C entry point of the same name
with the device pointers of torch tensors, the sizes read off their shapes and
the current CUDA stream.  No computation happens in Python; there is no CPU or
PyTorch fallback: if the library is missing or the device is not sm_103 the
call raises.  PyTorch supplies device memory and streams only.
"""
from __future__ import annotations

import ctypes
import dataclasses
import os
from typing import Optional, Sequence

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libcer.so")

TASK_UND = 0
TASK_GEN = 1

STATUS_NAMES = {0: "CER_OK", 1: "CER_ERR_NULL", 2: "CER_ERR_SHAPE", 3: "CER_ERR_ALIGN", 4: "CER_ERR_RANGE",
                5: "CER_ERR_NAN", 6: "CER_ERR_DEVICE", 7: "CER_ERR_TIMEOUT", 8: "CER_ERR_LAUNCH",
                9: "CER_ERR_WORKSPACE", 10: "CER_ERR_INDEX"}

# Every symbol include/cer_api.h declares.
EXPORTS = ("cer_score", "cer_score_workspace_size", "cer_score_static", "cer_select_topk", "cer_gather", "cer_routed_ffn",
           "cer_routed_ffn_workspace_size", "cer_pack_ffn_weights", "cer_scatter_add", "cer_scatter_add_checked", "cer_routed_block",
           "cer_routed_block_workspace_size", "cer_ffn_channel_norms", "cer_routed_ffn_gated",
           "cer_routed_ffn_gated_workspace_size", "cer_routed_block_gated", "cer_routed_block_gated_workspace_size",
           "cer_drop_set_stats", "cer_redundancy_gap",
           "cer_redundancy_gap_workspace_size", "cer_rope_packed", "cer_packed_attention",
           "cer_routed_attention", "cer_routed_attention_workspace_size", "cer_selftest_bounded_wait", "cer_sync_status",
           "cer_get_error", "cer_status_string", "cer_version")


class CerError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"{STATUS_NAMES.get(status, status)}: {message}")
        self.status = status


class CerScorerC(ctypes.Structure):
    _fields_ = [("W1", ctypes.c_void_p), ("b1", ctypes.c_void_p), ("w2", ctypes.c_void_p),
                ("U", ctypes.c_void_p), ("hidden", ctypes.c_int), ("emb_dim", ctypes.c_int),
                ("n_segments", ctypes.c_int)]


_lib = None

_vp, _i, _sz, _f = ctypes.c_void_p, ctypes.c_int, ctypes.c_size_t, ctypes.c_float
_SCP = ctypes.POINTER(CerScorerC)
_SIGS = {
    "cer_score": ([_vp, _i, _i, _i, _SCP, _SCP, _vp, _i, _vp, _vp, _vp, _sz, _vp], _i),
    "cer_score_workspace_size": ([_i, _i, _i, _i, _i], _sz),
    "cer_score_static": ([_vp, _i, _i, _i, _SCP, _SCP, _vp, _i, _vp, _vp, _vp], _i),
    "cer_select_topk": ([_vp, _i, _i, _i, _i, _i, _vp, _vp, _vp], _i),
    "cer_gather": ([_vp, _i, _i, _i, _vp, _i, _vp, _vp], _i),
    "cer_routed_ffn": ([_vp, _i, _i, _vp, _vp, _vp, _i, _vp, _i, _vp, _vp, _sz, _vp], _i),
    "cer_routed_ffn_workspace_size": ([_i, _i, _i, _i], _sz),
    "cer_pack_ffn_weights": ([_vp, _vp, _vp, _i, _i, _vp, _i, _vp, _vp, _vp, _vp], _i),
    "cer_scatter_add": ([_vp, _i, _i, _i, _vp, _i, _vp, _vp], _i),
    "cer_scatter_add_checked": ([_vp, _i, _i, _i, _vp, _i, _vp, _vp], _i),
    "cer_routed_block": ([_vp, _vp, _i, _i, _i, _SCP, _SCP, _vp, _i, _i, _i, _i, _vp, _vp, _vp, _i, _vp, _i,
                          _vp, _vp, _vp, _vp, _sz, _vp, _i, _vp], _i),
    "cer_routed_block_workspace_size": ([_i, _i, _i, _i, _i, _i, _i, _i, _i, _i, _i], _sz),
    "cer_ffn_channel_norms": ([_vp, _i, _i, _vp, _vp], _i),
    "cer_routed_ffn_gated": ([_vp, _i, _i, _vp, _vp, _vp, _i, _i, _vp, _f, _vp, _vp, _vp, _vp, _vp, _sz, _vp], _i),
    "cer_routed_ffn_gated_workspace_size": ([_i, _i, _i], _sz),
    "cer_routed_block_gated": ([_vp, _vp, _i, _i, _i, _SCP, _SCP, _vp, _i, _i, _i, _i, _vp, _vp, _vp, _i, _i, _vp,
                                _f, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _sz, _vp, _i, _vp], _i),
    "cer_routed_block_gated_workspace_size": ([_i, _i, _i, _i, _i, _i, _i, _i, _i, _i], _sz),
    "cer_drop_set_stats": ([_vp, _vp, _i, _i, _i, _i, _vp, _vp, _vp, _vp, _vp], _i),
    "cer_redundancy_gap": ([_vp, _vp, _vp, _i, _i, _i, _f, _vp, _vp, _vp, _sz, _vp], _i),
    "cer_redundancy_gap_workspace_size": ([_i, _i], _sz),
    "cer_rope_packed": ([_vp, _i, _i, _i, _i, _vp, ctypes.c_double, _vp], _i),
    "cer_packed_attention": ([_vp, _i, _i, _i, _i, _i, _vp, _vp], _i),
    "cer_routed_attention": ([_vp, _vp, _i, _i, _i, _vp, _i, _vp, _vp, _i, _i, _i, ctypes.c_double, _vp, _vp,
                              _sz, _vp], _i),
    "cer_routed_attention_workspace_size": ([_i, _i, _i, _i, _i], _sz),
    "cer_selftest_bounded_wait": ([_i, _vp, ctypes.c_ulonglong, _i, _i, _vp], _i),
    "cer_sync_status": ([_vp], _i),
    "cer_get_error": ([], ctypes.c_char_p),
    "cer_status_string": ([_i], ctypes.c_char_p),
    "cer_version": ([], _i),
}


def load(path: str = LIB_PATH) -> ctypes.CDLL:
    """Load libcer.so (once).  Raises if it has not been built."""
    global _lib
    if _lib is None:
        if not os.path.exists(path):
            raise RuntimeError(f"{path} is missing: build it with __graft_entry__.build()")
        lib = ctypes.CDLL(path)
        for name, (args, res) in _SIGS.items():
            fn = getattr(lib, name)
            fn.argtypes = args
            fn.restype = res
        _lib = lib
    return _lib


def _check(status: int) -> None:
    if status != 0:
        raise CerError(status, load().cer_get_error().decode())


def _p(t: Optional[torch.Tensor]):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream) -> ctypes.c_void_p:
    s = torch.cuda.current_stream() if stream is None else stream
    return ctypes.c_void_p(s.cuda_stream)


@dataclasses.dataclass
class Scorer:
    """One scorer MLP (core: W1 [H, d]; expansions: W1 [S, H, d]) on the device.

    W1 and U are bf16, w2 and b1 fp32.  See ``cer_scorer`` in cer_api.h.
    """
    W1: torch.Tensor
    w2: torch.Tensor
    b1: Optional[torch.Tensor] = None
    U: Optional[torch.Tensor] = None

    def c_struct(self) -> CerScorerC:
        S = 1 if self.W1.dim() == 2 else self.W1.shape[0]
        return CerScorerC(_p(self.W1), _p(self.b1), _p(self.w2), _p(self.U), int(self.W1.shape[-2]),
                          int(self.U.shape[-1]) if self.U is not None else 0, int(S))


def _sref(s: Optional[Scorer]):
    return None if s is None else ctypes.pointer(s.c_struct())


def workspace(nbytes: int, device) -> torch.Tensor:
    return torch.empty(max(int(nbytes), 256), dtype=torch.uint8, device=device)


# ------------------------------------------------------------------ entry points

def cer_score_workspace_size(B, N, core_hidden, exp_hidden, task) -> int:
    return load().cer_score_workspace_size(B, N, core_hidden, exp_hidden, task)


def cer_score(h, core: Scorer, exp: Optional[Scorer], t, task, logits, probs=None, ws=None, stream=None):
    B, N, d = h.shape
    need = cer_score_workspace_size(B, N, core.W1.shape[-2], exp.W1.shape[-2] if exp is not None else 0, task)
    if ws is None:
        ws = workspace(need, h.device)
    _check(load().cer_score(_p(h), B, N, d, _sref(core), _sref(exp), _p(t), task, _p(logits), _p(probs),
                            _p(ws), ws.numel(), _stream(stream)))


def cer_score_static(h, core: Scorer, exp: Optional[Scorer], t, task, logits, probs=None, stream=None):
    """cer_score without a workspace: the scratch is the library's static
    4 MiB device array (for callers that cannot allocate; see cer_api.h)."""
    B, N, d = h.shape
    _check(load().cer_score_static(_p(h), B, N, d, _sref(core), _sref(exp), _p(t), task, _p(logits), _p(probs),
                                   _stream(stream)))


def cer_select_topk(logits, r0, r1, K, idx, mask=None, stream=None):
    B, N = logits.shape
    _check(load().cer_select_topk(_p(logits), B, N, r0, r1, K, _p(idx), _p(mask), _stream(stream)))


def cer_gather(h, idx, X, stream=None):
    B, N, d = h.shape
    _check(load().cer_gather(_p(h), B, N, d, _p(idx), idx.shape[1], _p(X), _stream(stream)))


def cer_routed_ffn_workspace_size(M, d, C, with_chan) -> int:
    return load().cer_routed_ffn_workspace_size(M, d, C, int(bool(with_chan)))


def cer_routed_ffn(X, Wg, Wu, WdT, chan, Y, ws=None, stream=None):
    M, d = X.shape
    I = Wg.shape[0]
    C = I if chan is None else chan.numel()
    if ws is None:
        ws = workspace(cer_routed_ffn_workspace_size(M, d, C, chan is not None), X.device)
    _check(load().cer_routed_ffn(_p(X), M, d, _p(Wg), _p(Wu), _p(WdT), I, _p(chan), C, _p(Y), _p(ws), ws.numel(),
                                 _stream(stream)))


def cer_pack_ffn_weights(Wg, Wu, WdT, chan, Wg_out, Wu_out, WdT_out, stream=None):
    I, d = Wg.shape
    _check(load().cer_pack_ffn_weights(_p(Wg), _p(Wu), _p(WdT), I, d, _p(chan), chan.numel(), _p(Wg_out),
                                       _p(Wu_out), _p(WdT_out), _stream(stream)))


def pack_ffn_weights(Wg, Wu, WdT, chan, stream=None):
    """Kept-channel slices (new [C, d] tensors) of the three FFN weights."""
    C, d = chan.numel(), Wg.shape[1]
    outs = [torch.empty((C, d), dtype=Wg.dtype, device=Wg.device) for _ in range(3)]
    cer_pack_ffn_weights(Wg, Wu, WdT, chan, *outs, stream=stream)
    return tuple(outs)


def cer_scatter_add(h, idx, Y, stream=None):
    B, N, d = h.shape
    _check(load().cer_scatter_add(_p(h), B, N, d, _p(idx), idx.shape[1], _p(Y), _stream(stream)))


def cer_scatter_add_checked(h, idx, Y, stream=None):
    """cer_scatter_add that first checks each sequence's index list on the
    device (range, no repeats); a bad sequence is left unwritten and
    cer_sync_status raises CER_ERR_INDEX."""
    B, N, d = h.shape
    _check(load().cer_scatter_add_checked(_p(h), B, N, d, _p(idx), idx.shape[1], _p(Y), _stream(stream)))


def cer_routed_block_workspace_size(B, N, d, core_hidden, exp_hidden, task, r0, r1, K, C, with_chan) -> int:
    return load().cer_routed_block_workspace_size(B, N, d, core_hidden, exp_hidden, task, r0, r1, K, C,
                                                  int(bool(with_chan)))


def cer_routed_block(h, core: Scorer, exp: Optional[Scorer], t, task, r0, r1, K, Wg, Wu, WdT, chan,
                     out=None, logits=None, idx=None, mask=None, ws=None,
                     stage_events: Optional[Sequence[torch.cuda.Event]] = None, stream=None):
    """The fused routed block; updates h in place when ``out`` is None or h.

    With ``chan`` None the weights are used as given (all their rows are the
    channels to run: the full FFN or slices from pack_ffn_weights)."""
    B, N, d = h.shape
    I = Wg.shape[0]
    C = I if chan is None else chan.numel()
    eh = exp.W1.shape[-2] if exp is not None else 0
    if ws is None:
        ws = workspace(cer_routed_block_workspace_size(B, N, d, core.W1.shape[-2], eh, task, r0, r1, K, C,
                                                       chan is not None), h.device)
    ev_arr, n_ev = _event_array(stage_events)
    _check(load().cer_routed_block(_p(h), _p(out), B, N, d, _sref(core), _sref(exp), _p(t), task, r0, r1, K,
                                   _p(Wg), _p(Wu), _p(WdT), I, _p(chan), C, _p(logits), _p(idx), _p(mask),
                                   _p(ws), ws.numel(), ev_arr, n_ev, _stream(stream)))


def _event_array(stage_events):
    if stage_events is None:
        return None, 0
    handles = []
    for ev in stage_events:
        if ev.cuda_event == 0:     # torch creates the event lazily: force it
            ev.record()
        handles.append(ev.cuda_event)
    return (ctypes.c_void_p * len(handles))(*handles), len(handles)


def cer_ffn_channel_norms(WdT, norms, stream=None):
    I, d = WdT.shape
    _check(load().cer_ffn_channel_norms(_p(WdT), I, d, _p(norms), _stream(stream)))


def gate_weights(Wg, Wu, WdT, chan, stream=None):
    """Weights for the UCS FFN gate: all I channels, the kept ones (chan) first,
    then the rest in ascending order; plus their W_down column norms."""
    I = Wg.shape[0]
    keep = chan.to(torch.int64)
    rest = torch.ones(I, dtype=torch.bool, device=chan.device)
    rest[keep] = False
    perm = torch.cat([keep, torch.nonzero(rest).flatten()]).to(torch.int32).contiguous()
    Wg_p, Wu_p, WdT_p = pack_ffn_weights(Wg, Wu, WdT, perm, stream=stream)
    norms = torch.empty(I, dtype=torch.float32, device=Wg.device)
    cer_ffn_channel_norms(WdT_p, norms, stream=stream)
    return Wg_p, Wu_p, WdT_p, norms, perm


def cer_routed_ffn_gated(X, Wg, Wu, WdT, C_keep, norms, delta, Y, saliency=None, leakage=None, use_pruned=None,
                         ws=None, stream=None):
    M, d = X.shape
    I = Wg.shape[0]
    if ws is None:
        ws = workspace(load().cer_routed_ffn_gated_workspace_size(M, d, I), X.device)
    _check(load().cer_routed_ffn_gated(_p(X), M, d, _p(Wg), _p(Wu), _p(WdT), I, C_keep, _p(norms), float(delta),
                                       _p(Y), _p(saliency), _p(leakage), _p(use_pruned), _p(ws), ws.numel(),
                                       _stream(stream)))


def cer_routed_block_gated(h, core: Scorer, exp: Optional[Scorer], t, task, r0, r1, K, Wg, Wu, WdT, C_keep, norms,
                           delta, saliency=None, leakage=None, use_pruned=None, out=None, logits=None, idx=None,
                           mask=None, ws=None, stage_events=None, stream=None):
    B, N, d = h.shape
    I = Wg.shape[0]
    eh = exp.W1.shape[-2] if exp is not None else 0
    if ws is None:
        ws = workspace(load().cer_routed_block_gated_workspace_size(B, N, d, core.W1.shape[-2], eh, task, r0, r1, K,
                                                                    I), h.device)
    ev_arr, n_ev = _event_array(stage_events)
    _check(load().cer_routed_block_gated(_p(h), _p(out), B, N, d, _sref(core), _sref(exp), _p(t), task, r0, r1, K,
                                         _p(Wg), _p(Wu), _p(WdT), I, C_keep, _p(norms), float(delta), _p(saliency),
                                         _p(leakage), _p(use_pruned), _p(logits), _p(idx), _p(mask), _p(ws),
                                         ws.numel(), ev_arr, n_ev, _stream(stream)))


def cer_drop_set_stats(mask_t, mask_ref, r0, r1, jaccard, j_rand=None, rda=None, counts=None, stream=None):
    B, N = mask_t.shape
    _check(load().cer_drop_set_stats(_p(mask_t), _p(mask_ref), B, N, r0, r1, _p(jaccard), _p(j_rand), _p(rda),
                                     _p(counts), _stream(stream)))


def cer_redundancy_gap(h_in, h_out, mask, delta, gap, skip=None, ws=None, stream=None):
    B, N, d = h_in.shape
    if ws is None:
        ws = workspace(load().cer_redundancy_gap_workspace_size(B, N), h_in.device)
    _check(load().cer_redundancy_gap(_p(h_in), _p(h_out), _p(mask), B, N, d, float(delta), _p(gap), _p(skip),
                                     _p(ws), ws.numel(), _stream(stream)))


def cer_rope_packed(qkv, B, L, Hq, Hkv, pos, base=1e6, stream=None):
    """Rotary embedding of the packed query and key heads in place (qkv bf16 [B*L, (Hq+2Hkv)*128])."""
    _check(load().cer_rope_packed(_p(qkv), B, L, Hq, Hkv, _p(pos), float(base), _stream(stream)))


def cer_packed_attention(qkv, B, L, Hq, Hkv, causal, out=None, stream=None):
    """Softmax attention over each packed sequence; returns out bf16 [B*L, Hq*128]."""
    import torch
    if out is None:
        out = torch.empty((B * L, Hq * 128), dtype=torch.bfloat16, device=qkv.device)
    _check(load().cer_packed_attention(_p(qkv), B, L, Hq, Hkv, int(causal), _p(out), _stream(stream)))
    return out


def cer_routed_attention(h, idx, WqkvT, WoT, Hq, Hkv, causal, base=1e6, out=None, qkv=None, ws=None,
                         stream=None):
    """Attention sublayer on the packed sequence; h [B, N, d] updated in place unless out is given."""
    B, N, d = h.shape
    L = idx.shape[1]
    if ws is None:
        ws = workspace(load().cer_routed_attention_workspace_size(B, L, d, Hq, Hkv), h.device)
    _check(load().cer_routed_attention(_p(h), _p(out), B, N, d, _p(idx), L, _p(WqkvT), _p(WoT), Hq, Hkv,
                                       int(causal), float(base), _p(qkv), _p(ws), ws.numel(), _stream(stream)))
    return h if out is None else out


def cer_selftest_bounded_wait(kind, flag=None, token=0, arrive=False, limit_us=1000, stream=None):
    """One bounded wait on the device (kind 0: *flag == token; kind 1: an
    mbarrier phase, completed only when ``arrive``); a wait that runs out
    shows as CER_ERR_TIMEOUT at the next cer_sync_status."""
    _check(load().cer_selftest_bounded_wait(int(kind), _p(flag), int(token), int(bool(arrive)), int(limit_us),
                                            _stream(stream)))


def cer_sync_status(stream=None) -> None:
    """Synchronise the stream and raise if a kernel recorded an error."""
    _check(load().cer_sync_status(_stream(stream)))
