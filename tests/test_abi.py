"""Host-side checks of the C ABI that need no GPU: the library builds and loads,
exports every entry point include/cer_api.h declares, sizes workspaces, and
rejects bad arguments before touching a device.  A well-formed call on a
machine without an sm_103 GPU must fail loudly (CER_ERR_DEVICE), never fall
back to anything."""
import ctypes
import os
import re

import pytest
import torch

from paper_2608_29291_gb300 import cer

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "cer_api.h")


@pytest.fixture(scope="module")
def lib():
    if not os.path.exists(cer.LIB_PATH):
        from paper_2608_29291_gb300 import build_lib
        build_lib.build()
    return cer.load()


def declared_functions():
    text = open(HEADER).read()
    return sorted(set(re.findall(r"^\s*(?:cer_status|size_t|const char\*|int)\s+(cer_\w+)\s*\(", text, re.M)))


def test_header_declares_the_expected_entry_points():
    assert declared_functions() == sorted(cer.EXPORTS)


def test_library_exports_every_declared_symbol(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name
    assert lib.cer_version() == 1
    for code, name in cer.STATUS_NAMES.items():
        assert lib.cer_status_string(code).decode() == name


def _r256(x):
    return (x + 255) // 256 * 256


def test_workspace_sizes(lib):
    # scorer: bias + w2 tables [B][Ht] and at most Ht/64 partial-score rows of B*N
    assert lib.cer_score_workspace_size(4, 1024, 256, 0, 0) == 2 * 4096 + 4 * 4 * 1024 * 4
    assert lib.cer_score_workspace_size(2, 4096, 512, 512, 1) == 2 * 8192 + 16 * 2 * 4096 * 4
    assert lib.cer_score_workspace_size(1, 256, 64, 64, 1) == 2 * 512 + 2 * 256 * 4
    assert lib.cer_score_workspace_size(1, 10, 100, 0, 0) == 0          # hidden not a multiple of 64
    # FFN: act [M, C] bf16, plus three [C, d] slices when a channel list is packed per call
    sk = (24 << 20) + 8192     # stream-K partial accumulators and flags of the GEMMs
    assert lib.cer_routed_ffn_workspace_size(2348, 1536, 6720, 0) == _r256(2348 * 6720 * 2) + sk
    assert lib.cer_routed_ffn_workspace_size(2348, 1536, 6720, 1) == _r256(2348 * 6720 * 2) + sk + \
        3 * _r256(6720 * 1536 * 2)
    assert lib.cer_routed_ffn_workspace_size(0, 1536, 6720, 0) == 0
    M = 4 * (292 + 1024 - 729)
    for wc in (0, 1):
        ws = lib.cer_routed_block_workspace_size(4, 1024, 1536, 256, 0, 0, 0, 729, 292, 6720, wc)
        assert ws == lib.cer_score_workspace_size(4, 1024, 256, 0, 0) + _r256(M * 4) + _r256(M * 1536 * 2) + \
            lib.cer_routed_ffn_workspace_size(M, 1536, 6720, wc)
    assert lib.cer_routed_block_workspace_size(4, 1024, 1536, 256, 0, 0, 0, 729, 730, 6720, 0) == 0  # K > N_r


FAKE = ctypes.c_void_p(1 << 20)      # 16-byte aligned, never dereferenced: checks fail first


def _err(lib):
    return lib.cer_get_error().decode()


def test_select_argument_checks(lib):
    assert lib.cer_select_topk(None, 1, 8, 0, 8, 4, FAKE, None, None) == 1          # NULL logits
    assert lib.cer_select_topk(FAKE, 1, 8, 0, 8, 9, FAKE, None, None) == 4          # K > N_r
    assert "K=9" in _err(lib)
    assert lib.cer_select_topk(FAKE, 1, 8, 5, 3, 0, FAKE, None, None) == 4          # r0 > r1
    assert lib.cer_select_topk(FAKE, 1, 8, 0, 9, 1, FAKE, None, None) == 4          # r1 > N
    assert lib.cer_select_topk(FAKE, 1, 60000, 0, 8, 1, FAKE, None, None) == 2      # N too large
    assert lib.cer_select_topk(ctypes.c_void_p((1 << 20) + 4), 1, 8, 0, 8, 1, FAKE, None, None) == 3


def test_ffn_argument_checks(lib):
    f = lib.cer_routed_ffn
    assert f(FAKE, 10, 100, FAKE, FAKE, FAKE, 512, None, 512, FAKE, FAKE, 1 << 20, None) == 2   # d % 64
    assert f(FAKE, 10, 128, FAKE, FAKE, FAKE, 512, None, 256, FAKE, FAKE, 1 << 20, None) == 2   # NULL chan, C != I
    assert f(FAKE, 10, 128, FAKE, FAKE, FAKE, 512, FAKE, 100, FAKE, FAKE, 1 << 20, None) == 2   # C % 64
    assert f(FAKE, 10, 128, FAKE, FAKE, FAKE, 512, FAKE, 576, FAKE, FAKE, 1 << 20, None) == 2   # C > I
    assert f(FAKE, 1000, 128, FAKE, FAKE, FAKE, 512, FAKE, 256, FAKE, FAKE, 16, None) == 9      # workspace
    assert f(FAKE, 10, 128, None, FAKE, FAKE, 512, FAKE, 256, FAKE, FAKE, 1 << 20, None) == 1   # NULL Wg


def test_pack_argument_checks(lib):
    f = lib.cer_pack_ffn_weights
    assert f(FAKE, FAKE, FAKE, 512, 128, None, 256, FAKE, FAKE, FAKE, None) == 1      # NULL chan
    assert f(FAKE, FAKE, FAKE, 512, 100, FAKE, 256, FAKE, FAKE, FAKE, None) == 2      # d % 8
    assert f(FAKE, FAKE, FAKE, 512, 128, FAKE, 600, FAKE, FAKE, FAKE, None) == 2      # C > I


def test_score_argument_checks(lib):
    core = cer.CerScorerC(FAKE.value, None, FAKE.value, None, 256, 0, 1)
    bad_core = cer.CerScorerC(FAKE.value, None, FAKE.value, FAKE.value, 256, 64, 1)   # core with U
    s = lib.cer_score
    assert s(FAKE, 1, 16, 1536, ctypes.pointer(core), None, None, 1, FAKE, None, FAKE, 1 << 30, None) == 1  # GEN, no exp
    assert s(FAKE, 1, 16, 1500, ctypes.pointer(core), None, None, 0, FAKE, None, FAKE, 1 << 30, None) == 2  # d % 64
    assert s(FAKE, 1, 16, 1536, ctypes.pointer(bad_core), None, None, 0, FAKE, None, FAKE, 1 << 30, None) == 2
    assert s(FAKE, 1, 16, 1536, ctypes.pointer(core), None, None, 7, FAKE, None, FAKE, 1 << 30, None) == 4  # task
    assert s(FAKE, 1, 16, 1536, ctypes.pointer(core), None, None, 0, FAKE, None, FAKE, 8, None) == 9        # workspace


def test_attention_argument_checks(lib):
    r, a = lib.cer_rope_packed, lib.cer_packed_attention
    assert r(FAKE, 1, 8, 3, 2, FAKE, 1e6, None) == 2        # Hq not a multiple of Hkv
    assert r(FAKE, 1, 8, 4, 0, FAKE, 1e6, None) == 2        # no key/value head
    assert r(FAKE, 1, 8, 4, 2, None, 1e6, None) == 1        # NULL positions
    assert r(FAKE, 1, 8, 4, 2, FAKE, 0.5, None) == 4        # rotary base <= 1
    assert r(FAKE, 1, 8, 4, 2, FAKE, float("inf"), None) == 4
    assert a(FAKE, 1, 8, 6, 4, 1, FAKE, None) == 2          # Hq not a multiple of Hkv
    assert a(FAKE, 1, 8, 4, 2, 2, FAKE, None) == 4          # causal not 0 or 1
    assert a(FAKE, 1, 8, 4, 2, 1, None, None) == 1          # NULL out
    assert a(FAKE, -1, 8, 4, 2, 1, FAKE, None) == 2         # negative B
    assert a(ctypes.c_void_p((1 << 20) + 4), 1, 8, 4, 2, 1, FAKE, None) == 3   # misaligned qkv
    ra, big = lib.cer_routed_attention, 1 << 30
    assert ra(FAKE, None, 1, 16, 100, FAKE, 8, FAKE, FAKE, 4, 2, 1, 1e6, None, FAKE, big, None) == 2   # d % 64
    assert ra(FAKE, None, 1, 16, 128, FAKE, 20, FAKE, FAKE, 4, 2, 1, 1e6, None, FAKE, big, None) == 2  # L > N
    assert ra(FAKE, None, 1, 16, 128, FAKE, 8, None, FAKE, 4, 2, 1, 1e6, None, FAKE, big, None) == 1   # NULL WqkvT
    assert ra(FAKE, None, 1, 16, 128, FAKE, 8, FAKE, FAKE, 4, 2, 1, 1e6, None, FAKE, 64, None) == 9    # workspace
    W = (4 + 2 * 2) * 128
    assert lib.cer_routed_attention_workspace_size(2, 10, 128, 4, 2) == \
        _r256(20 * 128 * 2) + _r256(20 * W * 2) + _r256(20 * 512 * 2) + _r256(20 * 64 * 8) + (24 << 20) + 8192
    assert lib.cer_routed_attention_workspace_size(2, 0, 128, 4, 2) == 0


def test_checked_scatter_argument_checks(lib):
    f = lib.cer_scatter_add_checked
    assert f(FAKE, 1, 500000, 64, FAKE, 10, FAKE, None) == 2     # N beyond the bitmap
    assert f(FAKE, 1, 100, 60, FAKE, 10, FAKE, None) == 2        # d % 8
    assert f(FAKE, 1, 100, 64, FAKE, 101, FAKE, None) == 2       # k_tot > N
    assert f(FAKE, 1, 100, 64, None, 10, FAKE, None) == 1        # NULL idx


@pytest.mark.skipif(torch.cuda.is_available(), reason="checks the behaviour without a GPU")
def test_static_scorer_refuses_an_unusable_device_like_cer_score(lib):
    """cer_score_static asks whether the device is one this library runs on
    before it looks up its static array: without a usable GPU it fails with the
    same status and message as cer_score on the same well-formed call."""
    core = cer.CerScorerC(FAKE.value, None, FAKE.value, None, 256, 0, 1)
    st = lib.cer_score_static(FAKE, 1, 16, 1536, ctypes.pointer(core), None, None, 0, FAKE, None, None)
    msg_static = _err(lib)
    st_ws = lib.cer_score(FAKE, 1, 16, 1536, ctypes.pointer(core), None, None, 0, FAKE, None, FAKE, 1 << 30, None)
    assert st == st_ws == 6, (st, st_ws)
    assert msg_static == _err(lib)
    assert "static scratch" not in msg_static


@pytest.mark.skipif(torch.cuda.is_available(), reason="checks the behaviour without a GPU")
def test_well_formed_call_without_gpu_fails_loudly(lib):
    st = lib.cer_select_topk(FAKE, 1, 8, 0, 8, 4, FAKE, None, None)
    assert st == 6, (st, _err(lib))   # CER_ERR_DEVICE: no device, no fallback
    with pytest.raises(cer.CerError):
        cer._check(st)
