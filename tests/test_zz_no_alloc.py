"""cer_score_static: the scorer entry point that allocates nothing.

Callers such as a plug-in host that gives its operators no workspace, or a
real-time loop whose device memory is fixed at start-up, cannot allocate the
scratch cer_score asks for.  cer_score_static keeps that scratch in one static
4 MiB device array instead.  These tests check that it returns what cer_score
returns (same tolerance as the other score tests), on two calls in a row --
the second call reuses the array the first one left behind -- and that sizes
beyond the array are refused before any GPU work.  This file is collected last
on purpose, so a run that stops at the first failure has run everything else.
"""
import ctypes

import numpy as np
import pytest
import torch

from paper_2608_29291_gb300 import cer
from paper_2608_29291_gb300 import inputs as gen
from tests.gpu_helpers import bf16_dev, f32_dev, rel_err, scorers

SCORE_TOL = 1e-4


def _case(w):
    inp = gen.make_inputs(w)
    core, exp = scorers(inp)
    return inp, core, (exp if w.task == 1 else None)


@pytest.mark.gpu
def test_static_scratch_scorer_matches_workspace_scorer_twice():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    big = gen.Workload("und_small", B=3, N=700, d=512, I=64, C=64, r0=0, r1=700, K=100, Hc=256, He=0, E=0,
                       task=0, seed=7)
    for w in (gen.tiny(), big):            # two calls in a row, different sizes and tasks
        inp, core, exp = _case(w)
        h, t = bf16_dev(inp["h"]), f32_dev(inp["t"])
        ref = torch.empty((w.B, w.N), dtype=torch.float32, device="cuda")
        ref_p = torch.empty_like(ref)
        cer.cer_score(h, core, exp, t, w.task, ref, ref_p)
        got = torch.full_like(ref, float("nan"))
        got_p = torch.full_like(ref, float("nan"))
        cer.cer_score_static(h, core, exp, t, w.task, got, got_p)
        cer.cer_sync_status()
        assert rel_err(got.cpu().numpy(), ref.cpu().numpy()) <= SCORE_TOL
        assert np.max(np.abs(got_p.cpu().numpy() - ref_p.cpu().numpy())) <= 1e-5


def test_static_scratch_refuses_sizes_beyond_its_capacity():
    lib = cer.load()
    fake = ctypes.c_void_p(1 << 20)
    core = cer.CerScorerC(fake.value, None, fake.value, None, 2048, 0, 1)
    # B*N = 65536 tokens x 32 partial rows (hidden 2048 / 64) x 4 bytes = 8 MiB of partial scores > 4 MiB
    st = lib.cer_score_static(fake, 4, 16384, 1536, ctypes.pointer(core), None, None, 0, fake, None, None)
    assert st == 9, lib.cer_get_error()
    assert b"static scratch holds 4194304 bytes" in lib.cer_get_error()
