"""The bounded waits inside the decode kernel, made to run out on purpose without a
fault or a hang: the test hook's stage barriers expect more bytes than each copy
delivers, every wait gives up after ~1 ms, the kernel lets its copies land, writes
nothing and reports DAMP_DEV_WAIT_TIMEOUT; the next ordinary step is unaffected."""
import time

import numpy as np
import pytest
import torch

import paper_2608_27513_gb300 as damp
import workloads as wl
from tests import parity as P

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda:0")


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2608_27513_gb300 import build
    build.build()
    torch.cuda.init()
    assert damp.device_status() == 0
    yield
    assert damp.device_status() == 0


def test_wait_runs_out_reports_and_writes_nothing():
    w = wl.KDA_B256.replace(batch=4, heads=4, qk_heads=4)   # d = 128, K_hi = 10, format 0, BF16
    L = P.layout_of(w)
    state = damp.new_state(L, w.batch, DEV)
    S = P.to_dev(wl.random_states(5, w.batch * w.heads, 128, 128).reshape(w.batch, w.heads, 128, 128), DEV)
    perms = P.to_dev(np.stack([np.random.default_rng(h).permutation(128) for h in range(w.heads)]).astype(np.uint8),
                     DEV)
    damp.quantize_state(L, S, perms, state)
    before = state.clone()
    d = P.inputs_to_dev(w, wl.step_inputs(w, 0), DEV)
    o = torch.full((w.batch, w.heads, 128), 7.0, device=DEV)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    damp.test_kda_wait_timeout(L, state, perms, d["q"], d["k"], d["v"], d["g"], d["beta"], o=o)
    assert damp.device_status() == damp.DEV_WAIT_TIMEOUT
    assert time.perf_counter() - t0 < 2.0          # ~1 ms waits, not the decode step's 2 s
    assert torch.equal(state, before)               # no record written
    assert bool((o == 7.0).all())                   # no output written
    assert damp.device_status() == 0                # the read cleared the word
    # the same pool steps normally afterwards, and matches the ordinary step bit for bit
    ref = before.clone()
    o1 = damp.kda_decode_step(L, state, perms, d["q"], d["k"], d["v"], d["g"], d["beta"])
    o2 = damp.kda_decode_step(L, ref, perms, d["q"], d["k"], d["v"], d["g"], d["beta"])
    assert torch.equal(state, ref) and torch.equal(o1, o2) and not torch.equal(state, before)
    assert damp.device_status() == 0


def test_step_after_a_timeout_matches_the_oracle():
    w = wl.KDA_B256.replace(batch=2, heads=4, qk_heads=4)
    L = P.layout_of(w)
    state = damp.new_state(L, w.batch, DEV)
    d = P.inputs_to_dev(w, wl.step_inputs(w, 0), DEV)
    perms = P.to_dev(np.tile(np.arange(128, dtype=np.uint8), (w.heads, 1)), DEV)
    damp.test_kda_wait_timeout(L, state, perms, d["q"], d["k"], d["v"], d["g"], d["beta"])
    assert damp.device_status() == damp.DEV_WAIT_TIMEOUT
    P.run_teacher_forced(w, 2, DEV)
    assert damp.device_status() == 0
