"""Out-of-bounds write checks on the GPU: every output buffer and state pool sits
between poisoned guard regions, and each call must leave the guards (and the
outputs it was not asked to write) untouched.  Plus a packed-state checkpoint
round trip through the logical tiers."""
import numpy as np
import pytest
import torch

import paper_2608_27513_gb300 as damp
import workloads as wl
from paper_2608_27513_gb300 import checkpoint
from tests import parity as P

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda:0")
GUARD = 4096
POISON = 0xA5


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2608_27513_gb300 import build
    build.build()
    torch.cuda.init()
    assert damp.device_status() == 0
    yield
    assert damp.device_status() == 0


class Guarded:
    """A tensor of `shape`/`dtype` inside a byte buffer with poisoned guards on both sides."""

    def __init__(self, shape, dtype, fill=None):
        n = int(np.prod(shape)) * torch.empty((), dtype=dtype).element_size()
        self.raw = torch.full((GUARD + n + GUARD,), POISON, dtype=torch.uint8, device=DEV)
        self.t = self.raw[GUARD:GUARD + n].view(dtype).view(shape)
        if fill is not None:
            self.t.copy_(fill)

    def check(self):
        torch.cuda.synchronize()
        assert bool((self.raw[:GUARD] == POISON).all()), "write before the buffer"
        assert bool((self.raw[-GUARD:] == POISON).all()), "write after the buffer"


def _inputs(w, T=None):
    dt = torch.bfloat16 if w.in_dtype == "bf16" else torch.float32
    if T is None:
        inp = wl.step_inputs(w, 0)
    else:
        steps = [wl.step_inputs(w, t) for t in range(T)]
        inp = {k: np.stack([s[k] for s in steps], axis=1) for k in steps[0]}
    return {k: P.to_dev(v, DEV, dt if k in ("q", "k", "v") else None) for k, v in inp.items()}


def _pool(L, slots):
    g = Guarded((slots, damp.slot_bytes(L)), torch.uint8)
    g.t.zero_()
    return g


@pytest.mark.parametrize("fmt,K", [(0, 10), (0, 13), (1, 0), (2, 8), (3, 6), (5, 16)])
def test_decode_step_writes_only_its_slots_and_o(fmt, K):
    w = wl.KDA_B256.replace(batch=3, heads=4, qk_heads=2, k_hi=K, lo_format=fmt)
    L = P.layout_of(w)
    pool = _pool(L, 6)
    S = P.to_dev(wl.random_states(71, 12, 128, 128).reshape(3, 4, 128, 128), DEV)
    perm = P.to_dev(np.tile(np.random.default_rng(1).permutation(128).astype(np.uint8), (4, 1)), DEV)
    slot_idx = torch.tensor([5, 1, 3], dtype=torch.int32, device=DEV)
    damp.quantize_state(L, S, perm, pool.t, slot_idx=slot_idx)
    before = pool.t.clone()
    o = Guarded((3, 4, 128), torch.float32)
    d = _inputs(w)
    damp.kda_decode_step(L, pool.t, perm, d["q"], d["k"], d["v"], d["g"], d["beta"], o=o.t, slot_idx=slot_idx)
    pool.check()
    o.check()
    for s in (0, 2, 4):
        assert torch.equal(pool.t[s], before[s])
    assert bool(torch.isfinite(o.t).all())


@pytest.mark.parametrize("T", [5, 32])
def test_prefill_leaves_rows_past_their_length_and_guards_alone(T):
    w = wl.KDA_B256.replace(batch=3, heads=4, qk_heads=4)
    L = P.layout_of(w)
    pool = _pool(L, 3)
    S = P.to_dev(wl.random_states(72, 12, 128, 128).reshape(3, 4, 128, 128), DEV)
    perm = P.to_dev(np.tile(np.arange(128, dtype=np.uint8), (4, 1)), DEV)
    damp.quantize_state(L, S, perm, pool.t)
    before = pool.t.clone()
    o = Guarded((3, T, 4, 128), torch.float32)
    o.t.fill_(7.0)
    d = _inputs(w, T)
    lens = torch.tensor([T, 2, 0], dtype=torch.int32, device=DEV)
    damp.kda_prefill_chunk(L, pool.t, perm, d["q"], d["k"], d["v"], d["g"], d["beta"], o=o.t, lengths=lens)
    pool.check()
    o.check()
    assert bool((o.t[1, 2:] == 7.0).all()) and bool((o.t[2] == 7.0).all())
    assert torch.equal(pool.t[2], before[2]) and not torch.equal(pool.t[0], before[0])


def test_conversions_and_calibration_write_only_their_outputs():
    w = wl.GDN_B1_D64.replace(batch=2)
    L = P.layout_of(w)
    pool = _pool(L, 2)
    S = Guarded((2, w.heads, w.d_k, w.d_v), torch.float32,
                fill=P.to_dev(wl.random_states(73, 2 * w.heads, w.d_k, w.d_v).reshape(2, w.heads, w.d_k, w.d_v), DEV))
    perm = P.to_dev(np.tile(np.arange(w.d_k, dtype=np.uint8), (w.heads, 1)), DEV)
    damp.quantize_state(L, S.t, perm, pool.t)
    out = Guarded(S.t.shape, torch.float32)
    damp.dequantize_state(L, pool.t, perm, S=out.t)
    pool.check(), S.check(), out.check()
    E = Guarded((w.heads, w.d_k), torch.float32, fill=torch.zeros((w.heads, w.d_k), device=DEV))
    G = Guarded((w.heads, w.d_k), torch.float32, fill=torch.zeros((w.heads, w.d_k), device=DEV))
    damp.calib_error_energy(L, S.t, E.t)
    damp.calib_log_decay(L, _inputs(w)["g"], G.t)
    C = Guarded((w.heads, w.d_k), torch.float32)
    pi = Guarded((w.heads, w.d_k), torch.uint8)
    lib = damp._lib.lib()
    import ctypes
    c = L.c()
    assert lib.damp_calib_select(ctypes.byref(c), ctypes.c_void_p(E.t.data_ptr()), 1, ctypes.c_void_p(G.t.data_ptr()),
                                 1, ctypes.c_float(1e-4), ctypes.c_void_p(C.t.data_ptr()),
                                 ctypes.c_void_p(pi.t.data_ptr()), None) == 0
    for g in (E, G, C, pi):
        g.check()


def test_state_checkpoint_round_trip(tmp_path):
    w = wl.KDA_B256.replace(batch=3, heads=4, qk_heads=4, k_hi=7)
    L = P.layout_of(w)
    pool = damp.new_state(L, 3, DEV)
    S = P.to_dev(wl.random_states(74, 12, 128, 128).reshape(3, 4, 128, 128), DEV)
    perm = P.to_dev(np.tile(np.arange(128, dtype=np.uint8), (4, 1)), DEV)
    damp.quantize_state(L, S, perm, pool)
    path = str(tmp_path / "state.npz")
    checkpoint.save_state(path, L, pool)
    fresh = damp.new_state(L, 3, DEV)
    checkpoint.load_state(path, L, fresh)
    assert torch.equal(fresh, pool)
    with pytest.raises(ValueError):
        checkpoint.load_state(path, damp.Layout(4, 4, 128, 128, 8, 0), fresh)
