"""GPU parity of the 4-bit and FP8 low tiers (formats 3-5, App. A.1) against the
oracle: logical tiers bit for bit through pack/unpack, whole-state conversions,
decode steps (the fused packed step's 4-bit and FP8 instances) and prefill chunks, at the
decode tolerances with each format's tie rule."""
import numpy as np
import pytest
import torch

import paper_2608_27513_gb300 as damp
import workloads as wl
from oracle import core
from tests import parity as P
from tests.test_gpu_prefill import _run as run_chunks

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda:0")
NEW = [core.FMT_U4_H32, core.FMT_U4, core.FMT_E4M3]


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2608_27513_gb300 import build
    build.build()
    torch.cuda.init()
    assert damp.device_status() == 0
    yield
    assert damp.device_status() == 0


@pytest.mark.parametrize("fmt", NEW)
@pytest.mark.parametrize("dk,dv,K", [(128, 128, 10), (64, 96, 5), (32, 64, 0)])
def test_pack_unpack_tiers_bit_exact(fmt, dk, dv, K):
    w = wl.Workload("t", "kda", 3, 4, 2, dk, dv, K, 1, 1, "fp32", 7, fmt)
    rng = np.random.default_rng(61)
    hi = rng.integers(0, 1 << 16, (3, 4, K, dv)).astype(np.uint16)
    cols = dv // 2 if fmt != core.FMT_E4M3 else dv
    codes = rng.integers(0, 256, (3, 4, dk - K, cols)).astype(np.uint8)
    meta = (rng.random((3, 4, dk - K, dv // 32)).astype(np.float32) if fmt == core.FMT_E4M3 else
            rng.integers(0, 1 << 16, (3, 4, dk - K, dv // 32, 2)).astype(np.uint16))
    L = P.layout_of(w)
    state = damp.new_state(L, 5, DEV)
    slot_idx = torch.tensor([4, 0, 2], dtype=torch.int32, device=DEV)
    damp.pack_tiers(L, *P.tiers_to_dev(w, (hi, codes, meta), 3, DEV), state, slot_idx=slot_idx)
    got = P.tiers_from_dev(w, damp.unpack_tiers(L, state, slot_idx=slot_idx), 12)
    assert np.array_equal(got[0], hi.reshape(12, K, dv))
    assert np.array_equal(got[1], codes.reshape(12, dk - K, cols))
    assert np.array_equal(got[2], meta.reshape(got[2].shape))


@pytest.mark.parametrize("fmt", NEW)
def test_quantize_and_dequantize_match_oracle(fmt):
    n_rows, H, dk, dv, K = 3, 3, 64, 96, 6
    w = wl.Workload("t", "kda", n_rows, H, H, dk, dv, K, 1, 1, "fp32", 7, fmt)
    S = wl.random_states(62, n_rows * H, dk, dv).reshape(n_rows, H, dk, dv)
    perms = np.stack([np.random.default_rng(h).permutation(dk) for h in range(H)]).astype(np.uint8)
    perm_units = np.tile(perms, (n_rows, 1))
    ref = core.pack_heads(perm_units, S.reshape(-1, dk, dv), K, fmt)
    L = P.layout_of(w)
    state = damp.new_state(L, n_rows, DEV)
    damp.quantize_state(L, P.to_dev(S, DEV), P.to_dev(perms, DEV), state)
    got = P.tiers_from_dev(w, damp.unpack_tiers(L, state), n_rows * H)
    lo_pre = np.stack([S.reshape(-1, dk, dv)[i][perm_units[i][K:]] for i in range(n_rows * H)])
    if fmt == core.FMT_U4_H32:
        lo_pre = core.hadamard32(lo_pre.reshape(-1, 32)).reshape(lo_pre.shape)
    stats = P.CodeStats()
    P.compare_tiers(w, ref, got, lo_pre, stats, "quantize_state")
    stats.check_fraction()
    assert np.array_equal(got[0], ref[0])
    if fmt == core.FMT_E4M3:  # same FP32 input, correctly rounded division and E4M3 rounding
        assert np.array_equal(got[1], ref[1]) and np.array_equal(got[2], ref[2])
    # the reconstruction of the oracle's own tiers
    damp.pack_tiers(L, *P.tiers_to_dev(w, ref, n_rows, DEV), state)
    back = damp.dequantize_state(L, state, P.to_dev(perms, DEV)).cpu().numpy()
    want = core.unpack_heads(perm_units, *ref, K, fmt, dk, dv).reshape(back.shape)
    scale = np.abs(want).max(axis=-1, keepdims=True) + 1e-30
    assert np.all(np.abs(back - want) <= 1e-6 * scale)


@pytest.mark.parametrize("fmt", NEW)
@pytest.mark.parametrize("kind", ["gdn", "kda"])
@pytest.mark.parametrize("K", [10, 16])
def test_decode_steps_match_oracle(kind, fmt, K):
    """d_k = 128: K_hi = 10 runs the general instance of the format's step, K_hi = 16
    its compile-time layout (the instance the K_hi sweep times)."""
    w = wl.sweep(kind, K, fmt).replace(batch=2, heads=4, qk_heads=4)
    P.run_teacher_forced(w, 3, DEV)


@pytest.mark.parametrize("fmt", NEW)
def test_decode_k16_full_batch_sampled_rows(fmt):
    """KDA B=256, H=32, d=128, K_hi=16 in the 4-bit and FP8 formats, the whole batch in
    one launch (compile-time instances), rows 9 and 250 against the oracle."""
    from tests.test_gpu_fullsize import _fullsize
    _fullsize(wl.sweep("kda", 16, fmt), [9, 250], 1)


@pytest.mark.parametrize("fmt", NEW)
def test_uniform_entry_point(fmt):
    w = wl.sweep("kda", 0, fmt).replace(batch=1, heads=4, qk_heads=4)
    P.run_teacher_forced(w, 2, DEV, u8=True)


@pytest.mark.parametrize("fmt", NEW)
def test_prefill_chunks_match_oracle(fmt):
    run_chunks(wl.KDA_B256.replace(batch=2, heads=4, qk_heads=4, lo_format=fmt), 6, lengths=[6, 2])


@pytest.mark.parametrize("fmt", NEW)
@pytest.mark.parametrize("dk,dv,K", [(64, 96, 5), (32, 64, 0), (32, 32, 3)])
def test_decode_steps_small_heads(fmt, dk, dv, K):
    """The general instances of the 4-bit and FP8 steps (fewer row slots per lane,
    ragged value blocks)."""
    w = wl.Workload("t", "kda", 2, 4, 2, dk, dv, K, 1, 1, "bf16", 17, fmt)
    P.run_teacher_forced(w, 2, DEV)
