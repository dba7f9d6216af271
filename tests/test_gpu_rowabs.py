"""GPU parity of the per-row symmetric absmax INT8 low tier (lo_format 2) against
the oracle: conversions bit for bit, decode steps teacher-forced at the decode
tolerances (codes within 1 LSB at float-ordering ties, row scales within float
ordering)."""
import numpy as np
import pytest
import torch

import paper_2608_27513_gb300 as damp
import workloads as wl
from oracle import core
from tests import parity as P

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda:0")
S8 = core.FMT_S8_ROW


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2608_27513_gb300 import build
    build.build()
    torch.cuda.init()
    assert damp.device_status() == 0
    yield
    assert damp.device_status() == 0


@pytest.mark.parametrize("dk,dv,K", [(128, 128, 10), (64, 64, 8), (32, 96, 0), (64, 160, 33), (128, 64, 128)])
def test_pack_unpack_tiers_bit_exact(dk, dv, K):
    w = wl.Workload("t", "gdn", 3, 4, 2, dk, dv, K, 1, 1, "fp32", 7, S8)
    rng = np.random.default_rng(2)
    hi = rng.integers(0, 1 << 16, (3, 4, K, dv)).astype(np.uint16)
    codes = rng.integers(-127, 128, (3, 4, dk - K, dv)).astype(np.int8)
    meta = rng.random((3, 4, dk - K)).astype(np.float32)
    L = P.layout_of(w)
    state = damp.new_state(L, 5, DEV)
    slot_idx = torch.tensor([4, 0, 2], dtype=torch.int32, device=DEV)
    damp.pack_tiers(L, *P.tiers_to_dev(w, (hi, codes, meta), 3, DEV), state, slot_idx=slot_idx)
    got = P.tiers_from_dev(w, damp.unpack_tiers(L, state, slot_idx=slot_idx), 12)
    assert np.array_equal(got[0], hi.reshape(12, K, dv))
    assert np.array_equal(got[1], codes.reshape(12, dk - K, dv))
    assert np.array_equal(got[2], meta.reshape(12, dk - K))
    assert int(state[1].abs().sum()) == 0 and int(state[3].abs().sum()) == 0


@pytest.mark.parametrize("dk,dv,K", [(128, 128, 10), (64, 64, 8), (128, 96, 0), (32, 64, 32), (64, 1024, 7)])
def test_quantize_state_bit_exact(dk, dv, K):
    """Same FP32 input: max|x| is exact, s = max/127 and x/s are correctly rounded,
    so every code and scale matches the oracle bit for bit."""
    n_rows, H = 3, 3
    w = wl.Workload("t", "kda", n_rows, H, H, dk, dv, K, 1, 1, "fp32", 7, S8)
    S = wl.random_states(5, n_rows * H, dk, dv).reshape(n_rows, H, dk, dv)
    perms = np.stack([np.random.default_rng(h).permutation(dk) for h in range(H)]).astype(np.uint8)
    perm_units = np.tile(perms, (n_rows, 1))
    ref = core.pack_heads(perm_units, S.reshape(-1, dk, dv), K, S8)
    L = P.layout_of(w)
    state = damp.new_state(L, n_rows, DEV)
    damp.quantize_state(L, P.to_dev(S, DEV), P.to_dev(perms, DEV), state)
    got = P.tiers_from_dev(w, damp.unpack_tiers(L, state), n_rows * H)
    for g, r in zip(got, ref):
        assert np.array_equal(g, r)


def test_dequantize_state_bit_exact():
    dk, dv, K, H, n_rows = 128, 128, 16, 4, 3
    w = wl.Workload("t", "gdn", n_rows, H, H, dk, dv, K, 1, 1, "fp32", 7, S8)
    S = wl.random_states(6, n_rows * H, dk, dv)
    perms = np.stack([np.random.default_rng(h + 9).permutation(dk) for h in range(H)]).astype(np.uint8)
    perm_units = np.tile(perms, (n_rows, 1))
    tiers = core.pack_heads(perm_units, S, K, S8)
    ref = core.unpack_heads(perm_units, *tiers, K, S8, dk, dv).reshape(n_rows, H, dk, dv)
    L = P.layout_of(w)
    state = damp.new_state(L, n_rows, DEV)
    damp.pack_tiers(L, *P.tiers_to_dev(w, tiers, n_rows, DEV), state)
    got = damp.dequantize_state(L, state, P.to_dev(perms, DEV)).cpu().numpy()
    assert np.array_equal(got, ref)


def test_gdn_b1_d64_k8_row_absmax_matches_oracle():
    """The small GDN case (B=1, H=4, d=64, K_hi=8, T=16, FP32 inputs) with the
    row-absmax low tier."""
    w = wl.GDN_B1_D64.replace(lo_format=S8)
    P.run_teacher_forced(w, w.steps, DEV)


def test_kda_row_absmax_matches_oracle():
    P.run_teacher_forced(wl.KDA_B256.replace(batch=2, heads=8, qk_heads=8, lo_format=S8), 3, DEV)


def test_gdn_gqa_row_absmax_matches_oracle():
    P.run_teacher_forced(wl.GDN_B64_GQA.replace(batch=2, lo_format=S8), 3, DEV)


def test_odd_k_ragged_value_blocks():
    w = wl.Workload("kda_k5_dv96", "kda", 2, 4, 2, 64, 96, 5, 2, 8, "bf16", 13, S8)
    P.run_teacher_forced(w, 2, DEV)


@pytest.mark.parametrize("kind", ["gdn", "kda"])
def test_uniform_row_absmax_entry_point(kind):
    w = wl.sweep(kind, 0, lo_format=S8).replace(batch=1, heads=4, qk_heads=4)
    P.run_teacher_forced(w, 2, DEV, u8=True)


def test_all_fp16_and_widest_rows():
    """K_hi = d_k (no low tier) and d_v = 1024 (the widest row a scale spans)."""
    P.run_teacher_forced(wl.Workload("allhi", "gdn", 1, 2, 2, 32, 64, 32, 2, 8, "fp32", 14, S8), 2, DEV)
    P.run_teacher_forced(wl.Workload("dv1024", "kda", 1, 2, 2, 64, 1024, 6, 2, 8, "bf16", 15, S8), 2, DEV)


def test_slot_indirection_row_absmax():
    w = wl.KDA_B256.replace(batch=3, heads=4, qk_heads=4, lo_format=S8)
    P.run_teacher_forced(w, 2, DEV, slot_of={0: 5, 1: 0, 2: 2}, pool=6)


@pytest.mark.parametrize("dv,lengths", [(128, [6, 2]), (96, [6, 0]), (64, [3, 6])])
def test_row_absmax_prefill_chunks_match_oracle(dv, lengths):
    """Prefill chunks of the row-absmax format: the four warps of a head share each row's
    maximum over the value blocks (d_v = 96 and 64 leave warps without a block)."""
    from tests.test_gpu_prefill import _run as run_chunks
    w = wl.KDA_B256.replace(batch=2, heads=4, qk_heads=4, d_v=dv, lo_format=S8)
    run_chunks(w, 6, lengths=lengths)


@pytest.mark.parametrize("dk,dv,K", [(32, 32, 4), (64, 64, 0)])
def test_row_absmax_small_heads(dk, dv, K):
    """One or two value blocks per head: three or two warps of each group only meet."""
    w = wl.Workload("t", "gdn", 3, 4, 4, dk, dv, K, 1, 1, "fp32", 18, S8)
    P.run_teacher_forced(w, 2, DEV)


@pytest.mark.parametrize("kind,K", [("kda", 10), ("gdn", 16)])
def test_row_absmax_full_batch_sampled_rows(kind, K):
    """B=256, H=32, d=128, BF16 (the four-warp row-absmax step at a compile-time K_hi):
    rows 0, 77, 255 against the oracle over two steps."""
    from tests.test_gpu_fullsize import _fullsize
    w = (wl.KDA_B256 if kind == "kda" else wl.sweep("gdn", K)).replace(lo_format=S8)
    _fullsize(w, [0, 77, 255], 2)
