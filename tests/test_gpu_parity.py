"""GPU parity: the CUDA path through the C ABI against the CPU oracle on the same
seeded inputs.  Steps are teacher-forced: each GPU step starts from the
oracle's packed state, so one rounding tie never compounds."""
import numpy as np
import pytest
import torch

import paper_2608_27513_gb300 as damp
import workloads as wl
from oracle import core, runs
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


def _small(w, **kw):
    return w.replace(**kw)


# ------------------------------------------------------------- conversions ---

@pytest.mark.parametrize("fmt", [0, 1])
@pytest.mark.parametrize("dk,dv,K", [(128, 128, 10), (64, 64, 8), (32, 96, 0), (128, 64, 128), (64, 160, 33)])
def test_pack_unpack_tiers_bit_exact(fmt, dk, dv, K):
    w = wl.Workload("t", "kda", 3, 4, 2, dk, dv, K, 1, 1, "fp32", 7, fmt)
    rng = np.random.default_rng(1)
    hi = rng.integers(0, 1 << 16, (3, 4, K, dv)).astype(np.uint16)
    codes = rng.integers(0, 256, (3, 4, dk - K, dv)).astype(np.uint8)
    meta = rng.integers(0, 1 << 16, (3, 4, dk - K, dv // 32, 2)).astype(np.uint16)
    L = P.layout_of(w)
    state = damp.new_state(L, 5, DEV)
    slot_idx = torch.tensor([4, 0, 2], dtype=torch.int32, device=DEV)
    damp.pack_tiers(L, *P.tiers_to_dev(w, (hi, codes, meta), 3, DEV), state, slot_idx=slot_idx)
    back = damp.unpack_tiers(L, state, slot_idx=slot_idx)
    got = P.tiers_from_dev(w, back, 12)
    assert np.array_equal(got[0], hi.reshape(12, K, dv))
    assert np.array_equal(got[1], codes.reshape(12, dk - K, dv))
    assert np.array_equal(got[2], meta.reshape(12, dk - K, dv // 32, 2))
    # untouched slots stay zero
    assert int(state[1].abs().sum()) == 0 and int(state[3].abs().sum()) == 0


@pytest.mark.parametrize("fmt", [0, 1])
@pytest.mark.parametrize("dk,dv,K", [(128, 128, 10), (64, 64, 8), (128, 96, 0), (32, 64, 32)])
def test_quantize_state_matches_oracle(fmt, dk, dv, K):
    n_rows, H = 4, 3
    w = wl.Workload("t", "kda", n_rows, H, H, dk, dv, K, 1, 1, "fp32", 7, fmt)
    S = wl.random_states(5, n_rows * H, dk, dv).reshape(n_rows, H, dk, dv)
    perms = np.stack([np.random.default_rng(h).permutation(dk) for h in range(H)]).astype(np.uint8)
    perm_units = np.tile(perms, (n_rows, 1))
    ref = core.pack_heads(perm_units, S.reshape(-1, dk, dv), K, fmt)
    L = P.layout_of(w)
    state = damp.new_state(L, n_rows, DEV)
    damp.quantize_state(L, P.to_dev(S, DEV), P.to_dev(perms, DEV), state)
    got = P.tiers_from_dev(w, damp.unpack_tiers(L, state), n_rows * H)
    lo_pre = np.stack([S.reshape(-1, dk, dv)[i][perm_units[i][K:]] for i in range(n_rows * H)])
    if fmt == 0 and lo_pre.size:
        lo_pre = core.hadamard32(lo_pre.reshape(-1, 32)).reshape(lo_pre.shape)
    stats = P.CodeStats()
    P.compare_tiers(w, ref, got, lo_pre, stats, "quantize_state")
    stats.check_fraction()
    assert np.array_equal(got[0], ref[0])  # FP16 rows: same FP32 input, same RNE rounding


@pytest.mark.parametrize("fmt", [0, 1])
def test_dequantize_state_matches_oracle(fmt):
    dk, dv, K, H, n_rows = 128, 128, 16, 4, 3
    w = wl.Workload("t", "gdn", n_rows, H, H, dk, dv, K, 1, 1, "fp32", 7, fmt)
    S = wl.random_states(6, n_rows * H, dk, dv)
    perms = np.stack([np.random.default_rng(h + 9).permutation(dk) for h in range(H)]).astype(np.uint8)
    perm_units = np.tile(perms, (n_rows, 1))
    tiers = core.pack_heads(perm_units, S, K, fmt)
    ref = core.unpack_heads(perm_units, *tiers, K, fmt, dk, dv).reshape(n_rows, H, dk, dv)
    L = P.layout_of(w)
    state = damp.new_state(L, n_rows, DEV)
    damp.pack_tiers(L, *P.tiers_to_dev(w, tiers, n_rows, DEV), state)
    got = damp.dequantize_state(L, state, P.to_dev(perms, DEV)).cpu().numpy()
    scale = np.abs(ref).max(axis=-1, keepdims=True) + 1e-30
    assert np.all(np.abs(got - ref) <= 1e-6 * scale)


# --------------------------------------------------------- FP32 baseline ---

@pytest.mark.parametrize("w", [wl.GDN_B1_D64, wl.GDN_B64_GQA.replace(batch=3), wl.KDA_B256.replace(batch=3),
                               wl.KDA_B256.replace(batch=2, d_v=96, in_dtype="fp32")],
                         ids=["gdn_b1_d64", "gdn_gqa", "kda_b3", "kda_dv96_fp32in"])
def test_fp32_step_matches_oracle(w):
    S = wl.random_states(8, w.batch * w.heads, w.d_k, w.d_v, scale=0.3)
    L = P.layout_of(w)
    dS = P.to_dev(S.reshape(w.batch, w.heads, w.d_k, w.d_v), DEV)
    for t in range(3):
        inp = wl.step_inputs(w, t)
        u = runs.unit_operands(w, inp)
        o_ref = core.delta_step_heads(S, u["q"], u["k"], u["v"], u["g"], u["beta"], w.kind)
        d = P.inputs_to_dev(w, inp, DEV)
        step = damp.fp32_kda_decode_step if w.kind == "kda" else damp.fp32_gdn_decode_step
        o = step(L, dS, d["q"], d["k"], d["v"], d["g"], d["beta"])
        P.compare_o(o.cpu().numpy().reshape(-1, w.d_v), o_ref, f"fp32 step {t}")
        got = dS.cpu().numpy().reshape(S.shape)
        assert np.all(np.abs(got - S) <= P.ATOL + P.RTOL * np.abs(S))
        dS = P.to_dev(S.reshape(w.batch, w.heads, w.d_k, w.d_v), DEV)  # teacher-forced


# --------------------------------------------------- fused packed step ---

def _run_teacher_forced(w, steps, **kw):
    return P.run_teacher_forced(w, steps, DEV, **kw)


def test_gdn_b1_d64_k8_matches_oracle():
    """GDN decode, B=1, H=4, d=64, K_hi=8, T=16, FP32 inputs (the small paper-shaped case)."""
    _run_teacher_forced(wl.GDN_B1_D64, wl.GDN_B1_D64.steps)


def test_gdn_gqa_matches_oracle():
    """GDN, 32 value heads sharing 16 q/k heads, d=128, K_hi=8, BF16 inputs."""
    _run_teacher_forced(wl.GDN_B64_GQA.replace(batch=2), 4)


def test_kda_matches_oracle():
    """KDA, per-channel decay, H=32, d=128, K_hi=10, BF16 inputs."""
    _run_teacher_forced(wl.KDA_B256.replace(batch=2), 4)


@pytest.mark.parametrize("kind", ["gdn", "kda"])
@pytest.mark.parametrize("K", wl.SWEEP_K_HI)
def test_k_hi_sweep_matches_oracle(kind, K):
    _run_teacher_forced(wl.sweep(kind, K).replace(batch=1, heads=8, qk_heads=8), 2)


@pytest.mark.parametrize("kind", ["gdn", "kda"])
def test_uniform_int8_without_hadamard_matches_oracle(kind):
    w = wl.sweep(kind, 0, lo_format=1).replace(batch=1, heads=8, qk_heads=8)
    _run_teacher_forced(w, 2, u8=True)


@pytest.mark.parametrize("kind", ["gdn", "kda"])
def test_uniform_int8_hadamard_entry_point(kind):
    _run_teacher_forced(wl.sweep(kind, 0).replace(batch=1, heads=4, qk_heads=4), 2, u8=True)


def test_ragged_value_blocks_and_all_fp16():
    """d_v = 96 (3 value blocks), d_k = 32, K_hi = d_k (pure FP16 state)."""
    w = wl.Workload("kda_dv96_allhi", "kda", 2, 2, 1, 32, 96, 32, 2, 8, "fp32", 11)
    _run_teacher_forced(w, 2)


def test_k_hi_spanning_two_row_slots():
    """K_hi = 40 > 32: FP16 rows in two of a lane's row slots."""
    w = wl.Workload("gdn_k40", "gdn", 2, 4, 4, 128, 64, 40, 2, 8, "bf16", 12)
    _run_teacher_forced(w, 2)


@pytest.mark.parametrize("K,fmt", [(12, 0), (5, 0), (12, 1)])
def test_general_kernel_at_d128(K, fmt):
    """d_k = 128 layouts outside the compile-time list run the general kernel."""
    w = wl.KDA_B256.replace(batch=2, heads=4, qk_heads=4, k_hi=K, lo_format=fmt)
    _run_teacher_forced(w, 2)


def test_slot_indirection_into_a_larger_pool():
    w = wl.KDA_B256.replace(batch=3, heads=4, qk_heads=4)
    _run_teacher_forced(w, 2, slot_of={0: 6, 1: 1, 2: 3}, pool=7)


def test_bad_slot_index_is_skipped_and_reported():
    w = wl.KDA_B256.replace(batch=2, heads=2, qk_heads=2)
    L = P.layout_of(w)
    state = damp.new_state(L, 2, DEV)
    S = P.to_dev(wl.random_states(3, 4, 128, 128).reshape(2, 2, 128, 128), DEV)
    perms = P.to_dev(np.tile(np.arange(128, dtype=np.uint8), (2, 1)), DEV)
    damp.quantize_state(L, S, perms, state)
    before = state.clone()
    d = P.inputs_to_dev(w, wl.step_inputs(w, 0), DEV)
    slot_idx = torch.tensor([1, 9], dtype=torch.int32, device=DEV)
    o = torch.full((2, 2, 128), 7.0, device=DEV)
    damp.kda_decode_step(L, state, perms, d["q"], d["k"], d["v"], d["g"], d["beta"], o=o, slot_idx=slot_idx)
    torch.cuda.synchronize()
    assert damp.device_status() == damp.DEV_BAD_SLOT
    assert torch.equal(state[0], before[0])          # slot 0 not named: untouched
    assert not torch.equal(state[1], before[1])      # slot 1 updated
    assert torch.all(o[1] == 7.0)                    # the skipped row's output untouched
    assert damp.device_status() == 0


def test_status_of_a_side_stream_step_is_read_without_a_sync():
    """device_status() waits for kernels on every stream, including PyTorch's
    non-blocking side streams: a bad slot reported by a step still in flight there is
    returned, not cleared unread."""
    w = wl.KDA_B256.replace(batch=2, heads=2, qk_heads=2)
    L = P.layout_of(w)
    state = damp.new_state(L, 2, DEV)
    perms = P.to_dev(np.tile(np.arange(128, dtype=np.uint8), (2, 1)), DEV)
    d = P.inputs_to_dev(w, wl.step_inputs(w, 0), DEV)
    slot_idx = torch.tensor([0, 5], dtype=torch.int32, device=DEV)
    side = torch.cuda.Stream(device=DEV)
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        for _ in range(3):
            damp.kda_decode_step(L, state, perms, d["q"], d["k"], d["v"], d["g"], d["beta"], slot_idx=slot_idx,
                                 stream=side)
    assert damp.device_status() == damp.DEV_BAD_SLOT  # no synchronize before the read
    assert damp.device_status() == 0


def test_empty_batch_is_a_no_op():
    w = wl.KDA_B256.replace(batch=1, heads=2, qk_heads=2)
    L = P.layout_of(w)
    state = damp.new_state(L, 1, DEV)
    e = torch.empty((0, 2, 128), dtype=torch.bfloat16, device=DEV)
    o = damp.kda_decode_step(L, state, torch.zeros((2, 128), dtype=torch.uint8, device=DEV), e, e, e,
                             torch.empty((0, 2, 128), device=DEV), torch.empty((0, 2), device=DEV))
    assert o.shape == (0, 2, 128)
