"""The Python binding checks every tensor's shape (and dtype) against the layout and
the batch before it calls the library: the C ABI sees raw pointers only, so a
mis-sized tensor would otherwise be read or written out of bounds.  These tests run
on the host with CPU tensors and a library stand-in that fails the test if any
compute entry point is reached."""
import numpy as np
import pytest
import torch

import paper_2608_27513_gb300 as damp
from paper_2608_27513_gb300 import _lib, build, checkpoint

H, HQK, DK, DV, K = 4, 2, 64, 64, 8
B, T = 3, 5


class _NoCompute:
    """The real library for sizes and strings; any other call is an error."""
    SIZE_CALLS = {"damp_slot_bytes", "damp_record_bytes", "damp_validate_layout", "damp_status_string",
                  "damp_bits_per_value", "damp_version"}

    def __init__(self, real):
        self.real = real
        self.calls = []

    def __getattr__(self, name):
        if name in self.SIZE_CALLS:
            return getattr(self.real, name)

        def forbidden(*a, **kw):
            self.calls.append(name)
            raise AssertionError(f"{name} was called with mis-sized arguments")
        return forbidden


@pytest.fixture()
def fake(monkeypatch):
    build.build()
    f = _NoCompute(_lib.lib())
    monkeypatch.setattr(damp, "lib", lambda: f)
    yield f
    assert f.calls == []


def _layout(fmt=0, k=K):
    return damp.Layout(H, HQK, DK, DV, k, fmt)


def _ops(kind, lead=(B,), dt=torch.bfloat16):
    g = torch.zeros(lead + ((H, DK) if kind == "kda" else (H,)))
    return dict(q=torch.zeros(lead + (HQK, DK), dtype=dt), k=torch.zeros(lead + (HQK, DK), dtype=dt),
                v=torch.zeros(lead + (H, DV), dtype=dt), g=g, beta=torch.zeros(lead + (H,)))


def _pool(L, slots=8):
    return torch.zeros((slots, damp.slot_bytes(L)), dtype=torch.uint8)


def _perm():
    return torch.zeros((H, DK), dtype=torch.uint8)


def _bad_ops(kind, lead):
    """(what, operand dict) pairs, each with one operand of the wrong size or dtype."""
    good = _ops(kind, lead)
    out = []
    for name, t in good.items():
        shp = list(t.shape)
        shp[-1] += 1
        bad = dict(good)
        bad[name] = torch.zeros(shp, dtype=t.dtype)
        out.append((f"{name} last dim", bad))
    bad = dict(good)
    bad["q"] = torch.zeros(lead + (H, DK), dtype=torch.bfloat16)  # H instead of H_qk
    out.append(("q heads", bad))
    bad = dict(good)
    bad["g"] = torch.zeros(lead + ((H,) if kind == "kda" else (H, DK)))  # the other kind's gate
    out.append(("g rank", bad))
    bad = dict(good)
    bad["beta"] = torch.zeros(lead + (H,), dtype=torch.float64)
    out.append(("beta dtype", bad))
    return out


@pytest.mark.parametrize("kind", ["gdn", "kda"])
def test_decode_step_rejects_missized_operands(fake, kind):
    L = _layout()
    step = damp.gdn_decode_step if kind == "gdn" else damp.kda_decode_step
    for what, ops in _bad_ops(kind, (B,)):
        with pytest.raises(ValueError, match="shape|dtype"):
            step(L, _pool(L), _perm(), **ops)
    ops = _ops(kind)
    cases = [
        dict(state=torch.zeros((8, damp.slot_bytes(L) - 16), dtype=torch.uint8)),     # slot size
        dict(state=torch.zeros((8 * damp.slot_bytes(L),), dtype=torch.uint8)),       # not [slots, bytes]
        dict(perm=torch.zeros((H, DK - 1), dtype=torch.uint8)),
        dict(perm=torch.zeros((H + 1, DK), dtype=torch.uint8)),
        dict(o=torch.zeros((B, H, DV - 32))),
        dict(o=torch.zeros((B + 1, H, DV))),
        dict(slot_idx=torch.zeros((B + 1,), dtype=torch.int32)),
        dict(slot_idx=torch.zeros((B,), dtype=torch.int64)),
        dict(num_slots=9),                                                            # beyond the pool
        dict(state=_pool(L, slots=2)),                                                 # B > slots, no slot_idx
    ]
    for kw in cases:
        args = dict(state=_pool(L), perm=_perm())
        args.update(kw)
        state, perm = args.pop("state"), args.pop("perm")
        with pytest.raises(ValueError, match="shape|dtype|exceeds"):
            step(L, state, perm, **ops, **args)


def test_correct_shapes_pass_the_checks(fake):
    """Well-formed CPU tensors get through every size check and stop only at the
    device check, so the checks do not reject what the header allows."""
    L = _layout()
    for kind, step in (("gdn", damp.gdn_decode_step), ("kda", damp.kda_decode_step)):
        with pytest.raises(ValueError, match="CUDA"):
            step(L, _pool(L), _perm(), **_ops(kind), o=torch.zeros((B, H, DV)),
                 slot_idx=torch.zeros((B,), dtype=torch.int32))
    with pytest.raises(ValueError, match="CUDA"):
        damp.fp32_kda_decode_step(L, torch.zeros((B, H, DK, DV)), **_ops("kda"))
    with pytest.raises(ValueError, match="CUDA"):
        damp.kda_prefill_chunk(L, _pool(L), _perm(), **_ops("kda", (B, T)),
                               lengths=torch.zeros((B,), dtype=torch.int32))
    with pytest.raises(ValueError, match="CUDA"):
        damp.quantize_state(L, torch.zeros((B, H, DK, DV)), _perm(), _pool(L))
    with pytest.raises(ValueError, match="CUDA"):
        damp.pack_tiers(L, torch.zeros((B, H, K, DV), dtype=torch.int16),
                        torch.zeros((B, H, DK - K, DV), dtype=torch.uint8),
                        torch.zeros((B, H, DK - K, DV // 32, 2), dtype=torch.int16), _pool(L))


def test_fp32_step_rejects_missized_state(fake):
    L = _layout()
    for st in (torch.zeros((B, H, DK, DV + 32)), torch.zeros((B, H - 1, DK, DV)),
               torch.zeros((B, H, DK, DV), dtype=torch.float16)):
        with pytest.raises(ValueError, match="shape|dtype"):
            damp.fp32_gdn_decode_step(L, st, **_ops("gdn"))
    for what, ops in _bad_ops("gdn", (B,)):
        with pytest.raises(ValueError, match="shape|dtype"):
            damp.fp32_gdn_decode_step(L, torch.zeros((B, H, DK, DV)), **ops)


@pytest.mark.parametrize("kind", ["gdn", "kda"])
def test_prefill_rejects_missized_operands(fake, kind):
    L = _layout()
    fn = damp.gdn_prefill_chunk if kind == "gdn" else damp.kda_prefill_chunk
    for what, ops in _bad_ops(kind, (B, T)):
        with pytest.raises(ValueError, match="shape|dtype"):
            fn(L, _pool(L), _perm(), **ops)
    ops = _ops(kind, (B, T))
    ops["q"] = torch.zeros((B, T + 1, HQK, DK), dtype=torch.bfloat16)  # another chunk length
    with pytest.raises(ValueError, match="shape"):
        fn(L, _pool(L), _perm(), **ops)
    for kw in (dict(lengths=torch.zeros((B + 1,), dtype=torch.int32)), dict(o=torch.zeros((B, T, H, DV + 32))),
               dict(slot_idx=torch.zeros((B - 1,), dtype=torch.int32))):
        with pytest.raises(ValueError, match="shape|dtype"):
            fn(L, _pool(L), _perm(), **_ops(kind, (B, T)), **kw)


def test_conversions_and_tiers_reject_missized_tensors(fake):
    L = _layout()
    S = torch.zeros((B, H, DK, DV))
    for bad in (torch.zeros((B, H, DK, DV + 32)), torch.zeros((B, H + 1, DK, DV)),
                torch.zeros((B, H, DK, DV), dtype=torch.float64)):
        with pytest.raises(ValueError, match="shape|dtype"):
            damp.quantize_state(L, bad, _perm(), _pool(L))
    with pytest.raises(ValueError, match="shape"):
        damp.quantize_state(L, S, _perm(), _pool(L), slot_idx=torch.zeros((B + 2,), dtype=torch.int32))
    with pytest.raises(ValueError, match="shape"):
        damp.dequantize_state(L, _pool(L), _perm(), batch=B, S=torch.zeros((B, H, DK, DV - 32)))
    with pytest.raises(ValueError, match="shape"):
        damp.dequantize_state(L, _pool(L), torch.zeros((H, DK + 1), dtype=torch.uint8), batch=B)
    hi = torch.zeros((B, H, K, DV), dtype=torch.int16)
    codes = torch.zeros((B, H, DK - K, DV), dtype=torch.uint8)
    meta = torch.zeros((B, H, DK - K, DV // 32, 2), dtype=torch.int16)
    for h2, c2, m2 in ((torch.zeros((B, H, K + 1, DV), dtype=torch.int16), codes, meta),
                       (hi, torch.zeros((B, H, DK - K, DV // 2), dtype=torch.uint8), meta),
                       (hi, codes, torch.zeros((B, H, DK - K, DV // 32, 2), dtype=torch.float32)),
                       (hi, codes, torch.zeros((B - 1, H, DK - K, DV // 32, 2), dtype=torch.int16))):
        with pytest.raises(ValueError, match="shape|byte"):
            damp.pack_tiers(L, h2, c2, m2, _pool(L))
    with pytest.raises(ValueError, match="exceeds"):
        damp.unpack_tiers(L, _pool(L, slots=2), batch=3)


def test_calibration_rejects_missized_accumulators(fake):
    L = _layout(k=0)
    with pytest.raises(ValueError, match="shape"):
        damp.calib_error_energy(L, torch.zeros((B, H, DK, DV)), torch.zeros((H, DK + 1)))
    with pytest.raises(ValueError, match="shape"):
        damp.calib_error_energy(L, torch.zeros((B, H, DK - 1, DV)), torch.zeros((H, DK)))
    with pytest.raises(ValueError, match="shape"):
        damp.calib_log_decay(L, torch.zeros((B, H + 1)), torch.zeros((H, DK)))
    with pytest.raises(ValueError, match="shape"):
        damp.calib_log_decay(L, torch.zeros((B, H, DK)), torch.zeros((H - 1, DK)))
    with pytest.raises(ValueError, match="shape"):
        damp.calib_select(L, torch.zeros((H, DK)), 1, torch.zeros((H, DK - 1)), 1)


def test_checkpoint_restore_into_a_missized_target_is_rejected(fake, tmp_path):
    """A saved state restored into a pool of another layout, or for another number of
    slot indices, stops at the binding's checks."""
    L = _layout()
    path = str(tmp_path / "s.npz")
    hi = np.zeros((B, H, K, DV), np.int16)
    np.savez(path, hi=hi, codes=np.zeros((B, H, DK - K, DV), np.uint8),
             meta=np.zeros((B, H, DK - K, DV // 32, 2), np.int16),
             layout=np.array([H, HQK, DK, DV, K, 0], np.int32))
    with pytest.raises(ValueError, match="shape"):
        checkpoint.load_state(path, L, _pool(L), slot_idx=torch.zeros((B + 1,), dtype=torch.int32))
    with pytest.raises(ValueError, match="shape"):
        checkpoint.load_state(path, L, torch.zeros((8, damp.slot_bytes(L) + 16), dtype=torch.uint8))
