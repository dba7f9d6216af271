"""The C-ABI library on the host: it loads, exports every symbol include/damp.h
declares, sizes its records as documented, and rejects bad arguments before
enqueueing anything (no call here reaches the GPU)."""
import ctypes
import os
import re

import pytest

import paper_2608_27513_gb300 as damp
from paper_2608_27513_gb300 import _lib, build
from oracle import core
from tests.golden.load import paper_values

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def L():
    build.build()
    return _lib.lib()


def declared_functions():
    src = open(os.path.join(ROOT, "include", "damp.h")).read()
    return sorted(set(re.findall(r"DAMP_API\s+[\w\s\*]+?\b(damp_\w+)\s*\(", src)))


def test_header_declares_the_expected_entry_points():
    names = declared_functions()
    for n in ("damp_gdn_decode_step", "damp_kda_decode_step", "damp_quantize_state", "damp_dequantize_state",
              "damp_fp32_gdn_decode_step", "damp_fp32_kda_decode_step", "damp_u8_gdn_decode_step",
              "damp_u8_kda_decode_step", "damp_pack_tiers", "damp_unpack_tiers"):
        assert n in names


def test_library_exports_every_declared_symbol(L):
    for name in declared_functions():
        assert hasattr(L, name), name
    assert set(declared_functions()) == set(_lib.SIGNATURES)


def test_library_has_no_cpu_fallback_symbols(L):
    # the product library is CUDA only: it does not link the oracle
    out = os.popen(f"nm -D {_lib.LIB_PATH}").read()
    assert "dor_" not in out


def _layout(**kw):
    base = dict(num_heads=32, num_qk_heads=32, d_k=128, d_v=128, k_hi=16, lo_format=0)
    base.update(kw)
    return damp.Layout(**base)


def test_record_geometry_and_bits(L):
    pv = paper_values()
    for K in (0, 4, 8, 10, 16, 32, 128):
        lay = _layout(k_hi=K)
        logical = 64 * K + 32 * (128 - K) + 4 * (128 - K)  # per value block: FP16 rows, codes, (s, z)
        assert damp.record_bytes(lay) == (logical + 15) // 16 * 16
        assert damp.slot_bytes(lay) == 32 * 4 * damp.record_bytes(lay)
        assert damp.bits_per_value(lay) == 8.0 * logical / (128 * 32)
    assert damp.bits_per_value(_layout(k_hi=16)) == pv["damp_bits_k16_dk128"]
    # row-absmax INT8: one FP32 scale per row counted once, as the oracle's logical tiers
    for K in (0, 5, 16, 128):
        for dv in (64, 128, 1024):
            lay = _layout(k_hi=K, lo_format=2, d_v=dv)
            assert damp.bits_per_value(lay) == pytest.approx(core.bits_per_value(128, dv, K, core.FMT_S8_ROW), rel=1e-12)
            assert damp.record_bytes(lay) == damp.record_bytes(_layout(k_hi=K, d_v=dv))
    # 4-bit and FP8 tiers: bits from the oracle's logical tiers; 4-bit code rows take 16 bytes
    for fmt in (3, 4, 5):
        for K in (0, 10, 16):
            lay = _layout(k_hi=K, lo_format=fmt)
            assert damp.bits_per_value(lay) == pytest.approx(core.bits_per_value(128, 128, K, fmt), rel=1e-12)
            code_row = 16 if fmt in (3, 4) else 32
            logical = 128 * ((K + 1) // 2) + (code_row + 4) * (128 - K)
            assert damp.record_bytes(lay) == (logical + 15) // 16 * 16
    assert damp.bits_per_value(_layout(k_hi=0)) == pv["bits_int8_hadamard"]


@pytest.mark.parametrize("kw,status", [
    (dict(d_k=96), 2), (dict(d_k=256), 2), (dict(d_v=48), 2), (dict(d_v=2048), 2), (dict(k_hi=129), 2),
    (dict(k_hi=-1), 2), (dict(num_qk_heads=5), 2), (dict(num_heads=0), 2), (dict(lo_format=6), 5)])
def test_layout_validation(L, kw, status):
    c = _layout(**kw).c()
    assert L.damp_validate_layout(ctypes.byref(c)) == status
    assert L.damp_record_bytes(ctypes.byref(c)) == 0
    assert L.damp_bits_per_value(ctypes.byref(c)) == -1.0


def test_head_group_layouts(L):
    """Head groups (layers with per-head K_hi): held heads, model heads and the map."""
    fb = FakeBuffers(n=2, size=4096)

    def v(H, Hq, Hm, m):
        c = _lib.DampLayout(H, Hq, 128, 128, 16, 0, Hm, m)
        return L.damp_validate_layout(ctypes.byref(c)), c

    st, ok = v(4, 4, 8, fb[0])
    assert st == 0
    assert L.damp_slot_bytes(ctypes.byref(ok)) == 4 * 4 * damp.record_bytes(_layout(k_hi=16))
    assert v(3, 4, 8, fb[0])[0] == 0                      # a group need not hold whole q/k groups
    assert v(4, 4, 0, None)[0] == 0                       # model_heads 0: the held heads
    assert v(4, 4, 8, None)[0] == 2                       # more model heads but no map
    assert v(8, 4, 4, fb[0])[0] == 2                      # fewer model heads than held heads
    assert v(4, 3, 8, fb[0])[0] == 2                      # model heads not a multiple of the q/k heads
    assert v(4, 4, -1, fb[0])[0] == 2
    assert v(4, 4, 8, ctypes.c_void_p(fb.ptrs[0] + 2))[0] == 3   # a misaligned map
    # the FP32-state baseline holds every model head: a head map is rejected before launch
    _, c = v(4, 4, 4, fb[0])
    assert L.damp_fp32_kda_decode_step(ctypes.byref(c), fb[1], 4, None, 4, fb[1], fb[1], fb[1], fb[1], fb[1],
                                       fb[1], 0, None) == 2


class FakeBuffers:
    """Distinct, aligned host addresses standing in for device buffers (never dereferenced)."""

    def __init__(self, n=16, size=1 << 24):
        self.bufs = [ctypes.create_string_buffer(size + 256) for _ in range(n)]
        self.ptrs = [(ctypes.addressof(b) + 255) // 256 * 256 for b in self.bufs]

    def __getitem__(self, i):
        return ctypes.c_void_p(self.ptrs[i])


def _call_step(L, lay, fb, **over):
    c = lay.c()
    args = dict(layout=ctypes.byref(c), state=fb[0], num_slots=4, slot_idx=None, batch=4, perm=fb[1], q=fb[2],
                k=fb[3], v=fb[4], g=fb[5], beta=fb[6], o=fb[7], in_dtype=0, stream=None)
    args.update(over)
    return L.damp_kda_decode_step(*args.values())


def test_step_rejects_bad_arguments_before_launch(L):
    fb = FakeBuffers()
    lay = _layout()
    off = lambda i, d: ctypes.c_void_p(fb.ptrs[i] + d)
    assert _call_step(L, lay, fb, batch=0) == 0                      # empty batch: nothing enqueued
    assert _call_step(L, lay, fb, batch=-1) == 2
    assert _call_step(L, lay, fb, state=None) == 1
    assert _call_step(L, lay, fb, perm=None) == 1
    assert _call_step(L, lay, fb, o=None) == 1
    assert _call_step(L, lay, fb, num_slots=3) == 2                   # fewer slots than rows, no slot_idx
    assert _call_step(L, lay, fb, state=off(0, 8)) == 3
    assert _call_step(L, lay, fb, q=off(2, 4)) == 3
    assert _call_step(L, lay, fb, g=off(5, 4)) == 3                   # KDA gates are bulk-copied: 16 B
    assert _call_step(L, lay, fb, o=off(7, 2)) == 3
    assert _call_step(L, lay, fb, in_dtype=7) == 5
    assert _call_step(L, lay, fb, o=off(0, 4096)) == 4                # o inside the pool
    assert _call_step(L, lay, fb, q=off(0, 1 << 12)) == 4             # an input inside the pool
    assert _call_step(L, lay, fb, o=fb[2]) == 4                       # o over q
    assert _call_step(L, _layout(lo_format=6), fb) == 5
    c = _layout(k_hi=8).c()
    assert L.damp_u8_kda_decode_step(ctypes.byref(c), *[fb[0], 4, None, 4, fb[1], fb[2], fb[3], fb[4], fb[5],
                                                        fb[6], fb[7], 0, None]) == 2


def _call_prefill(L, lay, fb, **over):
    c = lay.c()
    args = dict(layout=ctypes.byref(c), state=fb[0], num_slots=4, slot_idx=None, batch=4, chunk_len=8, lengths=None,
                perm=fb[1], q=fb[2], k=fb[3], v=fb[4], g=fb[5], beta=fb[6], o=fb[7], in_dtype=0, stream=None)
    args.update(over)
    return L.damp_kda_prefill_chunk(*args.values())


def test_prefill_rejects_bad_arguments_before_launch(L):
    fb = FakeBuffers()
    lay = _layout()
    off = lambda i, d: ctypes.c_void_p(fb.ptrs[i] + d)
    assert _call_prefill(L, lay, fb, batch=0) == 0                   # nothing enqueued
    assert _call_prefill(L, lay, fb, chunk_len=0) == 0
    assert _call_prefill(L, lay, fb, chunk_len=-1) == 2
    assert _call_prefill(L, lay, fb, v=None) == 1
    assert _call_prefill(L, lay, fb, lengths=off(8, 2)) == 3
    assert _call_prefill(L, lay, fb, q=off(2, 8)) == 3
    assert _call_prefill(L, lay, fb, o=off(0, 64)) == 4               # o inside the pool
    assert _call_prefill(L, lay, fb, lengths=off(7, 0)) == 4          # lengths under o
    assert _call_prefill(L, _layout(lo_format=2, d_v=256), fb) == 2   # row-absmax chunks need d_v <= 128
    assert _call_prefill(L, lay, fb, in_dtype=3) == 5


def test_calibration_calls_reject_bad_arguments(L):
    fb = FakeBuffers()
    c = _layout().c()
    off = lambda i, d: ctypes.c_void_p(fb.ptrs[i] + d)
    assert L.damp_calib_error_energy(ctypes.byref(c), fb[0], 0, fb[1], None) == 0   # empty batch
    assert L.damp_calib_error_energy(ctypes.byref(c), None, 4, fb[1], None) == 1
    assert L.damp_calib_error_energy(ctypes.byref(c), off(0, 4), 4, fb[1], None) == 3
    assert L.damp_calib_error_energy(ctypes.byref(c), fb[0], 4, off(0, 64), None) == 4  # accumulator inside S
    assert L.damp_calib_log_decay(ctypes.byref(c), fb[0], -1, 1, fb[1], None) == 2
    assert L.damp_calib_log_decay(ctypes.byref(c), fb[0], 4, 1, off(1, 2), None) == 3
    sel = lambda **kw: L.damp_calib_select(ctypes.byref(c), *dict(dict(E=fb[0], ns=4, G=fb[1], nt=8,
                                                                       tau=ctypes.c_float(1e-4), C=fb[2],
                                                                       perm=fb[3], stream=None), **kw).values())
    assert sel(ns=0) == 2
    assert sel(tau=ctypes.c_float(0.0)) == 2
    assert sel(perm=None) == 1
    assert sel(perm=off(2, 16)) == 4                                                  # pi over the scores


def test_a_launch_failure_is_reported_not_raised(L):
    """With no CUDA device, a call that passes every host check returns DAMP_ERR_CUDA
    (the launcher's error, mapped at the boundary).  Skipped where a GPU is visible: the
    fake host addresses must never reach a kernel."""
    import torch
    if torch.cuda.is_available():
        pytest.skip("a GPU is visible")
    fb = FakeBuffers()
    assert _call_step(L, _layout(), fb) == 6
    assert L.damp_status_string(6).decode().startswith("DAMP_ERR_CUDA")


def test_gdn_gate_alignment_is_4_bytes(L):
    fb = FakeBuffers()
    c = _layout().c()
    args = [ctypes.byref(c), fb[0], 4, None, 4, fb[1], fb[2], fb[3], fb[4], ctypes.c_void_p(fb.ptrs[5] + 5),
            fb[6], fb[7], 0, None]
    assert L.damp_gdn_decode_step(*args) == 3


def test_conversions_reject_bad_arguments(L):
    fb = FakeBuffers()
    c = _layout().c()
    assert L.damp_quantize_state(ctypes.byref(c), None, fb[1], fb[0], 4, None, 4, None) == 1
    assert L.damp_quantize_state(ctypes.byref(c), fb[2], fb[1], fb[0], 4, None, 8, None) == 2
    assert L.damp_dequantize_state(ctypes.byref(c), fb[0], 4, None, 4, fb[1], fb[0], None) == 4
    assert L.damp_pack_tiers(ctypes.byref(c), fb[2], None, fb[4], fb[0], 4, None, 4, None) == 1
    assert L.damp_unpack_tiers(ctypes.byref(c), fb[0], 4, None, 4, fb[2], fb[2], fb[4], None) == 4
    assert L.damp_device_status(None) == 1


def test_status_strings(L):
    for s in range(7):
        assert L.damp_status_string(s).decode().startswith("DAMP_")


def test_wait_test_hook_accepts_only_its_layout(L):
    """The bounded-wait test hook runs one kernel instance: any other layout or input
    type is rejected on the host, before a launch."""
    fb = FakeBuffers()
    for kw in (dict(k_hi=16), dict(d_k=64, k_hi=10), dict(lo_format=1, k_hi=10)):
        c = _layout(**kw).c()
        assert L.damp_test_kda_wait_timeout(ctypes.byref(c), fb[0], 4, None, 4, fb[1], fb[2], fb[3], fb[4], fb[5],
                                            fb[6], fb[7], 0, None) == 2
    c = _layout(k_hi=10).c()
    assert L.damp_test_kda_wait_timeout(ctypes.byref(c), fb[0], 4, None, 4, fb[1], fb[2], fb[3], fb[4], fb[5],
                                        fb[6], fb[7], 1, None) == 2  # FP32 inputs
    assert L.damp_test_kda_wait_timeout(ctypes.byref(c), fb[0], 4, None, 0, fb[1], fb[2], fb[3], fb[4], fb[5],
                                        fb[6], fb[7], 0, None) == 0  # empty batch: nothing enqueued


def test_group_step_rejects_bad_arguments_before_launch(L):
    """damp_*_decode_step_groups checks every group and the groups against each other
    before anything is enqueued (fake host pointers: nothing is dereferenced)."""
    fb = FakeBuffers()

    def grp(k_hi, map_buf, **kw):
        base = dict(num_heads=4, num_qk_heads=4, d_k=128, d_v=128, k_hi=k_hi, lo_format=0, model_heads=8)
        base.update(kw)
        c = _lib.DampLayout(base["num_heads"], base["num_qk_heads"], base["d_k"], base["d_v"], base["k_hi"],
                            base["lo_format"], base["model_heads"], map_buf)
        return c

    def call(cs, states=None, perms=(10, 11), n=None, batch=4, slots=(4, 4), **kw):
        n = len(cs) if n is None else n
        arr = (_lib.DampLayout * max(len(cs), 1))(*cs)
        st = (ctypes.c_void_p * 2)(*(states or (fb.ptrs[8], fb.ptrs[9])))
        pm = (ctypes.c_void_p * 2)(*[fb.ptrs[i] for i in perms])
        ns = (ctypes.c_int64 * 2)(*slots)
        args = dict(slot_idx=None, q=fb[2], k=fb[3], v=fb[4], g=fb[5], beta=fb[6], o=fb[7], in_dtype=0, stream=None)
        args.update(kw)
        return L.damp_kda_decode_step_groups(arr, n, st, ns, pm, args["slot_idx"], batch, args["q"], args["k"],
                                             args["v"], args["g"], args["beta"], args["o"], args["in_dtype"],
                                             args["stream"])

    a, b = grp(8, fb.ptrs[12]), grp(24, fb.ptrs[13])
    assert call([a, b], batch=0) == 0                                         # empty batch: nothing enqueued
    assert call([a, b], n=0) == 2
    assert call([a, b], n=9) == 2
    assert call([a, grp(24, None, model_heads=0)]) == 2                       # a group without a head map
    assert call([a, grp(24, fb.ptrs[13], d_v=64)]) == 2                       # operand shapes differ
    assert call([a, grp(24, fb.ptrs[13], model_heads=16)]) == 2
    assert call([a, grp(24, fb.ptrs[13], lo_format=1)]) == 5                  # formats differ
    assert call([a, b], states=(fb.ptrs[8], fb.ptrs[8] + 4096)) == 4         # overlapping pools
    assert call([a, b], o=ctypes.c_void_p(fb.ptrs[9] + 64)) == 4              # o inside a pool
    assert call([a, b], in_dtype=7) == 5
    assert call([a, b], states=(fb.ptrs[8], fb.ptrs[9] + 8)) == 3            # a misaligned pool
    assert L.damp_kda_decode_step_groups(None, 2, None, None, None, None, 4, fb[2], fb[3], fb[4], fb[5], fb[6],
                                         fb[7], 0, None) == 1


def test_calib_accumulate_rejects_bad_arguments_before_launch(L):
    fb = FakeBuffers()
    off = lambda i, d: ctypes.c_void_p(fb.ptrs[i] + d)

    def call(lay=None, **over):
        c = (lay or _layout(k_hi=0)).c()
        args = dict(S=fb[0], n_docs=4, n_tokens=8, q=fb[1], k=fb[2], v=fb[3], g=fb[4], beta=fb[5], in_dtype=0,
                    kda=1, every=8, E=fb[6], G=fb[7], stream=None)
        args.update(over)
        return L.damp_calib_accumulate(ctypes.byref(c), *args.values())

    assert call(n_docs=0) == 0 and call(n_tokens=0) == 0            # nothing to do: nothing enqueued
    assert call(every=0) == 2 and call(n_docs=-1) == 2
    assert call(in_dtype=9) == 5
    assert call(S=None) == 1 and call(E=None) == 1 and call(beta=None) == 1
    assert call(S=off(0, 8)) == 3 and call(g=off(4, 4)) == 3          # KDA gates: 16-B aligned
    assert call(E=fb[7]) == 4                                          # E_acc over G_acc
    assert call(q=off(0, 4096)) == 4                                   # an input inside the states
    lay = damp.Layout(4, 4, 128, 128, 0, 0, model_heads=8, head_map=None)
    c = lay.c()
    c.head_map = fb.ptrs[8]
    assert L.damp_calib_accumulate(ctypes.byref(c), fb[0], 4, 8, fb[1], fb[2], fb[3], fb[4], fb[5], 0, 1, 8, fb[6],
                                   fb[7], None) == 2                   # a head group: not a whole layer
