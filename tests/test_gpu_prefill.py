"""GPU parity of the prefill chunk (App. A.5 "Prefill path") through the C ABI against
the oracle: outputs of every token within the decode tolerance, the chunk-final
packed state within the tie rules of the decode step."""
import numpy as np
import pytest
import torch

import paper_2608_27513_gb300 as damp
import workloads as wl
from oracle import runs
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


def _run(w, T, lengths=None, slot_of=None, pool=None, chunks=1, o_offset=None, g_scale=1.0):
    rows = list(range(w.batch))
    perms, _ = runs.calibrate_layout(w, n_docs=2, n_tokens=16)
    perm_units, tiers = P.initial_tiers(w, rows, perms, prefix=min(w.prefix, 24))
    L = P.layout_of(w)
    state = damp.new_state(L, pool or len(rows), DEV)
    slot_idx = None if slot_of is None else torch.tensor([slot_of[b] for b in rows], dtype=torch.int32, device=DEV)
    lens = np.full(len(rows), T, np.int32) if lengths is None else np.asarray(lengths, np.int32)
    lens_units = np.repeat(lens, w.heads)
    dperm = P.to_dev(perms, DEV)
    stats = P.CodeStats()
    fn = damp.kda_prefill_chunk if w.kind == "kda" else damp.gdn_prefill_chunk
    dt = torch.bfloat16 if w.in_dtype == "bf16" else torch.float32
    for ch in range(chunks):
        # teacher-forced: every chunk starts from the oracle's packed state
        damp.pack_tiers(L, *P.tiers_to_dev(w, tiers, len(rows), DEV), state, slot_idx=slot_idx)
        inp = P.chunk_inputs(w, ch * T, T, rows)
        if g_scale != 1.0:  # stronger decay (the same log-decays on both sides)
            inp["g"] = (inp["g"] * np.float32(g_scale)).astype(np.float32)
        u = P.unit_chunk(w, inp, T)
        o_ref, tiers, lo_pre = P.oracle_chunk(w, perm_units, tiers, u, lens_units)
        d = {key: P.to_dev(val, DEV, dt if key in ("q", "k", "v") else None) for key, val in inp.items()}
        o_arg = None
        if o_offset is not None:  # o at an offset of o_offset floats from a 16-byte boundary
            n = len(rows) * T * w.heads * w.d_v
            o_arg = torch.zeros(n + 4, device=DEV)[o_offset:o_offset + n].view(len(rows), T, w.heads, w.d_v)
        o = fn(L, state, dperm, d["q"], d["k"], d["v"], d["g"], d["beta"], o=o_arg,
               lengths=None if lengths is None else P.to_dev(lens, DEV), slot_idx=slot_idx)
        torch.cuda.synchronize()
        o = o.cpu().numpy().transpose(0, 2, 1, 3).reshape(len(rows) * w.heads, T, w.d_v)
        for i in range(o.shape[0]):
            P.compare_o(o[i, :lens_units[i]], o_ref[i, :lens_units[i]], f"{w.name} chunk {ch} unit {i}")
        got = P.tiers_from_dev(w, damp.unpack_tiers(L, state, batch=len(rows), slot_idx=slot_idx),
                               len(rows) * w.heads)
        P.compare_tiers(w, tiers, got, lo_pre, stats, f"{w.name} chunk {ch}")
    stats.check_fraction()
    return state, L, dperm, slot_idx


def test_kda_chunk_matches_oracle():
    """KDA, H = 8, d = 128, K_hi = 10, BF16 inputs, 16-token chunks, two chunks in a row."""
    _run(wl.KDA_B256.replace(batch=2, heads=8, qk_heads=8), 16, chunks=2)


def test_gdn_gqa_chunk_matches_oracle():
    _run(wl.GDN_B64_GQA.replace(batch=2), 8)


def test_ragged_lengths_and_slot_indirection():
    """Rows of 9, 3 and 0 tokens in a 9-token chunk, scattered over a larger pool; the
    zero-length row's slot stays as it was."""
    w = wl.KDA_B256.replace(batch=3, heads=4, qk_heads=4)
    _run(w, 9, lengths=[9, 3, 0], slot_of={0: 5, 1: 0, 2: 2}, pool=6)


@pytest.mark.parametrize("w", [
    wl.Workload("gdn_d64_dv96_k5_f1", "gdn", 2, 4, 2, 64, 96, 5, 4, 8, "fp32", 21, 1),
    wl.Workload("kda_uniform", "kda", 1, 4, 4, 128, 64, 0, 4, 8, "bf16", 22, 0),
    wl.Workload("kda_all_fp16", "kda", 1, 2, 2, 32, 64, 32, 4, 8, "fp32", 23, 0),
    wl.Workload("gdn_d32_k3", "gdn", 2, 2, 1, 32, 32, 3, 4, 8, "bf16", 24, 0),
], ids=lambda w: w.name)
def test_layouts(w):
    _run(w, 6)


@pytest.mark.parametrize("w", [
    wl.Workload("gdn_d64_dv96_k5_f1", "gdn", 2, 4, 2, 64, 96, 5, 4, 8, "fp32", 21, 1),
    wl.Workload("kda_uniform", "kda", 1, 4, 4, 128, 64, 0, 4, 8, "bf16", 22, 0),
    wl.Workload("kda_d64_all_fp16", "kda", 1, 2, 2, 64, 64, 64, 4, 8, "fp32", 23, 0),
    wl.Workload("kda_k31_f1", "kda", 2, 2, 1, 128, 32, 31, 4, 8, "bf16", 25, 1),
    wl.Workload("gdn_k127", "gdn", 1, 2, 2, 128, 64, 127, 4, 8, "fp32", 26, 0),
], ids=lambda w: w.name)
def test_layouts_long_chunks(w):
    """Chunks of 32 and more tokens on the UINT8 tiers (d_k 64 and 128) run the kernel
    that holds the tile in key-channel order: odd K_hi, all-FP16 and uniform tiers,
    d_v = 32 and 96."""
    _run(w, 32)


def test_long_chunk_ragged_lengths_and_slot_indirection():
    """Rows of 33, 17 and 0 tokens in a 33-token chunk, scattered over a larger pool."""
    w = wl.GDN_B64_GQA.replace(batch=3, heads=4, qk_heads=2)
    _run(w, 33, lengths=[33, 17, 0], slot_of={0: 4, 1: 1, 2: 0}, pool=5)


def test_unaligned_output_runs_the_short_chunk_kernel():
    """o that is not 16-byte aligned: a long chunk runs the kernel with 4-byte stores."""
    _run(wl.KDA_B256.replace(batch=2, heads=4, qk_heads=4), 32, o_offset=1)


def test_decode_after_prefill_reads_the_chunk_state():
    """The decode step continues from the chunk-final packed state that the GPU chunk
    wrote (the hand-off of the prefill path), matching the oracle's step from it."""
    w = wl.KDA_B256.replace(batch=2, heads=4, qk_heads=4)
    state, L, dperm, _ = _run(w, 5)
    got_tiers = P.tiers_from_dev(w, damp.unpack_tiers(L, state), w.batch * w.heads)
    inp = wl.step_inputs(w, 5, rows=list(range(w.batch)))
    perms = dperm.cpu().numpy()
    o_ref, new_ref, lo_pre = P.oracle_step(w, np.tile(perms, (w.batch, 1)), got_tiers, runs.unit_operands(w, inp))
    d = P.inputs_to_dev(w, inp, DEV)
    o = damp.kda_decode_step(L, state, dperm, d["q"], d["k"], d["v"], d["g"], d["beta"])
    P.compare_o(o.cpu().numpy().reshape(-1, w.d_v), o_ref, "decode after prefill")
    stats = P.CodeStats()
    P.compare_tiers(w, new_ref, P.tiers_from_dev(w, damp.unpack_tiers(L, state), w.batch * w.heads), lo_pre, stats,
                    "decode after prefill")
    stats.check_fraction()
