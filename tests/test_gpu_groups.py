"""Head groups: a layer whose heads keep different numbers of FP16 key channels (the
decay-tiered allocation of App. E) runs as one layout, pool and permutation table per
K_hi, each with a head map into the layer's heads.

  * Split at one K_hi, the groups must reproduce the uniform layer bit for bit, head
    for head (same kernels, same arithmetic; only the indexing of operands, outputs
    and S differs), for every call that takes a head map.
  * Split at two K_hi, each group must match the oracle at its own K_hi.
  * A head map entry outside the layer sets DAMP_DEV_BAD_HEAD and leaves that head alone.
"""
import numpy as np
import pytest
import torch

import paper_2608_27513_gb300 as damp
import workloads as wl
from oracle import core, runs
from paper_2608_27513_gb300 import calibration, checkpoint
from tests import parity as P

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda:0")
HEADS_A = [0, 3, 5, 6]
HEADS_B = [1, 2, 4, 7]


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2608_27513_gb300 import build
    build.build()
    torch.cuda.init()
    assert damp.device_status() == 0
    yield
    assert damp.device_status() == 0


def _group(L, heads, K=None):
    m = torch.tensor(heads, dtype=torch.int32, device=DEV)
    return damp.Layout(len(heads), L.num_qk_heads, L.d_k, L.d_v, L.k_hi if K is None else K, L.lo_format,
                       model_heads=L.num_heads, head_map=m)


def _layer(w, seed):
    S = P.to_dev(wl.random_states(seed, w.batch * w.heads, w.d_k, w.d_v, scale=0.3)
                 .reshape(w.batch, w.heads, w.d_k, w.d_v), DEV)
    rng = np.random.default_rng(seed)
    perm = P.to_dev(np.stack([rng.permutation(w.d_k) for _ in range(w.heads)]).astype(np.uint8), DEV)
    return S, perm


def _chunk(w, T):
    steps = [wl.step_inputs(w, t) for t in range(T)]
    dt = torch.bfloat16 if w.in_dtype == "bf16" else None
    return {k: P.to_dev(np.stack([s[k] for s in steps], axis=1), DEV, dt if k in ("q", "k", "v") else None)
            for k in steps[0]}


@pytest.mark.parametrize("kind", ["gdn", "kda"])
@pytest.mark.parametrize("fmt,K", [(0, 10), (1, 6), (2, 8), (3, 8), (5, 0)])
def test_groups_at_one_k_hi_reproduce_the_layer(kind, fmt, K):
    w = wl.sweep(kind, K, fmt).replace(batch=3, heads=8, qk_heads=4)  # GQA: pairs of heads share q/k
    L = P.layout_of(w)
    S, perm = _layer(w, 91)
    pool = damp.new_state(L, w.batch, DEV)
    damp.quantize_state(L, S, perm, pool)
    groups = [(_group(L, hs), hs) for hs in (HEADS_A, HEADS_B)]
    pools = []
    for G, hs in groups:
        pg = damp.new_state(G, w.batch, DEV)
        damp.quantize_state(G, S, perm[hs].contiguous(), pg)
        pools.append(pg)
    step = damp.kda_decode_step if kind == "kda" else damp.gdn_decode_step
    for t in range(2):
        d = P.inputs_to_dev(w, wl.step_inputs(w, t), DEV)
        o = step(L, pool, perm, d["q"], d["k"], d["v"], d["g"], d["beta"])
        og = torch.full_like(o, float("nan"))
        for (G, hs), pg in zip(groups, pools):
            step(G, pg, perm[hs].contiguous(), d["q"], d["k"], d["v"], d["g"], d["beta"], o=og)
        assert torch.equal(og, o), f"step {t}: o differs"
    whole = damp.unpack_tiers(L, pool)
    for (G, hs), pg in zip(groups, pools):
        part = damp.unpack_tiers(G, pg)
        for a, b in zip(part, whole):
            assert torch.equal(a, b[:, hs]), "packed tiers differ"
        # read-out into the layer's S rows of the group
        back = damp.dequantize_state(G, pg, perm[hs].contiguous())
        full = damp.dequantize_state(L, pool, perm)
        assert torch.equal(back[:, hs], full[:, hs])
        others = [h for h in range(w.heads) if h not in hs]
        assert bool((back[:, others] == 0).all())


@pytest.mark.parametrize("fmt,T", [(0, 5), (3, 5), (0, 32), (1, 40)])
def test_group_prefill_chunks_reproduce_the_layer(fmt, T):
    """Both chunk kernels (5 tokens; 32 and 40 tokens on the UINT8 tiers) with head maps."""
    w = wl.KDA_B256.replace(batch=2, heads=8, qk_heads=8, lo_format=fmt, k_hi=12)
    L = P.layout_of(w)
    S, perm = _layer(w, 92)
    pool = damp.new_state(L, w.batch, DEV)
    damp.quantize_state(L, S, perm, pool)
    c = _chunk(w, T)
    lens = torch.tensor([T, 3], dtype=torch.int32, device=DEV)
    o = damp.kda_prefill_chunk(L, pool, perm, c["q"], c["k"], c["v"], c["g"], c["beta"], lengths=lens)
    og = torch.zeros_like(o)
    for hs in (HEADS_A, HEADS_B):
        G = _group(L, hs)
        pg = damp.new_state(G, w.batch, DEV)
        damp.quantize_state(G, S, perm[hs].contiguous(), pg)
        damp.kda_prefill_chunk(G, pg, perm[hs].contiguous(), c["q"], c["k"], c["v"], c["g"], c["beta"], o=og,
                               lengths=lens)
        for a, b in zip(damp.unpack_tiers(G, pg), damp.unpack_tiers(L, pool)):
            assert torch.equal(a, b[:, hs])
    assert torch.equal(og, o)


@pytest.mark.parametrize("fmt,T", [(0, 64), (1, 40)])
def test_group_gdn_prefill_on_the_tensor_cores_reproduces_the_layer(fmt, T):
    """The GDN tensor-core chunk (d = 128, bf16, 32+ tokens) with head maps and GQA."""
    w = wl.sweep("gdn", 12, fmt).replace(batch=2, heads=8, qk_heads=4)
    L = P.layout_of(w)
    S, perm = _layer(w, 93)
    pool = damp.new_state(L, w.batch, DEV)
    damp.quantize_state(L, S, perm, pool)
    c = _chunk(w, T)
    lens = torch.tensor([T, 17], dtype=torch.int32, device=DEV)
    o = damp.gdn_prefill_chunk(L, pool, perm, c["q"], c["k"], c["v"], c["g"], c["beta"], lengths=lens)
    og = torch.zeros_like(o)
    for hs in (HEADS_A, HEADS_B):
        G = _group(L, hs)
        pg = damp.new_state(G, w.batch, DEV)
        damp.quantize_state(G, S, perm[hs].contiguous(), pg)
        damp.gdn_prefill_chunk(G, pg, perm[hs].contiguous(), c["q"], c["k"], c["v"], c["g"], c["beta"], o=og,
                               lengths=lens)
        for a, b in zip(damp.unpack_tiers(G, pg), damp.unpack_tiers(L, pool)):
            assert torch.equal(a, b[:, hs])
    assert torch.equal(og, o)


@pytest.mark.parametrize("kind", ["gdn", "kda"])
def test_decay_tiered_groups_match_oracle(kind):
    """Fast-decay heads with K_hi = 4, slow-decay heads with K_hi = 28 (mean 16, App. E):
    teacher-forced steps of each group against the oracle at its own K_hi."""
    w = wl.sweep(kind, 16, 0).replace(batch=2, heads=8, qk_heads=4)
    L = P.layout_of(w)
    rows = list(range(w.batch))
    perms, _ = runs.calibrate_layout(w, n_docs=2, n_tokens=16)
    S0 = runs.prefix_states(w, rows, steps=16)  # [B, H, d_k, d_v]
    step = damp.kda_decode_step if kind == "kda" else damp.gdn_decode_step
    for hs, K in ((HEADS_A, 4), (HEADS_B, 28)):
        G = _group(L, hs, K)
        wg = w.replace(heads=len(hs), k_hi=K)
        perm_units = np.tile(perms[hs], (w.batch, 1))
        tiers = core.pack_heads(perm_units, S0[:, hs].reshape(-1, w.d_k, w.d_v), K, 0)
        pg = damp.new_state(G, w.batch, DEV)
        dperm = P.to_dev(perms[hs], DEV)
        stats = P.CodeStats()
        for t in range(3):
            inp = wl.step_inputs(w, t)
            u = runs.unit_operands(w, inp, heads=hs)
            o_ref, new_ref, lo_pre = P.oracle_step(wg, perm_units, tiers, u)
            damp.pack_tiers(G, *P.tiers_to_dev(wg, tiers, w.batch, DEV), pg)
            d = P.inputs_to_dev(w, inp, DEV)
            o = step(G, pg, dperm, d["q"], d["k"], d["v"], d["g"], d["beta"])
            P.compare_o(o[:, hs].cpu().numpy().reshape(-1, w.d_v), o_ref, f"group K={K} step {t}")
            got = P.tiers_from_dev(wg, damp.unpack_tiers(G, pg), w.batch * len(hs))
            P.compare_tiers(wg, new_ref, got, lo_pre, stats, f"group K={K} step {t}")
            tiers = new_ref
        stats.check_fraction()


def test_head_groups_partition_and_calibration():
    ks = [4, 28, 28, 4, 28, 4, 4, 28]
    groups = damp.head_groups(ks, num_qk_heads=8, d_k=128, d_v=128, device=DEV)
    assert [K for K in (g.k_hi for g, _ in groups)] == [4, 28]
    assert sorted(h for _, hs in groups for h in hs) == list(range(8))
    # bytes of the ragged layer = the mean K_hi's (equal-sized groups)
    common = damp.Layout(8, 8, 128, 128, 16)
    assert sum(damp.slot_bytes(g) for g, _ in groups) == damp.slot_bytes(common)
    # calibration: one pass over all heads, each group selects at its own K_hi
    w = wl.sweep("kda", 16, 0).replace(batch=4, heads=8, qk_heads=8)
    inputs = wl.torch_step_inputs(w, 24, DEV)
    sel = calibration.calibrate_groups(groups, "kda", inputs)
    full = damp.Layout(8, 8, 128, 128, 0)
    E, n_s, G, n_t = calibration.accumulate(full, "kda", inputs)
    for (L, hs), (C, pi) in zip(groups, sel):
        Cf, pif = damp.calib_select(damp.Layout(8, 8, 128, 128, L.k_hi), E, n_s, G, n_t, 1e-4)
        assert torch.equal(C, Cf[hs]) and torch.equal(pi, pif[hs])


def test_bad_head_map_entry_is_flagged_and_skipped():
    w = wl.KDA_B256.replace(batch=2, heads=4, qk_heads=4, k_hi=8)
    L = P.layout_of(w)
    S, perm = _layer(w, 93)
    m = torch.tensor([0, 9, 2, 3], dtype=torch.int32, device=DEV)  # 9 is outside the layer's 4 heads
    G = damp.Layout(4, 4, 128, 128, 8, 0, model_heads=4, head_map=m)
    good = damp.Layout(4, 4, 128, 128, 8, 0, model_heads=4,
                       head_map=torch.tensor([0, 1, 2, 3], dtype=torch.int32, device=DEV))
    pool = damp.new_state(L, w.batch, DEV)
    damp.quantize_state(good, S, perm, pool)
    assert damp.device_status() == 0
    before = damp.unpack_tiers(L, pool)
    d = P.inputs_to_dev(w, wl.step_inputs(w, 0), DEV)
    o = damp.kda_decode_step(G, pool, perm, d["q"], d["k"], d["v"], d["g"], d["beta"])
    assert damp.device_status() == damp.DEV_BAD_HEAD
    after = damp.unpack_tiers(L, pool)
    for a, b in zip(after, before):
        assert torch.equal(a[:, 1], b[:, 1])          # the bad head's records are untouched
        assert not torch.equal(a[:, 0], b[:, 0])
    assert bool((o[:, 1] == 0).all())                  # and no output row was written for it


def test_group_layout_checkpoint_round_trip(tmp_path):
    L = damp.Layout(8, 4, 128, 128, 16)
    G = _group(L, HEADS_B, 28)
    perms = np.stack([np.random.default_rng(h).permutation(128) for h in range(4)]).astype(np.uint8)
    path = str(tmp_path / "group.json")
    checkpoint.save_layout(path, G, perms)
    G2, p2 = checkpoint.load_layout(path, device=DEV)
    assert G2 == G and G2.heads_of_operands == 8
    assert G2.head_map.cpu().tolist() == HEADS_B and np.array_equal(p2, perms)


def _same_up_to_ties(G, a, b, what):
    """Two pools of one group layout that hold the same updated states up to the rounding
    of float-ordering ties: the one-launch group step runs compile-time layouts, one call
    per group the general instance, and their instruction streams may round one value of
    a rare tie differently.  FP16 rows equal; codes within 1 LSB on at most 1e-5 of the
    entries; every reconstructed value within one quantization step of its group."""
    ha, ca, ma = damp.unpack_tiers(G, a)
    hb, cb, mb = damp.unpack_tiers(G, b)
    assert torch.equal(ha, hb), f"{what}: FP16 rows differ"
    dc = (ca.int() - cb.int()).abs()
    assert float((dc > 0).float().mean()) <= 1e-5, f"{what}: {int((dc > 0).sum())} codes differ"
    same_meta = (ma == mb).all(dim=-1)
    if bool(same_meta.all()):
        assert int(dc.max()) <= 1, f"{what}: a code moved by {int(dc.max())}"
    assert float((~same_meta).float().mean()) <= 1e-5, f"{what}: {int((~same_meta).sum())} group scales differ"
    perm = torch.stack([torch.arange(G.d_k, dtype=torch.uint8, device=DEV)] * G.num_heads)
    Sa = damp.dequantize_state(G, a, perm)
    Sb = damp.dequantize_state(G, b, perm)
    s = ma[..., 0].view(torch.float16).float().abs().amax()
    assert float((Sa - Sb).abs().max()) <= float(s) * 1.0001, f"{what}: reconstruction moved by more than a step"


@pytest.mark.parametrize("kind", ["gdn", "kda"])
@pytest.mark.parametrize("fmt,ka,kb", [(0, 12, 20), (0, 8, 24), (1, 4, 28), (0, 28, 4), (0, 10, 6)])
def test_group_step_reproduces_the_group_calls(kind, fmt, ka, kb):
    """damp_*_decode_step_groups: the K_hi pairs of the paper's head-budget table run as one
    launch (either order of the groups), other pairs as one launch per group; o equals one
    decode-step call per group bit for bit, the records up to float-ordering ties."""
    w = wl.sweep(kind, ka, fmt).replace(batch=3, heads=8, qk_heads=4)
    L = P.layout_of(w)
    S, perm = _layer(w, 93)
    groups = [(_group(L, HEADS_A, ka), HEADS_A), (_group(L, HEADS_B, kb), HEADS_B)]
    pools = {}
    for tag in ("one", "each"):
        pools[tag] = []
        for G, hs in groups:
            pg = damp.new_state(G, w.batch, DEV)
            damp.quantize_state(G, S, perm[hs].contiguous(), pg)
            pools[tag].append(pg)
    perms = [perm[hs].contiguous() for _, hs in groups]
    step = damp.kda_decode_step if kind == "kda" else damp.gdn_decode_step
    gstep = damp.kda_decode_step_groups if kind == "kda" else damp.gdn_decode_step_groups
    for t in range(3):
        d = P.inputs_to_dev(w, wl.step_inputs(w, t), DEV)
        o_each = torch.full((w.batch, w.heads, w.d_v), float("nan"), device=DEV)
        for (G, hs), pg, pm in zip(groups, pools["each"], perms):
            step(G, pg, pm, d["q"], d["k"], d["v"], d["g"], d["beta"], o=o_each)
        o_one = gstep([(G, pg, pm) for (G, _), pg, pm in zip(groups, pools["one"], perms)],
                      d["q"], d["k"], d["v"], d["g"], d["beta"])
        assert torch.equal(o_one, o_each), f"step {t}: o differs"
        for (G, _), a, b in zip(groups, pools["one"], pools["each"]):
            _same_up_to_ties(G, a, b, f"step {t}")


@pytest.mark.parametrize("kind", ["gdn", "kda"])
def test_group_step_full_batch_4_28(kind):
    """B=256, H=32, d=128, half the heads at K_hi = 4 and half at 28 (the tiered bench's
    split), with slot indirection: the one-launch step equals the per-group calls (o bit
    for bit, records up to float-ordering ties)."""
    w = wl.sweep(kind, 4).replace(batch=256)
    L = P.layout_of(w)
    S, perm = _layer(w.replace(batch=4), 94)
    S = S.repeat(64, 1, 1, 1)
    heads_fast = list(range(0, 32, 2))
    heads_slow = list(range(1, 32, 2))
    groups = [(_group(L, heads_fast, 4), heads_fast), (_group(L, heads_slow, 28), heads_slow)]
    perms = [perm[hs].contiguous() for _, hs in groups]
    slot_idx = torch.randperm(300, device=DEV)[:256].to(torch.int32)
    pools = {}
    for tag in ("one", "each"):
        pools[tag] = []
        for (G, hs), pm in zip(groups, perms):
            pg = damp.new_state(G, 300, DEV)
            damp.quantize_state(G, S, pm, pg, slot_idx=slot_idx)
            pools[tag].append(pg)
    step = damp.kda_decode_step if kind == "kda" else damp.gdn_decode_step
    gstep = damp.kda_decode_step_groups if kind == "kda" else damp.gdn_decode_step_groups
    d = P.inputs_to_dev(w, wl.step_inputs(w, 0), DEV)
    o_each = torch.zeros((w.batch, w.heads, w.d_v), device=DEV)
    for (G, _), pg, pm in zip(groups, pools["each"], perms):
        step(G, pg, pm, d["q"], d["k"], d["v"], d["g"], d["beta"], o=o_each, slot_idx=slot_idx)
    o_one = gstep([(G, pg, pm) for (G, _), pg, pm in zip(groups, pools["one"], perms)],
                  d["q"], d["k"], d["v"], d["g"], d["beta"], slot_idx=slot_idx)
    assert torch.equal(o_one, o_each)
    for (G, _), a, b in zip(groups, pools["one"], pools["each"]):
        _same_up_to_ties(G, a, b, "full batch")


@pytest.mark.parametrize("kind", ["gdn", "kda"])
def test_group_step_skips_a_bad_slot_and_head_in_the_second_group(kind):
    """One-launch group step (K_hi 8/24) whose second group maps a head outside the layer
    and whose slot list names a slot outside the pool (every warp meets the skipped tiles
    in its second body, after a first body that ran whole).  Both flags are raised, the
    bad slot's and head's records and output rows stay as they were, and the rest equals
    the per-group calls."""
    w = wl.sweep(kind, 8, 0).replace(batch=3, heads=8, qk_heads=4)
    L = P.layout_of(w)
    S, perm = _layer(w, 95)
    heads_b = [1, 2, 11, 7]  # 11 is outside the layer's 8 heads
    ga = _group(L, HEADS_A, 8)
    gb = damp.Layout(4, L.num_qk_heads, L.d_k, L.d_v, 24, L.lo_format, model_heads=L.num_heads,
                     head_map=torch.tensor(heads_b, dtype=torch.int32, device=DEV))
    good_b = _group(L, [1, 2, 4, 7], 24)
    perms = [perm[HEADS_A].contiguous(), perm[[1, 2, 4, 7]].contiguous()]
    setup = torch.tensor([2, 1, 0], dtype=torch.int32, device=DEV)
    slot_idx = torch.tensor([2, 7, 0], dtype=torch.int32, device=DEV)  # a pool of 3 slots: 7 is outside
    pools = {}
    for tag in ("one", "each"):
        pools[tag] = []
        for G, pm in ((ga, perms[0]), (good_b, perms[1])):
            pg = damp.new_state(G, 3, DEV)
            damp.quantize_state(G, S, pm, pg, slot_idx=setup)
            pools[tag].append(pg)
    assert damp.device_status() == 0
    before = [damp.unpack_tiers(G, pg) for G, pg in zip((ga, good_b), pools["one"])]
    step = damp.kda_decode_step if kind == "kda" else damp.gdn_decode_step
    gstep = damp.kda_decode_step_groups if kind == "kda" else damp.gdn_decode_step_groups
    d = P.inputs_to_dev(w, wl.step_inputs(w, 0), DEV)
    o_each = torch.zeros((w.batch, w.heads, w.d_v), device=DEV)
    for G, pg, pm in zip((ga, gb), pools["each"], perms):
        step(G, pg, pm, d["q"], d["k"], d["v"], d["g"], d["beta"], o=o_each, slot_idx=slot_idx)
    assert damp.device_status() == damp.DEV_BAD_SLOT | damp.DEV_BAD_HEAD
    o_one = torch.zeros_like(o_each)
    gstep([(G, pg, pm) for G, pg, pm in zip((ga, gb), pools["one"], perms)],
          d["q"], d["k"], d["v"], d["g"], d["beta"], o=o_one, slot_idx=slot_idx)
    assert damp.device_status() == damp.DEV_BAD_SLOT | damp.DEV_BAD_HEAD
    assert torch.equal(o_one, o_each)
    assert bool((o_one[1] == 0).all()) and bool((o_one[:, 4] == 0).all())  # the bad slot's row, head 4 (unmapped)
    after = [damp.unpack_tiers(G, pg) for G, pg in zip((ga, good_b), pools["one"])]
    for a, b in zip(after[1], before[1]):
        assert torch.equal(a[1], b[1])        # slot 1 was not named by the step
        assert torch.equal(a[2, 2], b[2, 2])  # the unmapped held head (slot 2 = batch row 0)
        assert not torch.equal(a[2, 0], b[2, 0])
    for (G, a, b) in zip((ga, good_b), pools["one"], pools["each"]):
        _same_up_to_ties(G, a, b, "bad slot and head")
