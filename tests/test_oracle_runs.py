"""The oracle's plain drivers on the small GDN workload (B=1, H=4, d=64) and the input recipe."""
import numpy as np

import workloads as wl
from oracle import calibrate, core, runs


def test_inputs_are_seeded_and_rowwise_reproducible():
    w = wl.GDN_B64_GQA
    a = wl.step_inputs(w, 3, rows=[5, 9])
    b = wl.step_inputs(w, 3, rows=[9])
    assert np.array_equal(a["q"][1], b["q"][0]) and np.array_equal(a["g"][1], b["g"][0])
    c = wl.step_inputs(w, 4, rows=[9])
    assert not np.array_equal(b["v"], c["v"])
    # recipe: unit-norm q/k (before bf16 rounding), beta in (0,1), decay in (0,1)
    assert np.allclose(np.linalg.norm(a["q"], axis=-1), 1, atol=1e-2)
    assert np.all((a["beta"] > 0) & (a["beta"] < 1)) and np.all(a["g"] < 0)
    # bf16 values: low 16 bits clear
    assert np.all((a["v"].view(np.uint32) & 0xFFFF) == 0)


def test_round_bf16_matches_torch():
    import torch
    x = np.random.default_rng(0).standard_normal(10000).astype(np.float32) * 100
    ours = wl.round_bf16(x)
    ref = torch.from_numpy(x).to(torch.bfloat16).float().numpy()
    assert np.array_equal(ours, ref)


def test_kda_decay_profile_range():
    w = wl.KDA_B256
    g = wl.step_inputs(w, 0, rows=[0])["g"]
    a = np.exp(g)
    assert a.min() > 0.3 and a.max() < 0.9999


def test_calibrated_layout_on_small_gdn():
    w = wl.GDN_B1_D64
    perms, scores = runs.calibrate_layout(w, n_docs=4, n_tokens=32)
    assert perms.shape == (w.heads, w.d_k)
    for h in range(w.heads):
        assert sorted(perms[h].tolist()) == list(range(w.d_k))
        prot = perms[h][: w.k_hi]
        assert np.all(np.diff(prot.astype(int)) > 0)
        # the protected channels carry the K_hi largest scores
        assert scores[h][prot].min() >= np.delete(scores[h], prot).max()


def test_prefix_then_quantized_decode_stays_close_to_fp32():
    w = wl.GDN_B1_D64
    perms, _ = runs.calibrate_layout(w, n_docs=2, n_tokens=16)
    S0 = runs.prefix_states(w, rows=[0]).reshape(w.heads, w.d_k, w.d_v)
    tiers = core.pack_heads(perms, S0, w.k_hi, w.lo_format)
    S_ref = core.unpack_heads(perms, *tiers, w.k_hi, w.lo_format, w.d_k, w.d_v)
    num = den = 0.0
    for t, o, _ in runs.decode_trajectory(w, perms, tiers, [0], range(w.heads), w.steps):
        u = runs.unit_operands(w, wl.step_inputs(w, t, rows=[0]))
        o_ref = core.delta_step_heads(S_ref, u["q"], u["k"], u["v"], u["g"], u["beta"], w.kind)
        num += float(((o - o_ref) ** 2).sum())
        den += float((o_ref ** 2).sum())
    rrmse = np.sqrt(num / den)  # App. E trajectory RRMSE of the output
    assert 0 < rrmse < 0.05


def test_gqa_mapping_is_consecutive_pairs():
    """Reading of the GQA mapping (not in the paper): value head h reads q/k head
    floor(h * H_qk / H), so with 32 value heads over 16 q/k heads heads 2j and 2j+1 share
    q/k head j; without GQA the map is the identity.  unit_operands takes q and k rows
    through that map and v, beta, g through the value head."""
    w = wl.GDN_B64_GQA
    assert (w.heads, w.qk_heads) == (32, 16)
    assert [wl.qk_head_of(w, h) for h in range(32)] == [h // 2 for h in range(32)]
    assert [wl.qk_head_of(wl.KDA_B256, h) for h in range(32)] == list(range(32))
    inp = wl.step_inputs(w, 0, rows=[2])
    u = runs.unit_operands(w, inp, heads=[5, 6])
    assert np.array_equal(u["q"][0], inp["q"][0, 2]) and np.array_equal(u["k"][1], inp["k"][0, 3])
    assert np.array_equal(u["v"][1], inp["v"][0, 6]) and u["beta"][0] == inp["beta"][0, 5]
