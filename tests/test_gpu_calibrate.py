"""GPU key-channel selection (Algorithm 1) against the oracle: error energy and
log-decay accumulators within FP32 summation tolerance, the selection bit for bit
on the same scores, and a whole calibration run against the oracle's."""
import numpy as np
import pytest
import torch

import paper_2608_27513_gb300 as damp
import workloads as wl
from oracle import calibrate, core, runs
from paper_2608_27513_gb300 import calibration
from tests import parity as P

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda:0")


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2608_27513_gb300 import build
    build.build()
    torch.cuda.init()
    yield
    assert damp.device_status() == 0


@pytest.mark.parametrize("fmt", [0, 1, 2, 3, 4, 5])
def test_error_energy_matches_oracle(fmt):
    B, H, dk, dv = 6, 3, 64, 96
    L = damp.Layout(H, H, dk, dv, 8, fmt)
    S1 = wl.random_states(41, B * H, dk, dv).reshape(B, H, dk, dv)
    S2 = wl.random_states(42, B * H, dk, dv, scale=0.1).reshape(B, H, dk, dv)
    E = torch.zeros((H, dk), device=DEV)
    for S in (S1, S2):
        damp.calib_error_energy(L, P.to_dev(S, DEV), E)
    ref = np.zeros((H, dk))
    for S in (S1, S2):
        for h in range(H):
            ref[h] += calibrate.error_energy_samples(np.ascontiguousarray(S[:, h]), fmt).sum(axis=0)
    got = E.cpu().numpy().astype(np.float64)
    # a group whose s sits at a binary16 rounding midpoint may take the neighbouring s
    # (the decode parity's tie rule): its error energy, quadratic in s, moves by up to
    # 2 * 2^-10 relative
    tol = 2.5e-3 if fmt != 2 else 1e-4
    assert np.all(np.abs(got - ref) <= tol * ref + 1e-12), np.max(np.abs(got - ref) / (ref + 1e-30))


@pytest.mark.parametrize("kda", [False, True])
def test_log_decay_accumulates(kda):
    B, H, dk = 5, 4, 32
    L = damp.Layout(H, H, dk, 64, 0, 0)
    rng = np.random.default_rng(43)
    gs = [(-np.exp(rng.uniform(-6, 0, (B, H, dk) if kda else (B, H)))).astype(np.float32) for _ in range(3)]
    G = torch.zeros((H, dk), device=DEV)
    for g in gs:
        damp.calib_log_decay(L, P.to_dev(g, DEV), G)
    ref = sum(g.astype(np.float64).sum(axis=0) for g in gs)
    ref = ref if kda else np.repeat(ref[:, None], dk, axis=1)
    assert np.all(np.abs(G.cpu().numpy() - ref) <= 1e-5 * np.abs(ref) + 1e-6)


@pytest.mark.parametrize("k_hi", [0, 5, 16, 64])
def test_selection_matches_oracle_on_the_same_scores(k_hi):
    """pi from the GPU's FP32 scores equals the oracle's TopK + stable partition of the
    same scores, ties included; the scores follow the float64 definition."""
    H, dk = 6, 64
    L = damp.Layout(H, H, dk, 64, k_hi, 0)
    rng = np.random.default_rng(44 + k_hi)
    E = rng.random((H, dk)).astype(np.float32)
    E[:, ::7] = E[:, 1:2]                                   # repeated error energies: ties in C
    G = (-np.exp(rng.uniform(-8, 0, (H, dk)))).astype(np.float32)
    G[0] = G[0, 0]                                          # a GDN-like head: one decay for all channels
    G[1, :8] = -1e-7                                        # decays at the persistence cap
    n_s, n_t = 3, 4
    C, perm = damp.calib_select(L, P.to_dev(E * n_s, DEV), n_s, P.to_dev(G * n_t, DEV), n_t, 1e-4)
    C, perm = C.cpu().numpy(), perm.cpu().numpy()
    for h in range(H):
        _, pi = calibrate.select_layout(C[h], np.ones(dk), k_hi)
        assert np.array_equal(perm[h], pi)
    Cref = E.astype(np.float64) * calibrate.persistence(np.exp(G.astype(np.float64)))
    assert np.all(np.abs(C - Cref) <= 1e-4 * Cref + 1e-12)
    assert np.allclose(C[1, :8] / E[1, :8], 1e4, rtol=1e-3)  # persistence at its cap 1/tau


@pytest.mark.parametrize("kind", ["gdn", "kda"])
def test_calibration_run_matches_oracle(kind):
    """A whole calibration run (FP32 trajectories, samples every 8 tokens) on the GPU
    against the oracle's on the same documents: scores close, protected sets equal
    except between channels whose oracle scores are within 1 % at the K_hi boundary."""
    w = wl.stack_layer(0 if kind == "gdn" else 1, 16).replace(heads=4, qk_heads=4)
    n_docs, n_tokens = 8, 64
    docs = list(range(n_docs))
    dt = torch.bfloat16 if w.in_dtype == "bf16" else torch.float32
    inputs = []
    for t in range(n_tokens):
        inp = wl.step_inputs(w, t, wl.STREAM_CALIB, docs)
        inputs.append({key: P.to_dev(val, DEV, dt if key in ("q", "k", "v") else None) for key, val in inp.items()})
    L = P.layout_of(w)
    C, perm = calibration.calibrate(L, kind, inputs)
    E, a_eff = runs.calibration_stats(w, n_docs, n_tokens)
    Cref = E * calibrate.persistence(a_eff)
    C = C.cpu().numpy().astype(np.float64)
    assert np.all(np.abs(C - Cref) <= 2e-2 * Cref + 1e-12), np.max(np.abs(C - Cref) / Cref)
    perm = perm.cpu().numpy()
    for h in range(w.heads):
        ref_prot = set(calibrate.topk(Cref[h], w.k_hi).tolist())
        got_prot = set(perm[h][:w.k_hi].tolist())
        kth = np.sort(Cref[h])[::-1][w.k_hi - 1]
        for u in ref_prot ^ got_prot:
            assert abs(Cref[h][u] - kth) <= 1e-2 * kth, (h, u)


@pytest.mark.parametrize("kind,fmt", [("kda", 0), ("gdn", 2), ("kda", 3)])
def test_accumulate_in_one_call_equals_the_per_token_calls(kind, fmt):
    """damp_calib_accumulate enqueues the same kernels in the same order as one FP32 step
    per token, an error-energy pass every 8 tokens and one log-decay call over all rows:
    the FP32 states and both accumulators are identical, bit for bit."""
    w = (wl.stack_layer(1, 16) if kind == "kda" else wl.stack_layer(0, 16)).replace(batch=4, lo_format=fmt)
    L = damp.Layout(w.heads, w.qk_heads, w.d_k, w.d_v, w.k_hi, w.lo_format)
    T, every = 20, 8
    inputs = wl.torch_step_inputs(w, T, DEV)
    stacked = {n: torch.stack([d[n] for d in inputs]) for n in ("q", "k", "v", "g", "beta")}
    S1 = damp.new_fp32_state(L, w.batch, DEV)
    E1 = torch.zeros((w.heads, w.d_k), device=DEV)
    G1 = torch.zeros_like(E1)
    n_samples, n_rows = damp.calib_accumulate(L, kind, S1, stacked["q"], stacked["k"], stacked["v"], stacked["g"],
                                              stacked["beta"], E1, G1, every)
    assert (n_samples, n_rows) == (w.batch * (T // every), w.batch * T)
    S2 = damp.new_fp32_state(L, w.batch, DEV)
    E2 = torch.zeros_like(E1)
    G2 = torch.zeros_like(E1)
    step = damp.fp32_kda_decode_step if kind == "kda" else damp.fp32_gdn_decode_step
    for t, d in enumerate(inputs):
        step(L, S2, d["q"], d["k"], d["v"], d["g"], d["beta"])
        if (t + 1) % every == 0:
            damp.calib_error_energy(L, S2, E2)
    damp.calib_log_decay(L, stacked["g"].flatten(0, 1), G2)
    torch.cuda.synchronize()
    assert torch.equal(S1, S2)
    assert torch.equal(E1, E2)
    assert torch.equal(G1, G2)
    assert damp.device_status() == 0
