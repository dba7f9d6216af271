"""Free-running drift of the packed state against the FP32-state trajectory.

A stack of alternating GDN / KDA layers runs many decode steps from the same FP32
prefix state twice: once on the packed state, once on the FP32 state (the FP32
kernel is itself checked against the oracle).  Drift is the held-out trajectory
RRMSE of App. E, (sum_t ||Y^_t - Y_t||^2 / sum_t ||Y_t||^2)^(1/2), of the outputs and
of the states.  Protecting the calibrated high-risk channels (K_hi = 16, error
energy x persistence, Algorithm 1) must drift less than uniform INT8 + H_32.
"""
import numpy as np
import pytest
import torch

import paper_2608_27513_gb300 as damp
import workloads as wl
from oracle import runs
from tests import parity as P

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda:0")


def _layer_drift(w: wl.Workload, perms: np.ndarray, steps: int):
    L = P.layout_of(w)
    S = torch.zeros((w.batch, w.heads, w.d_k, w.d_v), device=DEV)
    o = torch.empty((w.batch, w.heads, w.d_v), device=DEV)
    fp32_step = damp.fp32_kda_decode_step if w.kind == "kda" else damp.fp32_gdn_decode_step
    for t in range(w.prefix):
        d = P.inputs_to_dev(w, wl.step_inputs(w, t, wl.STREAM_PREFIX), DEV)
        fp32_step(L, S, d["q"], d["k"], d["v"], d["g"], d["beta"], o=o)
    dperm = P.to_dev(perms, DEV)
    state = damp.new_state(L, w.batch, DEV)
    damp.quantize_state(L, S, dperm, state)
    step = damp.kda_decode_step if w.kind == "kda" else damp.gdn_decode_step
    num_o = den_o = num_s = den_s = 0.0
    for t in range(steps):
        d = P.inputs_to_dev(w, wl.step_inputs(w, t), DEV)
        oq = step(L, state, dperm, d["q"], d["k"], d["v"], d["g"], d["beta"])
        fp32_step(L, S, d["q"], d["k"], d["v"], d["g"], d["beta"], o=o)
        num_o += float(((oq - o) ** 2).sum())
        den_o += float((o ** 2).sum())
        if (t + 1) % 16 == 0:
            Sq = damp.dequantize_state(L, state, dperm)
            num_s += float(((Sq - S) ** 2).sum())
            den_s += float((S ** 2).sum())
    assert damp.device_status() == 0
    return np.sqrt(num_o / den_o), np.sqrt(num_s / den_s)


@pytest.mark.parametrize("layer", [0, 1])  # GDN, KDA
def test_calibrated_mixed_precision_drifts_less_than_uniform_int8(layer):
    base = wl.stack_layer(layer, 16).replace(batch=16, heads=8, qk_heads=8, prefix=64)
    perms, _ = runs.calibrate_layout(base, n_docs=4, n_tokens=64)
    rr_damp = _layer_drift(base, perms, 96)
    uniform = base.replace(k_hi=0)
    rr_int8 = _layer_drift(uniform, np.tile(np.arange(base.d_k, dtype=np.uint8), (base.heads, 1)), 96)
    assert all(np.isfinite(rr_damp)) and all(np.isfinite(rr_int8))
    assert rr_damp[0] < 0.05 and rr_damp[1] < 0.05
    assert rr_damp[0] < rr_int8[0] and rr_damp[1] < rr_int8[1], (rr_damp, rr_int8)
