"""CUDA-graph capture of the decode step and the prefill chunk: after one eager call
(which performs the per-device set-up: symbol addresses, shared-memory limits), the
launches capture into a graph whose replays give the same bits as eager launches."""
import numpy as np
import pytest
import torch

import paper_2608_27513_gb300 as damp
import workloads as wl
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


def _setup(w, seed):
    L = P.layout_of(w)
    S = P.to_dev(wl.random_states(seed, w.batch * w.heads, w.d_k, w.d_v, scale=0.3)
                 .reshape(w.batch, w.heads, w.d_k, w.d_v), DEV)
    perm = P.to_dev(np.tile(np.random.default_rng(seed).permutation(w.d_k).astype(np.uint8), (w.heads, 1)), DEV)
    state = damp.new_state(L, w.batch, DEV)
    damp.quantize_state(L, S, perm, state)
    return L, perm, state


@pytest.mark.parametrize("fmt,K", [(0, 10), (0, 13), (3, 8)])
def test_decode_steps_replay_from_a_graph(fmt, K):
    w = wl.KDA_B256.replace(batch=4, heads=8, qk_heads=8, k_hi=K, lo_format=fmt)
    L, perm, state = _setup(w, 81)
    eager = state.clone()
    inputs = [P.inputs_to_dev(w, wl.step_inputs(w, t), DEV) for t in range(3)]
    o_e = torch.empty((w.batch, w.heads, w.d_v), device=DEV)
    o_g = torch.empty_like(o_e)
    d0 = inputs[0]
    damp.kda_decode_step(L, eager, perm, d0["q"], d0["k"], d0["v"], d0["g"], d0["beta"], o=o_e)  # set-up
    damp.kda_decode_step(L, state, perm, d0["q"], d0["k"], d0["v"], d0["g"], d0["beta"], o=o_g)
    static = {k: v.clone() for k, v in d0.items()}
    stream = torch.cuda.Stream()
    stream.wait_stream(torch.cuda.current_stream())
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=stream):
        damp.kda_decode_step(L, state, perm, static["q"], static["k"], static["v"], static["g"], static["beta"],
                             o=o_g)
    torch.cuda.current_stream().wait_stream(stream)
    for d in inputs[1:]:
        for k in static:
            static[k].copy_(d[k])
        graph.replay()
        damp.kda_decode_step(L, eager, perm, d["q"], d["k"], d["v"], d["g"], d["beta"], o=o_e)
        torch.cuda.synchronize()
        assert torch.equal(o_g, o_e)
        assert torch.equal(state, eager)


@pytest.mark.parametrize("T", [4, 32])
def test_prefill_chunk_replays_from_a_graph(T):
    w = wl.GDN_B64_GQA.replace(batch=2)
    L, perm, state = _setup(w, 82)
    eager = state.clone()
    steps = [wl.step_inputs(w, t) for t in range(T)]
    dt = torch.bfloat16
    chunk = {k: P.to_dev(np.stack([s[k] for s in steps], axis=1), DEV, dt if k in ("q", "k", "v") else None)
             for k in steps[0]}
    o_e = torch.empty((w.batch, T, w.heads, w.d_v), device=DEV)
    o_g = torch.empty_like(o_e)
    args = (chunk["q"], chunk["k"], chunk["v"], chunk["g"], chunk["beta"])
    damp.gdn_prefill_chunk(L, eager, perm, *args, o=o_e)  # set-up and the first eager chunk
    stream = torch.cuda.Stream()
    stream.wait_stream(torch.cuda.current_stream())
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=stream):
        damp.gdn_prefill_chunk(L, state, perm, *args, o=o_g)
    torch.cuda.current_stream().wait_stream(stream)
    graph.replay()
    torch.cuda.synchronize()
    assert torch.equal(o_g, o_e) and torch.equal(state, eager)
