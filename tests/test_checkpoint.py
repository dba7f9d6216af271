"""Layout checkpoints on the CPU: the calibrated permutation table round-trips through
the JSON artifact, and malformed files are rejected."""
import json

import numpy as np
import pytest

import paper_2608_27513_gb300 as damp
import workloads as wl
from oracle import runs
from paper_2608_27513_gb300 import checkpoint


def test_layout_round_trip(tmp_path):
    w = wl.GDN_B1_D64
    perms, _ = runs.calibrate_layout(w, n_docs=2, n_tokens=16)
    L = damp.Layout(w.heads, w.qk_heads, w.d_k, w.d_v, w.k_hi, w.lo_format)
    path = str(tmp_path / "layer.json")
    checkpoint.save_layout(path, L, perms)
    L2, p2 = checkpoint.load_layout(path)
    assert L2 == L and np.array_equal(p2, perms) and p2.dtype == np.uint8


def test_malformed_layouts_are_rejected(tmp_path):
    L = damp.Layout(2, 2, 32, 64, 4, 0)
    bad = np.tile(np.arange(32, dtype=np.uint8), (2, 1))
    bad[1, 3] = 5  # not a permutation
    with pytest.raises(ValueError):
        checkpoint.save_layout(str(tmp_path / "a.json"), L, bad)
    with pytest.raises(ValueError):
        checkpoint.save_layout(str(tmp_path / "a.json"), L, bad[:1])
    path = tmp_path / "b.json"
    checkpoint.save_layout(str(path), L, np.tile(np.arange(32, dtype=np.uint8), (2, 1)))
    doc = json.loads(path.read_text())
    doc["version"] = 99
    path.write_text(json.dumps(doc))
    with pytest.raises(ValueError):
        checkpoint.load_layout(str(path))
    doc["version"] = checkpoint.LAYOUT_VERSION
    doc["d_k"] = 48  # a layout libdamp does not take
    doc["perm"] = [list(range(48))] * 2
    path.write_text(json.dumps(doc))
    with pytest.raises(ValueError):
        checkpoint.load_layout(str(path))
