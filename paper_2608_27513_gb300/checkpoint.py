"""Checkpoint artifacts: the calibrated layout of a layer and packed states.

The paper stores the key-channel permutation once with the model, not per request
(App. A.1 "DAMP storage"; App. A.5 "Persistent representation"); a layer's layout is
(H, H_qk, d_k, d_v, K_hi, lo_format) plus pi [H][d_k].  Packed states are saved as
their logical tiers (FP16 rows, codes, metadata) through damp_unpack_tiers and
restored bit for bit through damp_pack_tiers, so a file does not depend on the
private record layout.
"""
from __future__ import annotations

import json

import numpy as np

import paper_2608_27513_gb300 as damp

LAYOUT_VERSION = 1


def save_layout(path: str, layout: "damp.Layout", perms) -> None:
    """Write a layer's layout and per-head permutations (uint8 [H, d_k]) as JSON."""
    perms = np.asarray(perms.cpu() if hasattr(perms, "cpu") else perms, dtype=np.uint8)
    if perms.shape != (layout.num_heads, layout.d_k):
        raise ValueError(f"perms must be [{layout.num_heads}, {layout.d_k}], got {list(perms.shape)}")
    for row in perms:
        if sorted(row.tolist()) != list(range(layout.d_k)):
            raise ValueError("every row of perms must be a permutation of 0..d_k-1")
    doc = {"version": LAYOUT_VERSION, "num_heads": layout.num_heads, "num_qk_heads": layout.num_qk_heads,
           "d_k": layout.d_k, "d_v": layout.d_v, "k_hi": layout.k_hi, "lo_format": layout.lo_format,
           "perm": perms.tolist()}
    if layout.head_map is not None:  # one head group of a layer: its model heads
        doc["model_heads"] = layout.heads_of_operands
        doc["heads"] = [int(h) for h in layout.head_map.cpu().tolist()]
    with open(path, "w") as f:
        json.dump(doc, f)


def load_layout(path: str, device="cuda"):
    """Read (Layout, perms uint8 [H, d_k]) written by save_layout; the layout is validated.
    A head group's map is placed on `device`."""
    with open(path) as f:
        doc = json.load(f)
    if doc.get("version") != LAYOUT_VERSION:
        raise ValueError(f"unknown layout file version {doc.get('version')}")
    head_map = None
    if "heads" in doc:
        import torch
        heads = [int(h) for h in doc["heads"]]
        if len(heads) != doc["num_heads"] or len(set(heads)) != len(heads) or \
                not all(0 <= h < doc["model_heads"] for h in heads):
            raise ValueError("the head map does not match the layout")
        head_map = torch.tensor(heads, dtype=torch.int32, device=device)
    layout = damp.Layout(doc["num_heads"], doc["num_qk_heads"], doc["d_k"], doc["d_v"], doc["k_hi"],
                         doc["lo_format"], model_heads=doc.get("model_heads", 0), head_map=head_map)
    perms = np.asarray(doc["perm"], dtype=np.uint8)
    if perms.shape != (layout.num_heads, layout.d_k):
        raise ValueError("perm table does not match the layout")
    if damp.record_bytes(layout) == 0:
        raise ValueError("the layout is not one libdamp accepts")
    return layout, perms


def save_state(path: str, layout: "damp.Layout", state, slot_idx=None) -> None:
    """Write packed slots (all of `state`, or the rows named by slot_idx) as logical tiers (.npz)."""
    hi, codes, meta = damp.unpack_tiers(layout, state, slot_idx=slot_idx)
    np.savez(path, hi=hi.cpu().numpy(), codes=codes.cpu().numpy(), meta=meta.cpu().numpy(),
             layout=np.array([layout.num_heads, layout.num_qk_heads, layout.d_k, layout.d_v, layout.k_hi,
                              layout.lo_format], np.int32))


def load_state(path: str, layout: "damp.Layout", state, slot_idx=None) -> None:
    """Restore logical tiers written by save_state into packed slots, bit for bit."""
    import torch
    with np.load(path) as z:
        saved = tuple(int(v) for v in z["layout"])
        want = (layout.num_heads, layout.num_qk_heads, layout.d_k, layout.d_v, layout.k_hi, layout.lo_format)
        if saved != want:
            raise ValueError(f"state file layout {saved} does not match {want}")
        dev = state.device
        hi, codes, meta = (torch.from_numpy(z[k]).to(dev) for k in ("hi", "codes", "meta"))
    damp.pack_tiers(layout, hi, codes, meta, state, slot_idx=slot_idx)
