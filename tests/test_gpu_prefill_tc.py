"""GPU parity of the GDN prefill chunk on the tensor cores (chunkwise closed form of
Sec. 3.1 Eq. delta_update, App. A.5 "Prefill path") against the oracle's per-token
chunk: GDN, d_k = d_v = 128, bf16 q/k/v, chunks of at least 32 tokens (one or more
pieces of 64 tokens, ragged rows masked); the UINT8, UINT4 and FP8 low tiers."""
import pytest

import workloads as wl
from tests.test_gpu_prefill import _built, _run  # noqa: F401  (module fixture and runner)

pytestmark = pytest.mark.gpu


def _gdn(name, batch, heads, qk_heads, k_hi, fmt=0, seed=31):
    return wl.Workload(name, "gdn", batch, heads, qk_heads, 128, 128, k_hi, 4, 24, "bf16", seed, fmt)


def test_one_piece_gqa():
    """64 tokens (one full piece), GQA (two value heads per q/k head), K_hi = 8."""
    _run(_gdn("tc_gqa_k8", 2, 4, 2, 8), 64)


def test_two_pieces_two_chunks():
    """128 tokens (two pieces in one launch), two chunks in a row."""
    _run(_gdn("tc_two_pieces", 1, 2, 2, 10, seed=32), 128, chunks=2)


def test_ragged_rows_and_slot_indirection():
    """Rows of 40, 17 and 0 tokens in a 40-token chunk (a partial piece: masked tokens),
    scattered over a larger pool; the zero-length row's slot stays as it was."""
    _run(_gdn("tc_ragged", 3, 2, 2, 6, seed=33), 40, lengths=[40, 17, 0], slot_of={0: 4, 1: 1, 2: 0}, pool=5)


@pytest.mark.parametrize("k_hi,fmt", [(0, 0), (16, 1), (40, 0), (127, 1), (10, 3), (16, 4), (10, 5), (0, 3)])
def test_tiers(k_hi, fmt):
    """No FP16 rows, FP16 rows in one warp or over two, all but one row FP16; the UINT8 and
    UINT4 tiers with and without H_32, FP8 E4M3."""
    _run(_gdn(f"tc_k{k_hi}_f{fmt}", 1, 2, 1, k_hi, fmt, seed=34 + k_hi), 64)


def test_full_piece_and_a_partial_one():
    """97 tokens: a full piece and a partial one of 33."""
    _run(_gdn("tc_97", 1, 2, 2, 12, seed=35), 97)
