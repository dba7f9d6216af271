"""GPU parity of the prefill chunk on the tensor cores (chunkwise closed form of Sec. 3.1
Eq. delta_update, App. A.5 "Prefill path") against the oracle's per-token chunk: GDN and
KDA, d_k = d_v = 128, bf16 q/k/v, chunks of at least 32 tokens (one or more pieces of up
to 64 tokens, ragged rows masked); the UINT8 and UINT4 low tiers.  KDA pieces are cut
short where a channel's decay would leave FP32 on either side of the reference token."""
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


@pytest.mark.parametrize("k_hi,fmt", [(0, 0), (16, 1), (40, 0), (127, 1), (10, 3), (16, 4), (0, 3)])
def test_tiers(k_hi, fmt):
    """No FP16 rows, FP16 rows in one warp or over two, all but one row FP16; the UINT8 and
    UINT4 tiers with and without H_32."""
    _run(_gdn(f"tc_k{k_hi}_f{fmt}", 1, 2, 1, k_hi, fmt, seed=34 + k_hi), 64)


def test_full_piece_and_a_partial_one():
    """97 tokens: a full piece and a partial one of 33."""
    _run(_gdn("tc_97", 1, 2, 2, 12, seed=35), 97)


def _kda(name, batch, heads, qk_heads, k_hi, fmt=0, seed=41):
    return wl.Workload(name, "kda", batch, heads, qk_heads, 128, 128, k_hi, 4, 24, "bf16", seed, fmt)


def test_kda_one_piece_gqa():
    """KDA, 64 tokens (one full piece), GQA, K_hi = 10."""
    _run(_kda("tck_gqa_k10", 2, 4, 2, 10), 64)


def test_kda_two_pieces_two_chunks():
    _run(_kda("tck_two_pieces", 1, 2, 2, 16, seed=42), 128, chunks=2)


def test_kda_ragged_rows_and_slot_indirection():
    _run(_kda("tck_ragged", 3, 2, 2, 6, seed=43), 40, lengths=[40, 17, 0], slot_of={0: 4, 1: 1, 2: 0}, pool=5)


@pytest.mark.parametrize("k_hi,fmt", [(0, 0), (16, 1), (40, 0), (127, 1), (10, 3), (16, 4)])
def test_kda_tiers(k_hi, fmt):
    _run(_kda(f"tck_k{k_hi}_f{fmt}", 1, 2, 1, k_hi, fmt, seed=44 + k_hi), 64)


@pytest.mark.parametrize("g_scale", [8.0, 60.0])
def test_kda_strong_decay_shortens_the_pieces(g_scale):
    """Log-decays 8x and 60x the workload's (down to about -8 and -60 per token and
    channel): the pieces are cut to 32 tokens or fewer, down to single tokens, and the
    chunk still matches the per-token recurrence."""
    _run(_kda(f"tck_decay{int(g_scale)}", 1, 2, 2, 12, seed=45), 64, g_scale=g_scale)
