"""Host-side planning of a generation (no GPU): the prefill is cut into
passes that every attention call of the stack accepts (at most 32 new
tokens, at most 200 queries per key/value head)."""
import pytest

from paper_2609_21704_gb300.generate import ATTN_MAX_GROUP_QUERIES, ATTN_MAX_T, prefill_chunk
from paper_2609_21704_gb300.shapes import STACKS


@pytest.mark.parametrize("name", sorted(STACKS))
def test_prefill_chunk_fits_one_attention_call(name):
    sh = STACKS[name]
    T = prefill_chunk(sh.q_heads, sh.kv_heads)
    G = sh.q_heads // sh.kv_heads
    assert 1 <= T <= ATTN_MAX_T
    assert G * T <= ATTN_MAX_GROUP_QUERIES
    # the largest chunk that fits: one more token would not
    assert T == ATTN_MAX_T or G * (T + 1) > ATTN_MAX_GROUP_QUERIES


def test_prefill_chunk_values():
    assert prefill_chunk(12, 2) == 32    # 1.5B: 6 query heads per key/value head
    assert prefill_chunk(28, 4) == 28    # 7B: 7 per group, 7 * 32 = 224 > 200
    assert prefill_chunk(40, 8) == 32    # 14B: 5 per group
    assert prefill_chunk(200, 1) == 1
    assert prefill_chunk(40, 8, 12) == 21   # 12 sequences: 21 x 12 = 252 rows <= 256
    assert prefill_chunk(12, 2, 300) == 1
