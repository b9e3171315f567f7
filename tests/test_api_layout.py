"""Host logic of the host-buffer API: the staging buffer's layout (no GPU)."""
import torch

from paper_2608_08721_gb300.api import _layout


def test_regions_are_aligned_ordered_and_disjoint():
    B, K, V, n, Hq, Hkv, d = 3, 5, 1001, 2, 8, 2, 64
    regions = [("draft_logits", (B, K, V), torch.float32), ("draft_tokens", (B, K), torch.int32),
               ("temperature", (B,), torch.float32), ("cost_table", (K + 1,), torch.float32),
               ("Q", (n, B, K + 1, Hq, d), torch.bfloat16), ("kv_new", (n, 2, B, Hkv, K + 1, d), torch.bfloat16),
               ("target_logits", (B, K + 1, V), torch.bfloat16), ("rng", (3,), torch.int64)]
    offs, total = _layout(regions)
    ends = []
    prev = -1
    for name, shape, dtype in regions:
        nbytes = torch.empty((), dtype=dtype).element_size()
        for s in shape:
            nbytes *= s
        o = offs[name]
        assert o % 256 == 0 and o > prev          # 256-byte aligned (TMA and 16-byte loads), in order
        assert not ends or o >= ends[-1]          # no overlap with the region before
        ends.append(o + nbytes)
        prev = o
    assert total % 256 == 0 and total >= ends[-1] and total - ends[-1] < 256
    assert offs["draft_logits"] == 0
    assert offs["draft_tokens"] == (B * K * V * 4 + 255) // 256 * 256


def test_empty_region_takes_no_room():
    offs, total = _layout([("a", (0, 7), torch.float32), ("b", (3,), torch.int32)])
    assert offs == {"a": 0, "b": 0} and total == 256
