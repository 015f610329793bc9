"""Host logic of the benchmark (no GPU): the decoded positions the diffusion
head is driven with, against the mask schedule they come from."""
import numpy as np
import pytest

import bench
import synth


@pytest.mark.parametrize("name", ["mar_b", "hires", "tiny"])
def test_decoded_positions_partition_the_image(name):
    """Across the 64 steps every pair decodes each image position exactly once.
    Step k decodes m[k-1] - m[k] positions (n_img - m[0] at step 0), the same
    count in every pair, each masked at step k and known at step k + 1."""
    cfg = synth.config(name)
    _, masks, _ = bench.decode_inputs(cfg, 0)
    pos = bench.decoded_positions(masks)
    m = synth.mask_counts(cfg["steps"], cfg["n_img"])
    B, n_img = cfg["batch"], cfg["n_img"]
    seen = np.zeros((B, n_img), np.int32)
    for k, p in enumerate(pos):
        # the input of step k still shows n_img - (positions decoded before k) masked
        before = n_img if k == 0 else m[k - 1]
        assert int(masks[k][0].sum()) == (n_img if k == 0 else before)
        want = before - m[k] if k > 0 else n_img - m[0]
        if p is None:
            assert want == 0
            continue
        assert p.shape == (B, want)
        for b in range(B):
            assert np.all(masks[k][b][p[b]] == 1)
            if k + 1 < len(pos):
                assert np.all(masks[k + 1][b][p[b]] == 0)
            seen[b, p[b]] += 1
    assert np.all(seen == 1)


def test_decoded_positions_need_equal_counts():
    masks = np.ones((2, 2, 4), np.uint8)
    masks[1, 0, :2] = 0      # pair 0 decodes two positions at step 0, pair 1 none
    with pytest.raises(AssertionError):
        bench.decoded_positions(masks)
