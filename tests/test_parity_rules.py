"""The comparison rules of tests/parity.py on hand-made cases (CPU): the
order the CUDA path sorts into, the order near-tie that lets an end-to-end
budget differ, and the decode bound."""
import numpy as np
import torch

import parity


def test_gpu_order_is_descending_with_lower_index_first():
    a = np.array([0.1, 0.3, 0.3, 0.2, 0.3], np.float32)
    assert parity.gpu_order(a).tolist() == [1, 2, 4, 3, 0]


def test_order_near_tie_accepts_only_float32_level_swaps():
    a64 = np.array([0.5, 0.142857113, 0.142857106, 0.01])
    ref = np.array([0, 1, 2, 3])
    swapped = np.array([0, 2, 1, 3])     # 5e-8 relative apart: fp32 cannot order them
    assert parity.order_near_tie(swapped, ref, a64)
    assert not parity.order_near_tie(ref, ref, a64)          # no difference at all
    a64_far = np.array([0.5, 0.143, 0.142, 0.01])
    assert not parity.order_near_tie(swapped, ref, a64_far)  # 7e-3 apart: a real error
    wrong = np.array([3, 0, 1, 2])
    assert not parity.order_near_tie(wrong, ref, a64)


def test_end_to_end_budget_difference_needs_a_cause():
    """Two heads, n = 4: the GPU moved one token between the heads.  Without an
    order near-tie the objective gap fails the check; with the float64 scores
    of head 0 tied at fp32 level (and the GPU order swapping them) it passes."""
    c = np.array([[4.0, 3.0, 2.0, 1.0], [4.0, 2.6, 1.5, 1.0]])
    ref = dict(counts=np.array([2, 1]), c=c, perm=np.array([[0, 1, 2, 3], [0, 1, 2, 3]]),
               a=np.array([[0.4, 0.3, 0.2, 0.1], [0.4, 0.3, 0.2, 0.1]]))
    got = dict(counts=np.array([1, 2]), offsets=np.array([0, 2, 5]),
               positions=np.array([0, -1, 0, 1, -1]))
    a_gpu = np.array([[0.4, 0.3, 0.2, 0.1], [0.4, 0.3, 0.2, 0.1]], np.float32)
    try:
        parity.check_end_to_end(got, ref, a_gpu, H=2)
        raise AssertionError("a budget difference without a near-tie was accepted")
    except AssertionError as e:
        assert "no order near-tie" in str(e)
    ref_tied = dict(ref, a=np.array([[0.4, 0.2000000001, 0.2, 0.1], [0.4, 0.3, 0.2, 0.1]]))
    a_gpu_tied = np.array([[0.4, 0.2, 0.2, 0.1], [0.4, 0.3, 0.2, 0.1]], np.float32)
    ref_tied["perm"] = np.array([[0, 1, 2, 3], [0, 1, 2, 3]])
    # the GPU's fp32 scores of tokens 1 and 2 are equal: order 0, 1, 2, 3 by index,
    # the same as float64 here, so swap the float64 order to make them differ
    ref_tied["a"][0, 1], ref_tied["a"][0, 2] = 0.2, 0.2000000001
    ref_tied["perm"][0] = [0, 2, 1, 3]
    assert parity.check_end_to_end(got, ref_tied, a_gpu_tied, H=2) == 1


def test_decode_bound_grows_by_half_a_bf16_ulp():
    ref = np.array([[0.5, 9.0]])
    got = ref + np.array([[0.0199, 0.0199 + 2.0 ** -5]])
    parity.check_decode(torch.tensor(got), ref)
    try:
        parity.check_decode(torch.tensor(ref + np.array([[0.0201, 0.0]])), ref)
        raise AssertionError("an error above 2e-2 + half an ulp was accepted")
    except AssertionError as e:
        assert "decode" in str(e) or "err" in str(e).lower()
