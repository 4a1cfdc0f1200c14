"""The comparison helpers of the GPU parity tests, checked on CPU against hand
cases: they must accept what is correct and reject each kind of wrong answer,
or the GPU comparisons would pass vacuously."""
import numpy as np
import pytest

from tests.parity import GAP_REL, SCORE_REL, check_topk_rows, map_rel_err, recall_allowance


def test_exact_rows_accept_the_right_set_in_any_order():
    s = [np.array([5.0, 1.0, 4.0, 3.0, 0.0])]
    assert check_topk_rows(np.array([[2, 0, 3]]), s, 3) == (1, 0)
    assert check_topk_rows(np.array([[0, 2, 3]]), s, 3, gpu_scores=np.array([[5.0, 4.0, 3.0]])) == (1, 0)


@pytest.mark.parametrize("got", [
    [[0, 2, 1]],        # a wrong key on a well-separated row
    [[0, 2, 2]],        # a duplicate
    [[0, 2, -1]],       # padding although enough keys are visible
    [[0, 2, 5]],        # an index past the visible prefix
    [[-1, 0, 2]],       # padding before valid entries
])
def test_exact_rows_reject_wrong_lists(got):
    s = [np.array([5.0, 1.0, 4.0, 3.0, 0.0])]
    with pytest.raises(AssertionError):
        check_topk_rows(np.array(got), s, 3)


def test_short_rows_take_every_visible_key():
    s = [np.array([1.0, 2.0]), np.array([])]
    assert check_topk_rows(np.array([[1, 0, -1], [-1, -1, -1]]), s, 3) == (1, 0)
    with pytest.raises(AssertionError):
        check_topk_rows(np.array([[1, -1, -1], [-1, -1, -1]]), s, 3)


def test_near_ties_are_waived_only_within_the_margin():
    mx = 10.0
    tie = [np.array([mx, 3.0, 3.0 - 0.5 * GAP_REL * mx, 1.0])]   # k = 2: the 2nd/3rd gap is below the margin
    assert check_topk_rows(np.array([[0, 2]]), tie, 2) == (0, 1)
    assert check_topk_rows(np.array([[0, 1]]), tie, 2) == (0, 1)
    with pytest.raises(AssertionError):                           # key 3 is far below the k-th
        check_topk_rows(np.array([[0, 3]]), tie, 2)


def test_reported_scores_are_checked():
    s = [np.array([5.0, 1.0, 4.0])]
    check_topk_rows(np.array([[0, 2]]), s, 2, gpu_scores=np.array([[5.0 + 0.5 * SCORE_REL * 5, 4.0]]))
    with pytest.raises(AssertionError):
        check_topk_rows(np.array([[0, 2]]), s, 2, gpu_scores=np.array([[5.0 + 2 * SCORE_REL * 5, 4.0]]))


def test_recall_allowance_counts_keys_near_the_kth_score():
    """k = 2.  Row 1: one score moves by 0.3, and two keys (9 and 8.8) lie within
    2 x 0.3 of the k-th score 9: allowance 2/2.  Row 2: nothing moves: 0.  Row 3
    has too few visible keys and does not count.  Mean over the two rows: 0.5."""
    ref = [np.array([10.0, 9.0, 8.8, 5.0]), np.array([3.0, 2.0, 1.0]), np.array([1.0])]
    alt = [np.array([10.0, 9.0, 9.1, 5.0]), np.array([3.0, 2.0, 1.0]), np.array([7.0])]
    assert recall_allowance(ref, alt, 2, 3) == pytest.approx(0.5)


def test_map_error_is_relative_frobenius():
    L = np.eye(4)[:, :2]
    M = L @ L.T
    assert map_rel_err(L, L, M) == 0.0
    assert map_rel_err(2 * L, L, M) == pytest.approx(1.0)
