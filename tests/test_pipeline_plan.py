"""Host-side layer-group plan of the pipelined end-to-end query (no GPU needed)."""
import pytest

from paper_2607_19547_gb300.pipeline import plan_layer_groups


def _covers(groups, n_layers):
    assert groups[0][0] == 0 and groups[-1][1] == n_layers
    for (a, b), (c, d) in zip(groups[:-1], groups[1:]):
        assert a < b == c < d


def test_default_plan_for_36_layers():
    """A 2-layer first group holding the score layer, groups of 4, and a 2-layer last group."""
    assert plan_layer_groups(36, 1) == [(0, 2), (2, 6), (6, 10), (10, 14), (14, 18), (18, 22),
                                        (22, 26), (26, 30), (30, 34), (34, 36)]


@pytest.mark.parametrize("n_layers", list(range(1, 41)))
@pytest.mark.parametrize("group_layers", [1, 3, 4, 6, 36])
def test_default_plan_covers_every_layer_once(n_layers, group_layers):
    score_layer = min(1, n_layers - 1)
    groups = plan_layer_groups(n_layers, score_layer, group_layers)
    _covers(groups, n_layers)
    # the first group reaches the score layer, and no middle group exceeds group_layers
    assert groups[0][0] <= score_layer < groups[0][1]
    for a, b in groups[1:-1]:
        assert b - a <= max(group_layers, 2)


def test_score_layer_deeper_than_two_lengthens_the_first_group():
    groups = plan_layer_groups(12, 5, 4)
    _covers(groups, 12)
    assert groups[0] == (0, 6)


def test_explicit_bounds_are_taken_as_given():
    assert plan_layer_groups(10, 1, bounds=[0, 3, 4, 10]) == [(0, 3), (3, 4), (4, 10)]


@pytest.mark.parametrize("bounds", [[1, 10], [0, 9], [0, 5, 5, 10], [0, 6, 4, 10], [10], [],
                                    [0, 1, 10]])
def test_bad_bounds_raise(bounds):
    """Including a first group that ends before the score layer (layer 1): the other groups'
    attention would run before the selection exists."""
    with pytest.raises(ValueError):
        plan_layer_groups(10, 1, bounds=bounds)


@pytest.mark.parametrize("args", [(0, 0), (10, 10), (10, -1), (10, 1, 0)])
def test_bad_sizes_raise(args):
    with pytest.raises(ValueError):
        plan_layer_groups(*args)
