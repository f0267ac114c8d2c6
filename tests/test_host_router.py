"""Host logic: the query-complexity router (Sec. III-B; the estimator and its
cut points are this library's own, the paper gives none)."""
import pytest

from paper_2609_21704_gb300 import router
from paper_2609_21704_gb300.router import PromptFeatures, complexity, route, route_batch


def test_score_is_the_weighted_mean_of_clipped_features():
    assert complexity(PromptFeatures(0)) == 0.0
    assert complexity(PromptFeatures(512, 8, 0.2)) == pytest.approx(1.0)
    assert complexity(PromptFeatures(10_000, 100, 5.0)) == pytest.approx(1.0)  # clipped
    assert complexity(PromptFeatures(256)) == pytest.approx(0.4 * 0.5)
    assert complexity(PromptFeatures(0, 4)) == pytest.approx(0.3 * 0.5)
    assert complexity(PromptFeatures(0, 0, 0.1)) == pytest.approx(0.3 * 0.5)


def test_three_classes_and_cut_points():
    assert route(PromptFeatures(16, 1, 0.0)) == "int4"
    assert route(PromptFeatures(512, 0, 0.0)) == "fp8"       # score 0.4
    assert route(PromptFeatures(512, 8, 0.0)) == "fp16"      # score 0.7
    # either side of the cut points (1/3 and 2/3)
    assert route(PromptFeatures(422)) == "int4"          # 0.3297
    assert route(PromptFeatures(428)) == "fp8"           # 0.3344
    assert route(PromptFeatures(512, 7.0)) == "fp8"      # 0.6625
    assert route(PromptFeatures(512, 7.2)) == "fp16"     # 0.67


def test_monotone_in_every_feature():
    order = {r: i for i, r in enumerate(router.ROUTES)}
    base = PromptFeatures(100, 2, 0.05)
    for f in (PromptFeatures(400, 2, 0.05), PromptFeatures(100, 6, 0.05), PromptFeatures(100, 2, 0.15)):
        assert complexity(f) > complexity(base)
        assert order[route(f)] >= order[route(base)]


def test_route_batch_keeps_input_order():
    fs = [PromptFeatures(16), PromptFeatures(512, 8, 0.2), PromptFeatures(512), PromptFeatures(20)]
    assert route_batch(fs) == {"int4": [0, 3], "fp8": [2], "fp16": [1]}


@pytest.mark.parametrize("bad", [dict(length=-1), dict(length=3.5), dict(length=5, depth=float("nan")),
                                 dict(length=5, entity_density=-0.1)])
def test_invalid_features_rejected(bad):
    with pytest.raises(ValueError):
        PromptFeatures(**bad)
