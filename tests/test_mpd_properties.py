"""Property tests of Algorithm 1's scheduler (hypothesis draws the pages): for any pages, fork
offsets (ties, any order, 0 and L), branch lengths, admission times and a pool just large enough,
the loop decodes exactly the packed pages' layout and branch tokens, each token's reachable rows are
the Algorithm 1 simulator's mask row, the pool never hands out a row still visible to a live
stream, and every block comes back."""
import numpy as np
import pytest

hyp = pytest.importorskip("hypothesis")
st = pytest.importorskip("hypothesis.strategies")

from paper_2608_06146_gb300 import build as pbuild  # noqa: E402
from paper_2608_06146_gb300 import padoc_attn as pa  # noqa: E402
from paper_2608_06146_gb300.inputs import LoopTokenSource, PageSpec  # noqa: E402
from tests.test_mpd_host import _blocks_needed, run_loop  # noqa: E402


@pytest.fixture(scope="module", autouse=True)
def lib():
    pbuild.build()
    return pa.load_library()


@st.composite
def page_sets(draw):
    n = draw(st.integers(1, 4))
    pages, admit = [], []
    for _ in range(n):
        P = draw(st.integers(0, 50))
        L = draw(st.integers(0, 20))
        N = draw(st.integers(0, 6))
        forks = draw(st.lists(st.integers(0, L), min_size=N, max_size=N))
        lens = draw(st.lists(st.integers(1, 40), min_size=N, max_size=N))
        pages.append(PageSpec(P, L, forks, lens))
        admit.append(draw(st.integers(0, 30)))
    return pages, admit


@hyp.settings(max_examples=60, deadline=None)
@hyp.given(page_sets(), st.integers(0, 2 ** 31 - 1))
def test_scheduler_matches_algorithm_1(case, seed):
    pages, admit = case
    need = _blocks_needed(pages)
    order = np.random.default_rng(seed).permutation(need).astype(np.int32)
    decoded, steps, mpd = run_loop(pages, need, order, admit_at=admit)
    src = LoopTokenSource(pages)
    want = sorted(int(src.base[p]) + j for p, pg in enumerate(pages) for j in range(pg.prefix_len, pg.packed_len))
    assert sorted(decoded) == want
    assert mpd.status() == (0, 0, need)
