"""Host logic of the diagnostics (acceptance by candidate position, scaling
efficiency, phase shares) on hand-made outputs."""
import numpy as np

from paper_2608_24411_gb300 import diagnostics as dg


def test_accepted_position_and_rates():
    # k = 3: seq 0 accepts candidate 1 (node 0), seq 1 candidate 3 (node 2),
    # seq 2 rejects all, seq 3 errors
    alen = np.array([1, 1, 0, -1])
    nodes = np.array([[0], [2], [-1], [-1]])
    pos = dg.accepted_position(alen, nodes, 3)
    np.testing.assert_array_equal(pos, [0, 2, 3, -1])
    reached, accepted, rate = dg.position_rates(pos, 3)
    np.testing.assert_array_equal(reached, [3, 2, 2])
    np.testing.assert_array_equal(accepted, [1, 0, 1])
    np.testing.assert_allclose(rate, [1 / 3, 0.0, 0.5])


def test_scaling_table_reproduces_the_papers_arithmetic():
    """The paper's scaling table (App., depth 4, N = 1, 2, 4, 8): EAL 1.89,
    2.17, 2.48, 2.76 give marginal gains 0.28, 0.31, 0.28 and efficiencies
    0.280, 0.155, 0.070 (eta = delta EAL / delta N)."""
    rows = dg.scaling_table({1: 1.89, 2: 2.17, 4: 2.48, 8: 2.76})
    assert rows[0] == (1, 1.89, None, None)
    np.testing.assert_allclose([r[2] for r in rows[1:]], [0.28, 0.31, 0.28], atol=1e-12)
    np.testing.assert_allclose([r[3] for r in rows[1:]], [0.280, 0.155, 0.070], atol=1e-12)


def test_phase_shares():
    cyc = np.array([[0, 10, 5, 5, 20, 10], [0, 30, 5, 5, 0, 10]])
    sh = dg.phase_shares(cyc)
    assert abs(sum(sh.values()) - 1) < 1e-12
    assert sh["norm"] == 0.4 and sh["reject"] == 0.2 and sh["setup"] == 0.0
