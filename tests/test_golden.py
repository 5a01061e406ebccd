"""Golden fixtures: values fixed by the paper's statements, and an oracle regression case."""
import os
import sys

import numpy as np
import pytest

HERE = os.path.dirname(os.path.abspath(__file__))
GOLD = os.path.join(HERE, "golden")
sys.path.insert(0, GOLD)


def _statements():
    out = {}
    with open(os.path.join(GOLD, "paper_statements.txt")) as f:
        for line in f:
            if not line.strip() or line.startswith("#"):
                continue
            name, cite, params, vals = (x.strip() for x in line.split("|"))
            out[name] = np.array([float(x) for x in vals.split()])
    return out


def test_paper_statements(orc):
    g = _statements()
    np.testing.assert_allclose(orc.dirichlet(4, np.arange(7), 2 * np.pi / 7), g["dirichlet_samples_M4"], atol=1e-14)
    np.testing.assert_allclose(orc.dirichlet(2, np.arange(3), 2 * np.pi / 3), g["dirichlet_samples_M2"], atol=1e-14)
    delta, A, B = orc.tables(2, 3, 3.0)
    np.testing.assert_allclose(A.ravel(), g["translated_A_M2"], atol=1e-15)
    np.testing.assert_allclose(B.ravel(), g["translated_B_M2"], atol=1e-15)
    np.testing.assert_array_equal(orc.tables(4, 7, 14.0)[0], g["dilated_grid_M4_T14"])
    np.testing.assert_array_equal(orc.tables(3, 5, 20.0)[0], g["dilated_grid_M3_T20"])
    assert orc.period(4, 3.0) == g["period_clamp_M4_T3"][0]


@pytest.mark.parametrize("key,H,dk,dv,M", [("state_size_bla", 16, 128, 128, 128),
                                            ("state_size_bla_small", 2, 32, 32, 16)])
def test_state_size_matches_table1(orc, key, H, dk, dv, M):
    """The recurrent state layout [2][M][2][d] per head holds exactly Table 1's H(dk+dv)(2M-1)
    live elements; the only other row is the sine of mode 0, which the recurrence keeps at 0."""
    g = _statements()
    rng = np.random.default_rng(0)
    q = rng.standard_normal((1, H, 5, dk))
    k = rng.standard_normal((1, H, 5, dk))
    v = rng.standard_normal((1, H, 5, dv))
    st = orc.forward(q, k, v, M, 2 * M - 1, 2 * M - 1, return_state=True)["state"]
    assert st.size == H * 2 * M * (dk + dv)
    assert np.all(st[..., 0, 1, :] == 0.0)
    live = st.size - H * (dk + dv)
    assert live == g[key][0]


def test_oracle_regression_case(orc):
    import make_golden
    ref = {}
    with open(os.path.join(GOLD, "oracle_small_case.txt")) as f:
        for line in f:
            if line.startswith("#"):
                continue
            name, *vals = line.split()
            ref[name] = np.array([float(x) for x in vals])
    out = make_golden.compute()
    for name, arr in out.items():
        np.testing.assert_allclose(np.ravel(arr), ref[name], rtol=1e-12, atol=1e-14, err_msg=name)
