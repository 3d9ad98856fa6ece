"""The field tolerance of the parity tests where the corrected Nesterov step
(Eq. autoloco-corrected-nesterov) cancels.  v' = mu v + Dtil is formed in
fp32 from terms that can be far larger than v' itself; on a vector of a few
elements there is no rms to fall back on, so the tolerance scales with the
terms (step_terms).  The scaling must admit an error of the size of fp32
rounding of the terms and still catch a dropped or mis-signed term."""
import numpy as np
import pytest

import oracle as O
from _parity import RTOL_FIELD, field_error, step_terms

U32 = 2.0 ** -24  # fp32 unit roundoff
MU, ETA, INV = 0.8, 0.7, 1.0


def _cancelling_round(M=4):
    """One element whose momentum term nearly cancels the averaged
    pseudo-gradient: v' is about 1e-4 of mu v."""
    g = np.array([0.5], np.float32)
    xs = [np.array([0.5 - 1e-3 * (m + 1)], np.float32) for m in range(M)]
    dtil = INV * float(np.mean([float(g[0]) - float(x[0]) for x in xs]))
    v = np.array([-dtil / MU * (1 + 1e-4)], np.float32)
    g_out, v_out, _, nf = O.pass2(g, v, xs, O.F32, MU, ETA, INV)
    assert nf == 0
    tg, tv = step_terms(g, v, xs, O.F32, MU, ETA, INV)
    return g, v, xs, g_out, v_out, tg, tv


def test_cancellation_is_what_the_terms_cover():
    g, v, xs, g_out, v_out, tg, tv = _cancelling_round()
    # v' is orders of magnitude below its terms
    assert abs(v_out[0]) < 1e-3 * tv[0]
    # an error of a few fp32 roundings of the terms: beyond the plain
    # relative tolerance, within the term-scaled one
    err = 8 * U32 * tv
    assert field_error(v_out + err, v_out) > RTOL_FIELD
    assert field_error(v_out + err, v_out, tv) <= RTOL_FIELD


@pytest.mark.parametrize("mistake", ["no_momentum", "dtil_sign", "eta_sign"])
def test_term_scaling_still_catches_mistakes(mistake):
    g, v, xs, g_out, v_out, tg, tv = _cancelling_round()
    if mistake == "no_momentum":
        _, bad_v, _, _ = O.pass2(g, v * 0, xs, O.F32, MU, ETA, INV)
        assert field_error(bad_v, v_out, tv) > RTOL_FIELD
    elif mistake == "dtil_sign":
        # the replicas reflected about theta: Dtil changes sign
        flipped = [(2 * g.astype(np.float64) - x).astype(np.float32) for x in xs]
        _, bad_v, _, _ = O.pass2(g, v, flipped, O.F32, MU, ETA, INV)
        assert field_error(bad_v, v_out, tv) > RTOL_FIELD
    else:
        bad_g, _, _, _ = O.pass2(g, v, xs, O.F32, MU, -ETA, INV)
        assert field_error(bad_g, g_out, tg) > RTOL_FIELD


def test_terms_reduce_to_the_plain_scale_without_cancellation():
    """With no cancellation the terms are of the size of the result, so the
    check is as strict as before: a 1e-4 relative error fails."""
    rng = np.random.default_rng(5)
    g = rng.standard_normal(64).astype(np.float32)
    xs = [(g + 1e-3 * rng.standard_normal(64)).astype(np.float32) for _ in range(4)]
    v = (1e-3 * rng.standard_normal(64)).astype(np.float32)
    g_out, v_out, _, _ = O.pass2(g, v, xs, O.F32, MU, ETA, INV)
    tg, tv = step_terms(g, v, xs, O.F32, MU, ETA, INV)
    assert field_error(v_out * (1 + 1e-4), v_out, tv) > RTOL_FIELD
    assert field_error(g_out * (1 + 1e-4), g_out, tg) > RTOL_FIELD
