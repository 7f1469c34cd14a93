"""The live-value bound of tests/_cmp.py against planted mistakes (CPU only):
it accepts the oracle's own values and a one-step rounding difference, and
rejects a two-step error at ordinary magnitudes, a flipped sign and a value
taken from the wrong element; near a cancellation it admits the fp32
evaluation error of the operands and nothing of the size of a wrong term."""
import numpy as np
import pytest

from tests._cmp import assert_live_close, fp16_step


def test_fp16_step_values():
    assert fp16_step(1.0) == 2.0 ** -10
    assert fp16_step(1.5) == 2.0 ** -10
    assert fp16_step(65504.0) == 32.0
    assert fp16_step(2.0 ** -14) == 2.0 ** -24
    assert fp16_step(1e-7) == 2.0 ** -24
    assert fp16_step(0.0) == 2.0 ** -24


def _case(orc, seed=3):
    cfg = dict(n_shards=2, hidden=64, n_canaries=3, tokens=8, malicious=(1,), noise=1,
               benign_sigma=0.05, tamper=0, tamper_param=0.05, seed=seed)
    D = orc.desc_from_dict(cfg)
    return orc.generate_coefs(D)


def _bits(x):
    return np.asarray(x, np.float16).view(np.uint16)


def test_accepts_the_oracle_and_one_step(orc):
    acts, refs, coef = _case(orc)
    assert assert_live_close(acts, acts, refs, refs, coef) == 0
    g = acts.copy().view(np.float16)
    flat = g.reshape(-1)
    i = int(np.argmax(np.abs(flat.astype(np.float64))))
    flat[i] = np.nextafter(flat[i], np.float16(np.inf), dtype=np.float16)
    assert assert_live_close(g.view(np.uint16), acts, refs, refs, coef) == 1


@pytest.mark.parametrize("mistake", ["two_steps", "sign", "wrong_element"])
def test_rejects_planted_mistakes(orc, mistake):
    acts, refs, coef = _case(orc)
    g = acts.copy().view(np.float16).astype(np.float64)
    o = acts.view(np.float16).astype(np.float64)
    # an element of ordinary size, inside a binade (|h| near 1.5)
    i = np.unravel_index(int(np.argmin(np.abs(np.abs(o) - 1.5))), o.shape)
    if mistake == "two_steps":
        g[i] += 2 * fp16_step(o[i])
    elif mistake == "sign":
        g[i] = -g[i]
    else:
        j = (i[0], i[1], (i[2] + 1) % o.shape[2])
        g[i] = o[j]
    with pytest.raises(AssertionError):
        assert_live_close(_bits(g), acts, refs, refs, coef)


def test_cancellation_admits_evaluation_error_only():
    """a + c z ~ 0: an fp32 evaluation error of 2^-22 |a| is admitted (many
    subnormal steps), an error of 1e-3 |a| (a dropped term's size) is not."""
    a = np.array([[1.25]], np.float32)
    c = np.array([0.5])
    o = _bits([[0.0]])
    ok = _bits([[1.25 * 2.0 ** -22]])
    assert assert_live_close(ok, o, a, a, c) > 1
    with pytest.raises(AssertionError):
        assert_live_close(_bits([[1.25e-3]]), o, a, a, c)
