"""Helpers that compare the CUDA path's trial records with the oracle's (used by the -m gpu tests)."""
import numpy as np

from oracle import mca_oracle as O

TIE_REL = 1e-5     # |dS| < 1e-5 * S: either decision is correct (candidate losses agree to 1e-5)


def oracle_trace(wl, n_trials, seed=0, mode="incremental", domain=None):
    run = O.run_incremental if mode == "incremental" else O.run_full
    tr, params, S = run(wl.layers, wl.loss, wl.X, wl.y, wl.init, n_trials, seed,
                        domain or wl.domain)
    return tr, params, S


def tie_band(tr, theta=0.0):
    """Trials where the oracle's dS lies within TIE_REL * S of the acceptance threshold theta (0 for
    the greedy rule, Eq. 6; per trial for the Metropolis rule, Eq. 7), except exact zeros of
    proposals that leave the parameter unchanged (new == old): those are no-ops and must match.
    An exact zero of a changed parameter is a tie like any other: it comes from an invariance of
    the network (a key bias adds the same q . b_k to every score of an attention row, which the
    softmax removes), which the fp64 oracle resolves to 0 and an fp32 evaluation to a
    rounding-size value of either sign."""
    d = np.abs(tr["dS"] - theta)
    noop = (tr["dS"] == 0.0) & (tr["new"] == tr["old"])
    return tr["valid"] & (d < TIE_REL * np.abs(tr["S"])) & ~noop


def forced_from_oracle(tr, theta=0.0):
    m = tie_band(tr, theta)
    return tr["tau"][m].astype(np.uint64), tr["accept"][m]


def compare(gpu, ora, check_dS=True):
    """gpu: structured array from mca_get_trace; ora: oracle trace dict. Proposals bit-exact,
    decisions equal, dS within TIE_REL * S."""
    n = len(ora["tau"])
    assert len(gpu) == n, (len(gpu), n)
    assert np.array_equal(gpu["tau"].astype(np.int64), ora["tau"])
    assert np.array_equal(gpu["idx"].astype(np.int64), ora["idx"])
    assert np.array_equal(gpu["new_w"], ora["new"].astype(np.float32))
    assert np.array_equal(gpu["old_w"], ora["old"].astype(np.float32))
    assert np.array_equal(gpu["valid"].astype(bool), ora["valid"])
    bad = np.nonzero(gpu["accept"].astype(bool) != ora["accept"])[0]
    assert len(bad) == 0, f"first decision mismatch at trial {bad[:5]}: gpu dS {gpu['dS'][bad[:5]]}, " \
                          f"oracle dS {ora['dS'][bad[:5]]}, S {ora['S'][bad[:5]]}"
    if check_dS:
        v = ora["valid"]
        err = np.abs(gpu["dS"][v] - ora["dS"][v])
        tol = TIE_REL * np.abs(ora["S"][v])
        worst = int(np.argmax(err / tol)) if v.any() else 0
        assert np.all(err <= tol), f"dS error {err[worst]} > {tol[worst]}"
        assert np.allclose(gpu["S"], ora["S"], rtol=TIE_REL, atol=0)
