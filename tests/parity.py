"""Comparison of CUDA outputs with the oracle, shared by the GPU tests.

Tolerances: the kernels compute every latency bound in fp32 from exact
integer aggregates (int64 prefix sums of lengths and of r (r + 1) / 2 terms),
with a handful of fp32 roundings per bound (about 5, each at most 2^-24
relative of the term it rounds), so a bound of magnitude B carries an error
of order 1e-6 B; 1e-5 relative of the bound's scale is the bar, a 10x margin.
KV bounds are integers below 2^24 and exact in fp32.
Feasibility flags are compared exactly except on pairs whose smallest latency
slack is within 1e-5 of its scale in the oracle's fp64 arithmetic ("near"
pairs), where fp32 may take the other side; those are counted and reported.
"""
import numpy as np

NEAR = 1e-5
REL = 1e-5


def margin_tol(ref_margin, ref_mscale, cand_in):
    bound = np.abs(ref_margin + cand_in[:, None]) if ref_margin.ndim == 2 else np.abs(ref_margin + cand_in)
    return REL * np.maximum(np.maximum(bound, ref_mscale), 1.0)


def compare_pairs(ref, flags, margin, cand_in, kvpeak=None, tcand=None, label=""):
    """ref: oracle dict (2-D [C, W] arrays or 1-D per-pair arrays)."""
    near = ref["near"] <= NEAR
    far = ~near
    bad = far & (flags != ref["flags"])
    assert not bad.any(), "%s: %d flag mismatches (first at %s): gpu %s oracle %s" % (
        label, int(bad.sum()), np.argwhere(bad)[0], flags[bad][:5], ref["flags"][bad][:5])
    m = margin.astype(np.float64)
    fin = np.isfinite(ref["margin"])
    assert np.all(np.isneginf(m[~fin])), "%s: -inf margins differ" % label
    tol = margin_tol(ref["margin"], ref["mscale"], cand_in)
    err = np.where(fin, np.abs(np.where(fin, m, 0.0) - np.where(fin, ref["margin"], 0.0)), 0.0)
    badm = fin & (err > tol)
    assert not badm.any(), "%s: %d margin mismatches, worst %s vs %s" % (
        label, int(badm.sum()), m[badm][:3], ref["margin"][badm][:3])
    # feasible <=> margin >= 0 on the GPU side
    assert np.array_equal(flags == 15, m >= 0), "%s: flags and margin disagree" % label
    if kvpeak is not None:
        assert np.array_equal(kvpeak, ref["kvpeak"]), "%s: kv peaks differ" % label
    if tcand is not None:
        assert np.allclose(tcand, ref["tcand"], rtol=REL, atol=0), "%s: t_cand differs" % label
    return int(near.sum())


def check_argbest(order, flags, argbest, label=""):
    """argbest[c] must be the first worker in capacity_norm order whose flags
    are all set (flags checked against the oracle separately)."""
    C = flags.shape[0]
    for c in range(C):
        feas = flags[c][order] == 15
        want = int(order[np.argmax(feas)]) if feas.any() else -1
        assert argbest[c] == want, "%s: argbest[%d] = %d, expected %d" % (label, c, argbest[c], want)
