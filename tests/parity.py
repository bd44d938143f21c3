"""Comparison of CUDA outputs with the oracle, shared by the GPU tests.

Tolerances: the kernels compute every latency bound in fp32 from exact
integer aggregates (int64 prefix sums of lengths and of r (r + 1) / 2 terms),
with a handful of fp32 roundings per bound (about 5, each at most 2^-24
relative of the term it rounds), so a bound of magnitude B carries an error
of order 1e-6 B; 1e-5 relative of the bound's scale is the bar, a 10x margin.
KV bounds are integers below 2^24 and exact in fp32.
Feasibility flags are compared exactly except on "near" pairs: a flag bit is
the sign of its group's smallest slack, and a pair is near when, for some
latency group, that smallest slack is within 1e-5 of its scale in the oracle's
fp64 arithmetic, where fp32 may take the other side. Near pairs are counted
and bounded: a group is near when its smallest relative slack falls in a band
of width 2e-5; with relative slacks spread over O(1) and four groups a pair,
the expected near fraction is of order 1e-4 (the workloads here measure up to
a few 1e-4), so more than NEAR_FRAC_MAX = 1e-3 of the pairs would mean the
comparison excludes too much. Flags of near pairs that do differ are counted
by direction; arithmetic without bias flips them either way and only a
fraction of them (rounding errors are ~10x below the band).
"""
import numpy as np

NEAR = 1e-5
REL = 1e-5
NEAR_FRAC_MAX = 1e-3


def margin_tol(ref_margin, ref_mscale, cand_in):
    bound = np.abs(ref_margin + cand_in[:, None]) if ref_margin.ndim == 2 else np.abs(ref_margin + cand_in)
    return REL * np.maximum(np.maximum(bound, ref_mscale), 1.0)


def near_report(ref, flags):
    """Near pairs and, among them, the pairs whose feasibility differs: GPU
    feasible where the oracle is not, and the other way round."""
    near = ref["near"] <= NEAR
    gf, of = flags == 15, ref["flags"] == 15
    return {"pairs": int(near.size), "near": int(near.sum()),
            "near_gpu_only": int((near & gf & ~of).sum()),
            "near_oracle_only": int((near & ~gf & of).sum())}


def compare_pairs(ref, flags, margin, cand_in, kvpeak=None, tcand=None, label="", report=None):
    """ref: oracle dict (2-D [C, W] arrays or 1-D per-pair arrays). Returns
    the number of near pairs; `report` (a dict) receives near_report()."""
    near = ref["near"] <= NEAR
    far = ~near
    rep = near_report(ref, flags)
    if report is not None:
        report.update(rep)
    assert rep["near"] <= max(NEAR_FRAC_MAX * rep["pairs"], 2), "%s: %d near pairs of %d" % (
        label, rep["near"], rep["pairs"])
    flips = rep["near_gpu_only"] + rep["near_oracle_only"]
    assert flips <= max(rep["near"] // 2, 1), "%s: %d of %d near pairs flip" % (
        label, flips, rep["near"])
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
