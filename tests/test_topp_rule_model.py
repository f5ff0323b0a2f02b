"""The top-p builder's selection rule, modelled in numpy float32, against the
top-p contract of Appendix Eq. 9 and the retention rule after it, on rows the
GPU parity tests rarely produce (exact ties, constant rows, planted spikes,
tau_p = 1). The model follows the kernel's documented arithmetic: a 14-bit
key q = min(2^14 - 1, floor((max - x) 2^14 / (max - min))), a radix select on
its digits (3, 3, 4, 4 bits, top first) with the boundary where the
cumulative mass from the top reaches tau_p Z (else the last non-empty digit
value), then every key below the boundary plus the boundary key's blocks in id
order while the mass before them is below the target. The contract: the kept
mass reaches tau_p; dropping the least kept block falls below it; and no
dropped block outranks a kept one by more than the key's resolution,
(max - min) / 16384 in log2 p. The fast path's rule (select_fast: the same
key from fused roundings, two 3-bit digits over every block, the last 8 bits
over a list of the window's blocks) is checked against the same contract."""
import numpy as np
import pytest

QBITS = 14
WIDTHS = (3, 3, 4, 4)
EPS = 2e-5


def select(x, tau):
    """x: float32 logits in log2 units over H_i, in block-id order. Returns the kept mask."""
    x = np.asarray(x, dtype=np.float32)
    if x.size == 0:
        return np.zeros(0, bool)
    m, lo = x.max(), x.min()
    u = (m - x).astype(np.float32)
    p = np.exp2(-u).astype(np.float32)
    z = np.float32(p.sum(dtype=np.float32))
    target = np.float32(tau) * z
    inv_r = np.float32(2 ** QBITS) / max(np.float32(m - lo), np.float32(1e-30))
    key = np.minimum(2 ** QBITS - 1, np.floor((u * inv_r).astype(np.float32))).astype(np.int64)
    wkey, above, shift = 0, np.float32(0), QBITS
    for width in WIDTHS:
        pshift, shift = shift, shift - width
        inwin = (key >> pshift) == wkey
        acc = np.zeros(16, np.float32)
        for j in np.nonzero(inwin)[0]:            # id order, as the kernel adds them
            d = (key[j] >> shift) & ((1 << width) - 1)
            acc[d] = np.float32(acc[d] + p[j])
        run, before_last, found, last = above, above, -1, 0
        for d in range(16):
            if acc[d] > 0:
                last, before_last = d, run
            if found < 0:
                if np.float32(run + acc[d]) >= target:
                    found = d
                else:
                    run = np.float32(run + acc[d])
        above = run if found >= 0 else before_last
        wkey = (wkey << width) | (found if found >= 0 else last)
    kept = key < wkey
    tie = np.float32(0)
    for j in np.nonzero(key == wkey)[0]:
        kept[j] = np.float32(above + tie) < target
        tie = np.float32(tie + p[j])
    return kept


LIST_CAP = 32
SC = np.float32(0.125 * np.log2(np.e))          # softmax scale 1/sqrt(64) in log2 units


def _f32_up(v):
    """The float32 nearest v from above (v exact in float64)."""
    r = np.float32(v)
    return r if float(r) >= v else np.nextafter(r, np.float32(np.inf))


def _cum(w, f, tops, base):
    """float32 sums, in id order, of the w with key below each top, from base."""
    out = []
    for t in tops:
        acc = np.float32(base)
        for wj, fj in zip(w, f):
            if fj < t:
                acc = np.float32(acc + wj)
        out.append(acc)
    return out


def _digit(cm, target, n_vals, lo, hi, step, above):
    d = n_vals - 1
    for k in range(len(cm) - 1, -1, -1):
        if cm[k] >= target:
            d = k
    above = above if d == 0 else cm[d - 1]
    hi = lo + step * (d + 1) if d < n_vals - 1 else hi
    return lo + step * d, hi, above


def select_fast(s, tau):
    """The builder's fast path on raw scores s (float32, block-id order; the
    logits are s * SC in log2 units): m = max x rounded up, u = fma(s, -SC, m),
    the key floor(u inv_r) (one fma toward zero), two 3-bit digits by
    cumulative masses over all blocks, the window's blocks listed (at most
    LIST_CAP, else the radix rule decides), two 4-bit digits over the list from
    the mass below the window, then the boundary key's blocks in id order.
    Returns (kept mask, whether the list held the window)."""
    s = np.asarray(s, dtype=np.float32)
    if s.size == 0:
        return np.zeros(0, bool), True
    smax, smin = s.max(), s.min()
    m = _f32_up(float(smax) * float(SC))
    inv_r = np.float32(2 ** QBITS) / max(np.float32(np.float32(smax - smin) * SC), np.float32(1e-30))
    u = np.array([np.float32(float(v) * -float(SC) + float(m)) for v in s], np.float32)
    w = np.exp2(-u).astype(np.float32)
    f = np.floor(u.astype(np.float64) * float(inv_r))       # the key, exact product floored
    z = np.float32(0)
    for wj in w:
        z = np.float32(z + wj)
    target = np.float32(tau) * z
    lo, hi, above = 0.0, np.inf, np.float32(0)
    for step in (2048.0, 256.0):
        cm = _cum(w, f, [lo + step * (k + 1) for k in range(7)], 0.0)
        lo, hi, above = _digit(cm, target, 8, lo, hi, step, above)
    kept = f < lo
    win = np.nonzero((f >= lo) & (f < hi))[0]
    if win.size > LIST_CAP:
        return select(s * SC, tau), False
    base = above
    for step in (16.0, 1.0):
        cm = _cum(w[win], f[win], [lo + step * (k + 1) for k in range(15)], base)
        lo, hi, above = _digit(cm, target, 16, lo, hi, step, above)
    tie = np.float32(0)
    for j in win:
        if f[j] < lo:
            kept[j] = True
        elif f[j] < hi:
            kept[j] = np.float32(above + tie) < target
            tie = np.float32(tie + w[j])
    return kept, True


def _check(lg, tau, fast=False):
    x = (lg / np.log(2)).astype(np.float32)
    kept = select_fast((x / SC).astype(np.float32), tau)[0] if fast else select(x, tau)
    p = np.exp(lg - lg.max())
    p /= p.sum()
    t = min(tau, 1 - 1e-6)
    mass = p[kept].sum()
    assert mass >= t - EPS, ("mass", mass)
    assert mass - p[kept].min() < t + EPS, ("not minimal", mass, p[kept].min())
    if (~kept).any():
        lp = np.log2(p)
        res = (lp.max() - lp.min()) / 16384 + 3e-5
        assert lp[kept].min() >= lp[~kept].max() - res, "not a top set"


@pytest.mark.parametrize("fast", [False, True], ids=["radix", "fast"])
@pytest.mark.parametrize("kind", ["gauss_small", "gauss_wide", "rounded_ties", "constant", "spikes", "near_uniform"])
@pytest.mark.parametrize("tau", [0.3, 0.9, 0.97, 1.0])
def test_rule_meets_the_top_p_contract(kind, tau, fast):
    rng = np.random.default_rng(hash((kind, tau)) % 2 ** 32)
    for _ in range(60):
        n = int(rng.integers(1, 300))
        if kind == "gauss_small":
            lg = rng.normal(0, 0.3, n)
        elif kind == "gauss_wide":
            lg = rng.normal(0, 4, n)
        elif kind == "rounded_ties":
            lg = np.round(rng.normal(0, 2, n), 1)          # many exactly equal logits
        elif kind == "constant":
            lg = np.zeros(n)
        elif kind == "spikes":
            lg = rng.normal(0, 1, n)
            lg[rng.integers(0, n, 3)] += 12
        else:
            lg = rng.normal(0, 1e-3, n)                    # the workloads' nearly uniform rows
        _check(lg, tau, fast)


def test_ties_go_to_the_lower_id():
    lg = np.zeros(10)
    kept = select((lg / np.log(2)).astype(np.float32), 0.35)
    assert kept.tolist() == [True] * 4 + [False] * 6        # 4 x 0.1 is the first prefix >= 0.35
    kept, listed = select_fast(np.zeros(10, np.float32), 0.35)
    assert listed and kept.tolist() == [True] * 4 + [False] * 6


def test_fast_path_lists_the_window_on_spread_rows():
    """Rows like the workloads' (a few hundred blocks of spread logits) resolve
    on the fast path; a constant row longer than the list goes to the radix rule."""
    rng = np.random.default_rng(9)
    listed = [select_fast((rng.normal(0, 1, 600) / np.log(2) / SC).astype(np.float32), 0.97)[1] for _ in range(20)]
    assert all(listed)
    assert not select_fast(np.zeros(100, np.float32), 0.97)[1]


def test_tau_one_drops_only_rounding_level_mass():
    """At tau_p = 1 the target is the fp32 total itself: the cumulative sums can
    reach it before the last blocks of the tail, whose mass is below fp32
    rounding of the total; nothing larger is dropped."""
    rng = np.random.default_rng(5)
    for _ in range(40):
        lg = rng.normal(0, 3, int(rng.integers(1, 200)))
        kept = select((lg / np.log(2)).astype(np.float32), 1.0)
        p = np.exp(lg - lg.max())
        p /= p.sum()
        assert p[~kept].sum() < 1e-6 * len(lg)
