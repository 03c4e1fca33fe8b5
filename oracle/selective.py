"""Float64 oracle of the verifier's operating-point calibration and its
selective-prediction metrics (Pro-Router, Section 3.1 and Section 4.1).

TEST INFRASTRUCTURE ONLY: used by the tests, the smoke check and the
benchmark's CPU baseline; the product path never imports it.  Plain numpy
written from the definitions in the text:

* Calibration (Section 3.1, Section 4.1): the threshold tau is fixed on a
  validation pool by the coverage rule of selective prediction -- choose the
  ship fraction q and take the tau that ships that fraction.  Reading: with n
  requests in the pool, k = floor(q n + 1/2) of them ship; tau is the k-th
  largest finite score (ties at tau ship too, so at least k ship); k = 0 gives
  tau = +inf (nothing ships); requests with a NaN score (escalated by a flag)
  never ship, so k is capped at the number of finite scores.
* AUROC (Section 4.1): the probability that a randomly chosen correct answer
  scores above a randomly chosen incorrect one, a tie counting one half.
* AUARC (Section 4.1): the area under the curve of the accuracy of what ships
  against the fraction shipped.  Reading: ship in
  order of decreasing score; after k of the n requests the accuracy is
  C_k / k, where C_k is the number of correct answers among the k shipped;
  AUARC = (1/n) sum_{k=1..n} C_k / k.  Inside a group of tied scores the order
  is not defined, so C_k is its expectation over the orders of the group
  (correct answers spread evenly over the group).  The same computation with
  the pairwise label gives AUACC.
Requests with a NaN score are left out of AUROC and AUARC.

Parity status: AUROC is pinned against brute-force pair counting and
scikit-learn's roc_auc_score; AUARC against brute-force averaging over every
order of tied groups on small cases and closed forms (perfect ranking, equal
scores, all correct); the calibration against its definition by counting.
The array forms (auroc, auarc) are pinned against the loop forms.
"""
from __future__ import annotations

import numpy as np


def ship_count(n: int, q: float) -> int:
    """Requests the coverage rule ships out of n for ship fraction q."""
    return int(np.floor(float(q) * n + 0.5))


def calibrate(scores, q: float):
    """(tau, k, n_ship): tau is the k-th largest finite score; n_ship counts
    the scores >= tau (ties included)."""
    s = np.asarray(scores, np.float64)
    fin = s[np.isfinite(s)]
    k = min(ship_count(s.size, q), fin.size)
    if k <= 0:
        return np.inf, 0, 0
    desc = np.sort(fin)[::-1]
    tau = desc[k - 1]
    return float(tau), k, int(np.count_nonzero(fin >= tau))


def auroc_pairs(scores, labels) -> float:
    """AUROC by counting every (correct, incorrect) pair: O(P N)."""
    s = np.asarray(scores, np.float64)
    y = np.asarray(labels).astype(bool)
    keep = np.isfinite(s)
    s, y = s[keep], y[keep]
    pos, neg = s[y], s[~y]
    if pos.size == 0 or neg.size == 0:
        return float("nan")
    diff = pos[:, None] - neg[None, :]
    return float(((diff > 0).sum() + 0.5 * (diff == 0).sum()) / (pos.size * neg.size))


def auroc_ranks(scores, labels) -> float:
    """AUROC from average ranks (Mann-Whitney), tie groups walked in a loop:
    the same number as auroc_pairs in O(n log n)."""
    s = np.asarray(scores, np.float64)
    y = np.asarray(labels).astype(bool)
    keep = np.isfinite(s)
    s, y = s[keep], y[keep]
    P, N = int(y.sum()), int((~y).sum())
    if P == 0 or N == 0:
        return float("nan")
    order = np.argsort(s, kind="stable")
    ss = s[order]
    ranks = np.empty(s.size)
    i = 0
    while i < ss.size:  # average rank of each tie group (1-based)
        j = i
        while j + 1 < ss.size and ss[j + 1] == ss[i]:
            j += 1
        ranks[order[i:j + 1]] = 0.5 * (i + j) + 1.0
        i = j + 1
    return float((ranks[y].sum() - P * (P + 1) / 2.0) / (P * N))


def auroc(scores, labels) -> float:
    """auroc_ranks with the tie groups found by array operations (for pools of
    millions of scores)."""
    s = np.asarray(scores, np.float64)
    y = np.asarray(labels).astype(bool)
    keep = np.isfinite(s)
    s, y = s[keep], y[keep]
    P, N = int(y.sum()), int((~y).sum())
    if P == 0 or N == 0:
        return float("nan")
    order = np.argsort(s, kind="stable")
    ss = s[order]
    start = np.flatnonzero(np.r_[True, ss[1:] != ss[:-1]])
    end = np.r_[start[1:], ss.size]             # group [start, end), 0-based
    grp = np.cumsum(np.r_[True, ss[1:] != ss[:-1]]) - 1
    avg_rank = 0.5 * (start + end - 1) + 1.0    # 1-based average rank of each group
    rank_sum = avg_rank[grp][y[order]].sum()
    return float((rank_sum - P * (P + 1) / 2.0) / (P * N))


def auarc_loop(scores, labels) -> float:
    """AUARC with tie groups averaged, computed one shipped request at a
    time."""
    s = np.asarray(scores, np.float64)
    y = np.asarray(labels).astype(np.float64)
    keep = np.isfinite(s)
    s, y = s[keep], y[keep]
    n = s.size
    if n == 0:
        return float("nan")
    order = np.argsort(-s, kind="stable")
    ss, yy = s[order], y[order]
    total = 0.0
    shipped, correct = 0, 0.0
    i = 0
    while i < n:
        j = i
        while j + 1 < n and ss[j + 1] == ss[i]:
            j += 1
        g, cg = j - i + 1, yy[i:j + 1].sum()
        for m in range(1, g + 1):  # m members of the tie group shipped
            total += (correct + m * cg / g) / (shipped + m)
        shipped += g
        correct += cg
        i = j + 1
    return total / n


def auarc(scores, labels) -> float:
    """auarc_loop with the tie groups found by array operations."""
    s = np.asarray(scores, np.float64)
    y = np.asarray(labels).astype(np.float64)
    keep = np.isfinite(s)
    s, y = s[keep], y[keep]
    n = s.size
    if n == 0:
        return float("nan")
    order = np.argsort(-s, kind="stable")
    ss, yy = s[order], y[order]
    new = np.r_[True, ss[1:] != ss[:-1]]
    start = np.flatnonzero(new)                  # group starts in shipping order
    size = np.diff(np.r_[start, n])
    correct = np.add.reduceat(yy, start)
    before = np.r_[0.0, np.cumsum(correct)[:-1]]  # correct answers shipped before the group
    grp = np.cumsum(new) - 1
    k = np.arange(1, n + 1, dtype=np.float64)     # requests shipped
    m = k - start[grp]                            # members of the own group shipped
    Ck = before[grp] + m * correct[grp] / size[grp]
    return float(np.sum(Ck / k) / n)


def accuracy_at(scores, labels, tau: float):
    """(ship rate, accuracy among shipped) at threshold tau over all n requests."""
    s = np.asarray(scores, np.float64)
    y = np.asarray(labels).astype(bool)
    shipped = np.isfinite(s) & (s >= tau)
    k = int(shipped.sum())
    return k / max(s.size, 1), (float(y[shipped].mean()) if k else float("nan"))


def selective_metrics(scores, labels, q: float) -> dict:
    """Everything the library's selective-metrics call reports."""
    s = np.asarray(scores, np.float64)
    tau, k, n_ship = calibrate(s, q)
    out = {"tau": tau, "k": k, "n_ship": n_ship, "n_finite": int(np.isfinite(s).sum())}
    if labels is not None:
        y = np.asarray(labels).astype(bool)
        fin = np.isfinite(s)
        out["n_pos"] = int(y[fin].sum())
        out["auroc"] = auroc(s, labels)
        out["auarc"] = auarc(s, labels)
        out["acc_shipped"] = (float(y[fin & (s >= tau)].mean()) if n_ship else float("nan"))
    return out
