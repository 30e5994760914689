"""Plain reference of the plan constructor's host statistics (Sec. 3.2-3.3).

TEST INFRASTRUCTURE ONLY: written from the paper with Python loops and fp64
arithmetic, one function per definition; the product library never imports
it, and it never touches the product library.  Only the test suite may use it.
"""
from __future__ import annotations

import math

# Operator numbering of the oracle (its own).
FULL, SNAPKV, H2O, STREAMING, TOVA = 0, 1, 2, 3, 4
PREFILL_OPS = (FULL, SNAPKV, H2O, STREAMING)
DECODE_OPS = (FULL, H2O, TOVA, STREAMING)
SCOPE_PREFILL, SCOPE_DECODE, SCOPE_BOTH = 1, 2, 3


def cosine_profile(h_full, h_cand):
    """Sec. 3.2: C[l][r] = cos(h_full_l, h_r_l) = <a, b> / (|a| |b|).
    h_full: L lists of D floats; h_cand: R lists of L lists of D floats."""
    L, R = len(h_full), len(h_cand)
    out = [[0.0] * R for _ in range(L)]
    for l in range(L):
        a = [float(x) for x in h_full[l]]
        na = math.sqrt(sum(x * x for x in a))
        for r in range(R):
            b = [float(x) for x in h_cand[r][l]]
            nb = math.sqrt(sum(x * x for x in b))
            out[l][r] = sum(x * y for x, y in zip(a, b)) / (na * nb)
    return out


def ppl_score(ppl, ppl_full):
    """Sec. 3.3: S^ppl_l = max over the profiled operators r of
    Delta PPL_{l,r} = PPL_{l,r} - PPL_full."""
    return [max(float(v) - float(ppl_full) for v in row) for row in ppl]


def entropy_score(A):
    """Sec. 3.3: H_l = E_{x,h,q}[ H(A^(l)_{h,q,:}) ], the mean Shannon entropy
    (natural log) of layer l's attention rows; A[l] is a list of rows, each a
    probability distribution over keys (0 log 0 = 0)."""
    out = []
    for rows in A:
        tot = 0.0
        for row in rows:
            tot += -sum(float(p) * math.log(float(p)) for p in row if p > 0)
        out.append(tot / len(rows))
    return out


def toprank(g, ops, higher_is_better, covered=None):
    """Sec. 3.2, Eq. (policy_routing): rho_l = TopRank over the covered
    operators r of g_{l,r} (highest for the cosine profile, lowest for the
    PPL profile).  Reading where the paper is silent: equal statistics keep
    the operator listed first; a layer with no covered operator stays FULL."""
    out = []
    for l, row in enumerate(g):
        cand = [r for r in range(len(row)) if covered is None or covered[l][r]]
        if not cand:
            out.append(FULL)
            continue
        best = cand[0]
        for r in cand[1:]:
            if (row[r] > row[best]) if higher_is_better else (row[r] < row[best]):
                best = r
        out.append(ops[best])
    return out


def install(route, scope):
    """Sec. 3.2: the selected operator is installed in every active phase of
    the scope, inactive phases use FULL.  Returns (route_prefill,
    route_decode), or None if an operator is not valid in an active phase."""
    pre_on, dec_on = bool(scope & SCOPE_PREFILL), bool(scope & SCOPE_DECODE)
    for m in route:
        if (pre_on and m not in PREFILL_OPS) or (dec_on and m not in DECODE_OPS):
            return None
    return ([m if pre_on else FULL for m in route], [m if dec_on else FULL for m in route])
