"""The fixed layer-timestep schedule (Section 3.3, Eq. 5), plain Python.

The paper fixes, before evaluation, the base policy's full-refresh timesteps
and a sparse site set S of (timestep, layer) pairs, shared by every sample and
by both the Verify and FeatFix arms.  Steps and layers are 0-based here.

Per (step i, layer l) the decision is
  EXACT  if i is a full-refresh step (or every step in the vanilla arm),
  SITE   if (i, l) is in S  (paid check: draft and exact from the same u),
  DRAFT  otherwise.
The draft order at step i is K_eff(i) = min(K, r(i) - 1) where r(i) counts
the refresh steps <= i.

Schedule rules (violations raise ScheduleError): step 0 must be a refresh
(no history exists before it), refresh steps lie in [0, steps) and are
distinct, a site lies in range and not on a refresh step (a paid check is
defined at skipped sites), sites are distinct, 0 <= K <= 3.

Test infrastructure only.
"""

EXACT, DRAFT, SITE = 0, 1, 2

MODES = ("featfix", "verify", "exact_only", "vanilla")


class ScheduleError(ValueError):
    pass


def validate(steps, L, refresh, K, sites):
    if steps <= 0 or L <= 0:
        raise ScheduleError("steps and layers must be positive")
    if not 0 <= K <= 3:
        raise ScheduleError("draft order must be in [0, 3]")
    if len(set(refresh)) != len(refresh):
        raise ScheduleError("duplicate refresh step")
    if any(not 0 <= s < steps for s in refresh):
        raise ScheduleError("refresh step out of range")
    if 0 not in refresh:
        raise ScheduleError("step 0 must be a full refresh")
    rs = set(refresh)
    seen = set()
    for (i, l) in sites:
        if not (0 <= i < steps and 0 <= l < L):
            raise ScheduleError("site out of range")
        if i in rs:
            raise ScheduleError("site on a refresh step")
        if (i, l) in seen:
            raise ScheduleError("duplicate site")
        seen.add((i, l))


def block_history_steps(steps, L, refresh, K, sites, mode, site_updates_history=False):
    """Per (step, layer) the steps of the history entries a draft at that
    point reads, newest first (at most K + 1), or None where no draft is
    formed (exact blocks, the vanilla arm).  Refreshes push every block; with
    ``site_updates_history`` a site pushes its own block after its draft."""
    kind, _ = build_plan(steps, L, refresh, K, sites, mode)
    nodes = [[] for _ in range(L)]
    out = []
    for i in range(steps):
        row = []
        for l in range(L):
            if kind[i][l] == EXACT:
                row.append(None)
                if mode != "vanilla":
                    nodes[l] = ([i] + nodes[l])[:K + 1]
            else:
                row.append(list(nodes[l]))
                if kind[i][l] == SITE and site_updates_history:
                    nodes[l] = ([i] + nodes[l])[:K + 1]
        out.append(row)
    return out


def build_plan(steps, L, refresh, K, sites, mode):
    """Return (kind[steps][L], k_eff[steps]).

    ``sites`` holds (step, layer) pairs.  In the vanilla arm every block is
    exact and S is unused.
    """
    if mode not in MODES:
        raise ScheduleError("unknown mode")
    validate(steps, L, refresh, K, sites)
    rs = set(refresh)
    S = set((int(i), int(l)) for (i, l) in sites)
    kind = []
    k_eff = []
    r = 0
    for i in range(steps):
        if i in rs:
            r += 1
        row = []
        for l in range(L):
            if mode == "vanilla" or i in rs:
                row.append(EXACT)
            elif (i, l) in S:
                row.append(SITE)
            else:
                row.append(DRAFT)
        kind.append(row)
        k_eff.append(min(K, r - 1))
    return kind, k_eff
