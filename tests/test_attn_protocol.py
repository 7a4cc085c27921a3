"""A model of the attention kernel's barrier protocol, checked over every interleaving.

The roles of csrc/attn.cu as state machines over its mbarriers: the TMA thread (Q once, then K_t
once S_t-2 has completed and V_t-1 once its stage is free), the UMMA thread (S_0, S_1, then per
tile PV_j after P_j and V_j, and S_j+2 after K_j+2, one commit each), and the softmax warps (S_j,
an optional rescale of O that waits for PV_j-1, the P_j arrival, the dual snapshot and the
epilogue).  TMA loads land in any order; a UMMA commit arrives when every UMMA issued before it
has completed, so commits complete in issue order.  Whether tile j needs a rescale is data: both
choices are explored.  For small tile counts every reachable state is visited, and the test
checks:

* parity waits: an mbarrier wait on completion k tests the parity k & 1, which passes whenever
  the barrier's completed-phase count has the other parity.  So from the moment a role starts
  waiting until it passes, the count must stay k or k + 1: at k - 1 the wait would pass too early,
  at k + 2 it would miss its phase;
* stage reuse: a K or V shared-memory stage is reloaded only after the UMMAs that read its
  previous tile have completed, and S_j+2 (which overwrites P_j's TMEM columns) is issued only
  after the softmax warps have published P_j; the softmax warps touch O (rescale, snapshot,
  epilogue) only between the completion of PV_j-1 and the issue of PV_j;
* progress: every interleaving runs to the end (no state without an enabled step before then).

This restates the kernel's schedule (no CUDA is run); the stage counts are those of its three
instances: bf16 with d = 128 (2 K, 2 V stages), 8-bit Q K^T (4 K, 2 V) and d = 64 (4 K, 4 V).
"""
import pytest

# barrier ids
Q, K0, V0, VE0, S0, P0, DRAIN = "q", "k", "v", "ve", "s", "p", "drain"


def tma_program(n, kst, vst):
    prog = [("issue", (Q, 0), ("Q",))]
    for t in range(n + 1):
        if t < n:
            if t >= 2:
                prog.append(("wait", (S0, (t - 2) & 1), (t - 2) >> 1))
            prog.append(("issue", (K0, t % kst), ("K", t)))
        if t >= 1:
            j = t - 1
            # stage free: the PV of tile j - vst has completed (k = -1: a fresh stage)
            prog.append(("wait", (VE0, j % vst), j // vst - 1))
            prog.append(("issue", (V0, j % vst), ("V", j)))
    # drain: every issued load has landed
    prog.append(("wait", (Q, 0), 0))
    for t in range(max(0, n - kst), n):
        prog.append(("wait", (K0, t % kst), t // kst))
    for t in range(max(0, n - vst), n):
        prog.append(("wait", (V0, t % vst), t // vst))
    return prog


def mma_program(n, kst, vst):
    prog = [("wait", (Q, 0), 0)]

    def s_tile(j):
        return [("wait", (K0, j % kst), j // kst), ("commit", (S0, j & 1), ("S", j))]

    prog += s_tile(0)
    if n > 1:
        prog += s_tile(1)
    for j in range(n):
        prog.append(("wait", (P0, j & 1), j >> 1))
        prog.append(("wait", (V0, j % vst), j // vst))
        prog.append(("commit", (VE0, j % vst), ("PV", j)))
        if j + 2 < n:
            prog += s_tile(j + 2)
    prog.append(("commit", (DRAIN, 0), ("drain",)))
    prog.append(("wait", (DRAIN, 0), 0))
    return prog


def softmax_program(n, vst, n_local, rescale):
    """n_local: None for the full/local modes, else the dual pass's local tile count."""
    prog = []
    for j in range(n):
        if n_local is not None and j == n_local and j > 0:
            prog.append(("wait", (VE0, (j - 1) % vst), (j - 1) // vst))
            prog.append(("o_access", j))      # A_loc snapshot
        prog.append(("wait", (S0, j & 1), j >> 1))
        if j > 0 and rescale[j]:
            prog.append(("wait", (VE0, (j - 1) % vst), (j - 1) // vst))
            prog.append(("o_access", j))      # O *= alpha
        prog.append(("arrive", (P0, j & 1), ("P", j)))
    prog.append(("wait", (VE0, (n - 1) % vst), (n - 1) // vst))
    prog.append(("o_access", n))              # epilogue
    return prog


class Violation(AssertionError):
    pass


def explore(n, kst, vst, n_local=None):
    """Visit every reachable state; returns the number of states.  Raises Violation."""
    rescale_choices = [tuple(bool(m >> j & 1) for j in range(n)) for m in range(1 << n)]
    n_states = 0
    for rescale in rescale_choices:
        if rescale[0]:
            continue   # tile 0 sets the running max; there is no O to rescale
        progs = (tma_program(n, kst, vst), mma_program(n, kst, vst), softmax_program(n, vst, n_local, rescale))
        n_states += _explore_one(progs, n, kst, vst)
    return n_states


def _explore_one(progs, n, kst, vst):
    # state: (pcs, done (sorted tuple of (barrier, count)), pending loads (frozenset), commit queue,
    #         issued PV tiles, completed S tiles, completed PV tiles, published P tiles)
    start = ((0, 0, 0), (), frozenset(), (), 0, 0, 0, 0)
    seen = set()
    stack = [start]

    def count(done, b):
        for bb, c in done:
            if bb == b:
                return c
        return 0

    def bump(done, b):
        d = dict(done)
        d[b] = d.get(b, 0) + 1
        return tuple(sorted(d.items())), d[b]

    def check_waiters(pcs, done, b, context):
        # every role waiting on b must see its completion count at k or k + 1
        c = count(done, b)
        for r, pc in enumerate(pcs):
            if pc < len(progs[r]) and progs[r][pc][0] == "wait" and progs[r][pc][1] == b:
                k = progs[r][pc][2]
                if not (k <= c <= k + 1):
                    raise Violation(f"{context}: role {r} waits for completion {k} of {b}, count is {c}")

    def enter(pcs, done, r, context):
        # role r has just reached pcs[r]: a wait it starts must not pass early
        pc = pcs[r]
        if pc < len(progs[r]) and progs[r][pc][0] == "wait":
            b, k = progs[r][pc][1], progs[r][pc][2]
            c = count(done, b)
            if not (k <= c <= k + 1):
                raise Violation(f"{context}: role {r} starts waiting for completion {k} of {b}, count is {c}")

    while stack:
        st = stack.pop()
        if st in seen:
            continue
        seen.add(st)
        pcs, done, pending, queue, pv_issued, s_done, pv_done, p_pub = st
        succ = []
        for r in range(3):
            pc = pcs[r]
            if pc >= len(progs[r]):
                continue
            op = progs[r][pc]
            npcs = tuple(pc + 1 if i == r else x for i, x in enumerate(pcs))
            kind = op[0]
            if kind == "wait":
                b, k = op[1], op[2]
                if count(done, b) == k + 1:
                    enter(npcs, done, r, f"after wait {op}")
                    succ.append((npcs, done, pending, queue, pv_issued, s_done, pv_done, p_pub))
            elif kind == "issue":   # TMA load with its barrier armed
                b, what = op[1], op[2]
                if b in pending:
                    raise Violation(f"load {what} re-arms {b} before its previous phase completed")
                if what[0] == "K" and s_done < what[1] - kst + 1:
                    raise Violation(f"K_{what[1]} overwrites a stage whose S has not completed ({s_done} S done)")
                if what[0] == "V" and pv_done < what[1] - vst + 1:
                    raise Violation(f"V_{what[1]} overwrites a stage whose PV has not completed ({pv_done} PV done)")
                enter(npcs, done, r, f"after {what}")
                succ.append((npcs, done, pending | {b}, queue, pv_issued, s_done, pv_done, p_pub))
            elif kind == "commit":
                b, what = op[1], op[2]
                npi = pv_issued
                if what[0] == "S" and what[1] >= 2 and p_pub < what[1] - 1:
                    raise Violation(f"S_{what[1]} issued before P_{what[1] - 2} was published")
                if what[0] == "PV":
                    npi = what[1] + 1
                enter(npcs, done, r, f"after {what}")
                succ.append((npcs, done, pending, queue + ((b, what),), npi, s_done, pv_done, p_pub))
            elif kind == "arrive":
                b = op[1]
                nd, _ = bump(done, b)
                check_waiters(npcs, nd, b, f"arrive {op[2]}")
                enter(npcs, nd, r, f"after {op[2]}")
                succ.append((npcs, nd, pending, queue, pv_issued, s_done, pv_done, p_pub + 1))
            elif kind == "o_access":
                j = op[1]
                if pv_done < j:
                    raise Violation(f"softmax touches O at tile {j} with {pv_done} PV completed")
                if pv_issued > j:
                    raise Violation(f"softmax touches O at tile {j} after PV_{pv_issued - 1} was issued")
                enter(npcs, done, r, f"O access {j}")
                succ.append((npcs, done, pending, queue, pv_issued, s_done, pv_done, p_pub))
        for b in pending:   # a TMA load lands
            nd, _ = bump(done, b)
            check_waiters(pcs, nd, b, f"load on {b} landed")
            succ.append((pcs, nd, pending - {b}, queue, pv_issued, s_done, pv_done, p_pub))
        if queue:           # the oldest commit arrives
            (b, what), rest = queue[0], queue[1:]
            nd, _ = bump(done, b)
            check_waiters(pcs, nd, b, f"commit {what}")
            succ.append((pcs, nd, pending, rest, pv_issued, s_done + (what[0] == "S"), pv_done + (what[0] == "PV"),
                         p_pub))
        if not succ:
            finished = all(pcs[r] >= len(progs[r]) for r in range(3)) and not pending and not queue
            if not finished:
                raise Violation(f"deadlock: pcs {pcs} of {[len(p) for p in progs]}, pending {set(pending)}, "
                                f"queue {queue}, done {done}")
        stack.extend(succ)
    return len(seen)


STAGES = [pytest.param(2, 2, id="bf16-d128"), pytest.param(4, 2, id="qk8-d128"), pytest.param(4, 4, id="bf16-d64")]


@pytest.mark.parametrize("kst,vst", STAGES)
@pytest.mark.parametrize("n", [1, 2, 3, 4, 5])
def test_full_and_local_passes(n, kst, vst):
    assert explore(n, kst, vst) > 0


@pytest.mark.parametrize("kst,vst", STAGES)
@pytest.mark.parametrize("n,n_local", [(2, 1), (3, 1), (3, 2), (4, 2), (4, 4), (5, 3)])
def test_dual_pass(n, n_local, kst, vst):
    assert explore(n, kst, vst, n_local) > 0


def _drop_waits(prog, barrier):
    return [op for op in prog if not (op[0] == "wait" and op[1][0] == barrier)]


def _retarget_s_waits(prog, back):
    """K_t released on S_t-back instead of S_t-2."""
    out = []
    for op in prog:
        if op[0] == "wait" and op[1][0] == S0:
            t = 2 * op[2] + op[1][1] + 2
            if t >= back:
                out.append(("wait", (S0, (t - back) & 1), (t - back) >> 1))
        else:
            out.append(op)
    return out


def _s_before_p(orig):
    """S_j+2 issued before the wait for P_j."""
    def prog_fn(n, kst, vst):
        out = []
        for op in orig(n, kst, vst):
            if op[0] == "commit" and op[2][0] == "S" and op[2][1] >= 2:
                # move this S (its K wait is the op before) ahead of the P wait of tile t - 2
                t = op[2][1]
                k_wait = out.pop()
                at = max(x for x, o in enumerate(out)
                         if o[0] == "wait" and o[1] == (P0, (t - 2) & 1) and o[2] == (t - 2) >> 1)
                out[at:at] = [k_wait, op]
            else:
                out.append(op)
        return out
    return prog_fn


# each planted mistake: the program it replaces, how, the check that must report it, and the case
PLANTED = {
    "k_released_on_s_t_3": ("tma_program", lambda f: lambda n, k, v: _retarget_s_waits(f(n, k, v), 3),
                            "starts waiting", (4, 2, 2)),
    "k_released_on_s_t_4_with_4_stages": ("tma_program", lambda f: lambda n, k, v: _retarget_s_waits(f(n, k, v), 4),
                                          "starts waiting", (6, 4, 2)),
    "k_never_released": ("tma_program", lambda f: lambda n, k, v: _drop_waits(f(n, k, v), S0),
                         "overwrites a stage whose S", (4, 2, 2)),
    "v_never_released": ("tma_program", lambda f: lambda n, k, v: _drop_waits(f(n, k, v), VE0),
                         "overwrites a stage whose PV", (4, 2, 2)),
    # (which report comes first depends on the search order: S_j+2 before P_j, or the softmax
    # warps running two tiles ahead of the UMMA thread's P wait)
    "s_issued_before_p": ("mma_program", _s_before_p, "was published|waits for completion", (4, 2, 2)),
}


@pytest.mark.parametrize("kind", sorted(PLANTED))
def test_checker_catches_planted_schedule_errors(kind, monkeypatch):
    import sys
    mod = sys.modules[__name__]
    name, transform, message, (n, kst, vst) = PLANTED[kind]
    monkeypatch.setattr(mod, name, transform(getattr(mod, name)))
    with pytest.raises(Violation, match=message):
        explore(n, kst, vst)


def test_checker_catches_rescale_without_pv_wait(monkeypatch):
    import sys
    mod = sys.modules[__name__]
    orig = softmax_program

    def no_wait(n, vst, n_local, rescale):
        prog = orig(n, vst, n_local, rescale)
        return [op for i, op in enumerate(prog)
                if not (op[0] == "wait" and op[1][0] == VE0 and i + 1 < len(prog) and prog[i + 1][0] == "o_access"
                        and prog[i + 1][1] < n)]
    monkeypatch.setattr(mod, "softmax_program", no_wait)
    with pytest.raises(Violation, match="touches O at tile 1 with 0 PV completed"):
        explore(3, 2, 2)
