"""A model of the attention kernel's barrier protocol, checked over every interleaving.

The roles of csrc/attn.cu as state machines over its mbarriers, for a CTA that works through m
items (query tile, head) of n key tiles each, the key tiles numbered g = k * n + j across items:

* the TMA thread: Q of the first item, then K_t once S_t-2 has completed and V_t-1 once its stage
  is free; at an item boundary the previous item's last V, then the next Q once the previous
  item's last S has completed; a try_cancel request per item (at its start for short items, four
  K tiles before its end otherwise), whose response it waits for at the item's end before it
  posts the next item (or none) to a two-slot mailbox, a slot being reused only after both
  consumers have read its previous item;
* the UMMA thread: S_0, S_1, then per tile PV_g after P_g and V_g and S_g+2 after K_g+2 within the
  item; at the item's end it reads the mailbox, waits for the next Q and issues the next item's
  first two S tiles (the next item's first PV, which overwrites O, follows P'_0, which the softmax
  warps publish after reading O in the epilogue);
* the softmax warps: S_g, an optional rescale of O that waits for PV_g-1, the P_g arrival, the dual
  snapshot and the epilogue, then the mailbox read.

TMA loads and try_cancel responses land in any order; a UMMA commit arrives when every UMMA issued
before it has completed, so commits complete in issue order.  Whether tile j needs a rescale is
data: both choices are explored.  For small tile and item counts every reachable state is visited,
and the test checks:

* parity waits: an mbarrier wait on completion k tests the parity k & 1, which passes whenever
  the barrier's completed-phase count has the other parity.  So from the moment a role starts
  waiting until it passes, the count must stay k or k + 1: at k - 1 the wait would pass too early,
  at k + 2 it would miss its phase;
* buffer reuse: a K or V shared-memory stage is reloaded only after the UMMAs that read its
  previous tile have completed; the Q tile of item k only after every S of the items before it
  has completed, and an S tile is issued only after its item's Q has landed; S_g+2 (which
  overwrites P_g's TMEM columns) only after the softmax warps have published P_g; the softmax
  warps touch O (rescale, snapshot, epilogue) only between the completion of PV_g-1 and the issue
  of PV_g, g counted across items; a mailbox slot is rewritten only after both readers are done
  with its previous item;
* progress: every interleaving runs to the end (no state without an enabled step before then).

This restates the kernel's schedule (no CUDA is run); the stage counts are those of its three
instances: bf16 with d = 128 (2 K, 2 V stages), 8-bit Q K^T (4 K, 2 V) and d = 64 (4 K, 4 V).
"""
import pytest

# barrier ids: Q, K stages, V full / empty, S, P, drain, try_cancel response, mailbox
Q, K0, V0, VE0, S0, P0, DRAIN, CLC, IF, IE = "q", "k", "v", "ve", "s", "p", "drain", "clc", "if", "ie"
ARRIVALS = {IE: 2}   # arrivals per phase where more than one (the UMMA thread and the softmax warps)


def tma_program(n, kst, vst, m=1):
    prog = []
    req_at = n - 4 if n > 4 else 0
    nreq, nresp = 0, 0

    def request():
        nonlocal nreq
        prog.append(("issue", (CLC, 0), ("R", nreq)))
        nreq += 1

    t = tv = 0
    kk = kj = 0
    k_live = True

    def issue_v():
        nonlocal tv
        # stage free: the PV of tile tv - vst has completed (k = -1: a fresh stage)
        prog.append(("wait", (VE0, tv % vst), tv // vst - 1))
        prog.append(("issue", (V0, tv % vst), ("V", tv)))
        tv += 1

    prog.append(("issue", (Q, 0), ("Q", 0)))
    if req_at == 0:
        request()
    while True:
        if k_live:
            if kj == 0 and kk > 0:
                if tv < t:
                    issue_v()
                prog.append(("wait", (S0, (t - 1) & 1), (t - 1) >> 1))
                prog.append(("issue", (Q, 0), ("Q", kk)))
                if req_at == 0:
                    request()
            if t >= 2:
                prog.append(("wait", (S0, (t - 2) & 1), (t - 2) >> 1))
            prog.append(("issue", (K0, t % kst), ("K", t)))
            t += 1
            kj += 1
            if kj == req_at and req_at > 0:
                request()
            if kj == n:
                if nreq > nresp:
                    prog.append(("wait", (CLC, 0), nresp))
                    nresp += 1
                sl = kk & 1
                prog.append(("wait", (IE, sl), (kk >> 1) - 1))
                prog.append(("arrive", (IF, sl), ("M", kk)))
                if kk + 1 < m:
                    kk += 1
                    kj = 0
                else:
                    k_live = False
        if tv < t - (1 if k_live else 0):
            issue_v()
        elif not k_live:
            break
    # drain: every issued load has landed
    prog.append(("wait", (Q, 0), m - 1))
    for g in range(max(0, t - kst), t):
        prog.append(("wait", (K0, g % kst), g // kst))
    for g in range(max(0, tv - vst), tv):
        prog.append(("wait", (V0, g % vst), g // vst))
    if nreq > nresp:
        prog.append(("wait", (CLC, 0), nresp))
    return prog


def mma_program(n, kst, vst, m=1):
    prog = [("wait", (Q, 0), 0)]

    def s_tile(g):
        return [("wait", (K0, g % kst), g // kst), ("commit", (S0, g & 1), ("S", g))]

    prog += s_tile(0)
    if n > 1:
        prog += s_tile(1)
    for k in range(m):
        base = k * n
        for j in range(n):
            g = base + j
            prog.append(("wait", (P0, g & 1), g >> 1))
            prog.append(("wait", (V0, g % vst), g // vst))
            prog.append(("commit", (VE0, g % vst), ("PV", g)))
            if j + 2 < n:
                prog += s_tile(g + 2)
        prog.append(("wait", (IF, k & 1), k >> 1))
        prog.append(("arrive", (IE, k & 1), ("E", k)))
        if k + 1 < m:
            prog.append(("wait", (Q, 0), k + 1))
            prog += s_tile(base + n)
            if n > 1:
                prog += s_tile(base + n + 1)
    prog.append(("commit", (DRAIN, 0), ("drain",)))
    prog.append(("wait", (DRAIN, 0), 0))
    return prog


def softmax_program(n, vst, n_local, rescale, m=1):
    """n_local: None for the full/local modes, else the dual pass's local tile count.
    rescale[g]: whether global tile g needs a rescale of O."""
    prog = []
    for k in range(m):
        base = k * n
        for j in range(n):
            g = base + j
            if n_local is not None and j == n_local and j > 0:
                prog.append(("wait", (VE0, (g - 1) % vst), (g - 1) // vst))
                prog.append(("o_access", g))      # A_loc snapshot
            prog.append(("wait", (S0, g & 1), g >> 1))
            if j > 0 and rescale[g]:
                prog.append(("wait", (VE0, (g - 1) % vst), (g - 1) // vst))
                prog.append(("o_access", g))      # O *= alpha
            prog.append(("arrive", (P0, g & 1), ("P", g)))
        g = base + n
        prog.append(("wait", (VE0, (g - 1) % vst), (g - 1) // vst))
        prog.append(("o_access", g))              # epilogue
        prog.append(("wait", (IF, k & 1), k >> 1))
        prog.append(("arrive", (IE, k & 1), ("E", k)))
    return prog


class Violation(AssertionError):
    pass


def explore(n, kst, vst, n_local=None, m=1):
    """Visit every reachable state; returns the number of states.  Raises Violation."""
    n_states = 0
    for mask in range(1 << (n * m)):
        rescale = tuple(bool(mask >> g & 1) for g in range(n * m))
        if any(rescale[k * n] for k in range(m)):
            continue   # an item's tile 0 sets the running max; there is no O to rescale
        if m > 1 and mask >> n:
            continue   # with several items the first item's choices suffice (fewer states)
        progs = (tma_program(n, kst, vst, m), mma_program(n, kst, vst, m),
                 softmax_program(n, vst, n_local, rescale, m))
        n_states += _explore_one(progs, n, kst, vst)
    return n_states


def _explore_one(progs, n, kst, vst):
    # state: (pcs, done (sorted (barrier, count)), partial arrivals, pending loads (frozenset),
    #         commit queue, counters (PV issued, S done, PV done, P published, mailbox posts,
    #         mailbox reads by the UMMA thread / the softmax warps))
    start = ((0, 0, 0), (), (), frozenset(), (), (0, 0, 0, 0, 0, 0, 0))
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
        return tuple(sorted(d.items()))

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
        pcs, done, partial, pending, queue, ctr = st
        pv_issued, s_done, pv_done, p_pub, posts, read_mma, read_soft = ctr
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
                    succ.append((npcs, done, partial, pending, queue, ctr))
            elif kind == "issue":   # TMA load (or try_cancel) with its barrier armed
                b, what = op[1], op[2]
                if b in pending:
                    raise Violation(f"load {what} re-arms {b} before its previous phase completed")
                if what[0] == "K" and s_done < what[1] - kst + 1:
                    raise Violation(f"K_{what[1]} overwrites a stage whose S has not completed ({s_done} S done)")
                if what[0] == "V" and pv_done < what[1] - vst + 1:
                    raise Violation(f"V_{what[1]} overwrites a stage whose PV has not completed ({pv_done} PV done)")
                if what[0] == "Q" and s_done < what[1] * n:
                    raise Violation(f"Q of item {what[1]} overwrites Q with {s_done} S done")
                enter(npcs, done, r, f"after {what}")
                succ.append((npcs, done, partial, pending | {b}, queue, ctr))
            elif kind == "commit":
                b, what = op[1], op[2]
                npi = pv_issued
                if what[0] == "S":
                    g = what[1]
                    if g >= 2 and p_pub < g - 1:
                        raise Violation(f"S_{g} issued before P_{g - 2} was published")
                    if count(done, (Q, 0)) < g // n + 1:
                        raise Violation(f"S_{g} issued before the Q of its item landed")
                if what[0] == "PV":
                    npi = what[1] + 1
                enter(npcs, done, r, f"after {what}")
                succ.append((npcs, done, partial, pending, queue + ((b, what),),
                             (npi, s_done, pv_done, p_pub, posts, read_mma, read_soft)))
            elif kind == "arrive":
                b, what = op[1], op[2]
                n_p, n_rm, n_rs, n_post = p_pub, read_mma, read_soft, posts
                if what[0] == "P":
                    n_p += 1
                elif what[0] == "M":
                    if min(read_mma, read_soft) < what[1] - 1:
                        raise Violation(f"mailbox slot of item {what[1]} rewritten before item {what[1] - 2} was read")
                    n_post += 1
                elif what[0] == "E":
                    if r == 1:
                        n_rm += 1
                    else:
                        n_rs += 1
                need = ARRIVALS.get(b[0], 1)
                pa = dict(partial)
                got = pa.get(b, 0) + 1
                nd = done
                if got == need:
                    pa.pop(b, None)
                    nd = bump(done, b)
                    check_waiters(npcs, nd, b, f"arrive {what}")
                else:
                    pa[b] = got
                enter(npcs, nd, r, f"after {what}")
                succ.append((npcs, nd, tuple(sorted(pa.items())), pending, queue,
                             (pv_issued, s_done, pv_done, n_p, n_post, n_rm, n_rs)))
            elif kind == "o_access":
                g = op[1]
                if pv_done < g:
                    raise Violation(f"softmax touches O at tile {g} with {pv_done} PV completed")
                if pv_issued > g:
                    raise Violation(f"softmax touches O at tile {g} after PV_{pv_issued - 1} was issued")
                enter(npcs, done, r, f"O access {g}")
                succ.append((npcs, done, partial, pending, queue, ctr))
        for b in pending:   # a TMA load (or a try_cancel response) lands
            nd = bump(done, b)
            check_waiters(pcs, nd, b, f"load on {b} landed")
            succ.append((pcs, nd, partial, pending - {b}, queue, ctr))
        if queue:           # the oldest commit arrives
            (b, what), rest = queue[0], queue[1:]
            nd = bump(done, b)
            check_waiters(pcs, nd, b, f"commit {what}")
            succ.append((pcs, nd, partial, pending, rest,
                         (pv_issued, s_done + (what[0] == "S"), pv_done + (what[0] == "PV"), p_pub, posts, read_mma,
                          read_soft)))
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


@pytest.mark.parametrize("kst,vst", STAGES)
@pytest.mark.parametrize("n,m", [(1, 2), (1, 3), (2, 2), (2, 3), (3, 2), (5, 2)])
def test_several_items(n, m, kst, vst):
    # items of 1-5 tiles back to back: Q, the O hand-over, the mailbox and the try_cancel
    # responses across item boundaries (5 tiles: the request goes out one K tile into the item)
    assert explore(n, kst, vst, None, m) > 0


@pytest.mark.parametrize("n,n_local,m", [(2, 1, 2), (3, 2, 2)])
def test_several_items_dual(n, n_local, m):
    assert explore(n, 2, 2, n_local, m) > 0


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
    def prog_fn(n, kst, vst, m=1):
        out = []
        for op in orig(n, kst, vst, m):
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
    "k_released_on_s_t_3": ("tma_program", lambda f: lambda n, k, v, m=1: _retarget_s_waits(f(n, k, v, m), 3),
                            "starts waiting", (4, 2, 2)),
    "k_released_on_s_t_4_with_4_stages": ("tma_program",
                                          lambda f: lambda n, k, v, m=1: _retarget_s_waits(f(n, k, v, m), 4),
                                          "starts waiting", (6, 4, 2)),
    "k_never_released": ("tma_program", lambda f: lambda n, k, v, m=1: _drop_waits(f(n, k, v, m), S0),
                         "overwrites a stage whose S", (4, 2, 2)),
    "v_never_released": ("tma_program", lambda f: lambda n, k, v, m=1: _drop_waits(f(n, k, v, m), VE0),
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

    def no_wait(n, vst, n_local, rescale, m=1):
        prog = orig(n, vst, n_local, rescale, m)
        return [op for i, op in enumerate(prog)
                if not (op[0] == "wait" and op[1][0] == VE0 and i + 1 < len(prog) and prog[i + 1][0] == "o_access"
                        and prog[i + 1][1] < n)]
    monkeypatch.setattr(mod, "softmax_program", no_wait)
    with pytest.raises(Violation, match="touches O at tile 1 with 0 PV completed"):
        explore(3, 2, 2)


def _drop_q_reuse_wait(prog):
    """The next item's Q goes out without waiting for the previous item's last S."""
    out = []
    for i, op in enumerate(prog):
        if op[0] == "wait" and op[1][0] == S0 and i + 1 < len(prog) and prog[i + 1][0] == "issue" \
                and prog[i + 1][2][0] == "Q":
            continue
        out.append(op)
    return out


MULTI_PLANTED = {
    "q_reloaded_before_last_s": ("tma_program", lambda f: lambda n, k, v, m=1: _drop_q_reuse_wait(f(n, k, v, m)),
                                 "overwrites Q", (3, 2, 2, 2)),
    "mailbox_slot_reused_early": ("tma_program", lambda f: lambda n, k, v, m=1: _drop_waits(f(n, k, v, m), IE),
                                  "rewritten before", (1, 2, 2, 3)),
}


@pytest.mark.parametrize("kind", sorted(MULTI_PLANTED))
def test_checker_catches_planted_item_boundary_errors(kind, monkeypatch):
    import sys
    mod = sys.modules[__name__]
    name, transform, message, (n, kst, vst, m) = MULTI_PLANTED[kind]
    monkeypatch.setattr(mod, name, transform(getattr(mod, name)))
    with pytest.raises(Violation, match=message):
        explore(n, kst, vst, None, m)
