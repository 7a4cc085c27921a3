"""A model of the barrier schedule shared by the Gram kernels and the W8A8 GEMM, checked over every
interleaving.

All three kernels (csrc/gram.cu: gram_kernel<128> and gram_wide_kernel; csrc/w8a8.cu) run the
same two hand-offs:

* a ring of ST shared-memory stages from the TMA thread to the UMMA thread: step i waits for
  empty[i % ST] (completion i / ST - 1, i.e. the UMMAs of step i - ST are done) before loading,
  and the UMMA thread waits for full[i % ST] (completion i / ST), issues the step's UMMAs and
  commits empty[i % ST];
* NB accumulators in TMEM from the UMMA thread to the epilogue warps: segment m (one output tile,
  or a stream-K piece of one) accumulates into accumulator m % NB after every epilogue group has
  released segment m - NB (acce, completion m / NB - 1), then commits accf (completion m / NB);
  each epilogue group waits for accf, reads the accumulator and arrives at its acce.

gram_kernel<128> and the W8A8 GEMM use NB = 2 accumulators and one epilogue group;
gram_wide_kernel uses NB = 1 (a 256 x 256 tile over all 512 TMEM columns) with two epilogue
groups, one per 128-row half, each releasing its half through its own barrier.  TMA loads land in
any order and commits complete in issue order; segments have 1-3 steps.  The checks are those of
the attention model: every parity wait sees its barrier at the completion it waits for or one
ahead, a stage is reloaded only after the UMMAs that read it completed, an accumulator is written
only after every epilogue group finished reading its previous segment and read only between its
segment's completion and the next write, and every interleaving runs to the end.
"""
import itertools

import pytest

FULL, EMPTY, ACCF, ACCE, DRAIN = "full", "empty", "accf", "acce", "drain"


def programs(segs, st, nb, groups):
    n_steps = sum(segs)
    tma = []
    for i in range(n_steps):
        tma.append(("wait", (EMPTY, i % st), i // st - 1))
        tma.append(("load", (FULL, i % st), i))
    for i in range(max(0, n_steps - st), n_steps):
        tma.append(("wait", (FULL, i % st), i // st))
    mma = []
    i = 0
    for m, n in enumerate(segs):
        b = m % nb
        for h in range(groups):
            mma.append(("wait", (ACCE, b, h), m // nb - 1))
        for s in range(n):
            mma.append(("wait", (FULL, i % st), i // st))
            mma.append(("umma", m, s == 0))
            mma.append(("commit", (EMPTY, i % st), ("step", i)))
            i += 1
        mma.append(("commit", (ACCF, b), ("seg", m)))
    mma.append(("commit", (DRAIN,), ("drain",)))
    mma.append(("wait", (DRAIN,), 0))
    epis = []
    for h in range(groups):
        e = []
        for m in range(len(segs)):
            b = m % nb
            e.append(("wait", (ACCF, b), m // nb))
            e.append(("read", m, h))
            e.append(("arrive", (ACCE, b, h)))
        epis.append(e)
    return [tma, mma] + epis


class Violation(AssertionError):
    pass


def explore(segs, st, nb, groups, progs=None):
    progs = progs or programs(segs, st, nb, groups)
    n_roles = len(progs)
    # state: pcs, done counts, pending loads, commit queue, steps completed, segments completed,
    #        segments whose first UMMA was issued, per-group segments read
    start = (tuple([0] * n_roles), (), frozenset(), (), 0, 0, 0, tuple([0] * groups))
    seen, stack = set(), [start]

    def count(done, b):
        return dict(done).get(b, 0)

    def bump(done, b):
        d = dict(done)
        d[b] = d.get(b, 0) + 1
        return tuple(sorted(d.items(), key=repr))

    def check_waiters(pcs, done, b, ctx):
        c = count(done, b)
        for r, pc in enumerate(pcs):
            if pc < len(progs[r]) and progs[r][pc][0] == "wait" and progs[r][pc][1] == b:
                k = progs[r][pc][2]
                if not (k <= c <= k + 1):
                    raise Violation(f"{ctx}: role {r} waits for completion {k} of {b}, count is {c}")

    def enter(pcs, done, r, ctx):
        pc = pcs[r]
        if pc < len(progs[r]) and progs[r][pc][0] == "wait":
            b, k = progs[r][pc][1], progs[r][pc][2]
            c = count(done, b)
            if not (k <= c <= k + 1):
                raise Violation(f"{ctx}: role {r} starts waiting for completion {k} of {b}, count is {c}")

    while stack:
        state = stack.pop()
        if state in seen:
            continue
        seen.add(state)
        pcs, done, pending, queue, steps_done, segs_done, segs_started, read = state
        succ = []
        for r in range(n_roles):
            pc = pcs[r]
            if pc >= len(progs[r]):
                continue
            op = progs[r][pc]
            npcs = tuple(pc + 1 if x == r else y for x, y in enumerate(pcs))
            kind = op[0]
            if kind == "wait":
                if count(done, op[1]) == op[2] + 1:
                    enter(npcs, done, r, f"after {op}")
                    succ.append((npcs, done, pending, queue, steps_done, segs_done, segs_started, read))
            elif kind == "load":
                b, i = op[1], op[2]
                if b in pending:
                    raise Violation(f"load {i} re-arms {b} before its previous phase completed")
                if steps_done < i - st + 1:
                    raise Violation(f"load {i} overwrites a stage whose UMMAs have not completed ({steps_done} done)")
                enter(npcs, done, r, f"after load {i}")
                succ.append((npcs, done, pending | {b}, queue, steps_done, segs_done, segs_started, read))
            elif kind == "umma":
                m, first = op[1], op[2]
                nss = segs_started
                if first:
                    if any(x < m - nb + 1 for x in read):
                        raise Violation(f"segment {m} overwrites an accumulator still being read ({read})")
                    nss = m + 1
                enter(npcs, done, r, f"umma of segment {m}")
                succ.append((npcs, done, pending, queue, steps_done, segs_done, nss, read))
            elif kind == "commit":
                enter(npcs, done, r, f"after commit {op[2]}")
                succ.append((npcs, done, pending, queue + ((op[1], op[2]),), steps_done, segs_done, segs_started, read))
            elif kind == "read":
                m, h = op[1], op[2]
                if segs_done < m + 1:
                    raise Violation(f"group {h} reads segment {m} before its UMMAs completed")
                if segs_started > m + nb:
                    raise Violation(f"group {h} reads segment {m} after segment {segs_started - 1} started writing")
                nread = tuple(x + 1 if y == h else x for y, x in enumerate(read))
                enter(npcs, done, r, f"read {m}")
                succ.append((npcs, done, pending, queue, steps_done, segs_done, segs_started, nread))
            elif kind == "arrive":
                nd = bump(done, op[1])
                check_waiters(npcs, nd, op[1], f"arrive {op[1]}")
                enter(npcs, nd, r, f"after arrive {op[1]}")
                succ.append((npcs, nd, pending, queue, steps_done, segs_done, segs_started, read))
        for b in pending:
            nd = bump(done, b)
            check_waiters(pcs, nd, b, f"load on {b} landed")
            succ.append((pcs, nd, pending - {b}, queue, steps_done, segs_done, segs_started, read))
        if queue:
            (b, what), rest = queue[0], queue[1:]
            nd = bump(done, b)
            check_waiters(pcs, nd, b, f"commit {what}")
            succ.append((pcs, nd, pending, rest, steps_done + (what[0] == "step"), segs_done + (what[0] == "seg"),
                         segs_started, read))
        if not succ:
            if not (all(pcs[r] >= len(progs[r]) for r in range(n_roles)) and not pending and not queue):
                raise Violation(f"deadlock: pcs {pcs}, pending {set(pending)}, queue {queue}, done {done}")
        stack.extend(succ)
    return len(seen)


# (stages, accumulators, epilogue groups) of gram_kernel<128> (GST), the W8A8 GEMM (QST) and
# gram_wide_kernel (W_ST); the two NB = 2 kernels differ only in how steps group into segments
KERNELS = [pytest.param(4, 2, 1, id="gram128-and-w8a8-4st"), pytest.param(3, 1, 2, id="gram_wide-3st"),
           pytest.param(2, 2, 1, id="two-stages")]
SEGS = [s for n in range(1, 4) for s in itertools.product([1, 2, 3], repeat=n)] + [(1, 1, 1, 1), (2, 1, 2, 1)]


@pytest.mark.parametrize("st,nb,groups", KERNELS)
def test_ring_and_accumulators(st, nb, groups):
    for segs in SEGS:
        assert explore(list(segs), st, nb, groups) > 0


def _mutate(progs, role, pred, repl):
    out = [list(p) for p in progs]
    out[role] = [x for op in out[role] for x in ([] if pred(op) and repl is None else [repl(op) if pred(op) else op])]
    return out


PLANTED = {
    # the TMA thread reloads a stage without waiting for its UMMAs
    "no_stage_release": (0, lambda op: op[0] == "wait" and op[1][0] == EMPTY, None, "overwrites a stage"),
    # the UMMA thread starts a segment without waiting for the epilogue to release the accumulator
    "no_accumulator_release": (1, lambda op: op[0] == "wait" and op[1][0] == ACCE, None,
                               "still being read|waits for completion"),
    # the epilogue waits one completion too early on accf
    "epilogue_off_by_one": (2, lambda op: op[0] == "wait" and op[1][0] == ACCF,
                            lambda op: ("wait", op[1], op[2] - 1), "starts waiting|before its UMMAs"),
}


@pytest.mark.parametrize("kind", sorted(PLANTED))
@pytest.mark.parametrize("st,nb,groups", KERNELS)
def test_checker_catches_planted_schedule_errors(kind, st, nb, groups):
    role, pred, repl, message = PLANTED[kind]
    segs = [2, 1, 2, 1]
    progs = _mutate(programs(segs, st, nb, groups), role, pred, repl)
    with pytest.raises(Violation, match=message):
        explore(segs, st, nb, groups, progs)
