"""An executable model of the attention kernel's synchronisation
(`csrc/attn_kernel.cuh`), checked by random interleavings on the CPU.

Each warp role is a Python generator that yields the mbarrier wait it is
about to make, in the kernel's order and with the kernel's phase arithmetic;
arrivals happen where the kernel arrives.  Two asynchronous engines complete
work in the background: the tensor pipe (MMAs and tcgen05.commit, in issue
order) and the copy engine (TMA loads, in any order).  mbarriers follow the
PTX semantics of `mbarrier.try_wait.parity`: a wait for the phase of parity P
passes whenever the barrier's current phase has the other parity.  The model
therefore flags

  * an aliased wait: it passes while the phase it means is not the last one
    completed (the barrier is a phase behind, or two ahead);
  * buffer hazards: a copy into a K, V or Q slot, a QK into an S/P buffer, a
    first PV into O, a row-sum slot or a queue slot reused before its previous
    reader is done, a QK reading a Q tile before its rotation;
  * deadlock: no role, engine or copy can move.

Both passes share the layout (Q in shared memory, three S/P buffers, NQ = 1
at d = 128 or 2 at d = 64, optional RoPE rotation of each Q tile by the
epilogue warps); the sink + window passes walk a static item sequence, the
strided dense pass claims its items in the producer and publishes them
through the eight-slot item queue.
Thread counts of an arrival (128 softmax or epilogue threads) are modelled as
one arrival on a barrier of count one."""
import random


class ModelError(Exception):
    pass


class Bar:
    """An mbarrier whose phase completes after `count` arrivals (a copy's
    completed bytes count as one arrival)."""

    def __init__(self, name, count=1):
        self.name, self.ph, self.count, self.pending = name, 0, count, 0

    def arrive(self):
        self.pending += 1
        if self.pending == self.count:
            self.pending = 0
            self.ph += 1


def _check_wait(bar, k):
    ok = (bar.ph & 1) != (k & 1)
    if ok and bar.ph != k + 1:
        raise ModelError("aliased wait on %s: wants phase %d, %d completed" % (bar.name, k, bar.ph))
    if not ok and bar.ph >= k + 2:
        raise ModelError("wait on %s for phase %d passed by: %d completed" % (bar.name, k, bar.ph))
    return ok


class Layout:
    def __init__(self, dense, nq=1, rope=False, nk=3, nv=2):
        self.dyn = dense  # items through the queue
        self.nq, self.nsb, self.nk, self.nv, self.rope = nq, 3, nk, nv, rope


def run(layout, tiles, seed, mutant=None, rescale_p=0.25, max_steps=10 ** 6):
    """Run one random interleaving; `tiles` lists each item's key-tile count
    (the CTA's items in order).  `mutant` names a deliberate protocol error
    (see MUTANTS) for the checker's own tests."""
    L, rnd = layout, random.Random(seed)
    n = len(tiles)
    bars = {}

    def bar(name):
        bars[name] = Bar(name)
        return bars[name]

    kfull = [bar("kfull%d" % s) for s in range(L.nk)]
    kempty = [bar("kempty%d" % s) for s in range(L.nk)]
    vfull = [bar("vfull%d" % s) for s in range(L.nv)]
    vempty = [bar("vempty%d" % s) for s in range(L.nv)]
    q_full = [bar("q_full%d" % b) for b in range(2)]
    q_free = [bar("q_free%d" % b) for b in range(2)]
    qt_ready = [bar("qt_ready%d" % b) for b in range(2)]
    s_full = [bar("s_full%d" % b) for b in range(L.nsb)]
    p_full = [bar("p_full%d" % b) for b in range(L.nsb)]
    pv_done = [bar("pv_done%d" % b) for b in range(L.nsb)]
    o_full, o_free = bar("o_full"), bar("o_free")
    l_ready = [bar("l_ready%d" % b) for b in range(2)]
    l_free = [bar("l_free%d" % b) for b in range(2)]
    kq = 8
    iq_full = [bar("iq_full%d" % s) for s in range(kq)]
    iq_empty_count = [0] * kq  # readers that released each queue slot (one completion = 5 roles)
    iq_empty = [bar("iq_empty%d" % s) for s in range(kq)]
    readers = 5  # V producer, QK, PV, softmax, epilogue (each warp group counted once)

    pipe, copies = [], []
    done = {"qk": set(), "pv": set(), "o_read": set(), "q_rot": set(), "l_read": set(), "iq_read": {}}
    first_g = []
    g = 0
    for T in tiles:
        first_g.append(g)
        g += T

    def iq_release(slot):
        iq_empty_count[slot] += 1
        if iq_empty_count[slot] == readers:
            iq_empty_count[slot] = 0
            iq_empty[slot].arrive()

    class Reader:
        """The item sequence as a role reads it: static, or from the queue."""

        def __init__(self, name):
            self.name, self.k = name, 0

        def next(self):
            if not L.dyn:
                i = self.k
                self.k += 1
                return i if i < n else -1
            slot = self.k % kq
            yield (iq_full[slot], self.k // kq)
            v = done["iq_read"][self.k]
            iq_release(slot)
            self.k += 1
            return v

    def producer():
        nq = 0
        c = 0
        np_ = 0
        claimed = 0

        def claim():
            nonlocal np_, claimed
            v = claimed if claimed < n else -1
            claimed += 1
            if L.dyn:
                slot = np_ % kq
                if np_ >= kq:
                    yield (iq_empty[slot], np_ // kq - 1)
                done["iq_read"][np_] = v
                iq_full[slot].arrive()
                np_ += 1
            return v

        def load_q(item):
            nonlocal nq
            qb = nq % L.nq
            if nq >= L.nq and mutant != "q_no_free_wait":
                yield (q_free[qb], nq // L.nq - 1)
            if nq >= L.nq:
                prev = nq - L.nq
                last = first_g[prev] + tiles[prev] - 1
                if last not in done["qk"]:
                    raise ModelError("Q buffer reloaded before the last QK of item %d" % prev)
            copies.append((q_full[qb], ("q", nq)))
            nq += 1

        item = yield from claim()
        if item >= 0:
            yield from load_q(item)
        while item >= 0:
            nxt = -1
            for j in range(tiles[item]):
                s = c % L.nk
                if c >= L.nk:
                    yield (kempty[s], c // L.nk - 1)
                    if (c - L.nk) not in done["qk"]:
                        raise ModelError("K slot reloaded before QK(%d) completed" % (c - L.nk))
                copies.append((kfull[s], ("k", c)))
                c += 1
                if j == 0:
                    nxt = yield from claim()
                    if L.nq >= 2 and nxt >= 0:
                        yield from load_q(nxt)
            if L.nq == 1 and nxt >= 0:
                yield from load_q(nxt)
            item = nxt
        if L.dyn and claimed <= n:
            yield from claim()

    def vprod():
        rd = Reader("v")
        c = 0
        while True:
            item = yield from rd.next()
            if item < 0:
                return
            for j in range(tiles[item]):
                s = c % L.nv
                if c >= L.nv:
                    yield (vempty[s], c // L.nv - 1)
                    if (c - L.nv) not in done["pv"]:
                        raise ModelError("V slot reloaded before PV(%d) completed" % (c - L.nv))
                copies.append((vfull[s], ("v", c)))
                c += 1

    def qk():
        rd = Reader("qk")
        g = 0
        i = 0
        while True:
            item = yield from rd.next()
            if item < 0:
                return
            qb = i % L.nq
            yield (qt_ready[qb] if L.rope else q_full[qb], i // L.nq)
            for j in range(tiles[item]):
                ks, sbi = g % L.nk, g % L.nsb
                yield (kfull[ks], g // L.nk)
                if g >= L.nsb and mutant != "qk_no_pv_wait":
                    yield (pv_done[sbi], g // L.nsb - 1)
                pipe.append(("qk", g, item))
                pipe.append(("commit", s_full[sbi]))
                g += 1
            pipe.append(("commit", q_free[qb]))
            i += 1

    def pv():
        rd = Reader("pv")
        g = 0
        i = 0
        while True:
            item = yield from rd.next()
            if item < 0:
                return
            T = tiles[item]
            for j in range(T):
                vs, sbi = g % L.nv, g % L.nsb
                yield (p_full[sbi], g // L.nsb)
                yield (vfull[vs], g // L.nv)
                if j == 0 and i >= 1 and mutant != "pv_no_o_free":
                    yield (o_free, i - 1)
                pipe.append(("pv", g, item, j == 0))
                pipe.append(("commit", pv_done[sbi]))
                pipe.append(("commit", vempty[vs]))
                if j == T - 1:
                    pipe.append(("commit", o_full))
                g += 1
            i += 1

    def softmax():
        rd = Reader("softmax")
        g = 0
        i = 0
        while True:
            item = yield from rd.next()
            if item < 0:
                return
            for j in range(tiles[item]):
                sbi = g % L.nsb
                yield (s_full[sbi], g // L.nsb)
                if g not in done["qk"]:
                    raise ModelError("softmax read S(%d) before its QK completed" % g)
                kempty[g % L.nk].arrive()
                if j >= 1 and rnd.random() < rescale_p:  # lazy O rescale: PV(g-1) must have landed
                    yield (pv_done[(g - 1) % L.nsb], (g - 1) // L.nsb)
                    if (g - 1) not in done["pv"]:
                        raise ModelError("O rescaled before PV(%d) completed" % (g - 1))
                p_full[sbi].arrive()
                yield None
                g += 1
            if i >= 2 and mutant != "softmax_no_l_free":
                yield (l_free[i & 1], (i >> 1) - 1)
            if i >= 2 and (i - 2) not in done["l_read"]:
                raise ModelError("row sums of item %d overwritten before the epilogue read them" % (i - 2))
            l_ready[i & 1].arrive()
            i += 1

    def epilogue():
        rd = Reader("epilogue")
        nq = 0

        def rotate(buf, qi):
            nonlocal nq
            if L.rope:
                yield (q_full[buf], nq // L.nq)
                nq += 1
                done["q_rot"].add(qi)
                qt_ready[buf].arrive()

        item = yield from rd.next()
        if item >= 0:
            yield from rotate(0, 0)
        i = 0
        while item >= 0:
            nxt = yield from rd.next()
            if nxt >= 0:
                yield from rotate((i + 1) % L.nq, i + 1)
            yield (l_ready[i & 1], i >> 1)
            done["l_read"].add(i)
            l_free[i & 1].arrive()
            yield (o_full, i + 1 if mutant == "o_full_phase_ahead" else i)
            done["o_read"].add(i)
            o_free.arrive()
            item = nxt
            i += 1

    roles = {"producer": producer(), "vprod": vprod(), "qk": qk(), "pv": pv(), "softmax": softmax(),
             "epilogue": epilogue()}
    waits = {}
    finished = set()

    def advance(name):
        try:
            waits[name] = next(roles[name])
        except StopIteration:
            finished.add(name)
            waits[name] = None

    for name in roles:
        advance(name)
    # each actor gets a random speed for this run, so that some runs starve
    # one role (a slow epilogue, a slow copy engine) and others the next
    speed = {name: rnd.choice([0.05, 0.3, 1.0, 1.0, 3.0]) for name in list(roles) + ["pipe", "copy"]}
    for _ in range(max_steps):
        cands = []
        for name in roles:
            if name in finished:
                continue
            w = waits[name]
            if w is None or _check_wait(*w):
                cands.append(("role", name))
        if pipe:
            cands.append(("pipe", None))
        if copies:
            cands.append(("copy", None))
        if not cands:
            if len(finished) == len(roles):
                return
            raise ModelError("deadlock: " + "; ".join(
                "%s waits %s for phase %d (%d completed)" % (nm, waits[nm][0].name, waits[nm][1], waits[nm][0].ph)
                for nm in roles if nm not in finished and waits[nm] is not None))
        kind, name = rnd.choices(cands, weights=[speed[c[1] if c[0] == "role" else c[0]] for c in cands])[0]
        if kind == "role":
            advance(name)
        elif kind == "pipe":
            op = pipe.pop(0)
            if op[0] == "qk":
                gg, item = op[1], op[2]
                if gg >= L.nsb and (gg - L.nsb) not in done["pv"]:
                    raise ModelError("QK(%d) overwrote S/P buffer before PV(%d) read it" % (gg, gg - L.nsb))
                if L.rope and item not in done["q_rot"]:
                    raise ModelError("QK of item %d read Q before its rotation" % item)
                done["qk"].add(gg)
            elif op[0] == "pv":
                gg, item, first = op[1], op[2], op[3]
                if first and item >= 1 and (item - 1) not in done["o_read"]:
                    raise ModelError("first PV of item %d overwrote O before item %d's was read" % (item, item - 1))
                done["pv"].add(gg)
            else:
                op[1].arrive()
        else:
            b, _ = copies.pop(rnd.randrange(len(copies)))
            b.arrive()
    raise ModelError("no end after %d steps" % max_steps)


# Each drops or misaims one wait of the protocol above.  The last waits for
# the next phase of o_full: with the barrier one phase behind, the parity
# test passes at once (the aliasing that a parity wait must never meet).
MUTANTS = ["qk_no_pv_wait", "pv_no_o_free", "softmax_no_l_free", "q_no_free_wait", "o_full_phase_ahead"]


def run_decode_ring(n_chunks, stages, warps, seed):
    """The decode kernel's ring (`csrc/decode.cu`): one producer thread loads
    chunk i into stage i % stages after the consumer of chunk i - stages
    released it; consumer warp w takes chunks w, w + warps, ... and waits for
    chunk i on stage i % stages with the parity of phase i / stages.  The
    kernel requires stages % warps == 0 so that every phase of a stage is
    consumed by one warp in order; the model flags the aliased waits
    otherwise."""
    rnd = random.Random(seed)
    full = [Bar("full%d" % s) for s in range(stages)]
    empty = [Bar("empty%d" % s) for s in range(stages)]
    in_stage, consumed, pending = {}, set(), []

    def producer():
        for i in range(n_chunks):
            st = i % stages
            if i >= stages:
                yield (empty[st], i // stages - 1)
                if (i - stages) not in consumed:
                    raise ModelError("stage %d reloaded before chunk %d was consumed" % (st, i - stages))
            pending.append((st, i))

    def consumer(w):
        for i in range(w, n_chunks, warps):
            st = i % stages
            yield (full[st], i // stages)
            if in_stage.get(st) != i:
                raise ModelError("warp %d read stage %d for chunk %d, found %s" % (w, st, i, in_stage.get(st)))
            consumed.add(i)
            yield None
            empty[st].arrive()

    roles = {"producer": producer()}
    roles.update({"warp%d" % w: consumer(w) for w in range(warps)})
    waits, finished = {}, set()

    def advance(name):
        try:
            waits[name] = next(roles[name])
        except StopIteration:
            finished.add(name)
            waits[name] = None

    for name in roles:
        advance(name)
    speed = {name: rnd.choice([0.1, 1.0, 3.0]) for name in list(roles) + ["copy"]}
    while True:
        cands = [nm for nm in roles if nm not in finished and (waits[nm] is None or _check_wait(*waits[nm]))]
        if pending:
            cands.append("copy")
        if not cands:
            if len(finished) == len(roles):
                return
            raise ModelError("deadlock in the decode ring")
        name = rnd.choices(cands, weights=[speed[c] for c in cands])[0]
        if name == "copy":
            st, i = pending.pop(rnd.randrange(len(pending)))
            in_stage[st] = i
            full[st].arrive()
        else:
            advance(name)


def run_pair(layout, tiles, seed, mutant=None, rescale_p=0.25, max_steps=10 ** 6):
    """The two-CTA sink + window kernel (`attn_kernel.cuh`, PAIR): CTAs 0 (the
    leader) and 1 run the same items (two heads of one row tile).  Each CTA
    has its own producer, V producer, softmax and epilogue; the leader's QK and
    PV threads issue the MMAs for both, which run in one tensor pipe.  Barriers
    the leader waits on count both CTAs: kfull / vfull (the leader's
    expect-tx arrival plus each CTA's copy of its half), p_full and o_free (one
    arrival per CTA, the kernel's per-warp arrivals lumped), qt_ready with
    RoPE; q_full without RoPE counts the leader's arrival and both Q copies.
    The commits of s_full, pv_done, vempty, o_full and q_free arrive on both
    CTAs' barriers; kempty, l_ready and l_free stay local.  Checked besides the
    one-CTA hazards: an MMA never reads a K or V half, a Q tile or a P that has
    not landed in either CTA."""
    L, rnd = layout, random.Random(seed)
    n = len(tiles)
    assert not L.dyn
    cnt_pair = 1 if mutant == "pair_one_cta_arrival" else 2
    cnt_copy = 2 if mutant == "pair_kfull_one_half" else 3

    def bars(name, k, count=1):
        return [Bar("%s%d" % (name, i), count) for i in range(k)]

    lead = {
        "kfull": bars("kfull", L.nk, cnt_copy), "vfull": bars("vfull", L.nv, 3),
        "q_full": bars("q_full", 2, 2 if L.rope else 3), "qt_ready": bars("qt_ready", 2, cnt_pair),
        "p_full": bars("p_full", L.nsb, cnt_pair), "o_free": Bar("o_free", cnt_pair),
    }
    cta = []
    for r in range(2):
        c = {
            "kempty": bars("kempty.%d." % r, L.nk), "vempty": bars("vempty.%d." % r, L.nv),
            "q_free": bars("q_free.%d." % r, 2), "s_full": bars("s_full.%d." % r, L.nsb),
            "pv_done": bars("pv_done.%d." % r, L.nsb), "o_full": Bar("o_full.%d" % r),
            "l_ready": bars("l_ready.%d." % r, 2, 1), "l_free": bars("l_free.%d." % r, 2, 1),
            # with RoPE each CTA's Q lands on its own barrier (its producer's arrival + the copy)
            "q_full": bars("q_full.%d." % r, 2, 2) if (L.rope and r == 1) else lead["q_full"],
        }
        cta.append(c)

    pipe, copies = [], []
    done = {"qk": set(), "pv": set(), "o_read": set(), "q_rot": set(), "l_read": set(), "k": set(), "v": set(),
            "q": set(), "p": set()}
    first_g = []
    g = 0
    for T in tiles:
        first_g.append(g)
        g += T

    def both(name, idx=None):
        return [c[name] if idx is None else c[name][idx] for c in cta]

    def producer(r):
        c, nq, kc = cta[r], 0, 0

        def load_q(item):
            nonlocal nq
            qb = nq % L.nq
            if nq >= L.nq:
                yield (c["q_free"][qb], nq // L.nq - 1)
                prev = nq - L.nq
                if first_g[prev] + tiles[prev] - 1 not in done["qk"]:
                    raise ModelError("CTA %d reloaded Q before the last QK of item %d" % (r, prev))
            if r == 0 or L.rope:
                c["q_full"][qb].arrive()  # the expect-tx arrival
            copies.append((c["q_full"][qb], ("q", r, nq)))
            nq += 1

        item = 0 if n > 0 else -1
        if item >= 0:
            yield from load_q(item)
        while item >= 0:
            for j in range(tiles[item]):
                s = kc % L.nk
                if kc >= L.nk:
                    yield (c["kempty"][s], kc // L.nk - 1)
                    if (kc - L.nk) not in done["qk"]:
                        raise ModelError("CTA %d reloaded K slot before QK(%d) completed" % (r, kc - L.nk))
                if r == 0:
                    lead["kfull"][s].arrive()
                copies.append((lead["kfull"][s], ("k", r, kc)))
                kc += 1
            nxt = item + 1 if item + 1 < n else -1
            if nxt >= 0:
                yield from load_q(nxt)
            item = nxt

    def vprod(r):
        c, vc = cta[r], 0
        for item in range(n):
            for j in range(tiles[item]):
                s = vc % L.nv
                if vc >= L.nv:
                    yield (c["vempty"][s], vc // L.nv - 1)
                    if (vc - L.nv) not in done["pv"]:
                        raise ModelError("CTA %d reloaded V slot before PV(%d) completed" % (r, vc - L.nv))
                if r == 0:
                    lead["vfull"][s].arrive()
                copies.append((lead["vfull"][s], ("v", r, vc)))
                vc += 1

    def qk():
        g = 0
        for i in range(n):
            qb = i % L.nq
            yield (lead["qt_ready"][qb] if L.rope else lead["q_full"][qb], i // L.nq)
            for j in range(tiles[i]):
                ks, sbi = g % L.nk, g % L.nsb
                yield (lead["kfull"][ks], g // L.nk)
                if g >= L.nsb:
                    yield (cta[0]["pv_done"][sbi], g // L.nsb - 1)
                pipe.append(("qk", g, i))
                pipe.append(("commit", both("s_full", sbi)))
                g += 1
            pipe.append(("commit", both("q_free", qb)))

    def pv():
        g = 0
        for i in range(n):
            T = tiles[i]
            for j in range(T):
                vs, sbi = g % L.nv, g % L.nsb
                yield (lead["p_full"][sbi], g // L.nsb)
                yield (lead["vfull"][vs], g // L.nv)
                if j == 0 and i >= 1:
                    yield (lead["o_free"], i - 1)
                pipe.append(("pv", g, i, j == 0))
                pipe.append(("commit", both("pv_done", sbi)))
                if mutant == "pair_vempty_leader_only":
                    pipe.append(("commit", [cta[0]["vempty"][vs]]))
                else:
                    pipe.append(("commit", both("vempty", vs)))
                if j == T - 1:
                    pipe.append(("commit", both("o_full")))
                g += 1

    def softmax(r):
        c, g = cta[r], 0
        for i in range(n):
            for j in range(tiles[i]):
                sbi = g % L.nsb
                yield (c["s_full"][sbi], g // L.nsb)
                if g not in done["qk"]:
                    raise ModelError("CTA %d softmax read S(%d) before its QK completed" % (r, g))
                c["kempty"][g % L.nk].arrive()
                if j >= 1 and rnd.random() < rescale_p:
                    yield (c["pv_done"][(g - 1) % L.nsb], (g - 1) // L.nsb)
                    if (g - 1) not in done["pv"]:
                        raise ModelError("CTA %d rescaled O before PV(%d) completed" % (r, g - 1))
                done["p"].add((r, g))
                lead["p_full"][sbi].arrive()
                yield None
                g += 1
            if i >= 2:
                yield (c["l_free"][i & 1], (i >> 1) - 1)
                if (r, i - 2) not in done["l_read"]:
                    raise ModelError("CTA %d row sums of item %d overwritten before read" % (r, i - 2))
            c["l_ready"][i & 1].arrive()

    def epilogue(r):
        c, nq = cta[r], 0

        def rotate(buf, qi):
            nonlocal nq
            if L.rope:
                yield (c["q_full"][buf], nq // L.nq)
                if (r, qi) not in done["q"]:
                    raise ModelError("CTA %d rotated Q of item %d before it landed" % (r, qi))
                nq += 1
                done["q_rot"].add((r, qi))
                lead["qt_ready"][buf].arrive()

        if n > 0:
            yield from rotate(0, 0)
        for i in range(n):
            if i + 1 < n:
                yield from rotate((i + 1) % L.nq, i + 1)
            yield (c["l_ready"][i & 1], i >> 1)
            done["l_read"].add((r, i))
            c["l_free"][i & 1].arrive()
            yield (c["o_full"], i)
            done["o_read"].add((r, i))
            lead["o_free"].arrive()

    roles = {"qk": qk(), "pv": pv()}
    for r in range(2):
        roles["producer%d" % r] = producer(r)
        roles["vprod%d" % r] = vprod(r)
        roles["softmax%d" % r] = softmax(r)
        roles["epilogue%d" % r] = epilogue(r)
    waits, finished = {}, set()

    def advance(name):
        try:
            waits[name] = next(roles[name])
        except StopIteration:
            finished.add(name)
            waits[name] = None

    for name in roles:
        advance(name)
    speed = {name: rnd.choice([0.05, 0.3, 1.0, 1.0, 3.0]) for name in list(roles) + ["pipe", "copy"]}
    for _ in range(max_steps):
        cands = [("role", nm) for nm in roles
                 if nm not in finished and (waits[nm] is None or _check_wait(*waits[nm]))]
        if pipe:
            cands.append(("pipe", None))
        if copies:
            cands.append(("copy", None))
        if not cands:
            if len(finished) == len(roles):
                return
            raise ModelError("deadlock: " + "; ".join(
                "%s waits %s for phase %d (%d completed)" % (nm, waits[nm][0].name, waits[nm][1], waits[nm][0].ph)
                for nm in roles if nm not in finished and waits[nm] is not None))
        kind, name = rnd.choices(cands, weights=[speed[c[1] if c[0] == "role" else c[0]] for c in cands])[0]
        if kind == "role":
            advance(name)
        elif kind == "pipe":
            op = pipe.pop(0)
            if op[0] == "qk":
                gg, item = op[1], op[2]
                if gg >= L.nsb and (gg - L.nsb) not in done["pv"]:
                    raise ModelError("QK(%d) overwrote S/P before PV(%d) read it" % (gg, gg - L.nsb))
                for r in range(2):
                    if ("k", r, gg) not in done["k"]:
                        raise ModelError("QK(%d) read CTA %d's K half before it landed" % (gg, r))
                    if (r, item) not in (done["q_rot"] if L.rope else done["q"]):
                        raise ModelError("QK of item %d read CTA %d's Q before it was ready" % (item, r))
                done["qk"].add(gg)
            elif op[0] == "pv":
                gg, item, first = op[1], op[2], op[3]
                for r in range(2):
                    if ("v", r, gg) not in done["v"]:
                        raise ModelError("PV(%d) read CTA %d's V half before it landed" % (gg, r))
                    if (r, gg) not in done["p"]:
                        raise ModelError("PV(%d) read CTA %d's P before it was written" % (gg, r))
                    if first and item >= 1 and (r, item - 1) not in done["o_read"]:
                        raise ModelError("first PV of item %d overwrote CTA %d's O before it was read" % (item, r))
                done["pv"].add(gg)
            else:
                for b in op[1]:
                    b.arrive()
        else:
            b, what = copies.pop(rnd.randrange(len(copies)))
            if what[0] == "q":
                done["q"].add((what[1], what[2]))
            else:
                done[what[0]].add(what)
            b.arrive()
    raise ModelError("no end after %d steps" % max_steps)


# Each breaks the pair protocol in one place: the leader waits for one CTA's
# arrival instead of both (P, O, rotated Q), for one K half instead of two, or
# the V slots are released in the leader only.
PAIR_MUTANTS = ["pair_one_cta_arrival", "pair_kfull_one_half", "pair_vempty_leader_only"]
