"""CPU check of the index arithmetic of the misaligned-tile paths: the
16-byte window path (`stage_issue_w`, `stage_drain_w`, `drain_full_w` in the
remap kernel source) and the one-element-per-lane path (`stage_issue_e`,
`load_a_e`, `stage_drain_e`, and `stage_drain_e1` for the kinds that do not
read A), replayed per lane for random tiles before any kernel runs them.

For a tile of nx x ny elements (nx, ny <= 32), transposed or not, with any
element-aligned start addresses and leading dimensions of source and target,
the replay checks that:
  - every 16-byte source copy is aligned and lies inside the aligned window
    of its run, [floor16(run start), ceil16(run end));
  - every shared-memory access stays inside the warp's buffer;
  - every 16-byte store to A is aligned;
  - every target element of the tile is written exactly once, with the staged
    value of its own source element, and nothing outside the tile is written.
The arithmetic below restates the kernel's (lane map, phases, window chunks,
swizzled slots, extra column); a change there must be mirrored here."""
import random

import pytest

TS = 32


def lane_map(chunks, lane):
    sh = 0 if chunks <= 1 else (chunks - 1).bit_length()
    return lane & ((1 << sh) - 1), lane >> sh, 32 >> sh


def replay(es, rnd):
    vec = 16 // es
    cpr = TS // vec
    xcol = TS * cpr * 16
    buf_bytes = (xcol + TS * 16 + 127) // 128 * 128

    def slot(r, c):
        assert 0 <= c < cpr and 0 <= r < TS
        return (r * cpr + (c ^ ((r // vec) & 7))) * 16

    def welem(r, q):
        j = q // vec
        return (slot(r, j) if j < cpr else xcol + r * 16) + (q % vec) * es

    def phase(p, ld, r):
        return ((p & 15) // es + r * (ld & (vec - 1))) & (vec - 1)

    def wchunks(n):
        return (n + 2 * vec - 2) // vec

    def wmain(n):
        return min(cpr, wchunks(n))

    nx = TS if rnd.random() < 0.3 else rnd.randint(1, TS)
    ny = TS if rnd.random() < 0.3 else rnd.randint(1, TS)
    tr = rnd.random() < 0.5
    runs, ln = (nx, ny) if tr else (ny, nx)
    sld = ln + rnd.randint(0, 9)
    dld = nx + rnd.randint(0, 9)
    src = (1 << 20) + rnd.randrange(64) * es
    dst = (1 << 24) + rnd.randrange(64) * es
    smem = {}

    def copy16(sa, ga, r):
        assert ga % 16 == 0 and sa % 16 == 0 and 0 <= sa and sa + 16 <= buf_bytes
        start, end = src + r * sld * es, src + (r * sld + ln) * es
        assert start // 16 * 16 <= ga and ga + 16 <= -(-end // 16) * 16
        for b in range(vec):
            smem[sa + b * es] = ga + b * es

    # stage_issue_w
    cm = wmain(ln)
    for lane in range(32):
        c, r0, rpp = lane_map(cm, lane)
        assert rpp % vec == 0
        ph = phase(src, sld, r0)
        if c < cm and c * vec < ph + ln:
            for r in range(r0, runs, rpp):
                assert phase(src, sld, r) == ph
                copy16(slot(r, c), src + (r * sld - ph + c * vec) * es, r)
        if wchunks(ln) > cpr and lane < runs:
            pr = phase(src, sld, lane)
            if cpr * vec < pr + ln:
                copy16(xcol + lane * 16, src + (lane * sld - pr + cpr * vec) * es, lane)

    written = set()

    def drain(x0, y, full):
        for i in range(vec):
            x = min(max(x0 + i, 0), nx - 1)
            if tr:
                sa, want = welem(x, phase(src, sld, x) + y), src + (x * sld + y) * es
            else:
                sa, want = welem(y, phase(src, sld, y) + x), src + (y * sld + x) * es
            assert 0 <= sa < buf_bytes and smem.get(sa) == want
        if full:
            assert (dst + (y * dld + x0) * es) % 16 == 0 and 0 <= x0 and x0 + vec <= nx
        for i in range(vec):
            if 0 <= x0 + i < nx:
                assert (y, x0 + i) not in written
                written.add((y, x0 + i))

    def hoisted(x0, r0, rpp, p, y):
        """drain_full_w's staged offsets for pass p (row y), per element."""
        row = cpr * 16
        if tr:
            out = []
            for e in range(vec):
                x = x0 + e
                q = phase(src, sld, x) + r0
                j = q // vec + p * (rpp // vec)
                off = x * row + (q % vec) * es
                out.append(off + ((j ^ ((x // vec) & 7)) << 4) if j < cpr else xcol + x * 16 + (q % vec) * es)
            return out
        q = phase(src, sld, r0) + x0
        j, w = q // vec, q % vec
        sw = (y // vec) & 7
        o0 = y * row + ((j ^ sw) << 4) if j < cpr else xcol + y * 16
        o1 = y * row + (((j + 1) ^ sw) << 4) if j + 1 < cpr else xcol + y * 16
        return [o0 + (w + e) * es if w + e < vec else o1 + (w + e - vec) * es for e in range(vec)]

    # stage_drain_w: full chunks (drain_full_w)
    cmd = wmain(nx)
    for lane in range(32):
        c, r0, rpp = lane_map(cmd, lane)
        x0 = c * vec - phase(dst, dld, r0)
        if c < cmd and x0 >= 0 and x0 + vec <= nx:
            for p, y in enumerate(range(r0, ny, rpp)):
                assert c * vec - phase(dst, dld, y) == x0
                want = [welem(x0 + e, phase(src, sld, x0 + e) + y) if tr else welem(y, phase(src, sld, y) + x0 + e)
                        for e in range(vec)]
                assert hoisted(x0, r0, rpp, p, y) == want
                drain(x0, y, True)
    # partial chunks (drain_partial_w): lane = tile row
    for lane in range(32):
        if lane < ny:
            ph = phase(dst, dld, lane)
            last = (ph + nx - 1) // vec
            xl = last * vec - ph
            if ph > 0:
                drain(-ph, lane, False)
            if xl + vec > nx and (last > 0 or ph == 0):
                drain(xl, lane, False)
    assert written == {(y, x) for y in range(ny) for x in range(nx)}


@pytest.mark.parametrize("es", [4, 8])
def test_window_map(es):
    rnd = random.Random(2106066010 + es)
    for _ in range(8000):
        replay(es, rnd)


def replay_elements(es, rnd):
    """The one-element-per-lane path.  Staging: every source element lands in
    the TS x TS buffer at c ^ (r mod TS) of its row, read from inside its
    run.  load_a_e: the A elements a lane loads are the target elements it
    later writes, each at dst + (y * dld + x) * es inside the tile's target
    rows, and only whole-chunk padding slots beyond the tile are left at
    zero.  stage_drain_e: each target element is written exactly once, at
    its own address, with the source element staged for it."""
    nx = TS if rnd.random() < 0.3 else rnd.randint(1, TS)
    ny = TS if rnd.random() < 0.3 else rnd.randint(1, TS)
    tr = rnd.random() < 0.5
    runs, ln = (nx, ny) if tr else (ny, nx)
    sld = ln + rnd.randint(0, 9)
    dld = nx + rnd.randint(0, 9)
    src = (1 << 20) + rnd.randrange(64) * es
    dst = (1 << 24) + rnd.randrange(64) * es
    vec = 16 // es
    ne = (TS // (32 // (TS // vec))) * vec  # NPASS * VEC: elements per lane of a full tile

    def slot_e(r, c):
        assert 0 <= r < TS and 0 <= c < TS
        return r * TS + (c ^ (r & (TS - 1)))

    def target(y, x):
        """Address of target element (y, x); inside the tile's rows."""
        a = dst + (y * dld + x) * es
        assert 0 <= y < ny and 0 <= x < nx
        assert dst + y * dld * es <= a < dst + (y * dld + nx) * es
        return a

    # stage_issue_e
    smem = {}
    for lane in range(32):
        c, r0, rpp = lane_map(ln, lane)
        if c >= ln:
            continue
        for r in range(r0, runs, rpp):
            ga = src + (r * sld + c) * es
            assert src + r * sld * es <= ga < src + (r * sld + ln) * es
            smem[slot_e(r, c)] = ga

    every = {target(y, x) for y in range(ny) for x in range(nx)}
    loaded, stored = [], []
    for lane in range(32):
        c, r0, rpp = lane_map(nx, lane)
        on = c < nx
        npass = (ny + rpp - 1) // rpp
        npad = (npass + vec - 1) // vec * vec
        assert npass <= ne and npad <= ne
        # load_a_e: register slot p holds A's element of pass p, or zero
        regs = {}
        for p in range(ne):
            if p >= npad:
                break
            y = p * rpp + r0
            regs[p] = target(y, c) if (on and p < npass and y < ny) else None
            if regs[p] is not None:
                loaded.append(regs[p])
        # stage_drain_e: writes pass p's element, combined with register slot p
        if not on:
            continue
        for p in range(ne):
            if p >= npass:
                break
            y = p * rpp + r0
            if y >= ny:
                continue
            a = target(y, c)
            assert regs[p] == a                     # the A value it combines is its own
            want = src + ((c * sld + y) if tr else (y * sld + c)) * es
            assert smem.get(slot_e(c, y) if tr else slot_e(y, c)) == want
            stored.append(a)
    assert len(stored) == len(set(stored)) and set(stored) == every
    assert len(loaded) == len(set(loaded)) and set(loaded) == every
    # stage_drain_e1 (kinds that do not read A): rows r0, r0 + rpp, ...
    stored1 = []
    for lane in range(32):
        c, r0, rpp = lane_map(nx, lane)
        if c >= nx:
            continue
        for y in range(r0, ny, rpp):
            want = src + ((c * sld + y) if tr else (y * sld + c)) * es
            assert smem.get(slot_e(c, y) if tr else slot_e(y, c)) == want
            stored1.append(target(y, c))
    assert len(stored1) == len(set(stored1)) and set(stored1) == every


@pytest.mark.parametrize("es", [4, 8])
def test_element_map(es):
    rnd = random.Random(2106066020 + es)
    for _ in range(8000):
        replay_elements(es, rnd)
