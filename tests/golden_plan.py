"""Independent construction of the exported plan bytes (test helper).

This is a second implementation of the compile phase (paper, Alg. 1 compile
phase: constant gates pre-multiplied and cached, parametric gates kept
symbolic) written from the plan format's documentation, not from the engine:
it does not call the library.  Tests compare its bytes with vqc_plan_export.

The lowering it restates:
  * single-qubit gates meeting consecutively on a qubit form a run (one table
    entry); consecutive constant factors of a run are multiplied in float64
    (later factor on the left); RX/RY/RZ with a parameter stay symbolic; U3
    with a parameter becomes RZ(lambda) RY(theta) RZ(phi) times the global
    phase e^{i(phi + lambda)/2} (a constant when both angles are);
  * a two-qubit gate closes the runs of its qubits; SWAP becomes three CX;
    CRZ and RZZ are diagonal phase entries;
  * every parametric constituent with an x or w angle is a gradient term
    (the U3 phase is not); an entry with terms gets an accumulator;
  * table slots number per-sample and shared entries apart; x / w occurrence
    lists hold term indices in increasing order;
  * stage schedules: ops are taken greedily in order into a stage while the
    active set (the qubits of non-diagonal targets) stays within K; CX gates
    with both qubits in the tile fold into the stage's store map; the active
    set is padded to K; thread bits take residues mod G first; addresses use
    the linear swizzle sw(u) = u ^ (fold_G(u >> G) & (2^G - 1));
  * HBM passes: tiles of m qubits always holding the low G qubits, filled
    greedily, padded with the deferred ops' targets, then from the top qubit.
"""
from __future__ import annotations

import math
import struct

import numpy as np

# ---------------------------------------------------------------- record layouts
DENTRY = np.dtype([("cfirst", "<u2"), ("ccount", "<u2"), ("slot", "<u2"), ("per_sample", "u1"),
                   ("phase", "u1"), ("acc", "<u2"), ("pad", "<u2")])
DCONST = np.dtype([("kind", "u1"), ("src0", "u1"), ("src1", "u1"), ("pad", "u1"),
                   ("idx0", "<i4"), ("idx1", "<i4"), ("term", "<i4")])
DOP = np.dtype([("code", "u1"), ("a", "u1"), ("b", "u1"), ("flags", "u1"), ("slot", "<u2"),
                ("aux", "<u2")])
DSTAGE = np.dtype([("op_begin", "<i4"), ("op_end", "<i4"), ("sigma", "<i4", 5), ("tau", "<i4", 16),
                   ("tmask", "<u4", 16), ("sigma_st", "<i4", 5), ("tau_st", "<i4", 16),
                   ("active", "u1", 5), ("nthreadbits", "u1"), ("nperm", "u1"), ("cl_local", "u1")])
DPASS = np.dtype([("stage_begin", "<i4"), ("stage_end", "<i4"), ("m", "<i4"), ("nout", "<i4"),
                  ("tile_q", "u1", 24), ("out_q", "u1", 24), ("ps_begin", "<i4"), ("ps_count", "<i4"),
                  ("sh_begin", "<i4"), ("sh_count", "<i4"), ("acc_begin", "<i4"), ("acc_count", "<i4")])

OP_M1, OP_CX, OP_CZ, OP_PH2 = 1, 2, 3, 4
OPF_PER_SAMPLE, OPF_GEN_CRZ, OPF_GEN_RZZ, OPF_HAS_ACC = 1, 2, 4, 8
DC_M1, DC_CX_LL, DC_CX_PL, DC_CZ_LL, DC_CZ_PL, DC_CZ_PP = 0, 5, 25, 30, 40, 45
DC_PH2_LL, DC_PH2_PL, DC_PH2_PP = 46, 56, 61
CK_CONST, CK_RX, CK_RY, CK_RZ, CK_GPHASE, CK_CRZ, CK_RZZ = 1, 2, 3, 4, 5, 6, 7
SRC_NONE, SRC_CONST, SRC_X, SRC_W = 0, 1, 2, 3
KIND_OF = {"c": SRC_CONST, "x": SRC_X, "w": SRC_W}
REF_PHYS = 8
MAX_K, MAX_TB = 5, 16
C64, C128 = 0, 1


def popcount(v):
    return bin(v).count("1")


def pair_index(lo, hi):
    return [(0, 1), (0, 2), (0, 3), (0, 4), (1, 2), (1, 3), (1, 4), (2, 3), (2, 4), (3, 4)].index((lo, hi))


def swz(u, G):
    v, f = u >> G, 0
    while v:
        f ^= v
        v >>= G
    return u ^ (f & ((1 << G) - 1))


# ---------------------------------------------------------------- complex arithmetic
# complex numbers as (re, im) float pairs; products written out (no fused
# multiply-add), as the definition of a complex product
def cmul(a, b):
    return (a[0] * b[0] - a[1] * b[1], a[0] * b[1] + a[1] * b[0])


def cadd(a, b):
    return (a[0] + b[0], a[1] + b[1])


def mmul(a, b):   # 2x2 row-major: a * b
    return [cadd(cmul(a[0], b[0]), cmul(a[1], b[2])), cadd(cmul(a[0], b[1]), cmul(a[1], b[3])),
            cadd(cmul(a[2], b[0]), cmul(a[3], b[2])), cadd(cmul(a[2], b[1]), cmul(a[3], b[3]))]


def polar(r, t):
    return (r * math.cos(t), r * math.sin(t))


def fixed_matrix(name, th=(0.0, 0.0, 0.0)):
    r2 = 1.0 / math.sqrt(2.0)
    z, one = (0.0, 0.0), (1.0, 0.0)
    if name == "H":
        return [(r2, 0.0), (r2, 0.0), (r2, 0.0), (-r2, 0.0)]
    if name == "X":
        return [z, one, one, z]
    if name == "Y":
        return [z, (-0.0, -1.0), (0.0, 1.0), z]
    if name == "Z":
        return [one, z, z, (-1.0, 0.0)]
    if name == "S":
        return [one, z, z, (0.0, 1.0)]
    if name == "T":
        return [one, z, z, polar(1.0, math.pi / 4)]
    if name == "SX":
        return [(0.5, 0.5), (0.5, -0.5), (0.5, -0.5), (0.5, 0.5)]
    c, s = math.cos(th[0] / 2), math.sin(th[0] / 2)
    if name == "RX":
        return [(c, 0.0), (0.0, -s), (0.0, -s), (c, 0.0)]
    if name == "RY":
        return [(c, 0.0), (-s, 0.0), (s, 0.0), (c, 0.0)]
    if name == "RZ":
        return [polar(1.0, -th[0] / 2), z, z, polar(1.0, th[0] / 2)]
    if name == "U3":
        m1 = polar(s, th[2])
        return [(c, 0.0), (-m1[0], -m1[1]), polar(s, th[1]), polar(c, th[1] + th[2])]
    raise ValueError(name)


# ---------------------------------------------------------------- lowering
class Lowered:
    """Fused ops, table entries and their constituents, constants, gradient
    terms and accumulators of a circuit (CircuitSpec)."""

    def __init__(self, spec, dtype):
        self.n, self.nx, self.nw = int(spec.n), int(spec.num_x), int(spec.num_w)
        self.dtype = C64 if dtype == "c64" else C128
        self.G = 4 if self.dtype == C64 else 3
        self.num_gates_in = len(spec.gates)
        self.ops = []            # (type, q0, q1, entry, gen)
        self.entries = []        # dicts
        self.consts = []         # dicts
        self.cmat, self.cang = [], []
        self.term_src, self.term_idx, self.accs = [], [], []
        self.n_runs = 0
        self.open = [[] for _ in range(self.n)]
        for name, qubits, params in spec.gates:
            self._gate(name, qubits, [(KIND_OF[k], v) for k, v in params])
        for q in range(self.n):
            self._flush(q)
        self.n_ps = self.n_sh = 0
        for e in self.entries:
            if e["per_sample"]:
                e["slot"], self.n_ps = self.n_ps, self.n_ps + 1
            else:
                e["slot"], self.n_sh = self.n_sh, self.n_sh + 1
        self.xocc_ptr, self.xocc = self._occ(SRC_X, self.nx)
        self.wocc_ptr, self.wocc = self._occ(SRC_W, self.nw)

    def _occ(self, kind, count):
        ptr = [0] * (count + 1)
        for s, i in zip(self.term_src, self.term_idx):
            if s == kind:
                ptr[i + 1] += 1
        for i in range(count):
            ptr[i + 1] += ptr[i]
        occ, fill = [0] * ptr[count], ptr[:-1]
        for t, (s, i) in enumerate(zip(self.term_src, self.term_idx)):
            if s == kind:
                occ[fill[i]] = t
                fill[i] += 1
        return ptr, occ

    # a constituent: dict(kind, s0=(srckind, value), s1=..., mat=4 complex)
    def _entry(self, cons, phase):
        cs = []
        for c in cons:
            if c["kind"] == CK_CONST and cs and cs[-1]["kind"] == CK_CONST:
                cs[-1] = dict(cs[-1], mat=mmul(c["mat"], cs[-1]["mat"]))
            else:
                cs.append(c)
        e = dict(cfirst=len(self.consts), ccount=len(cs), slot=0, per_sample=0, phase=int(phase),
                 acc=0xffff)
        has_term = False
        for c in cs:
            d = dict(kind=c["kind"], src0=0, src1=0, idx0=0, idx1=0, term=-1)
            if c["kind"] == CK_CONST:
                d["idx0"] = len(self.cmat) // 8
                for z in c["mat"]:
                    self.cmat += [z[0], z[1]]
            else:
                def put(src):
                    kind, val = src
                    if kind == SRC_CONST:
                        self.cang.append(float(val))
                        idx = len(self.cang) - 1
                    else:
                        idx = int(val)
                    if kind == SRC_X:
                        e["per_sample"] = 1
                    return kind, idx
                d["src0"], d["idx0"] = put(c["s0"])
                if c["kind"] == CK_GPHASE:
                    d["src1"], d["idx1"] = put(c["s1"])
                if c["kind"] != CK_GPHASE and c["s0"][0] in (SRC_X, SRC_W):
                    d["term"] = len(self.term_src)
                    self.term_src.append(c["s0"][0])
                    self.term_idx.append(int(c["s0"][1]))
                    has_term = True
            self.consts.append(d)
        eid = len(self.entries)
        if has_term:
            e["acc"] = len(self.accs)
            self.accs.append((eid, int(phase)))
        self.entries.append(e)
        return eid

    def _flush(self, q):
        if self.open[q]:
            eid = self._entry(self.open[q], False)
            self.open[q] = []
            self.ops.append((OP_M1, q, -1, eid, 0))
            self.n_runs += 1

    def _rotation(self, q, name, kind, src):
        if src[0] == SRC_CONST:
            self.open[q].append(dict(kind=CK_CONST, mat=fixed_matrix(name, (float(src[1]), 0.0, 0.0))))
        else:
            self.open[q].append(dict(kind=kind, s0=src))

    def _gate(self, name, qubits, src):
        q0 = qubits[0]
        if name in ("H", "X", "Y", "Z", "S", "T", "SX"):
            self.open[q0].append(dict(kind=CK_CONST, mat=fixed_matrix(name)))
        elif name in ("RX", "RY", "RZ"):
            self._rotation(q0, name, {"RX": CK_RX, "RY": CK_RY, "RZ": CK_RZ}[name], src[0])
        elif name == "U3":
            if all(s[0] == SRC_CONST for s in src):
                self.open[q0].append(dict(kind=CK_CONST, mat=fixed_matrix(
                    "U3", tuple(float(s[1]) for s in src))))
            else:
                # U3(t, p, l) = e^{i(p+l)/2} RZ(p) RY(t) RZ(l): RZ(l) first
                self._rotation(q0, "RZ", CK_RZ, src[2])
                self._rotation(q0, "RY", CK_RY, src[0])
                self._rotation(q0, "RZ", CK_RZ, src[1])
                if src[1][0] == SRC_CONST and src[2][0] == SRC_CONST:
                    ph = polar(1.0, 0.5 * (float(src[1][1]) + float(src[2][1])))
                    self.open[q0].append(dict(kind=CK_CONST, mat=[ph, (0.0, 0.0), (0.0, 0.0), ph]))
                else:
                    self.open[q0].append(dict(kind=CK_GPHASE, s0=src[1], s1=src[2]))
        else:
            q1 = qubits[1]
            self._flush(q0)
            self._flush(q1)
            if name == "CX":
                self.ops.append((OP_CX, q0, q1, -1, 0))
            elif name == "SWAP":
                self.ops += [(OP_CX, q0, q1, -1, 0), (OP_CX, q1, q0, -1, 0), (OP_CX, q0, q1, -1, 0)]
            elif name == "CZ":
                self.ops.append((OP_CZ, q0, q1, -1, 0))
            else:
                kind = CK_CRZ if name == "CRZ" else CK_RZZ
                eid = self._entry([dict(kind=kind, s0=src[0])], True)
                self.ops.append((OP_PH2, q0, q1, eid, OPF_GEN_CRZ if name == "CRZ" else OPF_GEN_RZZ))


# ---------------------------------------------------------------- schedules
def op_touch(o):
    t = 1 << o[1]
    if o[0] != OP_M1:
        t |= 1 << o[2]
    return t


def op_need(o):
    if o[0] == OP_M1:
        return 1 << o[1]
    if o[0] == OP_CX:
        return 1 << o[2]
    return 0


class Schedule:
    def __init__(self, mode, K, m, path):
        self.mode, self.K, self.m, self.path = mode, K, m, path
        self.thread_bits = m - K
        self.group_lanes_log2 = m - K
        self.cta_bits = 0
        self.ops, self.stages, self.passes = [], [], []
        self.pass_entries, self.pass_accs, self.store_masks = [], [], []


def cut_stages(L, opidx, tile, K, s, slot_of, acc_of):
    """Stages of K active qubits over the tile (tile-local addressing)."""
    G = L.G
    lpos = {q: i for i, q in enumerate(tile)}
    remaining = list(opidx)
    while True:
        active = blocked = pend = 0
        taken, deferred, perm = [], [], []
        for oi in remaining:
            o = L.ops[oi]
            touch, need = op_touch(o), op_need(o)
            if touch & blocked:
                blocked |= touch
                deferred.append(oi)
                continue
            if o[0] == OP_CX and o[1] in lpos and o[2] in lpos:   # folded into the store map
                pend |= touch
                perm.append(oi)
                continue
            if touch & pend:
                blocked |= touch
                deferred.append(oi)
                continue
            if popcount(active | need) <= K:
                active |= need
                taken.append(oi)
            else:
                blocked |= touch
                deferred.append(oi)
        while popcount(active) < K:   # pad, keeping residues mod G among the thread bits
            best, best_cnt = -1, -1
            for i in range(len(tile) - 1, -1, -1):
                q = tile[i]
                if active >> q & 1:
                    continue
                cnt = sum(1 for r in tile if not (active >> r & 1) and lpos[r] % G == i % G)
                if cnt > best_cnt:
                    best_cnt, best = cnt, q
            active |= 1 << best
        st = np.zeros((), DSTAGE)
        act = [q for q in tile if active >> q & 1]
        for j, q in enumerate(act):
            st["active"][j] = q
            st["sigma"][j] = swz(1 << lpos[q], G)
        outer = [q for q in tile if not (active >> q & 1)]
        used, order = [False] * len(outer), []
        for i in range(min(G, len(outer))):
            pick = next((c for c in range(len(outer)) if not used[c] and lpos[outer[c]] % G == i), -1)
            if pick < 0:
                pick = next(c for c in range(len(outer)) if not used[c])
            used[pick] = True
            order.append(outer[pick])
        order += [q for c, q in enumerate(outer) if not used[c]]
        st["nthreadbits"] = len(order)
        for i, q in enumerate(order):
            st["tau"][i] = swz(1 << lpos[q], G)
            st["tmask"][i] = 1 << q

        def pi(v):
            for oi in perm:
                o = L.ops[oi]
                if (v >> o[1]) & 1:
                    v ^= 1 << o[2]
            return v

        def tile_local(v):
            return sum(1 << i for i, q in enumerate(tile) if (v >> q) & 1)

        masks = [0] * (MAX_K + MAX_TB)
        for k, q in enumerate(act):
            v = pi(1 << q)
            st["sigma_st"][k] = swz(tile_local(v), G)
            masks[k] = v
        for i, q in enumerate(order):
            v = pi(1 << q)
            st["tau_st"][i] = swz(tile_local(v), G)
            masks[MAX_K + i] = v
        s.store_masks += masks
        st["nperm"] = min(len(perm), 255)

        def local(q):
            return act.index(q) if q in act else -1

        def ref(q):
            lq = local(q)
            return lq if lq >= 0 else REF_PHYS + q

        st["op_begin"] = len(s.ops)
        for oi in taken:
            typ, q0, q1, ent, gen = L.ops[oi]
            d = np.zeros((), DOP)
            if typ in (OP_M1, OP_PH2):
                e = L.entries[ent]
                d["slot"] = slot_of[ent]
                d["flags"] = (OPF_PER_SAMPLE if e["per_sample"] else 0) | \
                    (OPF_HAS_ACC if e["acc"] != 0xffff else 0) | gen
                d["aux"] = acc_of[e["acc"]] if e["acc"] != 0xffff else 0xffff
            if typ == OP_M1:
                d["a"] = local(q0)
                d["code"] = DC_M1 + local(q0)
            elif typ == OP_CX:
                a, b = ref(q0), local(q1)
                d["a"], d["b"] = a, b
                d["code"] = DC_CX_LL + 4 * a + (b if b < a else b - 1) if a < REF_PHYS else DC_CX_PL + b
            elif typ == OP_CZ:
                ra, rb = ref(q0), ref(q1)
                if ra >= REF_PHYS and rb >= REF_PHYS:
                    d["code"] = DC_CZ_PP
                elif ra >= REF_PHYS or rb >= REF_PHYS:
                    if ra >= REF_PHYS:
                        ra, rb = rb, ra
                    d["code"] = DC_CZ_PL + ra
                else:
                    ra, rb = min(ra, rb), max(ra, rb)
                    d["code"] = DC_CZ_LL + pair_index(ra, rb)
                d["a"], d["b"] = ra, rb
            else:
                a, b = ref(q0), ref(q1)
                d["a"], d["b"] = a, b
                la, lb = a < REF_PHYS, b < REF_PHYS
                if la and lb:
                    d["code"] = DC_PH2_LL + pair_index(min(a, b), max(a, b))
                elif la or lb:
                    d["code"] = DC_PH2_PL + (a if la else b)
                else:
                    d["code"] = DC_PH2_PP
            s.ops.append(d)
        st["op_end"] = len(s.ops)
        s.stages.append(st)
        remaining = deferred
        # a trailing permutation gets one more (empty) stage
        if not remaining and not perm:
            break


def hbm_passes(L, s):
    n, m, G = L.n, s.m, L.G
    remaining = list(range(len(L.ops)))
    low_mask = (1 << min(G, n)) - 1
    while True:
        tilem, blocked, taken, deferred = low_mask, 0, [], []
        for oi in remaining:
            o = L.ops[oi]
            touch, need = op_touch(o), op_need(o)
            if touch & blocked:
                blocked |= touch
                deferred.append(oi)
                continue
            if popcount(tilem | need) <= m:
                tilem |= need
                taken.append(oi)
            else:
                blocked |= touch
                deferred.append(oi)
        for oi in deferred:   # pad with the deferred ops' targets first
            if popcount(tilem) >= m:
                break
            need = op_need(L.ops[oi])
            if need and popcount(tilem | need) <= m:
                tilem |= need
        for q in range(n - 1, -1, -1):
            if popcount(tilem) >= m:
                break
            tilem |= 1 << q
        ps = np.zeros((), DPASS)
        ps["stage_begin"], ps["m"], ps["nout"] = len(s.stages), m, n - m
        tile = [q for q in range(n) if tilem >> q & 1]
        outq = [q for q in range(n) if not (tilem >> q & 1)]
        ps["tile_q"][:m] = tile
        ps["out_q"][:len(outq)] = outq
        slot_of, acc_of = {}, {}
        ps["ps_begin"] = len(s.pass_entries)
        for per in (1, 0):
            for oi in taken:
                ent = L.ops[oi][3]
                if ent >= 0 and L.entries[ent]["per_sample"] == per and ent not in slot_of:
                    slot_of[ent] = int(ps["ps_count" if per else "sh_count"])
                    ps["ps_count" if per else "sh_count"] += 1
                    s.pass_entries.append(ent)
            if per:
                ps["sh_begin"] = len(s.pass_entries)
        ps["acc_begin"] = len(s.pass_accs)
        for oi in taken:
            ent = L.ops[oi][3]
            if ent >= 0 and L.entries[ent]["acc"] != 0xffff and L.entries[ent]["acc"] not in acc_of:
                acc_of[L.entries[ent]["acc"]] = int(ps["acc_count"])
                ps["acc_count"] += 1
                s.pass_accs.append(L.entries[ent]["acc"])
        cut_stages(L, taken, tile, s.K, s, slot_of, acc_of)
        ps["stage_end"] = len(s.stages)
        s.passes.append(ps)
        remaining = deferred
        if not remaining:
            break


def cluster_locality(st, K, n, cl):
    """cl_local of a cluster-schedule stage, by enumerating every (thread,
    register) slot of both maps: bit 0 (loads) / bit 1 (stores) when each slot
    lies in the slice of the CTA whose rank is the thread's top cl index bits
    (slices of 2^(n - cl) slots, in rank order)."""
    nb = int(st["nthreadbits"])
    t = np.arange(1 << nb, dtype=np.int64)
    r = np.arange(1 << K, dtype=np.int64)
    flags = 0
    for bit, (sig, tau) in enumerate((("sigma", "tau"), ("sigma_st", "tau_st"))):
        base = np.zeros_like(t)
        for i in range(nb):
            base ^= np.where((t >> i) & 1, int(st[tau][i]), 0)
        off = np.zeros_like(r)
        for j in range(K):
            off ^= np.where((r >> j) & 1, int(st[sig][j]), 0)
        slots = base[:, None] ^ off[None, :]
        if np.all((slots >> (n - cl)) == (t >> (nb - cl))[:, None]):
            flags |= 1 << bit
    return flags


def schedules(L):
    """Resident schedules for every usable (mode, K), cluster schedules (one
    sample over 2-8 CTAs of 512 threads), then HBM passes."""
    c64 = L.dtype == C64
    max_k = {(0, True): 5, (1, True): 4, (0, False): 4, (1, False): 3}
    res_max = {(0, True): 14, (1, True): 13, (0, False): 13, (1, False): 12}
    tile_q = {(0, True): 13, (1, True): 12, (0, False): 12, (1, False): 11}
    n = L.n
    out = []
    for mode in (0, 1):
        for K in range(1, min(max_k[mode, c64], n) + 1):
            if n - K > 9 or n > res_max[mode, c64]:
                continue
            s = Schedule(mode, K, n, 0)
            cut_stages(L, range(len(L.ops)), list(range(n)), K, s,
                       {i: e["slot"] for i, e in enumerate(L.entries)}, {i: i for i in range(len(L.accs))})
            out.append(s)
    for mode in (0, 1):
        # one register block per thread, 512-thread CTAs, <= 128 KiB of state
        # (psi, and lam for the backward) per CTA
        K = max_k[mode, c64]
        cl = n - K - 9
        if n > res_max[mode, c64] and n <= 16 and 1 <= cl <= 3 and \
                ((mode + 1) << (n - cl)) * (8 if c64 else 16) <= 128 * 1024:
            s = Schedule(mode, K, n, 2)
            s.cta_bits = 9
            cut_stages(L, range(len(L.ops)), list(range(n)), K, s,
                       {i: e["slot"] for i, e in enumerate(L.entries)}, {i: i for i in range(len(L.accs))})
            for st in s.stages:
                st["cl_local"] = cluster_locality(st, K, n, cl)
            out.append(s)
    for mode in (0, 1):
        m = min(tile_q[mode, c64], n - 1)
        K = min(max_k[mode, c64], m - 1)
        if n < L.G + 2 or K < 1 or m <= L.G or K != max_k[mode, c64]:
            continue
        if mode == 1 and not any(s.path == 1 and s.mode == 0 for s in out):
            continue
        s = Schedule(mode, K, m, 1)
        hbm_passes(L, s)
        out.append(s)
    return out


# ---------------------------------------------------------------- bytes
def _vec(arr, dtype):
    a = np.asarray(arr, dtype=dtype)
    return struct.pack("<i", len(a)) + a.tobytes()


def _records(items, dtype):
    return struct.pack("<i", len(items)) + b"".join(np.asarray(r, dtype=dtype).tobytes() for r in items)


def plan_bytes(spec, dtype):
    """The bytes vqc_plan_export must return for spec compiled with dtype
    ("c64", "c128" or "c128df"; double-float plans are complex128 plans)."""
    L = Lowered(spec, dtype)
    out = b"VQCP" + struct.pack("<i", 3)
    out += struct.pack("<9i", L.n, L.nx, L.nw, L.dtype, L.num_gates_in, L.G, L.n_ps, L.n_sh, L.n_runs)
    out += _vec([v for o in L.ops for v in o], "<i4")
    ents = []
    for e in L.entries:
        r = np.zeros((), DENTRY)
        for k in ("cfirst", "ccount", "slot", "per_sample", "phase", "acc"):
            r[k] = e[k]
        ents.append(r)
    out += _records(ents, DENTRY)
    cons = []
    for c in L.consts:
        r = np.zeros((), DCONST)
        for k in ("kind", "src0", "src1", "idx0", "idx1", "term"):
            r[k] = c[k]
        cons.append(r)
    out += _records(cons, DCONST)
    out += _vec(L.cmat, "<f8") + _vec(L.cang, "<f8")
    out += _vec(L.term_src, "<i4") + _vec(L.term_idx, "<i4")
    out += struct.pack("<i", len(L.accs)) + np.asarray(L.accs, dtype="<i4").reshape(-1).tobytes()
    for v in (L.xocc_ptr, L.xocc, L.wocc_ptr, L.wocc):
        out += _vec(v, "<i4")
    sch = schedules(L)
    out += struct.pack("<i", len(sch))
    for s in sch:
        out += struct.pack("<7i", s.mode, s.K, s.m, s.path, s.thread_bits, s.group_lanes_log2, s.cta_bits)
        out += _records(s.ops, DOP) + _records(s.stages, DSTAGE) + _records(s.passes, DPASS)
        out += _vec(s.pass_entries, "<i4") + _vec(s.pass_accs, "<i4") + _vec(s.store_masks, "<u4")
    return out
