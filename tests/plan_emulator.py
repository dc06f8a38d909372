"""Test helper: parse an exported plan and execute its stage schedules on the CPU.

This checks the host compiler (fusion, constant pre-multiplication, stage
cutting, register-block addressing, gradient-term bookkeeping) without a GPU:
each schedule is run stage by stage, thread block by thread block, exactly as
the kernels address amplitudes, in numpy complex128, and the result is
compared with the oracle.  The emulator reads only the exported plan bytes.
"""
from __future__ import annotations

import struct

import numpy as np

DENTRY = np.dtype([("cfirst", "<u2"), ("ccount", "<u2"), ("slot", "<u2"), ("per_sample", "u1"),
                   ("phase", "u1"), ("acc", "<u2"), ("pad", "<u2")])
DCONST = np.dtype([("kind", "u1"), ("src0", "u1"), ("src1", "u1"), ("pad", "u1"),
                   ("idx0", "<i4"), ("idx1", "<i4"), ("term", "<i4")])
DACC = np.dtype([("entry", "<i4"), ("kind", "<i4")])
DOP = np.dtype([("code", "u1"), ("a", "u1"), ("b", "u1"), ("flags", "u1"), ("slot", "<u2"),
                ("aux", "<u2")])
DSTAGE = np.dtype([("op_begin", "<i4"), ("op_end", "<i4"), ("sigma", "<i4", 5), ("tau", "<i4", 16),
                   ("tmask", "<u4", 16), ("sigma_st", "<i4", 5), ("tau_st", "<i4", 16),
                   ("active", "u1", 5), ("nthreadbits", "u1"), ("nperm", "u1"), ("cl_local", "u1")])
DPASS = np.dtype([("stage_begin", "<i4"), ("stage_end", "<i4"), ("m", "<i4"), ("nout", "<i4"),
                  ("tile_q", "u1", 24), ("out_q", "u1", 24), ("ps_begin", "<i4"), ("ps_count", "<i4"),
                  ("sh_begin", "<i4"), ("sh_count", "<i4"), ("acc_begin", "<i4"), ("acc_count", "<i4")])
assert DENTRY.itemsize == 12 and DCONST.itemsize == 16 and DOP.itemsize == 8
assert DSTAGE.itemsize == 248 and DPASS.itemsize == 88
PATH_RESIDENT, PATH_HBM, PATH_CLUSTER = 0, 1, 2

OP_M1, OP_CX, OP_CZ, OP_PH2 = 1, 2, 3, 4
DC_M1, DC_CX_LL, DC_CX_PL, DC_CZ_LL, DC_CZ_PL, DC_CZ_PP = 0, 5, 25, 30, 40, 45
DC_PH2_LL, DC_PH2_PL, DC_PH2_PP, DC_NUM = 46, 56, 61, 62
CZ_PAIRS = [(0, 1), (0, 2), (0, 3), (0, 4), (1, 2), (1, 3), (1, 4), (2, 3), (2, 4), (3, 4)]


def op_type(op):
    """Decode an op's dispatch code into (type, a, b), checking that the code
    agrees with the refs it carries."""
    c, a, b = int(op["code"]), int(op["a"]), int(op["b"])
    if c < DC_CX_LL:
        assert a == c - DC_M1
        return OP_M1, a, b
    if c < DC_CX_PL:
        k = c - DC_CX_LL
        cc, tt = k // 4, k % 4
        tt = tt if tt < cc else tt + 1
        assert (a, b) == (cc, tt)
        return OP_CX, a, b
    if c < DC_CZ_LL:
        assert a >= REF_PHYS and b == c - DC_CX_PL
        return OP_CX, a, b
    if c < DC_CZ_PL:
        assert (a, b) == CZ_PAIRS[c - DC_CZ_LL]
        return OP_CZ, a, b
    if c < DC_CZ_PP:
        assert a == c - DC_CZ_PL and b >= REF_PHYS
        return OP_CZ, a, b
    if c == DC_CZ_PP:
        assert a >= REF_PHYS and b >= REF_PHYS
        return OP_CZ, a, b
    if c < DC_PH2_PL:
        lo, hi = CZ_PAIRS[c - DC_PH2_LL]
        assert a < REF_PHYS and b < REF_PHYS and (min(a, b), max(a, b)) == (lo, hi)
    elif c < DC_PH2_PP:
        assert (a < REF_PHYS) != (b < REF_PHYS) and min(a, b) == c - DC_PH2_PL
    else:
        assert c == DC_PH2_PP and a >= REF_PHYS and b >= REF_PHYS
    return OP_PH2, a, b
OPF_PER_SAMPLE, OPF_GEN_CRZ, OPF_GEN_RZZ, OPF_HAS_ACC = 1, 2, 4, 8
CK_CONST, CK_RX, CK_RY, CK_RZ, CK_GPHASE, CK_CRZ, CK_RZZ = 1, 2, 3, 4, 5, 6, 7
SRC_CONST, SRC_X, SRC_W = 1, 2, 3
REF_PHYS = 8


class Reader:
    def __init__(self, buf):
        self.buf, self.off = buf, 0

    def i32(self):
        v = struct.unpack_from("<i", self.buf, self.off)[0]
        self.off += 4
        return v

    def vec(self, dtype):
        n = self.i32()
        dt = np.dtype(dtype)
        a = np.frombuffer(self.buf, dtype=dt, count=n, offset=self.off).copy()
        self.off += n * dt.itemsize
        return a


class Plan:
    def __init__(self, blob: bytes):
        assert blob[:4] == b"VQCP"
        r = Reader(blob)
        r.off = 4
        assert r.i32() == 3
        (self.n, self.num_x, self.num_w, self.dtype, self.num_gates_in, self.G, self.n_ps,
         self.n_sh, self.n_runs) = [r.i32() for _ in range(9)]
        self.hops = r.vec("<i4").reshape(-1, 5)
        self.entries = r.vec(DENTRY)
        self.consts = r.vec(DCONST)
        self.cmat = r.vec("<f8").reshape(-1, 8)
        self.cang = r.vec("<f8")
        self.term_src = r.vec("<i4")
        self.term_idx = r.vec("<i4")
        self.accs = r.vec(DACC)
        self.xocc_ptr = r.vec("<i4")
        self.xocc = r.vec("<i4")
        self.wocc_ptr = r.vec("<i4")
        self.wocc = r.vec("<i4")
        self.scheds = []
        for _ in range(r.i32()):
            mode, K, m, path, tb, gl, ctb = [r.i32() for _ in range(7)]
            ops = r.vec(DOP)
            stages = r.vec(DSTAGE)
            passes = r.vec(DPASS)
            pass_entries = r.vec("<i4")
            pass_accs = r.vec("<i4")
            store_masks = r.vec("<u4").reshape(len(stages), 5 + 16)
            self.scheds.append(dict(mode=mode, K=K, m=m, path=path, thread_bits=tb, cta_bits=ctb, ops=ops,
                                    stages=stages, passes=passes, pass_entries=pass_entries,
                                    pass_accs=pass_accs, store_masks=store_masks))
        assert r.off == len(blob)

    # ------------------------------------------------------------------ tables
    def angle(self, src, idx, xb, w):
        if src == SRC_X:
            return xb[idx]
        if src == SRC_W:
            return w[idx]
        return self.cang[idx]

    def constituent(self, c, xb, w):
        if c["kind"] == CK_CONST:
            m = self.cmat[c["idx0"]]
            return np.array([[m[0] + 1j * m[1], m[2] + 1j * m[3]], [m[4] + 1j * m[5], m[6] + 1j * m[7]]])
        t = self.angle(c["src0"], c["idx0"], xb, w)
        if c["kind"] == CK_GPHASE:
            t += self.angle(c["src1"], c["idx1"], xb, w)
        co, s = np.cos(t / 2), np.sin(t / 2)
        if c["kind"] == CK_RX:
            return np.array([[co, -1j * s], [-1j * s, co]])
        if c["kind"] == CK_RY:
            return np.array([[co, -s], [s, co]])
        if c["kind"] == CK_RZ:
            return np.diag([np.exp(-0.5j * t), np.exp(0.5j * t)])
        assert c["kind"] == CK_GPHASE
        return np.exp(0.5j * t) * np.eye(2)

    def entry_value(self, eid, xb, w):
        e = self.entries[eid]
        cs = self.consts[e["cfirst"]:e["cfirst"] + e["ccount"]]
        if e["phase"]:
            c = cs[0]
            t = self.angle(c["src0"], c["idx0"], xb, w)
            a, b = np.exp(-0.5j * t), np.exp(0.5j * t)
            return np.array([1, a, 1, b]) if c["kind"] == CK_CRZ else np.array([a, b, b, a])
        M = np.eye(2, dtype=complex)
        for c in cs:
            M = self.constituent(c, xb, w) @ M
        return M

    def tables(self, xb, w):
        ps, sh = [None] * self.n_ps, [None] * self.n_sh
        for eid, e in enumerate(self.entries):
            (ps if e["per_sample"] else sh)[e["slot"]] = self.entry_value(eid, xb, w)
        return ps, sh

    # ------------------------------------------------------------------ blocks
    @staticmethod
    def block_index(st, K, t):
        base = 0
        for i in range(int(st["nthreadbits"])):
            if (t >> i) & 1:
                base |= int(st["tmask"][i])
        idx = np.array([base | sum(((r >> j) & 1) << int(st["active"][j]) for j in range(K))
                        for r in range(1 << K)])
        return base, idx

    @staticmethod
    def store_index(masks, K, nthreadbits, t):
        """Physical indices the block of thread t is stored to: the images of
        its indices under the stage's absorbed permutation (XOR-linear)."""
        base = 0
        for i in range(int(nthreadbits)):
            if (t >> i) & 1:
                base ^= int(masks[5 + i])
        idx = []
        for r in range(1 << K):
            v = base
            for j in range(K):
                if (r >> j) & 1:
                    v ^= int(masks[j])
            idx.append(v)
        return np.array(idx)

    @staticmethod
    def refbit(ref, r, base):
        ref, r, base = int(ref), int(r), int(base)
        return (base >> (ref - REF_PHYS)) & 1 if ref >= REF_PHYS else (r >> ref) & 1

    def apply_op(self, op, K, base, a, tabs, adjoint=False):
        ps, sh = tabs
        tab = ps if op["flags"] & OPF_PER_SAMPLE else sh
        t, oa, ob = op_type(op)
        if t == OP_M1:
            M = tab[op["slot"]]
            if adjoint:
                M = M.conj().T
            T = oa
            assert T < K
            for r in range(1 << K):
                if not (r >> T) & 1:
                    u, v = a[r], a[r | (1 << T)]
                    a[r], a[r | (1 << T)] = M[0, 0] * u + M[0, 1] * v, M[1, 0] * u + M[1, 1] * v
        elif t == OP_CX:
            T = ob
            assert T < K
            for r in range(1 << K):
                if not (r >> T) & 1 and self.refbit(oa, r, base):
                    a[r], a[r | (1 << T)] = a[r | (1 << T)], a[r]
        elif t == OP_CZ:
            for r in range(1 << K):
                if self.refbit(op["a"], r, base) and self.refbit(op["b"], r, base):
                    a[r] = -a[r]
        elif t == OP_PH2:
            ph = tab[op["slot"]]
            if adjoint:
                ph = ph.conj()
            for r in range(1 << K):
                s = self.refbit(op["a"], r, base) + 2 * self.refbit(op["b"], r, base)
                a[r] *= ph[s]
        else:
            raise AssertionError("bad op type %d" % t)

    # ------------------------------------------------------------------ runs
    def units(self, sched, xb, w):
        """(stages, tile bases, tables, acc map) of each pass; the resident path
        is one pass over one tile holding every qubit."""
        n = self.n
        if sched["path"] in (PATH_RESIDENT, PATH_CLUSTER):
            yield (sched["stages"], [0], self.tables(xb, w), np.arange(len(self.accs)),
                   sched["store_masks"])
            return
        pe = sched["pass_entries"]
        for ps in sched["passes"]:
            ps_ids = pe[ps["ps_begin"]:ps["ps_begin"] + ps["ps_count"]]
            sh_ids = pe[ps["sh_begin"]:ps["sh_begin"] + ps["sh_count"]]
            tabs = ([self.entry_value(int(e), xb, w) for e in ps_ids],
                    [self.entry_value(int(e), xb, w) for e in sh_ids])
            out_q = ps["out_q"][:ps["nout"]]
            bases = []
            for tau in range(1 << int(ps["nout"])):
                bases.append(sum(((tau >> j) & 1) << int(out_q[j]) for j in range(int(ps["nout"]))))
            accmap = sched["pass_accs"][ps["acc_begin"]:ps["acc_begin"] + ps["acc_count"]]
            yield (sched["stages"][ps["stage_begin"]:ps["stage_end"]], bases, tabs, accmap,
                   sched["store_masks"][ps["stage_begin"]:ps["stage_end"]])

    def forward(self, sched, xb, w, psi0=None):
        n, K = self.n, sched["K"]
        psi = np.zeros(1 << n, complex)
        if psi0 is None:
            psi[0] = 1
        else:
            psi[:] = psi0
        for stages, bases, tabs, _, smasks in self.units(sched, xb, w):
            for tb in bases:
                for st, sm in zip(stages, smasks):
                    new = psi.copy()
                    for t in range(1 << int(st["nthreadbits"])):
                        base, idx = self.block_index(st, K, t)
                        base |= tb
                        idx = idx | tb
                        a = psi[idx].copy()
                        for op in sched["ops"][st["op_begin"]:st["op_end"]]:
                            self.apply_op(op, K, base, a, tabs)
                        new[self.store_index(sm, K, st["nthreadbits"], t) | tb] = a
                    psi = new
        return psi

    def backward(self, sched, xb, w, gEb, psi0=None):
        """(dx row, dw contribution) of one sample by the plan's adjoint sweep:
        rho accumulated at each run's output, terms Im Tr(W P W^dag rho)."""
        n, K = self.n, sched["K"]
        psi = self.forward(sched, xb, w, psi0)
        k = np.arange(1 << n)
        O = sum(gEb[j] * (1 - 2 * ((k >> j) & 1)) for j in range(n))
        lam = O * psi
        acc = np.zeros((len(self.accs), 8))
        for stages, bases, tabs, accmap, smasks in list(self.units(sched, xb, w))[::-1]:
          for tb in bases:
           for st, sm in list(zip(stages, smasks))[::-1]:
            ops = sched["ops"][st["op_begin"]:st["op_end"]]
            npsi, nlam = psi.copy(), lam.copy()
            for t in range(1 << int(st["nthreadbits"])):
                base, idx = self.block_index(st, K, t)
                base |= tb
                idx = idx | tb
                sidx = self.store_index(sm, K, st["nthreadbits"], t) | tb
                a, l = psi[sidx].copy(), lam[sidx].copy()
                for op in ops[::-1]:
                    if op["flags"] & OPF_HAS_ACC:
                        if op_type(op)[0] == OP_M1:
                            T = int(op["a"])
                            for r in range(1 << K):
                                if not (r >> T) & 1:
                                    pp = [a[r], a[r | (1 << T)]]
                                    ll = [l[r], l[r | (1 << T)]]
                                    for ia in range(2):
                                        for ib in range(2):
                                            z = pp[ia] * np.conj(ll[ib])
                                            acc[accmap[op["aux"]], 2 * (2 * ia + ib)] += z.real
                                            acc[accmap[op["aux"]], 2 * (2 * ia + ib) + 1] += z.imag
                        else:
                            crz = op["flags"] & OPF_GEN_CRZ
                            for r in range(1 << K):
                                ba = self.refbit(op["a"], r, base)
                                bb = self.refbit(op["b"], r, base)
                                g = (1 - 2 * bb) * ba if crz else 1 - 2 * (ba ^ bb)
                                acc[accmap[op["aux"]], 0] += g * (np.conj(l[r]) * a[r]).imag
                    self.apply_op(op, K, base, a, tabs, adjoint=True)
                    self.apply_op(op, K, base, l, tabs, adjoint=True)
                npsi[idx], nlam[idx] = a, l
            psi, lam = npsi, nlam
        terms = np.zeros(len(self.term_src))
        P = {CK_RX: np.array([[0, 1], [1, 0]], complex),
             CK_RY: np.array([[0, -1j], [1j, 0]]),
             CK_RZ: np.array([[1, 0], [0, -1]], complex)}
        for k2, ac in enumerate(self.accs):
            e = self.entries[ac["entry"]]
            cs = self.consts[e["cfirst"]:e["cfirst"] + e["ccount"]]
            if ac["kind"] == 1:
                terms[cs[0]["term"]] = acc[k2, 0]
                continue
            v = acc[k2]
            rho = np.array([[v[0] + 1j * v[1], v[2] + 1j * v[3]], [v[4] + 1j * v[5], v[6] + 1j * v[7]]])
            W = np.eye(2, dtype=complex)
            for c in cs[::-1]:
                if c["term"] >= 0:
                    terms[c["term"]] = np.trace(W @ P[int(c["kind"])] @ W.conj().T @ rho).imag
                W = W @ self.constituent(c, xb, w)
        dx = np.array([terms[self.xocc[self.xocc_ptr[p]:self.xocc_ptr[p + 1]]].sum()
                       for p in range(self.num_x)])
        dw = np.array([terms[self.wocc[self.wocc_ptr[p]:self.wocc_ptr[p + 1]]].sum()
                       for p in range(self.num_w)])
        return dx, dw


def swz(u, G):
    v, f = u >> G, 0
    while v:
        f ^= v
        v >>= G
    return u ^ (f & ((1 << G) - 1))
