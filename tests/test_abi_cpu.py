"""CPU tests of the boundary and the host compiler (no kernel launches).

* libvqc.so loads and exports every entry point declared in include/vqc.h;
* vqc_compile validates its input (static-circuit scope, paper Sec. 3) and
  returns the documented status codes;
* vqc_plan_export is a deterministic function of the compile arguments;
* every exported stage schedule, executed on the CPU exactly as the kernels
  address it (tests/plan_emulator.py), reproduces the oracle's final state
  and the oracle's adjoint gradients;
* register-block addressing is a bijection onto the shared-memory slots.
"""
import os
import re

import numpy as np
import pytest

from oracle import oracle as orc
from paper_2607_11985_gb300 import binding as B
from paper_2607_11985_gb300 import workloads as wl
from tests.plan_emulator import Plan, op_type, swz

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2607_11985_gb300 import build
    build.build()


def header_functions():
    with open(os.path.join(ROOT, "include", "vqc.h")) as f:
        text = f.read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"^[A-Za-z_][\w\s\*]*?\b(vqc_\w+)\s*\(", text, flags=re.M)))


def test_library_exports_every_declared_symbol():
    names = header_functions()
    assert len(names) >= 11, names
    lib = B.lib()
    for name in names:
        assert hasattr(lib, name), name
    assert B.vqc_abi_version() == 1
    assert {s[0] for s in B.SIGNATURES} == set(names)


def compile_spec(spec, dtype=0):
    arr = B.gates_array(spec)
    return B.vqc_compile(arr, len(spec.gates), spec.n, spec.num_x, spec.num_w, dtype)


def status_of(spec, dtype=0, n=None, nx=None, nw=None, arr=None):
    import ctypes
    arr = arr if arr is not None else B.gates_array(spec)
    plan = ctypes.c_void_p()
    st = B.lib().vqc_compile(arr, len(spec.gates), spec.n if n is None else n,
                             spec.num_x if nx is None else nx, spec.num_w if nw is None else nw,
                             dtype, ctypes.byref(plan))
    if st == 0:
        B.vqc_free(plan.value)
    return st


def test_validation_codes():
    ok = wl.CircuitSpec(3, 1, 1).add("RY", (0,), [("x", 0)]).add("CX", (0, 2)).add("RZ", (1,), [("w", 0)])
    assert status_of(ok) == 0
    assert status_of(wl.CircuitSpec(3, 0, 0).add("H", (3,))) == 3            # qubit range
    assert status_of(wl.CircuitSpec(3, 0, 0).add("CX", (1, 1))) == 3         # repeated qubit
    assert status_of(wl.CircuitSpec(3, 1, 0).add("RX", (0,), [("x", 1)])) == 5   # x column
    assert status_of(wl.CircuitSpec(3, 0, 1).add("RX", (0,), [("w", 3)])) == 5   # w index
    assert status_of(ok, n=0) == 4
    assert status_of(ok, n=25) == 4
    assert status_of(ok, nx=-1) == 1
    assert status_of(ok, dtype=7) == 1
    arr = B.gates_array(ok)
    arr[0].op = 16
    assert status_of(ok, arr=arr) == 2
    arr = B.gates_array(ok)
    arr[1].reserved[0] = 1
    assert status_of(ok, arr=arr) == 1
    arr = B.gates_array(ok)
    arr[0].pkind[0] = 0
    assert status_of(ok, arr=arr) == 5
    assert "invalid source" in B.vqc_last_error()


def test_export_deterministic_and_info():
    for k in (1, 2, 3):
        spec = wl.config(k)[0].spec
        p1, p2 = compile_spec(spec), compile_spec(spec)
        assert B.vqc_plan_export(p1) == B.vqc_plan_export(p2)
        info = B.vqc_plan_info(p1, 1024)
        assert info["num_gates_in"] == len(spec.gates)
        assert info["fwd_path"] == 0 and info["fwd_stages"] >= 1
        B.vqc_free(p1)
        B.vqc_free(p2)


def test_double_float_plan_is_a_complex128_plan():
    # VQC_C128_DF changes only the kernels' arithmetic: the plan bytes (layouts,
    # schedules, tables) equal the complex128 plan's; plan_info reports the dtype
    for k in (2, 3, 5):
        spec = wl.config(k)[0].spec
        p1, p2 = compile_spec(spec, B.VQC_C128), compile_spec(spec, B.VQC_C128_DF)
        assert B.vqc_plan_export(p1) == B.vqc_plan_export(p2)
        i1, i2 = B.vqc_plan_info(p1, 512), B.vqc_plan_info(p2, 512)
        assert i1["dtype"] == B.VQC_C128 and i2["dtype"] == B.VQC_C128_DF
        assert {k: v for k, v in i1.items() if k != "dtype"} == {k: v for k, v in i2.items() if k != "dtype"}
        B.vqc_free(p1)
        B.vqc_free(p2)
    assert status_of(wl.config(1)[0].spec, dtype=3) == 1   # VQC_ERR_INVALID_ARG


def slot_of(st, K, t, r, sig, tau):
    sl = 0
    for i in range(int(st["nthreadbits"])):
        if (t >> i) & 1:
            sl ^= int(st[tau][i])
    for j in range(K):
        if (r >> j) & 1:
            sl ^= int(st[sig][j])
    return sl


def check_addressing(plan):
    """Load and store maps of every stage agree with the swizzle of the
    indices the emulator assigns to each (thread, register) and are
    bijections onto the tile's slots."""
    for s in plan.scheds:
        n, K, m = plan.n, s["K"], s["m"]
        if s["path"] in (0, 2):   # resident / cluster: one tile holding every qubit
            tiles = [(list(range(n)), range(len(s["stages"])))]
        else:
            tiles = [(list(ps["tile_q"][:ps["m"]]), range(ps["stage_begin"], ps["stage_end"]))
                     for ps in s["passes"]]
            # every pass's tile holds the low qubits of one 128-byte chunk
            for tq, _ in tiles:
                assert tq[:min(plan.G, n)] == list(range(min(plan.G, n)))
        for tq, srange in tiles:
            tq = [int(q) for q in tq]
            lpos = {q: i for i, q in enumerate(tq)}
            local = lambda v: sum(((int(v) >> q) & 1) << lpos[q] for q in tq)
            for si in srange:
                st, sm = s["stages"][si], s["store_masks"][si]
                assert sorted(st["active"][:K].tolist()) == st["active"][:K].tolist()
                assert set(st["active"][:K].tolist()) <= set(tq)
                assert int(st["nthreadbits"]) == m - K
                slots, slots_st = set(), set()
                for t in range(1 << (m - K)):
                    _, idx = Plan.block_index(st, K, t)
                    sidx = Plan.store_index(sm, K, st["nthreadbits"], t)
                    for r in range(1 << K):
                        sl = slot_of(st, K, t, r, "sigma", "tau")
                        assert sl == swz(local(idx[r]), plan.G)
                        slots.add(sl)
                        sl = slot_of(st, K, t, r, "sigma_st", "tau_st")
                        assert sl == swz(local(sidx[r]), plan.G)
                        slots_st.add(sl)
                assert slots == set(range(1 << m)) and slots_st == slots
                if s["path"] == 0:   # one register block per thread (<= 512 threads)
                    assert n - K <= 9
                if int(st["nperm"]) == 0:
                    assert list(st["sigma_st"][:K]) == list(st["sigma"][:K])
                    assert list(st["tau_st"]) == list(st["tau"])
                for op in s["ops"][st["op_begin"]:st["op_end"]]:
                    t, oa, ob = op_type(op)
                    if t == 1:
                        assert oa < K
                    if t == 2:
                        assert ob < K
                        assert s["path"] == 1   # resident and cluster schedules fold every CX
            # <Z> / lambda come from the last stage's registers (of each pass)
            assert int(s["stages"][srange[-1]]["nperm"]) == 0


SMALL_CASES = [(s, n, g) for s, n, g in [(101, 1, 12), (102, 2, 30), (103, 3, 60), (104, 4, 80),
                                        (105, 5, 120), (106, 6, 150), (107, 7, 150)]]


@pytest.mark.parametrize("seed,n,G", SMALL_CASES)
@pytest.mark.parametrize("dtype", [0, 1])
def test_schedules_reproduce_oracle_state(seed, n, G, dtype):
    w_, psi0 = wl.small_random(seed, n, G, batch=2, dtype="c128", with_psi0=(seed % 2 == 1))
    pl = Plan(B.vqc_plan_export(compile_spec(w_.spec, dtype)))
    check_addressing(pl)
    _, ref = orc.forward(w_.spec, w_.x, w_.w, psi0=psi0, want_state=True)
    assert len(pl.scheds) >= 2
    for s in pl.scheds:
        for b in range(2):
            xb = w_.x[b] if w_.spec.num_x else np.zeros(0)
            got = pl.forward(s, xb, w_.w, None if psi0 is None else psi0[b])
            assert np.allclose(got, ref[b], atol=1e-12), (s["mode"], s["K"])


@pytest.mark.parametrize("seed,n,G", SMALL_CASES[:6])
def test_schedules_reproduce_oracle_gradients(seed, n, G):
    w_, psi0 = wl.small_random(seed, n, G, batch=2, dtype="c128", with_psi0=(seed % 2 == 0))
    pl = Plan(B.vqc_plan_export(compile_spec(w_.spec, 1)))
    dx_ref, dw_ref = orc.backward(w_.spec, w_.x, w_.w, w_.gE, psi0=psi0)
    for s in pl.scheds:
        if s["mode"] != 1:
            continue
        dw = np.zeros(w_.spec.num_w)
        for b in range(2):
            xb = w_.x[b] if w_.spec.num_x else np.zeros(0)
            dx, dwb = pl.backward(s, xb, w_.w, w_.gE[b], None if psi0 is None else psi0[b])
            assert np.allclose(dx, dx_ref[b], atol=1e-10), s["K"]
            dw += dwb
        assert np.allclose(dw, dw_ref, atol=1e-10), s["K"]


@pytest.mark.parametrize("seed,n,G", [(501, 8, 120), (502, 9, 160), (503, 10, 200)])
def test_hbm_schedules_small_tiles(monkeypatch, seed, n, G):
    # force small tiles so the HBM pass schedules are exercised at emulator sizes
    monkeypatch.setenv("VQC_HBM_TILE_QUBITS", str(6))
    w_, psi0 = wl.small_random(seed, n, G, batch=1, dtype="c128", with_psi0=True)
    for dtype in (0, 1):
        pl = Plan(B.vqc_plan_export(compile_spec(w_.spec, dtype)))
        check_addressing(pl)
        hb = [s for s in pl.scheds if s["path"] == 1]
        assert len(hb) == 2 and all(len(s["passes"]) >= 2 for s in hb)
        _, ref = orc.forward(w_.spec, w_.x, w_.w, psi0=psi0, want_state=True)
        dx_ref, dw_ref = orc.backward(w_.spec, w_.x, w_.w, w_.gE, psi0=psi0)
        for s in hb:
            got = pl.forward(s, w_.x[0], w_.w, psi0[0])
            assert np.allclose(got, ref[0], atol=1e-12)
            if s["mode"] == 1 and dtype == 1:
                dx, dw = pl.backward(s, w_.x[0], w_.w, w_.gE[0], psi0[0])
                assert np.allclose(dx, dx_ref[0], atol=1e-10)
                assert np.allclose(dw, dw_ref, atol=1e-10)


@pytest.mark.parametrize("n", range(2, 14))
def test_hbm_backward_schedule_implies_forward(n):
    # the HBM backward recomputes the final state with the forward passes when
    # none is given, so a plan never holds the backward passes alone
    w_, _ = wl.small_random(520 + n, n, 4 * n, batch=1, dtype="c128")
    for dtype in (0, 1):
        pl = Plan(B.vqc_plan_export(compile_spec(w_.spec, dtype)))
        modes = {s["mode"] for s in pl.scheds if s["path"] == 1}
        assert 1 not in modes or 0 in modes, (n, dtype, modes)


def test_config5_hbm_schedule_structure():
    w_ = wl.config(5, batch=1)[0]
    for dtype in (0, 1):
        pl = Plan(B.vqc_plan_export(compile_spec(w_.spec, dtype)))
        assert not any(s["path"] == 0 for s in pl.scheds)
        hb = [s for s in pl.scheds if s["path"] == 1]
        assert len(hb) == 2
        for s in hb:
            # every op lands in exactly one stage of one pass: as an op record or
            # folded into a store map (CX gates with both qubits in the tile)
            assert sum(st["op_end"] - st["op_begin"] for st in s["stages"]) + \
                int(s["stages"]["nperm"].sum()) == len(pl.hops)
            assert int(s["stages"]["nperm"].sum()) > 0
            assert s["passes"][-1]["stage_end"] == len(s["stages"])


def slots_all(st, K, sig, tau):
    """slot_of for every (thread, register) pair at once: [threads, 2^K]."""
    nb = int(st["nthreadbits"])
    t = np.arange(1 << nb)
    base = np.zeros(1 << nb, np.int64)
    for i in range(nb):
        base ^= np.where((t >> i) & 1, int(st[tau][i]), 0)
    r = np.arange(1 << K)
    off = np.zeros(1 << K, np.int64)
    for j in range(K):
        off ^= np.where((r >> j) & 1, int(st[sig][j]), 0)
    return base[:, None] ^ off[None, :]


def test_cluster_locality_flags():
    """Cluster schedules (2^cta_bits threads per CTA, 2^(n-K-cta_bits) CTAs): a
    stage's cl_local bit 0 / bit 1 is set exactly when every slot its load /
    store map gives a thread lies in the slice of that thread's own CTA."""
    w_ = wl.config(5, batch=1)[0]
    seen = 0
    for dtype in (0, 1):
        pl = Plan(B.vqc_plan_export(compile_spec(w_.spec, dtype)))
        for s in (s for s in pl.scheds if s["path"] == 2):
            n, K, ctb = pl.n, s["K"], s["cta_bits"]
            assert ctb == 9 and 1 <= n - K - ctb <= 3
            slice_ = K + ctb
            rank = (np.arange(1 << (n - K)) >> ctb)[:, None]
            flags = []
            for st in s["stages"]:
                ld = bool(((slots_all(st, K, "sigma", "tau") >> slice_) == rank).all())
                sto = bool(((slots_all(st, K, "sigma_st", "tau_st") >> slice_) == rank).all())
                assert int(st["cl_local"]) == (ld | (sto << 1))
                flags.append(int(st["cl_local"]))
            # a non-permuting stage stores where it loads
            for st in s["stages"]:
                if int(st["nperm"]) == 0:
                    assert int(st["cl_local"]) in (0, 3)
            assert 3 in flags
            seen += 1
    assert seen >= 1


@pytest.mark.parametrize("k", [1, 2])
def test_config_schedules_gradients(k):
    w_ = wl.config(k, dtype="c128", batch=2)[0]
    pl = Plan(B.vqc_plan_export(compile_spec(w_.spec, 1)))
    check_addressing(pl)
    dx_ref, dw_ref = orc.backward(w_.spec, w_.x, w_.w, w_.gE)
    s = [s for s in pl.scheds if s["mode"] == 1][-1]
    dw = np.zeros(w_.spec.num_w)
    for b in range(2):
        dx, dwb = pl.backward(s, w_.x[b], w_.w, w_.gE[b])
        assert np.allclose(dx, dx_ref[b], atol=1e-10)
        dw += dwb
    assert np.allclose(dw, dw_ref, atol=1e-10)


def test_reupload_config_structure():
    # config 3 shape at 6 qubits: re-uploaded x, Rot layers, CX range ring
    spec = wl.layered(6, 3, ("RZ", "RY", "RZ"), "CX", reupload=True, ring_range=lambda l: (l % 5) + 1)
    rng = np.random.default_rng(3)
    x = rng.standard_normal((1, 6))
    w = rng.uniform(-np.pi, np.pi, spec.num_w)
    gE = rng.standard_normal((1, 6))
    pl = Plan(B.vqc_plan_export(compile_spec(spec, 1)))
    dx_ref, dw_ref = orc.backward(spec, x, w, gE)
    for s in pl.scheds:
        if s["mode"] == 1:
            dx, dw = pl.backward(s, x[0], w, gE[0])
            assert np.allclose(dx, dx_ref[0], atol=1e-10)
            assert np.allclose(dw, dw_ref, atol=1e-10)
