// compiler.cpp -- host compiler: gate list -> plan (paper, Alg. 1 compile phase).
//
// Steps, each O(G):
//   1. validate every gate (static-circuit scope, Sec. 3: fixed gate identity
//      and wiring, only angles vary at run time);
//   2. lower: SWAP -> CX CX CX; single-qubit gates become constituents of the
//      run open on their qubit; a two-qubit gate closes the runs on its qubits;
//   3. classify constituents as constant (pre-multiplied here in fp64, the
//      paper's cached static matrices) or parametric (x or w, evaluated in the
//      kernel prologue), and number the gradient terms;
//   4. cut the fused op list into register-block stages for each (mode, K).
#include <algorithm>
#include <cmath>
#include <complex>
#include <cstdlib>
#include <cstring>
#include <numeric>

#include "engine.h"

namespace vqc {
namespace {

using cd = std::complex<double>;

struct Mat2 {
    cd m[4];   // row-major [[m0, m1], [m2, m3]]
};

Mat2 mul(const Mat2& a, const Mat2& b) {   // a * b
    Mat2 r;
    r.m[0] = a.m[0] * b.m[0] + a.m[1] * b.m[2];
    r.m[1] = a.m[0] * b.m[1] + a.m[1] * b.m[3];
    r.m[2] = a.m[2] * b.m[0] + a.m[3] * b.m[2];
    r.m[3] = a.m[2] * b.m[1] + a.m[3] * b.m[3];
    return r;
}

Mat2 fixed_matrix(int op, const double* th) {
    const double r2 = 1.0 / std::sqrt(2.0);
    const cd i(0, 1);
    Mat2 u{};
    switch (op) {
    case VQC_H: u = {{r2, r2, r2, -r2}}; break;
    case VQC_X: u = {{0, 1, 1, 0}}; break;
    case VQC_Y: u = {{0, -i, i, 0}}; break;
    case VQC_Z: u = {{1, 0, 0, -1}}; break;
    case VQC_S: u = {{1, 0, 0, i}}; break;
    case VQC_T: u = {{1, 0, 0, std::polar(1.0, M_PI / 4)}}; break;
    case VQC_SX: u = {{cd(0.5, 0.5), cd(0.5, -0.5), cd(0.5, -0.5), cd(0.5, 0.5)}}; break;
    case VQC_RX: { double c = std::cos(th[0] / 2), s = std::sin(th[0] / 2);
                   u = {{c, cd(0, -s), cd(0, -s), c}}; break; }
    case VQC_RY: { double c = std::cos(th[0] / 2), s = std::sin(th[0] / 2);
                   u = {{c, -s, s, c}}; break; }
    case VQC_RZ: u = {{std::polar(1.0, -th[0] / 2), 0, 0, std::polar(1.0, th[0] / 2)}}; break;
    case VQC_U3: { double c = std::cos(th[0] / 2), s = std::sin(th[0] / 2);
                   u = {{c, -std::polar(s, th[2]), std::polar(s, th[1]),
                         std::polar(c, th[1] + th[2])}}; break; }
    default: break;
    }
    return u;
}

bool is_two_qubit(int op) { return op >= VQC_CX && op <= VQC_RZZ; }
int num_angles(int op) {
    switch (op) {
    case VQC_RX: case VQC_RY: case VQC_RZ: case VQC_CRZ: case VQC_RZZ: return 1;
    case VQC_U3: return 3;
    default: return 0;
    }
}

struct Src {
    uint8_t kind = SRC_NONE;
    int32_t idx = 0;
    double cval = 0;
};

struct Cons {            // constituent before packing
    uint8_t kind;
    Src s0, s1;
    Mat2 mat;            // CK_CONST
};

struct Builder {
    HostPlan& p;
    std::vector<std::vector<Cons>> open;   // per qubit

    explicit Builder(HostPlan& plan) : p(plan), open(plan.n) {}

    int32_t cang_index(double v) {
        p.cang.push_back(v);
        return (int32_t)p.cang.size() - 1;
    }

    // Pack a constituent list into an entry.  Consecutive constants are
    // multiplied here (time order: later factor on the left).
    int make_entry(std::vector<Cons>& in, bool phase) {
        std::vector<Cons> cs;
        for (auto& c : in) {
            if (c.kind == CK_CONST && !cs.empty() && cs.back().kind == CK_CONST)
                cs.back().mat = mul(c.mat, cs.back().mat);
            else
                cs.push_back(c);
        }
        DEntry e{};
        e.cfirst = (uint16_t)p.consts.size();
        e.ccount = (uint16_t)cs.size();
        e.phase = phase ? 1 : 0;
        e.per_sample = 0;
        bool has_term = false;
        for (auto& c : cs) {
            DConst d{};
            d.kind = c.kind;
            d.term = -1;
            if (c.kind == CK_CONST) {
                d.idx0 = (int32_t)(p.cmat.size() / 8);
                for (int k = 0; k < 4; ++k) {
                    p.cmat.push_back(c.mat.m[k].real());
                    p.cmat.push_back(c.mat.m[k].imag());
                }
            } else {
                auto put = [&](const Src& s, uint8_t& kind, int32_t& idx) {
                    kind = s.kind;
                    idx = s.kind == SRC_CONST ? cang_index(s.cval) : s.idx;
                    if (s.kind == SRC_X) e.per_sample = 1;
                };
                put(c.s0, d.src0, d.idx0);
                if (c.kind == CK_GPHASE) put(c.s1, d.src1, d.idx1);
                // Gradient terms: rotations and phase gates with an x or w source.
                // The global phase of U3 carries none: L is invariant under it.
                if (c.kind != CK_GPHASE && (c.s0.kind == SRC_X || c.s0.kind == SRC_W)) {
                    d.term = (int32_t)p.term_src.size();
                    p.term_src.push_back(c.s0.kind);
                    p.term_idx.push_back(c.s0.idx);
                    has_term = true;
                }
            }
            p.consts.push_back(d);
        }
        int id = (int)p.entries.size();
        e.acc = 0xffff;
        if (has_term) {
            e.acc = (uint16_t)p.accs.size();
            p.accs.push_back(DAcc{id, phase ? 1 : 0});
        }
        p.entries.push_back(e);
        return id;
    }

    void flush(int q) {
        if (open[q].empty()) return;
        int id = make_entry(open[q], false);
        open[q].clear();
        p.ops.push_back(HOp{OP_M1, q, -1, id, 0});
        ++p.n_runs;
    }

    void add_rotation(int q, uint8_t kind, const Src& s) {
        Cons c{};
        if (s.kind == SRC_CONST) {
            const double th[3] = {s.cval, 0, 0};
            c.kind = CK_CONST;
            c.mat = fixed_matrix(kind == CK_RX ? VQC_RX : kind == CK_RY ? VQC_RY : VQC_RZ, th);
        } else {
            c.kind = kind;
            c.s0 = s;
        }
        open[q].push_back(c);
    }

    void add_gate(const vqc_gate& g) {
        Src src[3];
        for (int k = 0; k < num_angles(g.op); ++k) {
            src[k].kind = g.pkind[k];
            src[k].idx = g.pidx[k];
            src[k].cval = g.pconst[k];
        }
        const int q0 = g.q0, q1 = g.q1;
        switch (g.op) {
        case VQC_H: case VQC_X: case VQC_Y: case VQC_Z: case VQC_S: case VQC_T: case VQC_SX: {
            Cons c{};
            c.kind = CK_CONST;
            c.mat = fixed_matrix(g.op, nullptr);
            open[q0].push_back(c);
            break;
        }
        case VQC_RX: add_rotation(q0, CK_RX, src[0]); break;
        case VQC_RY: add_rotation(q0, CK_RY, src[0]); break;
        case VQC_RZ: add_rotation(q0, CK_RZ, src[0]); break;
        case VQC_U3: {
            bool all_const = src[0].kind == SRC_CONST && src[1].kind == SRC_CONST &&
                             src[2].kind == SRC_CONST;
            if (all_const) {
                const double th[3] = {src[0].cval, src[1].cval, src[2].cval};
                Cons c{};
                c.kind = CK_CONST;
                c.mat = fixed_matrix(VQC_U3, th);
                open[q0].push_back(c);
            } else {
                // U3(t, p, l) = e^{i(p+l)/2} RZ(p) RY(t) RZ(l): RZ(l) first.
                add_rotation(q0, CK_RZ, src[2]);
                add_rotation(q0, CK_RY, src[0]);
                add_rotation(q0, CK_RZ, src[1]);
                Cons c{};
                if (src[1].kind == SRC_CONST && src[2].kind == SRC_CONST) {
                    c.kind = CK_CONST;
                    cd ph = std::polar(1.0, 0.5 * (src[1].cval + src[2].cval));
                    c.mat = {{ph, 0, 0, ph}};
                } else {
                    c.kind = CK_GPHASE;
                    c.s0 = src[1];
                    c.s1 = src[2];
                }
                open[q0].push_back(c);
            }
            break;
        }
        case VQC_CX: case VQC_CZ: case VQC_SWAP: case VQC_CRZ: case VQC_RZZ: {
            flush(q0);
            flush(q1);
            if (g.op == VQC_CX) {
                p.ops.push_back(HOp{OP_CX, q0, q1, -1, 0});
            } else if (g.op == VQC_SWAP) {
                p.ops.push_back(HOp{OP_CX, q0, q1, -1, 0});
                p.ops.push_back(HOp{OP_CX, q1, q0, -1, 0});
                p.ops.push_back(HOp{OP_CX, q0, q1, -1, 0});
            } else if (g.op == VQC_CZ) {
                p.ops.push_back(HOp{OP_CZ, q0, q1, -1, 0});
            } else {
                std::vector<Cons> one(1);
                one[0].kind = g.op == VQC_CRZ ? CK_CRZ : CK_RZZ;
                one[0].s0 = src[0];
                const int id = make_entry(one, true);   // constant angles come from the pool
                p.ops.push_back(HOp{OP_PH2, q0, q1, id,
                                    (uint8_t)(g.op == VQC_CRZ ? OPF_GEN_CRZ : OPF_GEN_RZZ)});
            }
            break;
        }
        default: break;
        }
    }
};

vqc_status validate(const vqc_gate* gates, int32_t G, int32_t n, int32_t nx, int32_t nw,
                    std::string& err) {
    for (int32_t g = 0; g < G; ++g) {
        const vqc_gate& x = gates[g];
        if (x.op >= VQC_NUM_GATE_OPS) {
            err = "gate " + std::to_string(g) + ": unsupported opcode " + std::to_string(x.op);
            return VQC_ERR_UNSUPPORTED_GATE;
        }
        if (x.reserved[0] || x.reserved[1] || x.reserved2) {
            err = "gate " + std::to_string(g) + ": reserved bytes must be zero";
            return VQC_ERR_INVALID_ARG;
        }
        if (x.q0 >= n || (is_two_qubit(x.op) && (x.q1 >= n || x.q1 == x.q0))) {
            err = "gate " + std::to_string(g) + ": qubit out of range or repeated";
            return VQC_ERR_QUBIT_RANGE;
        }
        for (int k = 0; k < num_angles(x.op); ++k) {
            int kind = x.pkind[k];
            bool ok = (kind == VQC_P_CONST && std::isfinite(x.pconst[k])) ||
                      (kind == VQC_P_X && x.pidx[k] >= 0 && x.pidx[k] < nx) ||
                      (kind == VQC_P_W && x.pidx[k] >= 0 && x.pidx[k] < nw);
            if (!ok) {
                err = "gate " + std::to_string(g) + ": angle " + std::to_string(k) +
                      " has an invalid source";
                return VQC_ERR_PARAM_RANGE;
            }
        }
    }
    return VQC_OK;
}

uint32_t swz(uint32_t u, int G) {
    uint32_t v = u >> G, f = 0;
    while (v) { f ^= v; v >>= G; }
    return u ^ (f & ((1u << G) - 1));
}

uint32_t op_touch(const HOp& o) {
    uint32_t t = 1u << o.q0;
    if (o.type != OP_M1) t |= 1u << o.q1;
    return t;
}
uint32_t op_need(const HOp& o) {
    if (o.type == OP_M1) return 1u << o.q0;
    if (o.type == OP_CX) return 1u << o.q1;
    return 0;
}

// Cut `ops` (indices into p.ops, time-valid order) into stages of K active
// qubits drawn from the tile qubit set `tile` (ascending).  Stage records use
// tile-local positions for shared-memory addressing and global qubits for the
// thread-bit masks.  `slot_of` / `acc_of` map entry ids / accumulator ids to the
// indices the kernel sees (identity on the resident path, pass-local on the
// HBM path).
void cut_stages(const HostPlan& p, const std::vector<int>& ops, const std::vector<int>& tile,
                int K, Schedule& s, const std::vector<int>& slot_of,
                const std::vector<int>& acc_of, bool absorb) {
    const int G = p.G_swz;
    std::vector<int> lpos(p.n, -1);   // tile-local bit of each global qubit
    uint32_t tile_mask = 0;
    for (size_t i = 0; i < tile.size(); ++i) {
        lpos[tile[i]] = (int)i;
        tile_mask |= 1u << tile[i];
    }
    std::vector<int> remaining = ops;
    bool last_perm = false;
    do {   // an empty op list still gets one (empty) stage
        uint32_t active = 0, blocked = 0, pend = 0;
        std::vector<int> taken, deferred, perm;
        for (int oi : remaining) {
            const HOp& o = p.ops[oi];
            uint32_t touch = op_touch(o), need = op_need(o);
            if (touch & blocked) {
                blocked |= touch;
                deferred.push_back(oi);
                continue;
            }
            if (absorb && o.type == OP_CX && lpos[o.q0] >= 0 && lpos[o.q1] >= 0) {
                // folded into this stage's store map (both qubits in the tile)
                pend |= touch;
                perm.push_back(oi);
                continue;
            }
            if (touch & pend) {   // would have to run after an absorbed CX
                blocked |= touch;
                deferred.push_back(oi);
                continue;
            }
            uint32_t na = active | need;
            if (__builtin_popcount(na) <= K) {
                active = na;
                taken.push_back(oi);
            } else {
                blocked |= touch;
                deferred.push_back(oi);
            }
        }
        // Pad the active set to exactly K tile qubits, keeping every residue
        // class (mod G, of tile-local positions) represented among the thread bits.
        while (__builtin_popcount(active) < K) {
            int best = -1, best_cnt = -1;
            for (int i = (int)tile.size() - 1; i >= 0; --i) {
                int q = tile[i];
                if (active >> q & 1) continue;
                int cnt = 0;
                for (int r : tile)
                    if (!(active >> r & 1) && lpos[r] % G == i % G) ++cnt;
                if (cnt > best_cnt) { best_cnt = cnt; best = q; }
            }
            active |= 1u << best;
        }
        DStage st{};
        int j = 0;
        for (int q : tile)
            if (active >> q & 1) st.active[j++] = (uint8_t)q;
        for (int k = 0; k < K; ++k) st.sigma[k] = (int32_t)swz(1u << lpos[st.active[k]], G);
        // Thread bits: bit i (i < G) takes a tile qubit whose tile-local
        // position has residue i (mod G) when one exists.
        std::vector<int> outer;
        for (int q : tile)
            if (!(active >> q & 1)) outer.push_back(q);
        std::vector<int> order;
        std::vector<bool> used(outer.size(), false);
        for (int i = 0; i < std::min<int>(G, (int)outer.size()); ++i) {
            int pick = -1;
            for (size_t c = 0; c < outer.size(); ++c)
                if (!used[c] && lpos[outer[c]] % G == i) { pick = (int)c; break; }
            if (pick < 0)
                for (size_t c = 0; c < outer.size(); ++c)
                    if (!used[c]) { pick = (int)c; break; }
            used[pick] = true;
            order.push_back(outer[pick]);
        }
        for (size_t c = 0; c < outer.size(); ++c)
            if (!used[c]) order.push_back(outer[c]);
        st.nthreadbits = (uint8_t)order.size();
        for (size_t i = 0; i < order.size(); ++i) {
            st.tau[i] = (int32_t)swz(1u << lpos[order[i]], G);
            st.tmask[i] = 1u << order[i];
        }
        // Store map: the image of each basis index under the absorbed CX gates.
        auto pi = [&](uint32_t v) {
            for (int oi : perm) {
                const HOp& o = p.ops[oi];
                if ((v >> o.q0) & 1) v ^= 1u << o.q1;
            }
            return v;
        };
        auto tile_local = [&](uint32_t v) {
            uint32_t u = 0;
            for (size_t i = 0; i < tile.size(); ++i)
                if ((v >> tile[i]) & 1) u |= 1u << i;
            return u;
        };
        const size_t mb = s.store_masks.size();
        s.store_masks.resize(mb + kMaxK + kMaxThreadBits, 0);
        for (int k = 0; k < K; ++k) {
            const uint32_t v = pi(1u << st.active[k]);
            st.sigma_st[k] = (int32_t)swz(tile_local(v), G);
            s.store_masks[mb + k] = v;
        }
        for (size_t i = 0; i < order.size(); ++i) {
            const uint32_t v = pi(1u << order[i]);
            st.tau_st[i] = (int32_t)swz(tile_local(v), G);
            s.store_masks[mb + kMaxK + i] = v;
        }
        st.nperm = (uint8_t)std::min<size_t>(perm.size(), 255);
        last_perm = !perm.empty();
        auto local = [&](int q) -> int {
            for (int k = 0; k < K; ++k)
                if (st.active[k] == q) return k;
            return -1;
        };
        auto ref = [&](int q) -> uint8_t {
            int l = local(q);
            return (uint8_t)(l >= 0 ? l : kRefPhys + q);
        };
        st.op_begin = (int32_t)s.ops.size();
        for (int oi : taken) {
            const HOp& o = p.ops[oi];
            DOp d{};
            if (o.type == OP_M1 || o.type == OP_PH2) {
                const DEntry& e = p.entries[o.entry];
                d.slot = (uint16_t)slot_of[o.entry];
                d.flags = (uint8_t)((e.per_sample ? OPF_PER_SAMPLE : 0) |
                                    (e.acc != 0xffff ? OPF_HAS_ACC : 0) | o.gen);
                d.aux = e.acc != 0xffff ? (uint16_t)acc_of[e.acc] : (uint16_t)0xffff;
            }
            if (o.type == OP_M1) {
                d.a = (uint8_t)local(o.q0);
                d.code = (uint8_t)(DC_M1 + d.a);
            } else if (o.type == OP_CX) {
                d.a = ref(o.q0);
                d.b = (uint8_t)local(o.q1);
                if (d.a < kRefPhys)
                    d.code = (uint8_t)(DC_CX_LL + 4 * d.a + (d.b < d.a ? d.b : d.b - 1));
                else
                    d.code = (uint8_t)(DC_CX_PL + d.b);
            } else if (o.type == OP_CZ) {
                uint8_t ra = ref(o.q0), rb = ref(o.q1);
                if (ra >= kRefPhys && rb >= kRefPhys) {
                    d.code = DC_CZ_PP;
                } else if (ra >= kRefPhys || rb >= kRefPhys) {
                    if (ra >= kRefPhys) std::swap(ra, rb);   // local qubit first
                    d.code = (uint8_t)(DC_CZ_PL + ra);
                } else {
                    if (ra > rb) std::swap(ra, rb);
                    d.code = (uint8_t)(DC_CZ_LL + cz_pair_index(ra, rb));
                }
                d.a = ra;
                d.b = rb;
            } else {
                d.a = ref(o.q0);
                d.b = ref(o.q1);
                const bool la = d.a < kRefPhys, lb = d.b < kRefPhys;
                if (la && lb)
                    d.code = (uint8_t)(DC_PH2_LL + cz_pair_index(std::min(d.a, d.b), std::max(d.a, d.b)));
                else if (la || lb)
                    d.code = (uint8_t)(DC_PH2_PL + (la ? d.a : d.b));
                else
                    d.code = DC_PH2_PP;
            }
            s.ops.push_back(d);
        }
        st.op_end = (int32_t)s.ops.size();
        s.stages.push_back(st);
        remaining.swap(deferred);
        // The last stage computes <Z> / lambda from its registers, in the frame
        // before its store map: a trailing permutation gets one more (empty) stage.
    } while (!remaining.empty() || last_perm);
    (void)tile_mask;
}

void build_schedule(const HostPlan& p, Schedule& s) {
    const int n = p.n;
    s.m = n;
    s.thread_bits = n - s.K;
    s.group_lanes_log2 = s.thread_bits;
    std::vector<int> ops(p.ops.size()), tile(n), slot_of(p.entries.size()), acc_of(p.accs.size());
    std::iota(ops.begin(), ops.end(), 0);
    std::iota(tile.begin(), tile.end(), 0);
    for (size_t i = 0; i < p.entries.size(); ++i) slot_of[i] = p.entries[i].slot;
    std::iota(acc_of.begin(), acc_of.end(), 0);
    // Resident schedules have one register block per thread (n - K <= 9, see
    // the schedule list), so every CX can be folded into a store map.
    cut_stages(p, ops, tile, s.K, s, slot_of, acc_of, true);
}

// HBM path: passes over tiles of m qubits (always containing the low qubits
// whose amplitudes form one 128-byte chunk), each pass cut into stages.
void build_hbm_schedule(const HostPlan& p, Schedule& s) {
    const int n = p.n, m = s.m, low = p.G_swz;   // 2^G amplitudes = 128 bytes
    s.thread_bits = m - s.K;
    s.group_lanes_log2 = s.thread_bits;
    std::vector<int> remaining(p.ops.size());
    std::iota(remaining.begin(), remaining.end(), 0);
    const uint32_t low_mask = (1u << std::min(low, n)) - 1;
    do {
        uint32_t tilem = low_mask, blocked = 0;
        std::vector<int> taken, deferred;
        for (int oi : remaining) {
            const HOp& o = p.ops[oi];
            uint32_t touch = op_touch(o), need = op_need(o);
            if (touch & blocked) {
                blocked |= touch;
                deferred.push_back(oi);
                continue;
            }
            uint32_t nt = tilem | need;
            if (__builtin_popcount(nt) <= m) {
                tilem = nt;
                taken.push_back(oi);
            } else {
                blocked |= touch;
                deferred.push_back(oi);
            }
        }
        // Pad the tile with the qubits the deferred ops need first.
        for (int oi : deferred) {
            if (__builtin_popcount(tilem) >= m) break;
            uint32_t need = op_need(p.ops[oi]);
            if (need && __builtin_popcount(tilem | need) <= m) tilem |= need;
        }
        for (int q = n - 1; q >= 0 && __builtin_popcount(tilem) < m; --q) tilem |= 1u << q;
        DPass ps{};
        ps.stage_begin = (int32_t)s.stages.size();
        ps.m = m;
        ps.nout = n - m;
        std::vector<int> tile;
        int no = 0;
        for (int q = 0; q < n; ++q) {
            if (tilem >> q & 1) tile.push_back(q);
            else ps.out_q[no++] = (uint8_t)q;
        }
        for (int i = 0; i < m; ++i) ps.tile_q[i] = (uint8_t)tile[i];
        // Pass-local table slots and accumulators.
        std::vector<int> slot_of(p.entries.size(), -1), acc_of(p.accs.size(), -1);
        ps.ps_begin = (int32_t)s.pass_entries.size();
        for (int oi : taken) {
            const HOp& o = p.ops[oi];
            if (o.entry >= 0 && p.entries[o.entry].per_sample && slot_of[o.entry] < 0) {
                slot_of[o.entry] = ps.ps_count++;
                s.pass_entries.push_back(o.entry);
            }
        }
        ps.sh_begin = (int32_t)s.pass_entries.size();
        for (int oi : taken) {
            const HOp& o = p.ops[oi];
            if (o.entry >= 0 && !p.entries[o.entry].per_sample && slot_of[o.entry] < 0) {
                slot_of[o.entry] = ps.sh_count++;
                s.pass_entries.push_back(o.entry);
            }
        }
        ps.acc_begin = (int32_t)s.pass_accs.size();
        for (int oi : taken) {
            const HOp& o = p.ops[oi];
            if (o.entry >= 0 && p.entries[o.entry].acc != 0xffff && acc_of[p.entries[o.entry].acc] < 0) {
                acc_of[p.entries[o.entry].acc] = ps.acc_count++;
                s.pass_accs.push_back(p.entries[o.entry].acc);
            }
        }
        cut_stages(p, taken, tile, s.K, s, slot_of, acc_of, true);
        ps.stage_end = (int32_t)s.stages.size();
        s.passes.push_back(ps);
        remaining.swap(deferred);
    } while (!remaining.empty());
}

template <class T>
void put_vec(std::vector<uint8_t>& out, const std::vector<T>& v) {
    int32_t count = (int32_t)v.size();
    const uint8_t* c = reinterpret_cast<const uint8_t*>(&count);
    out.insert(out.end(), c, c + 4);
    if (!v.empty()) {
        const uint8_t* b = reinterpret_cast<const uint8_t*>(v.data());
        out.insert(out.end(), b, b + v.size() * sizeof(T));
    }
}

void put_i32(std::vector<uint8_t>& out, int32_t v) {
    const uint8_t* c = reinterpret_cast<const uint8_t*>(&v);
    out.insert(out.end(), c, c + 4);
}

}  // namespace

vqc_status compile_host(const vqc_gate* gates, int32_t G, int32_t n, int32_t nx, int32_t nw,
                        int dtype, HostPlan& p, std::string& err) {
    vqc_status st = validate(gates, G, n, nx, nw, err);
    if (st != VQC_OK) return st;
    p.n = n;
    p.num_x = nx;
    p.num_w = nw;
    p.dtype = dtype;
    p.num_gates_in = G;
    p.G_swz = dtype == VQC_C64 ? 4 : 3;
    Builder b(p);
    for (int32_t g = 0; g < G; ++g) b.add_gate(gates[g]);
    for (int q = 0; q < n; ++q) b.flush(q);
    if (p.entries.size() > 0xfff0 || p.accs.size() > 0xfff0) {
        err = "circuit too large for one plan (table entries exceed 65520)";
        return VQC_ERR_UNSUPPORTED;
    }
    // Table slots: per-sample entries and shared entries are numbered apart.
    for (auto& e : p.entries) e.slot = (uint16_t)(e.per_sample ? p.n_ps++ : p.n_sh++);
    // Terms of each x column / w index, in increasing term order.
    p.xocc_ptr.assign(nx + 1, 0);
    p.wocc_ptr.assign(nw + 1, 0);
    for (size_t t = 0; t < p.term_src.size(); ++t)
        (p.term_src[t] == SRC_X ? p.xocc_ptr : p.wocc_ptr)[p.term_idx[t] + 1]++;
    for (int i = 0; i < nx; ++i) p.xocc_ptr[i + 1] += p.xocc_ptr[i];
    for (int i = 0; i < nw; ++i) p.wocc_ptr[i + 1] += p.wocc_ptr[i];
    p.xocc.assign(p.xocc_ptr[nx], 0);
    p.wocc.assign(p.wocc_ptr[nw], 0);
    {
        std::vector<int32_t> fx(p.xocc_ptr.begin(), p.xocc_ptr.end() - 1);
        std::vector<int32_t> fw(p.wocc_ptr.begin(), p.wocc_ptr.end() - 1);
        for (size_t t = 0; t < p.term_src.size(); ++t) {
            if (p.term_src[t] == SRC_X) p.xocc[fx[p.term_idx[t]]++] = (int32_t)t;
            else p.wocc[fw[p.term_idx[t]]++] = (int32_t)t;
        }
    }
    for (const HOp& o : p.ops) p.has_ph2 = p.has_ph2 || o.type == OP_PH2;
    // Algorithmic flops per evaluation (counted on the fused op list).
    const double dim = std::ldexp(1.0, n);
    double f = 0, fb = 0;
    for (const HOp& o : p.ops) {
        bool acc = (o.type == OP_M1 || o.type == OP_PH2) && p.entries[o.entry].acc != 0xffff;
        if (o.type == OP_M1) { f += 14; fb += acc ? 44 : 28; }
        else if (o.type == OP_PH2) {
            double half = o.gen == OPF_GEN_CRZ ? 0.5 : 1.0;
            f += 6 * half;
            fb += (acc ? 16 : 12) * half;
        }
    }
    p.recompute_flops = f * dim;
    p.fwd_flops = (f + 3 + n) * dim;
    p.bwd_flops = (fb + n + 2) * dim;
    // Stage schedules for every usable (mode, K) on the resident path.
    for (int mode = 0; mode < 2; ++mode) {
        for (int K = 1; K <= std::min(max_k(mode, dtype), n); ++K) {
            // at most 512 register blocks per sample: one block per thread, which
            // the folded CX gates need (a thread holding two blocks would store
            // one before loading the other)
            if (n - K > 9) continue;
            if (n > resident_max_qubits(mode, dtype)) continue;
            Schedule s;
            s.mode = mode;
            s.K = K;
            s.path = VQC_PATH_RESIDENT;
            build_schedule(p, s);
            p.scheds.push_back(std::move(s));
        }
    }
    // Cluster schedules: states up to 16 qubits over 2..8 CTAs of a thread-block
    // cluster, one register block per thread (2^(n-K) threads) and at most 128
    // KiB of state per CTA (the backward holds psi and lam: two slices).  CTAs of
    // 512 threads (2^cta_bits): 256-thread CTAs, two clusters' CTAs per SM,
    // measured 12% slower on the 16-qubit forward (more cross-CTA stages, wider
    // cluster barriers).
    for (int mode = 0; mode < 2; ++mode) {
        const int K = max_k(mode, dtype);
        const size_t cs = dtype == VQC_C128 ? 16 : 8;
        const int ctb = 9, cl = n - K - ctb;
        if (n > resident_max_qubits(mode, dtype) && n <= 16 && cl >= 1 && cl <= 3 &&
            (((size_t)(mode + 1) << (n - cl)) * cs) <= 128 * 1024) {
            Schedule s;
            s.mode = mode;
            s.K = K;
            s.path = VQC_PATH_CLUSTER;
            s.cta_bits = ctb;
            build_schedule(p, s);
            // A map keeps every block in its thread's own CTA when no local offset
            // reaches the top cl slot bits (those index the CTA) and the top cl
            // thread bits (the thread's rank) map onto them identically.
            const int slice = n - cl;
            for (DStage& st : s.stages) {
                const int nb = st.nthreadbits;
                auto local = [&](const int32_t* sig, const int32_t* tau) {
                    for (int j = 0; j < K; ++j)
                        if ((uint32_t)sig[j] >> slice) return false;
                    for (int i = 0; i < nb; ++i) {
                        const uint32_t top = (uint32_t)tau[i] >> slice;
                        const uint32_t want = i >= nb - cl ? 1u << (i - (nb - cl)) : 0u;
                        if (top != want) return false;
                    }
                    return true;
                };
                st.cl_local = (uint8_t)((local(st.sigma, st.tau) ? 1 : 0) |
                                        (local(st.sigma_st, st.tau_st) ? 2 : 0));
            }
            p.scheds.push_back(std::move(s));
        }
    }
    // HBM-tiled pass schedules (tile of m qubits, K fixed per mode and type).
    for (int mode = 0; mode < 2; ++mode) {
        int m = std::min(hbm_tile_qubits(mode, dtype, p.G_swz), n - 1);
        int K = std::min(hbm_k(mode, dtype), m - 1);
        if (n < p.G_swz + 2 || K < 1 || m <= p.G_swz) continue;
        const int env_m = std::getenv("VQC_HBM_TILE_QUBITS") ? std::atoi(std::getenv("VQC_HBM_TILE_QUBITS")) : 0;
        if (env_m > p.G_swz && env_m < n) {
            m = std::min(std::max(env_m, hbm_k(mode, dtype) + 1), hbm_k(mode, dtype) + 8);
            K = std::min(hbm_k(mode, dtype), m - 1);
        }
        if (K != hbm_k(mode, dtype)) continue;   // pass kernels exist for this K only
        // the backward passes recompute the final state with the forward passes
        // when the caller gives none: no backward schedule without a forward one
        if (mode == 1 && !find_hbm_schedule(p, 0)) continue;
        Schedule s;
        s.mode = mode;
        s.K = K;
        s.m = m;
        s.path = VQC_PATH_HBM;
        build_hbm_schedule(p, s);
        p.scheds.push_back(std::move(s));
    }
    return VQC_OK;
}

const Schedule* find_schedule(const HostPlan& p, int mode, int K) {
    for (const auto& s : p.scheds)
        if (s.mode == mode && s.K == K && s.path == VQC_PATH_RESIDENT) return &s;
    return nullptr;
}

const Schedule* find_cluster_schedule(const HostPlan& p, int mode) {
    for (const auto& s : p.scheds)
        if (s.mode == mode && s.path == VQC_PATH_CLUSTER) return &s;
    return nullptr;
}

const Schedule* find_hbm_schedule(const HostPlan& p, int mode) {
    for (const auto& s : p.scheds)
        if (s.mode == mode && s.path == VQC_PATH_HBM) return &s;
    return nullptr;
}

std::vector<uint8_t> export_plan(const HostPlan& p) {
    std::vector<uint8_t> out = {'V', 'Q', 'C', 'P'};
    put_i32(out, 3);   // export format version
    for (int v : {p.n, p.num_x, p.num_w, p.dtype, p.num_gates_in, p.G_swz, p.n_ps, p.n_sh,
                  p.n_runs})
        put_i32(out, v);
    std::vector<int32_t> hops;
    for (const HOp& o : p.ops) {
        hops.push_back(o.type);
        hops.push_back(o.q0);
        hops.push_back(o.q1);
        hops.push_back(o.entry);
        hops.push_back(o.gen);
    }
    put_vec(out, hops);
    put_vec(out, p.entries);
    put_vec(out, p.consts);
    put_vec(out, p.cmat);
    put_vec(out, p.cang);
    put_vec(out, p.term_src);
    put_vec(out, p.term_idx);
    put_vec(out, p.accs);
    put_vec(out, p.xocc_ptr);
    put_vec(out, p.xocc);
    put_vec(out, p.wocc_ptr);
    put_vec(out, p.wocc);
    put_i32(out, (int32_t)p.scheds.size());
    for (const auto& s : p.scheds) {
        for (int v : {s.mode, s.K, s.m, s.path, s.thread_bits, s.group_lanes_log2, s.cta_bits})
            put_i32(out, v);
        put_vec(out, s.ops);
        put_vec(out, s.stages);
        put_vec(out, s.passes);
        put_vec(out, s.pass_entries);
        put_vec(out, s.pass_accs);
        put_vec(out, s.store_masks);
    }
    return out;
}

}  // namespace vqc
