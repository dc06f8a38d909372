// qasm.cpp -- OpenQASM 2 front end: lowers a normalised program over the
// engine's gate set onto the vqc_gate list that vqc_compile takes.
//
// The paper's input is a static circuit given as normalised OpenQASM (Sec. 3
// "Static Circuit Scope": fixed gate sequence, no measurement-dependent control,
// only the angles vary; Fig. 2: the circuit source is parsed once and lowered).
// This front end accepts OPENQASM 2.0 with qreg/creg declarations, the gates of
// the engine's set under their qelib1 names, the single-qubit phase forms that
// are exact special cases of U3 (u1, p, u2, sdg, tdg, id), `barrier` and
// terminal `measure` (both ignored: the engine returns expectations; a gate or
// barrier on a qubit after its measurement is rejected, since a mid-circuit
// measurement is outside the static-circuit scope), and one extension
// for variational circuits: an angle may be a per-sample parameter `x[i]` or a
// shared weight `w[j]` instead of a constant expression.  Constant expressions
// use numbers, pi, + - * / ^, unary minus, parentheses and sin cos tan exp ln
// sqrt.  Everything else (gate definitions, opaque, if, reset, scaled
// parameters) is rejected with a message naming the line.
#include <algorithm>
#include <cctype>
#include <cmath>
#include <cstring>
#include <map>
#include <stdexcept>
#include <string>
#include <vector>

#include "vqc.h"

namespace vqc {
vqc_status set_error(vqc_status s, const std::string& msg);
}

namespace {

struct QasmError : std::runtime_error {
    vqc_status code;
    QasmError(vqc_status c, const std::string& m) : std::runtime_error(m), code(c) {}
};

struct Tok {
    enum Kind { ID, NUM, STR, SYM, END } kind;
    std::string text;
    double num = 0;
    int line = 0;
};

std::vector<Tok> tokenize(const char* src) {
    std::vector<Tok> out;
    int line = 1;
    const char* p = src;
    while (*p) {
        const char c = *p;
        if (c == '\n') { ++line; ++p; continue; }
        if (std::isspace((unsigned char)c)) { ++p; continue; }
        if (c == '/' && p[1] == '/') {   // comment to end of line
            while (*p && *p != '\n') ++p;
            continue;
        }
        Tok t;
        t.line = line;
        if (std::isalpha((unsigned char)c) || c == '_') {
            const char* b = p;
            while (std::isalnum((unsigned char)*p) || *p == '_') ++p;
            t.kind = Tok::ID;
            t.text.assign(b, p);
        } else if (std::isdigit((unsigned char)c) || (c == '.' && std::isdigit((unsigned char)p[1]))) {
            char* e = nullptr;
            t.num = std::strtod(p, &e);
            t.kind = Tok::NUM;
            t.text.assign(p, (const char*)e);
            p = e;
        } else if (c == '"') {
            const char* b = ++p;
            while (*p && *p != '"' && *p != '\n') ++p;
            if (*p != '"') throw QasmError(VQC_ERR_INVALID_ARG, "line " + std::to_string(line) + ": unterminated string");
            t.kind = Tok::STR;
            t.text.assign(b, p);
            ++p;
        } else if (c == '-' && p[1] == '>') {
            t.kind = Tok::SYM;
            t.text = "->";
            p += 2;
        } else if (std::strchr("()[]{},;+-*/^=", c)) {
            t.kind = Tok::SYM;
            t.text = std::string(1, c);
            ++p;
        } else {
            throw QasmError(VQC_ERR_INVALID_ARG, "line " + std::to_string(line) + ": unexpected character '" +
                                                     std::string(1, c) + "'");
        }
        out.push_back(t);
    }
    Tok e;
    e.kind = Tok::END;
    e.line = line;
    out.push_back(e);
    return out;
}

// An angle: a constant, or a reference to x[i] / w[j].
struct Angle {
    uint8_t kind = VQC_P_CONST;
    int32_t idx = 0;
    double value = 0;
};

struct Parser {
    std::vector<Tok> t;
    size_t i = 0;
    std::map<std::string, int> qbase, qsize;
    std::map<std::string, int> cregs;
    int nq = 0;
    std::vector<char> measured;   // per qubit: a measure statement has named it
    std::vector<vqc_gate> gates;
    int32_t max_x = -1, max_w = -1;

    int stmt_line = 0;   // line of the statement being parsed (for its errors)
    [[noreturn]] void err(const std::string& m, vqc_status c = VQC_ERR_INVALID_ARG) {
        throw QasmError(c, "line " + std::to_string(stmt_line ? stmt_line : t[i].line) + ": " + m);
    }
    bool is_sym(const char* s) const { return t[i].kind == Tok::SYM && t[i].text == s; }
    void expect_sym(const char* s) {
        if (!is_sym(s)) err(std::string("expected '") + s + "'");
        ++i;
    }
    std::string expect_id() {
        if (t[i].kind != Tok::ID) err("expected an identifier");
        return t[i++].text;
    }
    int expect_int() {
        if (t[i].kind != Tok::NUM) err("expected an integer");
        const double v = t[i].num;
        if (v != std::floor(v) || v < 0 || v > 1e9) err("expected a non-negative integer");
        ++i;
        return (int)v;
    }

    // constant expressions (recursive descent; ^ binds tighter than unary minus)
    double primary() {
        if (is_sym("(")) {
            ++i;
            const double v = expr();
            expect_sym(")");
            return v;
        }
        if (t[i].kind == Tok::NUM) return t[i++].num;
        if (t[i].kind == Tok::ID) {
            const std::string id = t[i++].text;
            if (id == "pi") return 3.14159265358979323846;
            static const std::map<std::string, double (*)(double)> fn = {
                {"sin", std::sin}, {"cos", std::cos}, {"tan", std::tan},
                {"exp", std::exp}, {"ln", std::log}, {"sqrt", std::sqrt}};
            auto f = fn.find(id);
            if (f != fn.end()) {
                expect_sym("(");
                const double v = expr();
                expect_sym(")");
                return f->second(v);
            }
            if (id == "x" || id == "w")
                err("a parameter reference must be the whole angle (no arithmetic on x[i] / w[j])");
            err("unknown identifier '" + id + "' in an angle");
        }
        err("expected an angle expression");
    }
    double power() {
        const double b = primary();
        if (is_sym("^")) {
            ++i;
            return std::pow(b, unary());
        }
        return b;
    }
    double unary() {
        if (is_sym("-")) { ++i; return -unary(); }
        if (is_sym("+")) { ++i; return unary(); }
        return power();
    }
    double term() {
        double v = unary();
        while (is_sym("*") || is_sym("/")) {
            const bool mul = is_sym("*");
            ++i;
            const double r = unary();
            v = mul ? v * r : v / r;
        }
        return v;
    }
    double expr() {
        double v = term();
        while (is_sym("+") || is_sym("-")) {
            const bool add = is_sym("+");
            ++i;
            const double r = term();
            v = add ? v + r : v - r;
        }
        return v;
    }
    Angle angle() {
        Angle a;
        if (t[i].kind == Tok::ID && (t[i].text == "x" || t[i].text == "w") &&
            t[i + 1].kind == Tok::SYM && t[i + 1].text == "[") {
            const bool isx = t[i].text == "x";
            i += 2;
            a.kind = isx ? VQC_P_X : VQC_P_W;
            a.idx = expect_int();
            expect_sym("]");
            if (!(is_sym(",") || is_sym(")")))
                err("a parameter reference must be the whole angle (no arithmetic on x[i] / w[j])");
            if (isx) max_x = std::max(max_x, a.idx);
            else max_w = std::max(max_w, a.idx);
            return a;
        }
        a.value = expr();
        if (!std::isfinite(a.value)) err("angle is not finite");
        return a;
    }

    // a qubit operand: reg[i] (one qubit) or reg (the whole register)
    std::vector<int> operand() {
        const std::string r = expect_id();
        auto b = qbase.find(r);
        if (b == qbase.end()) err("unknown quantum register '" + r + "'", VQC_ERR_QUBIT_RANGE);
        if (is_sym("[")) {
            ++i;
            const int k = expect_int();
            expect_sym("]");
            if (k >= qsize[r]) err("qubit " + r + "[" + std::to_string(k) + "] out of range", VQC_ERR_QUBIT_RANGE);
            return {b->second + k};
        }
        std::vector<int> all;
        for (int k = 0; k < qsize[r]; ++k) all.push_back(b->second + k);
        return all;
    }
    // Only terminal measurements: nothing may act on a qubit after its measure.
    void not_measured(const std::vector<int>& qs, const std::string& what) {
        for (int q : qs)
            if (measured[q])
                err(what + " on qubit " + std::to_string(q) +
                    " after its measurement (only terminal measurements are in the static-circuit scope)",
                    VQC_ERR_UNSUPPORTED_GATE);
    }
    void skip_classical_operand() {
        const std::string r = expect_id();
        if (!cregs.count(r)) err("unknown classical register '" + r + "'");
        if (is_sym("[")) { ++i; expect_int(); expect_sym("]"); }
    }

    void emit(uint8_t op, int q0, int q1, const std::vector<Angle>& a) {
        vqc_gate g;
        std::memset(&g, 0, sizeof g);
        g.op = op;
        g.q0 = (uint8_t)q0;
        g.q1 = (uint8_t)(q1 < 0 ? 0 : q1);
        for (size_t k = 0; k < a.size() && k < 3; ++k) {
            g.pkind[k] = a[k].kind;
            g.pidx[k] = a[k].kind == VQC_P_CONST ? 0 : a[k].idx;
            g.pconst[k] = a[k].kind == VQC_P_CONST ? a[k].value : 0.0;
        }
        gates.push_back(g);
    }
    static Angle cst(double v) { Angle a; a.value = v; return a; }

    void gate_statement(const std::string& name) {
        std::vector<Angle> args;
        if (is_sym("(")) {
            ++i;
            if (!is_sym(")")) {
                args.push_back(angle());
                while (is_sym(",")) { ++i; args.push_back(angle()); }
            }
            expect_sym(")");
        }
        std::vector<std::vector<int>> ops;
        ops.push_back(operand());
        while (is_sym(",")) { ++i; ops.push_back(operand()); }
        expect_sym(";");

        struct G { uint8_t op; int nq, na; };
        static const std::map<std::string, G> table = {
            {"h", {VQC_H, 1, 0}}, {"x", {VQC_X, 1, 0}}, {"y", {VQC_Y, 1, 0}}, {"z", {VQC_Z, 1, 0}},
            {"s", {VQC_S, 1, 0}}, {"t", {VQC_T, 1, 0}}, {"sx", {VQC_SX, 1, 0}},
            {"rx", {VQC_RX, 1, 1}}, {"ry", {VQC_RY, 1, 1}}, {"rz", {VQC_RZ, 1, 1}},
            {"u3", {VQC_U3, 1, 3}}, {"u", {VQC_U3, 1, 3}}, {"U", {VQC_U3, 1, 3}},
            {"cx", {VQC_CX, 2, 0}}, {"CX", {VQC_CX, 2, 0}}, {"cz", {VQC_CZ, 2, 0}},
            {"swap", {VQC_SWAP, 2, 0}}, {"crz", {VQC_CRZ, 2, 1}}, {"rzz", {VQC_RZZ, 2, 1}},
            // exact special cases of U3(theta, phi, lambda)
            {"u1", {VQC_U3, 1, -1}}, {"p", {VQC_U3, 1, -1}}, {"u2", {VQC_U3, 1, -2}},
            {"sdg", {VQC_U3, 1, -3}}, {"tdg", {VQC_U3, 1, -4}}, {"id", {0, 1, -5}}};
        auto it = table.find(name);
        if (it == table.end())
            err("gate '" + name + "' is not in the engine's gate set", VQC_ERR_UNSUPPORTED_GATE);
        const G g = it->second;
        const int want_args = g.na >= 0 ? g.na : g.na == -1 ? 1 : g.na == -2 ? 2 : 0;
        if ((int)args.size() != want_args)
            err("gate '" + name + "' takes " + std::to_string(want_args) + " angle(s)");
        if ((int)ops.size() != g.nq)
            err("gate '" + name + "' takes " + std::to_string(g.nq) + " qubit operand(s)");
        // expand register broadcasts
        size_t width = 1;
        for (auto& o : ops) {
            if (o.size() > 1) {
                if (width > 1 && o.size() != width) err("registers of different sizes in one gate");
                width = o.size();
            }
        }
        for (size_t k = 0; k < width; ++k) {
            const int q0 = ops[0].size() > 1 ? ops[0][k] : ops[0][0];
            const int q1 = g.nq == 2 ? (ops[1].size() > 1 ? ops[1][k] : ops[1][0]) : -1;
            if (g.nq == 2 && q0 == q1) err("a two-qubit gate needs two different qubits", VQC_ERR_QUBIT_RANGE);
            not_measured(g.nq == 2 ? std::vector<int>{q0, q1} : std::vector<int>{q0}, "gate '" + name + "'");
            const double pi = 3.14159265358979323846;
            switch (g.na) {
            case -1: emit(VQC_U3, q0, -1, {cst(0), cst(0), args[0]}); break;          // u1 / p
            case -2: emit(VQC_U3, q0, -1, {cst(pi / 2), args[0], args[1]}); break;    // u2
            case -3: emit(VQC_U3, q0, -1, {cst(0), cst(0), cst(-pi / 2)}); break;     // sdg
            case -4: emit(VQC_U3, q0, -1, {cst(0), cst(0), cst(-pi / 4)}); break;     // tdg
            case -5: break;                                                           // id
            default: emit(g.op, q0, q1, args); break;
            }
        }
    }

    void program() {
        if (!(t[i].kind == Tok::ID && t[i].text == "OPENQASM")) err("the program must start with 'OPENQASM 2.0;'");
        ++i;
        if (t[i].kind != Tok::NUM || t[i].num < 2.0 || t[i].num >= 3.0) err("only OpenQASM 2 is supported");
        ++i;
        expect_sym(";");
        while (t[i].kind != Tok::END) {
            stmt_line = t[i].line;
            if (t[i].kind != Tok::ID) err("expected a statement");
            const std::string kw = t[i++].text;
            if (kw == "include") {
                if (t[i].kind != Tok::STR) err("expected a file name");
                if (t[i].text != "qelib1.inc") err("only \"qelib1.inc\" can be included");
                ++i;
                expect_sym(";");
            } else if (kw == "qreg" || kw == "creg") {
                const std::string r = expect_id();
                expect_sym("[");
                const int n = expect_int();
                expect_sym("]");
                expect_sym(";");
                if (qbase.count(r) || cregs.count(r)) err("register '" + r + "' declared twice");
                if (kw == "qreg") {
                    if (n < 1) err("empty quantum register");
                    qbase[r] = nq;
                    qsize[r] = n;
                    nq += n;
                    measured.resize(nq > 0 ? nq : 0, 0);
                    if (nq > VQC_MAX_QUBITS) err("more than " + std::to_string(VQC_MAX_QUBITS) + " qubits",
                                                 VQC_ERR_TOO_MANY_QUBITS);
                } else {
                    cregs[r] = n;
                }
            } else if (kw == "barrier") {
                not_measured(operand(), "barrier");
                while (is_sym(",")) { ++i; not_measured(operand(), "barrier"); }
                expect_sym(";");
            } else if (kw == "measure") {   // expectations are returned instead
                for (int q : operand()) measured[q] = 1;
                expect_sym("->");
                skip_classical_operand();
                expect_sym(";");
            } else if (kw == "gate" || kw == "opaque" || kw == "if" || kw == "reset") {
                --i;
                err("'" + kw + "' is outside the static-circuit subset (normalise the program first)",
                    VQC_ERR_UNSUPPORTED_GATE);
            } else {
                gate_statement(kw);
            }
        }
        if (nq == 0) err("no quantum register declared", VQC_ERR_TOO_MANY_QUBITS);
    }
};

}  // namespace

extern "C" {

vqc_status vqc_parse_qasm(const char* source, vqc_gate* gates, int32_t* inout_num_gates,
                          int32_t* num_qubits, int32_t* num_x, int32_t* num_w) {
    try {
        if (!source || !inout_num_gates || !num_qubits || !num_x || !num_w)
            return vqc::set_error(VQC_ERR_INVALID_ARG, "NULL argument to vqc_parse_qasm");
        Parser P;
        P.t = tokenize(source);
        P.program();
        const int32_t ng = (int32_t)P.gates.size();
        const int32_t cap = *inout_num_gates;
        *inout_num_gates = ng;
        *num_qubits = P.nq;
        *num_x = P.max_x + 1;
        *num_w = P.max_w + 1;
        if (!gates) return VQC_OK;
        if (cap < ng)
            return vqc::set_error(VQC_ERR_INVALID_ARG, "gate buffer holds " + std::to_string(cap) +
                                                           " gates, the program has " + std::to_string(ng));
        if (ng) std::memcpy(gates, P.gates.data(), sizeof(vqc_gate) * (size_t)ng);
        return VQC_OK;
    } catch (const QasmError& e) {
        return vqc::set_error(e.code, std::string("qasm: ") + e.what());
    } catch (...) {
        return vqc::set_error(VQC_ERR_INVALID_ARG, "qasm: internal error");
    }
}

vqc_status vqc_compile_qasm(const char* source, int32_t num_x, int32_t num_w, vqc_dtype dtype,
                            vqc_plan** out_plan) {
    try {
        int32_t ng = 0, nq = 0, nx = 0, nw = 0;
        vqc_status st = vqc_parse_qasm(source, nullptr, &ng, &nq, &nx, &nw);
        if (st != VQC_OK) return st;
        std::vector<vqc_gate> g((size_t)ng);
        st = vqc_parse_qasm(source, g.data(), &ng, &nq, &nx, &nw);
        if (st != VQC_OK) return st;
        if (num_x >= 0) {
            if (num_x < nx) return vqc::set_error(VQC_ERR_PARAM_RANGE, "qasm: the program uses x[" +
                                                                           std::to_string(nx - 1) + "]");
            nx = num_x;
        }
        if (num_w >= 0) {
            if (num_w < nw) return vqc::set_error(VQC_ERR_PARAM_RANGE, "qasm: the program uses w[" +
                                                                           std::to_string(nw - 1) + "]");
            nw = num_w;
        }
        return vqc_compile(g.data(), ng, nq, nx, nw, dtype, out_plan);
    } catch (...) {
        return vqc::set_error(VQC_ERR_INVALID_ARG, "qasm: internal error");
    }
}

}  // extern "C"
