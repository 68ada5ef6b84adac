// Scheme-style front end: a tree-walking evaluator over the program as heap data
// that records the realized numeric trace.
//
// Runtime values follow section 3.1, Definition 1: a fixed-size record
// <tag, aux, pid>.  Structural values (integers, booleans, pairs, closures,
// primitives, symbols) live entirely in <tag, aux>; a numeric value's pid names
// its tape node.  Pairs live in a write-once arena (section 3.2), symbols are
// interned, environments are frames of (symbol, value) slots.  Control is the
// exact realized trace (section 3.3): `if` on a structural test takes one branch
// at trace time; `if` on a per-lane numeric test traces both branches and merges
// them with a lane mask (select), whose adjoint reaches only the taken side.
// Named let and closure calls in tail position run in a loop (proper tail calls).
#include <cmath>
#include <cstdlib>
#include <cstring>
#include <string>
#include <unordered_map>
#include <vector>

#include "status.h"
#include "tape.h"

namespace ndvm {
namespace {

enum Tag : uint8_t { T_NIL, T_BOOL, T_INT, T_FLT, T_NUM, T_PRED, T_PAIR, T_CLOS, T_PRIM, T_SYM };

struct Value {
  Tag tag = T_NIL;
  int64_t aux = 0;   // immediate: integer, boolean, symbol id, heap index, closure id, primitive id
  int32_t pid = -1;  // tape node of a numeric value (T_NUM, T_PRED)
};

enum Prim {
  PR_ADD, PR_SUB, PR_MUL, PR_DIV, PR_EXP, PR_LOG, PR_SIN, PR_COS, PR_TANH, PR_SQRT, PR_ABS, PR_POW,
  PR_EXPT, PR_LT, PR_LE, PR_GT, PR_GE, PR_EQ, PR_NOT, PR_QUOT, PR_REM, PR_PARAM, PR_OBS, PR_DOBS,
  PR_OBSVEC, PR_CONS, PR_CAR, PR_CDR, PR_LIST, PR_NULLP, PR_PAIRP, PR_LENGTH, PR_LISTREF, PR_MATRIX,
  PR_MREF, PR_MADD, PR_MSUB, PR_MSCALE, PR_MATMUL, PR_TRANSPOSE, PR_INV, PR_DET, PR_LOGDET, PR_TRACE,
  PR_IDENTITY, PR_ZEROS, PR_SUBMAT, PR_ROWS, PR_COLS, PR_EXACT, PR_DOT, PR_COUNT
};
const char* kPrimNames[PR_COUNT] = {
    "+", "-", "*", "/", "exp", "log", "sin", "cos", "tanh", "sqrt", "abs", "pow", "expt", "<", "<=", ">", ">=",
    "=", "not", "quotient", "remainder", "param", "obs", "dobs", "obs-vec", "cons", "car", "cdr", "list",
    "null?", "pair?", "length", "list-ref", "matrix", "mref", "m+", "m-", "mscale", "matmul", "transpose",
    "inv", "det", "logdet", "trace", "identity", "zeros", "submatrix", "rows", "cols", "exact->inexact", "dot"};

[[noreturn]] void parse_error(const std::string& m) { throw BuildError{NDVM_E_PARSE, m}; }
[[noreturn]] void unsupported(const std::string& m) { throw BuildError{NDVM_E_UNSUPPORTED, m}; }

struct Frame {
  int parent;
  std::vector<std::pair<int, Value>> slots;
};

struct Closure {
  std::vector<int> params;
  Value body;  // list of expressions
  int env;
};

class Tracer {
 public:
  Tracer(Builder& b) : B(b) {}

  void load(const char* s, size_t n) {
    src_ = s; n_ = n; i_ = 0;
    std::vector<Value> forms;
    for (;;) {
      skip();
      if (i_ >= n_) break;
      forms.push_back(read());
    }
    program_ = list_of(forms);
  }

  void run();

 private:
  Builder& B;
  const char* src_ = nullptr;
  size_t n_ = 0, i_ = 0;
  Value program_;

  std::vector<std::string> symnames_;
  std::unordered_map<std::string, int> symids_;
  std::vector<std::pair<Value, Value>> heap_;  // write-once pair arena
  std::vector<double> flits_;                  // float literals of the program text
  std::vector<Frame> frames_;
  std::vector<Closure> closures_;
  int globals_ = -1;
  int depth_ = 0;
  // interned special-form symbols
  int s_quote_, s_if_, s_let_, s_letstar_, s_lambda_, s_begin_, s_define_, s_and_, s_or_, s_datasum_,
      s_model_, s_params_;

  // ---------------- reader ----------------
  int intern(const std::string& s) {
    auto it = symids_.find(s);
    if (it != symids_.end()) return it->second;
    int id = (int)symnames_.size();
    symnames_.push_back(s);
    symids_[s] = id;
    return id;
  }
  Value cons(Value a, Value d) {
    heap_.push_back({a, d});
    Value v;
    v.tag = T_PAIR; v.aux = (int64_t)heap_.size() - 1;
    return v;
  }
  Value list_of(const std::vector<Value>& xs) {
    Value r;
    for (size_t k = xs.size(); k-- > 0;) r = cons(xs[k], r);
    return r;
  }
  Value car(Value p) const { return heap_[p.aux].first; }
  Value cdr(Value p) const { return heap_[p.aux].second; }
  void skip() {
    while (i_ < n_) {
      char c = src_[i_];
      if (c == ';') { while (i_ < n_ && src_[i_] != '\n') i_++; }
      else if (c == ' ' || c == '\t' || c == '\n' || c == '\r') i_++;
      else break;
    }
  }
  Value read() {
    skip();
    if (i_ >= n_) parse_error("unexpected end of program text");
    char c = src_[i_];
    if (c == ')') parse_error("unexpected ')' at offset " + std::to_string(i_));
    if (c == '(') {
      i_++;
      std::vector<Value> xs;
      for (;;) {
        skip();
        if (i_ >= n_) parse_error("missing ')'");
        if (src_[i_] == ')') { i_++; break; }
        xs.push_back(read());
      }
      return list_of(xs);
    }
    size_t st = i_;
    while (i_ < n_) {
      char d = src_[i_];
      if (d == '(' || d == ')' || d == ' ' || d == '\t' || d == '\n' || d == '\r' || d == ';') break;
      i_++;
    }
    std::string tok(src_ + st, i_ - st);
    Value v;
    if (tok == "#t" || tok == "#f") { v.tag = T_BOOL; v.aux = tok == "#t"; return v; }
    // integers: optional sign and digits only (structural)
    size_t k = (tok[0] == '+' || tok[0] == '-') ? 1 : 0;
    bool digits = k < tok.size();
    for (size_t j = k; j < tok.size(); j++) if (tok[j] < '0' || tok[j] > '9') { digits = false; break; }
    if (digits) {
      if (tok.size() > 18) parse_error("integer literal too long");
      v.tag = T_INT; v.aux = std::strtoll(tok.c_str(), nullptr, 10);
      return v;
    }
    char c0 = tok[0];
    bool numeric_start = (c0 >= '0' && c0 <= '9') || c0 == '.' ||
                         ((c0 == '-' || c0 == '+') && tok.size() > 1 && ((tok[1] >= '0' && tok[1] <= '9') || tok[1] == '.'));
    if (numeric_start) {
      char* end = nullptr;
      double d = std::strtod(tok.c_str(), &end);  // correctly rounded
      if (end == tok.c_str() + tok.size()) {
        flits_.push_back(d);
        v.tag = T_FLT; v.aux = (int64_t)flits_.size() - 1;
        return v;
      }
    }
    v.tag = T_SYM; v.aux = intern(tok);
    return v;
  }

  // ---------------- helpers ----------------
  static Value mkint(int64_t i) { Value v; v.tag = T_INT; v.aux = i; return v; }
  static Value mkbool(bool b) { Value v; v.tag = T_BOOL; v.aux = b; return v; }
  static Value mknum(int pid) { Value v; v.tag = T_NUM; v.pid = pid; return v; }
  static Value mkpred(int pid) { Value v; v.tag = T_PRED; v.pid = pid; return v; }
  int list_len(Value x) const { int n = 0; while (x.tag == T_PAIR) { n++; x = cdr(x); } return n; }
  Value nth(Value x, int i) const { while (i-- > 0) x = cdr(x); return car(x); }
  bool is_sym(Value x, int s) const { return x.tag == T_SYM && x.aux == s; }
  const std::string& name(int s) const { return symnames_[s]; }

  int num(Value v) {  // promote to a tape node
    if (v.tag == T_NUM) return v.pid;
    if (v.tag == T_INT) return B.konst((double)v.aux);
    parse_error("number expected");
  }
  int64_t integer(Value v, const char* what) {
    if (v.tag != T_INT) parse_error(std::string(what) + ": structural integer expected");
    return v.aux;
  }
  int new_frame(int parent) { frames_.push_back(Frame{parent, {}}); return (int)frames_.size() - 1; }
  Value lookup(int env, int sym) {
    for (int f = env; f >= 0; f = frames_[f].parent) {
      const auto& s = frames_[f].slots;
      for (size_t k = s.size(); k-- > 0;) if (s[k].first == sym) return s[k].second;
    }
    parse_error("unbound variable '" + name(sym) + "'");
  }
  void define(int env, int sym, Value v) {
    auto& s = frames_[env].slots;
    for (auto& p : s) if (p.first == sym) { p.second = v; return; }
    s.push_back({sym, v});
  }
  Value closure(Value params, Value body, int env) {
    Closure c;
    for (Value p = params; p.tag == T_PAIR; p = cdr(p)) {
      if (car(p).tag != T_SYM) parse_error("lambda parameter must be a symbol");
      c.params.push_back((int)car(p).aux);
    }
    c.body = body; c.env = env;
    closures_.push_back(c);
    Value v;
    v.tag = T_CLOS; v.aux = (int64_t)closures_.size() - 1;
    return v;
  }

  Value apply_prim(int p, std::vector<Value>& av);
  Value eval(Value x, int env);
  Value eval_branch(Value x, int env);
};

Value Tracer::apply_prim(int p, std::vector<Value>& av) {
  int argc = (int)av.size();
  auto need = [&](int k) {
    if (argc != k) parse_error(std::string(kPrimNames[p]) + " expects " + std::to_string(k) + " argument(s)");
  };
  switch (p) {
    case PR_ADD: case PR_SUB: case PR_MUL: case PR_DIV: {
      if (argc < 1) parse_error(std::string(kPrimNames[p]) + " needs at least one argument");
      bool allint = true;
      for (auto& v : av) {
        if (v.tag != T_INT && v.tag != T_NUM) parse_error(std::string(kPrimNames[p]) + ": number expected");
        if (v.tag != T_INT) allint = false;
      }
      if (allint && p != PR_DIV) {  // structural integer arithmetic: no tape node
        int64_t r = av[0].aux;
        if (p == PR_SUB && argc == 1) return mkint(-r);
        for (int k = 1; k < argc; k++) r = p == PR_ADD ? r + av[k].aux : p == PR_SUB ? r - av[k].aux : r * av[k].aux;
        return mkint(r);
      }
      std::vector<int> x(argc);
      for (int k = 0; k < argc; k++) x[k] = num(av[k]);
      if (p == PR_SUB && argc == 1) return mknum(B.unary(OP_NEG, x[0]));
      if (p == PR_DIV && argc == 1) return mknum(B.binary(OP_DIV, B.konst(1.0), x[0]));
      if (p == PR_ADD || p == PR_MUL) {
        Op op = p == PR_ADD ? OP_ADD : OP_MUL;
        int z = x[0];  // (+ x) and (* x) are x
        for (int k = 1; k < argc; k++) z = B.binary(op, z, x[k]);
        return mknum(z);
      }
      // z = x0 - (x1 + ... + xn), z = x0 / (x1 * ... * xn)  (Appendix C, n-ary sub/div)
      Op fold = p == PR_SUB ? OP_ADD : OP_MUL;
      int s = x[1];
      for (int k = 2; k < argc; k++) s = B.binary(fold, s, x[k]);
      return mknum(B.binary(p == PR_SUB ? OP_SUB : OP_DIV, x[0], s));
    }
    case PR_EXP: case PR_LOG: case PR_SIN: case PR_COS: case PR_TANH: case PR_SQRT: case PR_ABS: {
      need(1);
      Op op = p == PR_EXP ? OP_EXP : p == PR_LOG ? OP_LOG : p == PR_SIN ? OP_SIN : p == PR_COS ? OP_COS
            : p == PR_TANH ? OP_TANH : p == PR_SQRT ? OP_SQRT : OP_ABS;
      return mknum(B.unary(op, num(av[0])));
    }
    case PR_POW: case PR_EXPT:
      need(2);
      if (av[1].tag == T_INT) return mknum(B.powi(num(av[0]), (int)std::max<int64_t>(-1, std::min<int64_t>(av[1].aux, 65))));
      return mknum(B.binary(OP_POW, num(av[0]), num(av[1])));
    case PR_LT: case PR_LE: case PR_GT: case PR_GE: case PR_EQ: {
      need(2);
      if (av[0].tag == T_INT && av[1].tag == T_INT) {
        int64_t a = av[0].aux, b = av[1].aux;
        bool r = p == PR_LT ? a < b : p == PR_LE ? a <= b : p == PR_GT ? a > b : p == PR_GE ? a >= b : a == b;
        return mkbool(r);
      }
      Op op = p == PR_LT ? OP_LT : p == PR_LE ? OP_LE : p == PR_GT ? OP_GT : p == PR_GE ? OP_GE : OP_EQ;
      return mkpred(B.compare(op, num(av[0]), num(av[1])));
    }
    case PR_NOT:
      need(1);
      if (av[0].tag != T_BOOL) unsupported("not: structural boolean expected");
      return mkbool(!av[0].aux);
    case PR_QUOT: case PR_REM: {
      need(2);
      int64_t a = integer(av[0], kPrimNames[p]), b = integer(av[1], kPrimNames[p]);
      if (b == 0) parse_error(std::string(kPrimNames[p]) + " by zero");
      return mkint(p == PR_QUOT ? a / b : a % b);
    }
    case PR_PARAM: {
      need(1);
      int64_t k = integer(av[0], "param");
      if (k < 0 || k >= B.t.n_params) parse_error("param index out of range");
      return mknum(B.param((int)k));
    }
    case PR_OBS: need(1); return mknum(B.obs(integer(av[0], "obs"), 1));
    case PR_DOBS: need(1); return mknum(B.dobs((int)std::min<int64_t>(integer(av[0], "dobs"), 1 << 30)));
    case PR_OBSVEC: {
      need(2);
      int64_t k = integer(av[0], "obs-vec"), n = integer(av[1], "obs-vec");
      if (n < 1 || n > kMaxDim) unsupported("obs-vec length outside 1..64");
      return mknum(B.obs(k, (int)n));
    }
    case PR_CONS: need(2); return cons(av[0], av[1]);
    case PR_CAR: need(1); if (av[0].tag != T_PAIR) parse_error("car of a non-pair"); return car(av[0]);
    case PR_CDR: need(1); if (av[0].tag != T_PAIR) parse_error("cdr of a non-pair"); return cdr(av[0]);
    case PR_LIST: return list_of(av);
    case PR_NULLP: need(1); return mkbool(av[0].tag == T_NIL);
    case PR_PAIRP: need(1); return mkbool(av[0].tag == T_PAIR);
    case PR_LENGTH: need(1); return mkint(list_len(av[0]));
    case PR_LISTREF: {
      need(2);
      int64_t k = integer(av[1], "list-ref");
      if (k < 0 || k >= list_len(av[0])) parse_error("list-ref index out of range");
      return nth(av[0], (int)k);
    }
    case PR_MATRIX: {
      if (argc < 2) parse_error("matrix needs rows and cols");
      int64_t r = integer(av[0], "matrix"), c = integer(av[1], "matrix");
      if (r < 1 || c < 1 || r > kMaxDim || c > kMaxDim) throw BuildError{NDVM_E_SHAPE, "matrix shape outside 1..64"};
      if (argc != 2 + r * c) throw BuildError{NDVM_E_SHAPE, "matrix element count mismatch"};
      std::vector<int> el(r * c);
      for (int k = 0; k < r * c; k++) el[k] = num(av[2 + k]);
      return mknum(B.matfrom((int)r, (int)c, el));
    }
    case PR_MREF: need(3); return mknum(B.mref(num(av[0]), (int)integer(av[1], "mref"), (int)integer(av[2], "mref")));
    case PR_MADD: need(2); return mknum(B.madd(OP_MADD, num(av[0]), num(av[1])));
    case PR_MSUB: need(2); return mknum(B.madd(OP_MSUB, num(av[0]), num(av[1])));
    case PR_MSCALE: need(2); return mknum(B.mscale(num(av[0]), num(av[1])));
    case PR_MATMUL: need(2); return mknum(B.matmul(num(av[0]), num(av[1])));
    case PR_TRANSPOSE: need(1); return mknum(B.transpose(num(av[0])));
    case PR_INV: need(1); return mknum(B.matfun(OP_INV, num(av[0])));
    case PR_DET: need(1); return mknum(B.matfun(OP_DET, num(av[0])));
    case PR_LOGDET: need(1); return mknum(B.matfun(OP_LOGDET, num(av[0])));
    case PR_TRACE: need(1); return mknum(B.matfun(OP_TRACE, num(av[0])));
    case PR_IDENTITY: case PR_ZEROS: {
      int64_t r, c;
      if (p == PR_IDENTITY) { need(1); r = c = integer(av[0], "identity"); }
      else { need(2); r = integer(av[0], "zeros"); c = integer(av[1], "zeros"); }
      if (r < 1 || c < 1 || r > kMaxDim || c > kMaxDim) throw BuildError{NDVM_E_SHAPE, "matrix shape outside 1..64"};
      std::vector<double> v(r * c, 0.0);
      if (p == PR_IDENTITY) for (int k = 0; k < r; k++) v[k * c + k] = 1.0;
      return mknum(B.konst_matrix((int)r, (int)c, v.data()));
    }
    case PR_SUBMAT:
      need(5);
      return mknum(B.submat(num(av[0]), (int)integer(av[1], "submatrix"), (int)integer(av[2], "submatrix"),
                            (int)integer(av[3], "submatrix"), (int)integer(av[4], "submatrix")));
    case PR_ROWS: need(1); return mkint(B.rows(num(av[0])));
    case PR_COLS: need(1); return mkint(B.cols(num(av[0])));
    case PR_EXACT: need(1); return mknum(B.konst((double)integer(av[0], "exact->inexact")));
    case PR_DOT: {
      need(2);
      int a = num(av[0]), b = num(av[1]);
      if (B.cols(a) != 1 || B.cols(b) != 1 || B.rows(a) != B.rows(b))
        throw BuildError{NDVM_E_SHAPE, "dot needs two column vectors of equal length"};
      return mknum(B.mref(B.matmul(B.transpose(a), b), 0, 0));
    }
  }
  parse_error("unknown primitive");
}

// A branch of a per-lane numeric test: traced in full (not in tail position).
Value Tracer::eval_branch(Value x, int env) {
  Value r = eval(x, env);
  if (r.tag == T_INT) r = mknum(B.konst((double)r.aux));
  if (r.tag != T_NUM) unsupported("a branch on a numeric test must produce a number");
  return r;
}

Value Tracer::eval(Value x, int env) {
  if (++depth_ > 4000) unsupported("evaluation nested too deeply (a per-lane test may guard an unbounded recursion)");
  struct Guard { int& d; ~Guard() { d--; } } guard{depth_};
  for (;;) {
    switch (x.tag) {
      case T_SYM: return lookup(env, (int)x.aux);
      case T_INT: case T_BOOL: return x;
      case T_FLT: return mknum(B.konst(flits_[x.aux]));
      case T_PAIR: break;
      default: parse_error("cannot evaluate this form");
    }
    Value head = car(x), rest = cdr(x);
    if (head.tag == T_SYM) {
      int h = (int)head.aux;
      if (h == s_quote_) return car(rest);
      if (h == s_if_) {
        if (list_len(rest) != 3) parse_error("if needs a test, a consequent and an alternative");
        Value c = eval(nth(rest, 0), env);
        if (c.tag == T_BOOL) { x = nth(rest, c.aux ? 1 : 2); continue; }
        if (c.tag != T_PRED) parse_error("if: test must be a boolean");
        // per-lane divergence: both sides, merged by lane mask
        Value a = eval_branch(nth(rest, 1), env);
        Value b = eval_branch(nth(rest, 2), env);
        return mknum(B.select(c.pid, a.pid, b.pid));
      }
      if (h == s_and_ || h == s_or_) {
        bool isand = h == s_and_;
        Value r = mkbool(isand);
        for (Value e = rest; e.tag == T_PAIR; e = cdr(e)) {
          r = eval(car(e), env);
          if (r.tag != T_BOOL) unsupported(std::string(isand ? "and" : "or") + ": structural boolean expected");
          if (isand ? !r.aux : r.aux) break;
        }
        return r;
      }
      if (h == s_begin_) {
        if (rest.tag != T_PAIR) parse_error("empty begin");
        while (cdr(rest).tag == T_PAIR) { eval(car(rest), env); rest = cdr(rest); }
        x = car(rest);
        continue;
      }
      if (h == s_lambda_) return closure(car(rest), cdr(rest), env);
      if (h == s_let_ || h == s_letstar_) {
        Value b0 = car(rest);
        Value body;
        int f;
        if (h == s_let_ && b0.tag == T_SYM) {
          // named let: bind the loop procedure, then call it
          Value binds = nth(rest, 1);
          body = cdr(cdr(rest));
          int lf = new_frame(env);
          std::vector<Value> ps;
          for (Value e = binds; e.tag == T_PAIR; e = cdr(e)) ps.push_back(car(car(e)));
          Value clo = closure(list_of(ps), body, lf);
          define(lf, (int)b0.aux, clo);
          f = new_frame(lf);
          for (Value e = binds; e.tag == T_PAIR; e = cdr(e)) {
            Value bi = car(e);
            if (bi.tag != T_PAIR || list_len(bi) != 2 || car(bi).tag != T_SYM) parse_error("bad named-let binding");
            Value v = eval(nth(bi, 1), env);
            frames_[f].slots.push_back({(int)car(bi).aux, v});
          }
        } else {
          body = cdr(rest);
          if (h == s_letstar_) {
            f = env;
            for (Value e = b0; e.tag == T_PAIR; e = cdr(e)) {
              Value bi = car(e);
              if (bi.tag != T_PAIR || list_len(bi) != 2 || car(bi).tag != T_SYM) parse_error("bad let* binding");
              Value v = eval(nth(bi, 1), f);
              int nf = new_frame(f);
              frames_[nf].slots.push_back({(int)car(bi).aux, v});
              f = nf;
            }
          } else {
            std::vector<std::pair<int, Value>> vals;
            for (Value e = b0; e.tag == T_PAIR; e = cdr(e)) {
              Value bi = car(e);
              if (bi.tag != T_PAIR || list_len(bi) != 2 || car(bi).tag != T_SYM) parse_error("bad let binding");
              vals.push_back({(int)car(bi).aux, eval(nth(bi, 1), env)});
            }
            f = new_frame(env);
            frames_[f].slots = vals;
          }
        }
        if (body.tag != T_PAIR) parse_error("empty let body");
        while (cdr(body).tag == T_PAIR) { eval(car(body), f); body = cdr(body); }
        x = car(body);
        env = f;
        continue;
      }
      if (h == s_datasum_) {
        int n = list_len(rest);
        if (n != 3 && n != 4) parse_error("data-sum needs N S [BASE] body");
        int64_t N = integer(eval(nth(rest, 0), env), "data-sum N");
        int64_t S = integer(eval(nth(rest, 1), env), "data-sum S");
        int64_t base = n == 4 ? integer(eval(nth(rest, 2), env), "data-sum BASE") : 0;
        if (N < 0 || S < 0 || base < 0) parse_error("data-sum N, S and BASE must be >= 0");
        B.begin_region();
        Value r = eval(nth(rest, n - 1), env);
        if (r.tag == T_INT) r = mknum(B.konst((double)r.aux));
        if (r.tag != T_NUM) parse_error("data-sum body must produce a number");
        return mknum(B.end_region(r.pid, N, S, base));
      }
      if (h == s_define_ || h == s_model_) parse_error(name(h) + " is only allowed at top level");
    }
    // application
    Value f = eval(head, env);
    std::vector<Value> av;
    for (Value e = rest; e.tag == T_PAIR; e = cdr(e)) av.push_back(eval(car(e), env));
    if (f.tag == T_PRIM) return apply_prim((int)f.aux, av);
    if (f.tag != T_CLOS) parse_error("application of a non-procedure");
    const Closure& c = closures_[f.aux];
    if (c.params.size() != av.size())
      parse_error("procedure expects " + std::to_string(c.params.size()) + " argument(s), got " + std::to_string(av.size()));
    int nf = new_frame(c.env);
    for (size_t k = 0; k < av.size(); k++) frames_[nf].slots.push_back({c.params[k], av[k]});
    Value body = c.body;
    if (body.tag != T_PAIR) parse_error("empty procedure body");
    while (cdr(body).tag == T_PAIR) { eval(car(body), nf); body = cdr(body); }
    x = car(body);
    env = nf;  // proper tail call
  }
}

void Tracer::run() {
  s_quote_ = intern("quote"); s_if_ = intern("if"); s_let_ = intern("let"); s_letstar_ = intern("let*");
  s_lambda_ = intern("lambda"); s_begin_ = intern("begin"); s_define_ = intern("define"); s_and_ = intern("and");
  s_or_ = intern("or"); s_datasum_ = intern("data-sum"); s_model_ = intern("model"); s_params_ = intern("params");
  globals_ = new_frame(-1);
  for (int p = 0; p < PR_COUNT; p++) {
    Value v;
    v.tag = T_PRIM; v.aux = p;
    define(globals_, intern(kPrimNames[p]), v);
  }
  // first pass: the model form fixes the parameter count before anything is traced
  int nmodel = 0;
  for (Value fs = program_; fs.tag == T_PAIR; fs = cdr(fs)) {
    Value f = car(fs);
    if (f.tag == T_PAIR && is_sym(car(f), s_model_)) {
      nmodel++;
      Value ps = nth(f, 1);
      if (ps.tag != T_PAIR || !is_sym(car(ps), s_params_)) parse_error("model needs (params name...)");
      B.t.n_params = list_len(ps) - 1;
    }
  }
  if (nmodel != 1) parse_error(nmodel == 0 ? "no model form" : "more than one model form");
  for (Value fs = program_; fs.tag == T_PAIR; fs = cdr(fs)) {
    Value f = car(fs);
    if (f.tag == T_PAIR && is_sym(car(f), s_define_)) {
      Value t = nth(f, 1);
      if (t.tag == T_SYM) define(globals_, (int)t.aux, eval(nth(f, 2), globals_));
      else if (t.tag == T_PAIR && car(t).tag == T_SYM) define(globals_, (int)car(t).aux, closure(cdr(t), cdr(cdr(f)), globals_));
      else parse_error("bad define");
      continue;
    }
    if (f.tag == T_PAIR && is_sym(car(f), s_model_)) {
      Value ps = nth(f, 1);
      int fr = new_frame(globals_);
      int k = 0;
      for (Value e = cdr(ps); e.tag == T_PAIR; e = cdr(e), k++) {
        if (car(e).tag != T_SYM) parse_error("parameter name must be a symbol");
        frames_[fr].slots.push_back({(int)car(e).aux, mknum(B.param(k))});
      }
      Value body = cdr(cdr(f));
      if (body.tag != T_PAIR) parse_error("empty model body");
      while (cdr(body).tag == T_PAIR) { eval(car(body), fr); body = cdr(body); }
      Value r = eval(car(body), fr);
      if (r.tag == T_INT) r = mknum(B.konst((double)r.aux));
      if (r.tag != T_NUM) parse_error("the model must produce a number");
      if (!B.is_scalar(r.pid)) throw BuildError{NDVM_E_SHAPE, "the model must produce a scalar"};
      B.t.loss = r.pid;
      continue;
    }
    eval(f, globals_);
  }
}

}  // namespace

int trace_scheme(const char* text, size_t len, Builder& b, std::string& err) {
  Tracer t(b);
  t.load(text, len);
  t.run();
  (void)err;
  return NDVM_OK;
}

}  // namespace ndvm
