// Stack-bytecode front end (paper section 7, the second client): a linear
// instruction stream with an explicit operand stack, run once on the host.  Stack
// entries are structural records whose numeric payloads are tape nodes; counted
// loops are realized by re-walking their body, so the tape is the unrolled trace.
//
// Instruction set (one per line, ';' starts a comment):
//   PUSH c      push the numeric constant c        PARAM k   push parameter k
//   OBS k       push observation k                 OBSN      push obs[cursor++]
//   LOAD r      push register r (0..15)            STORE r   pop into register r
//   DUP SWAP POP
//   ADD SUB MUL DIV  (pop b, pop a, push a op b)
//   NEG EXP LOG SIN COS TANH SQRT ABS   POW (pop e, pop a, push a^e)   POWI n
//   LT GT LE GE (pop b, pop a, push the per-lane predicate a op b)
//   SEL         pop b, pop a, pop p: push p ? a : b (lane mask)
//   LOOP n ... END   counted loop (n >= 0), nestable
//   DOT n       pop n values b, pop n values a: push sum_i a_i b_i
// The program's result is the single value left on the stack.
#include <cstdlib>
#include <cstring>
#include <string>
#include <vector>

#include "status.h"
#include "tape.h"

namespace ndvm {
namespace {

enum BOp {
  BC_PUSH, BC_PARAM, BC_OBS, BC_OBSN, BC_LOAD, BC_STORE, BC_DUP, BC_SWAP, BC_POP, BC_ADD, BC_SUB, BC_MUL,
  BC_DIV, BC_NEG, BC_EXP, BC_LOG, BC_SIN, BC_COS, BC_TANH, BC_SQRT, BC_ABS, BC_POW, BC_POWI, BC_LT, BC_GT,
  BC_LE, BC_GE, BC_SEL, BC_LOOP, BC_END, BC_DOT, BC_COUNT
};
const char* kNames[BC_COUNT] = {"PUSH", "PARAM", "OBS", "OBSN", "LOAD", "STORE", "DUP", "SWAP", "POP", "ADD",
                                "SUB", "MUL", "DIV", "NEG", "EXP", "LOG", "SIN", "COS", "TANH", "SQRT", "ABS",
                                "POW", "POWI", "LT", "GT", "LE", "GE", "SEL", "LOOP", "END", "DOT"};

struct Ins {
  int op;
  double f = 0;
  int64_t i = 0;
  int match = -1;  // LOOP <-> END
};

// structural record on the operand stack: a tape node that is a number or a predicate
struct Slot {
  int pid;
  bool pred;
};

[[noreturn]] void perr(int line, const std::string& m) {
  throw BuildError{NDVM_E_PARSE, "line " + std::to_string(line) + ": " + m};
}

std::vector<Ins> assemble(const char* s, size_t n, int& max_param) {
  std::vector<Ins> code;
  std::vector<int> loops;
  size_t i = 0;
  int line = 0;
  max_param = -1;
  while (i < n) {
    line++;
    size_t st = i;
    while (i < n && s[i] != '\n') i++;
    std::string ln(s + st, i - st);
    if (i < n) i++;
    size_t semi = ln.find(';');
    if (semi != std::string::npos) ln.resize(semi);
    // split into tokens
    std::vector<std::string> tok;
    size_t k = 0;
    while (k < ln.size()) {
      while (k < ln.size() && (ln[k] == ' ' || ln[k] == '\t' || ln[k] == '\r')) k++;
      size_t b = k;
      while (k < ln.size() && ln[k] != ' ' && ln[k] != '\t' && ln[k] != '\r') k++;
      if (k > b) tok.push_back(ln.substr(b, k - b));
    }
    if (tok.empty()) continue;
    int op = -1;
    for (int c = 0; c < BC_COUNT; c++) if (tok[0] == kNames[c]) op = c;
    if (op < 0) perr(line, "unknown instruction '" + tok[0] + "'");
    bool needs = op == BC_PUSH || op == BC_PARAM || op == BC_OBS || op == BC_LOAD || op == BC_STORE ||
                 op == BC_POWI || op == BC_LOOP || op == BC_DOT;
    if (needs && tok.size() != 2) perr(line, tok[0] + " needs one operand");
    if (!needs && tok.size() != 1) perr(line, tok[0] + " takes no operand");
    Ins in;
    in.op = op;
    if (needs) {
      char* end = nullptr;
      if (op == BC_PUSH) in.f = std::strtod(tok[1].c_str(), &end);  // correctly rounded
      else in.i = std::strtoll(tok[1].c_str(), &end, 10);
      if (!end || *end || tok[1].empty()) perr(line, "bad operand '" + tok[1] + "'");
    }
    if (op == BC_PARAM && in.i > max_param) max_param = (int)std::min<int64_t>(in.i, 1 << 20);
    if (op == BC_LOOP) loops.push_back((int)code.size());
    if (op == BC_END) {
      if (loops.empty()) perr(line, "END without LOOP");
      in.match = loops.back();
      code[loops.back()].match = (int)code.size();
      loops.pop_back();
    }
    code.push_back(in);
  }
  if (!loops.empty()) throw BuildError{NDVM_E_PARSE, "LOOP without END"};
  return code;
}

}  // namespace

int trace_bytecode(const char* text, size_t len, Builder& B, std::string& err) {
  int max_param = -1;
  std::vector<Ins> code = assemble(text, len, max_param);
  B.t.n_params = max_param + 1;
  std::vector<Slot> st;
  Slot regs[16];
  bool set[16] = {false};
  int64_t cursor = 0;
  std::vector<std::pair<int, int64_t>> loops;  // (pc of LOOP, iterations left)
  auto pop = [&](const char* what) {
    if (st.empty()) throw BuildError{NDVM_E_PARSE, std::string("stack underflow at ") + what};
    Slot s = st.back();
    st.pop_back();
    return s;
  };
  auto popn = [&](const char* what) {
    Slot s = pop(what);
    if (s.pred) throw BuildError{NDVM_E_UNSUPPORTED, std::string(what) + ": a predicate is not a number"};
    return s.pid;
  };
  for (int pc = 0; pc < (int)code.size(); pc++) {
    const Ins& in = code[pc];
    switch (in.op) {
      case BC_PUSH: st.push_back({B.konst(in.f), false}); break;
      case BC_PARAM:
        if (in.i < 0) throw BuildError{NDVM_E_PARSE, "PARAM index must be >= 0"};
        st.push_back({B.param((int)in.i), false});
        break;
      case BC_OBS: st.push_back({B.obs(in.i, 1), false}); break;
      case BC_OBSN: st.push_back({B.obs(cursor++, 1), false}); break;
      case BC_LOAD:
        if (in.i < 0 || in.i > 15 || !set[in.i]) throw BuildError{NDVM_E_PARSE, "LOAD of an unset register"};
        st.push_back(regs[in.i]);
        break;
      case BC_STORE:
        if (in.i < 0 || in.i > 15) throw BuildError{NDVM_E_PARSE, "STORE register outside 0..15"};
        regs[in.i] = pop("STORE");
        set[in.i] = true;
        break;
      case BC_DUP: { Slot s = pop("DUP"); st.push_back(s); st.push_back(s); break; }
      case BC_SWAP: { Slot b = pop("SWAP"), a = pop("SWAP"); st.push_back(b); st.push_back(a); break; }
      case BC_POP: pop("POP"); break;
      case BC_ADD: case BC_SUB: case BC_MUL: case BC_DIV: case BC_POW: {
        int b = popn(kNames[in.op]), a = popn(kNames[in.op]);
        Op op = in.op == BC_ADD ? OP_ADD : in.op == BC_SUB ? OP_SUB : in.op == BC_MUL ? OP_MUL
              : in.op == BC_DIV ? OP_DIV : OP_POW;
        st.push_back({B.binary(op, a, b), false});
        break;
      }
      case BC_NEG: case BC_EXP: case BC_LOG: case BC_SIN: case BC_COS: case BC_TANH: case BC_SQRT: case BC_ABS: {
        int a = popn(kNames[in.op]);
        Op op = in.op == BC_NEG ? OP_NEG : in.op == BC_EXP ? OP_EXP : in.op == BC_LOG ? OP_LOG
              : in.op == BC_SIN ? OP_SIN : in.op == BC_COS ? OP_COS : in.op == BC_TANH ? OP_TANH
              : in.op == BC_SQRT ? OP_SQRT : OP_ABS;
        st.push_back({B.unary(op, a), false});
        break;
      }
      case BC_POWI: {
        int a = popn("POWI");
        if (in.i < 0 || in.i > 64) throw BuildError{NDVM_E_UNSUPPORTED, "POWI exponent outside 0..64"};
        st.push_back({B.powi(a, (int)in.i), false});
        break;
      }
      case BC_LT: case BC_GT: case BC_LE: case BC_GE: {
        int b = popn(kNames[in.op]), a = popn(kNames[in.op]);
        Op op = in.op == BC_LT ? OP_LT : in.op == BC_GT ? OP_GT : in.op == BC_LE ? OP_LE : OP_GE;
        st.push_back({B.compare(op, a, b), true});
        break;
      }
      case BC_SEL: {
        int b = popn("SEL"), a = popn("SEL");
        Slot p = pop("SEL");
        if (!p.pred) throw BuildError{NDVM_E_UNSUPPORTED, "SEL needs a predicate under its two values"};
        st.push_back({B.select(p.pid, a, b), false});
        break;
      }
      case BC_LOOP:
        if (in.i < 0) throw BuildError{NDVM_E_PARSE, "LOOP count must be >= 0"};
        if (in.i == 0) pc = in.match;  // skip the body
        else loops.push_back({pc, in.i});
        break;
      case BC_END:
        if (--loops.back().second > 0) pc = loops.back().first;
        else loops.pop_back();
        break;
      case BC_DOT: {
        if (in.i < 1 || in.i > 4096) throw BuildError{NDVM_E_UNSUPPORTED, "DOT length outside 1..4096"};
        int n = (int)in.i;
        std::vector<int> a(n), b(n);
        for (int k = n - 1; k >= 0; k--) b[k] = popn("DOT");
        for (int k = n - 1; k >= 0; k--) a[k] = popn("DOT");
        int s = B.binary(OP_MUL, a[0], b[0]);
        for (int k = 1; k < n; k++) s = B.binary(OP_ADD, s, B.binary(OP_MUL, a[k], b[k]));
        st.push_back({s, false});
        break;
      }
    }
  }
  if (st.size() != 1) throw BuildError{NDVM_E_PARSE, "the program must leave exactly one value on the stack"};
  if (st[0].pred) throw BuildError{NDVM_E_UNSUPPORTED, "the result must be a number"};
  B.t.loss = st[0].pid;
  (void)err;
  return NDVM_OK;
}

}  // namespace ndvm
