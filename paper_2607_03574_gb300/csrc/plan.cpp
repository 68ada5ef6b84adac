// Planner: lowers a Tape (SSA, section 3.4) to the device instruction stream.
//
// Forward sweep: one instruction per non-leaf node, in tape order.  A data-axis
// region (section 3.5) becomes a loop over the lane's data points whose body runs
// the region's forward instructions, then immediately its reverse instructions
// seeded with d(body)/d(body) = 1, accumulating the body value and the partial
// derivatives of the body with respect to its lane-level inputs.  Because the
// region's output is a sum, the adjoint of each region input is later
// g_sum * (sum over points of its partial) -- exact by linearity.
// Reverse sweep: one instruction per active node in reverse tape order, using
// the adjoint rules of Appendix C (and readings for tanh/neg/select/compare).
#include "plan.h"

#include <algorithm>
#include <climits>
#include <cstdlib>
#include <cstring>
#include <functional>
#include <map>
#include <set>

#include "cost.h"
#include "status.h"

namespace ndvm {
namespace {

[[noreturn]] void unsupported(const std::string& m) { throw BuildError{NDVM_E_UNSUPPORTED, m}; }

// NDVM_PREFETCH=0 disables the reverse sweep's workspace prefetch (a tuning knob).
bool prefetch_enabled() {
  const char* e = std::getenv("NDVM_PREFETCH");
  return !(e && e[0] == '0');
}

// NDVM_FETCHTRIM=0 keeps a fetch record, a commit and a wait in every window of the
// reverse sweep, also where nothing is fetched (a tuning knob).
bool fetch_trim_enabled() {
  const char* e = std::getenv("NDVM_FETCHTRIM");
  return !(e && e[0] == '0');
}

// NDVM_FETCH_STRIDE=n (1..64) sets the instructions per prefetch window of the reverse
// sweep (a tuning knob; default kFetchStride).
int fetch_stride() {
  const char* e = std::getenv("NDVM_FETCH_STRIDE");
  const int v = e ? std::atoi(e) : 0;
  return v >= 1 && v <= 64 ? v : kFetchStride;
}

// NDVM_DERIVE=0 computes the shared per-point values on every lane instead.
bool derive_enabled() {
  const char* e = std::getenv("NDVM_DERIVE");
  return !(e && e[0] == '0');
}

// NDVM_PAIR=0 keeps adjacent independent fused instructions in separate records.
bool pair_enabled() {
  const char* e = std::getenv("NDVM_PAIR");
  return !(e && e[0] == '0');
}

// NDVM_SAVEPAIR=0 leaves fused instructions that save their result unpaired (a tuning
// knob).
bool save_pair_enabled() {
  const char* e = std::getenv("NDVM_SAVEPAIR");
  return !(e && e[0] == '0');
}

// NDVM_DEPPAIR=0 pairs independent fused instructions only (a tuning knob).
bool dep_pair_enabled() {
  const char* e = std::getenv("NDVM_DEPPAIR");
  return !(e && e[0] == '0');
}

// Two adjacent D_FMA records become one D_FMA2: one dispatch for both (a save's
// workspace index travels in 24 bits of the record).
// Runs on the encoded stream (physical slots).  The kernel loads every operand of the
// pair before it stores either result, so a second destination that the first reads
// is safe.  When the second reads the first's result (a chain, e.g. two contributions
// accumulated into one adjoint), flags bit 2 tells the kernel to take that operand from
// the first's result in a register; the two stores then run in order, so a shared
// destination ends with the second's value.
std::vector<DInst> pair_fma(const std::vector<DInst>& code) {
  const int n = (int)code.size();
  const bool dep_ok = dep_pair_enabled();
  const bool save_pairs = save_pair_enabled();
  std::vector<DInst> out;
  out.reserve(n);
  std::vector<int> newpc(n, -1);
  for (int pc = 0; pc < n; pc++) {
    const DInst& a = code[pc];
    newpc[pc] = (int)out.size();
    auto save24 = [&](int32_t sv) { return sv == -1 || (sv >= 0 && sv < kNoSave24 && save_pairs); };
    if (pc + 1 < n && a.op == D_FMA && code[pc + 1].op == D_FMA && save24(a.f[5]) && save24(code[pc + 1].f[5])) {
      const DInst& b = code[pc + 1];
      const bool raw = b.f[1] == a.f[0] || b.f[2] == a.f[0] || b.f[3] == a.f[0] || b.f[4] == a.f[0];
      if (raw ? dep_ok : b.f[0] != a.f[0]) {
        DInst q;
        q.op = D_FMA2;
        const bool saves = a.f[5] != -1 || b.f[5] != -1;
        q.flags = (uint8_t)((a.flags & 1) | ((b.flags & 1) << 1) | (raw ? 4 : 0) | (saves ? 8 : 0));
        if (saves) {
          const uint32_t s1 = a.f[5] == -1 ? (uint32_t)kNoSave24 : (uint32_t)a.f[5];
          const uint32_t s2 = b.f[5] == -1 ? (uint32_t)kNoSave24 : (uint32_t)b.f[5];
          q.r = (uint8_t)s1; q.c = (uint8_t)(s1 >> 8); q.k = (uint8_t)(s1 >> 16);
          q.pad0 = (uint8_t)s2; q.pad1 = (uint8_t)(s2 >> 8); q.pad2 = (uint8_t)(s2 >> 16);
        }
        for (int k = 0; k < 5; k++) q.f[k] = a.f[k];
        q.f[5] = b.f[0]; q.f[6] = b.f[1]; q.f[7] = b.f[2]; q.pad3 = b.f[3]; q.pad4 = b.f[4];
        out.push_back(q);
        newpc[pc + 1] = newpc[pc];
        pc++;
        continue;
      }
    }
    out.push_back(a);
  }
  for (DInst& d : out) {
    if (d.op == D_LOOP) d.f[3] = newpc[d.f[3]];
    if (d.op == D_ENDLOOP) d.f[0] = newpc[d.f[0]];
  }
  return out;
}

// NDVM_HOIST=0 keeps the seed of a data-axis body's reverse sweep inside the loop (a
// tuning knob).
bool hoist_enabled() {
  const char* e = std::getenv("NDVM_HOIST");
  return !(e && e[0] == '0');
}

// NDVM_COALESCE=0 keeps every adjoint copy as its own instruction (a tuning knob).
bool coalesce_enabled() {
  const char* e = std::getenv("NDVM_COALESCE");
  return !(e && e[0] == '0');
}

// NDVM_MERGELOADS=0 keeps one record per observation load (a tuning knob).
bool merge_loads_enabled() {
  const char* e = std::getenv("NDVM_MERGELOADS");
  return !(e && e[0] == '0');
}

// Adjacent loads of the current point's observations (D_LOAD of a DOBS reference, which
// the planner places together at the start of a loop body) become D_FETCH records of up
// to kFetchPairs asynchronous copies from the observations (flags bit 5), each record
// committing its copies and waiting for all of them: one dispatch, the loads in flight
// together, and no registers held for the values.  Runs on the encoded stream and
// renumbers the loop links.
std::vector<DInst> merge_obs_loads(const std::vector<DInst>& code) {
  const int n = (int)code.size();
  auto obs_load = [&](int pc) { return pc < n && code[pc].op == D_LOAD && ref_kind(code[pc].f[1]) == RK_DOBS; };
  std::vector<DInst> out;
  out.reserve(n);
  std::vector<int> newpc(n, -1);
  for (int pc = 0; pc < n;) {
    if (!obs_load(pc)) {
      newpc[pc] = (int)out.size();
      out.push_back(code[pc++]);
      continue;
    }
    DInst q;
    q.op = D_FETCH;
    q.flags = 32 | 2 | 1;  // observation sources, commit, wait until none is pending
    int m = 0;
    newpc[pc] = (int)out.size();
    while (m < kFetchPairs && obs_load(pc)) {
      q.f[2 * m] = code[pc].f[1];
      q.f[2 * m + 1] = code[pc].f[0];
      newpc[pc] = (int)out.size();
      m++;
      pc++;
    }
    q.k = (uint8_t)m;
    out.push_back(q);
  }
  for (DInst& d : out) {
    if (d.op == D_LOOP) d.f[3] = newpc[d.f[3]];
    if (d.op == D_ENDLOOP) d.f[0] = newpc[d.f[0]];
  }
  return out;
}

// NDVM_FMA=0 keeps the general scalar instructions instead of the fused form (a tuning knob).
bool fma_enabled() {
  const char* e = std::getenv("NDVM_FMA");
  return !(e && e[0] == '0');
}

struct PRef {
  uint32_t kind = RK_SLOT;
  int32_t id = -1;  // VR id for slots; index otherwise
  int32_t off = 0;
};
struct PArg {
  bool isref = false;
  PRef r;
  int32_t v = -1;
};
inline PArg I(int32_t v) { PArg a; a.v = v; return a; }
inline PArg R(PRef r) { PArg a; a.isref = true; a.r = r; return a; }
inline PRef slotref(int vr, int off = 0) { PRef r; r.kind = RK_SLOT; r.id = vr; r.off = off; return r; }
inline PRef kref(uint32_t kind, int32_t idx) { PRef r; r.kind = kind; r.id = idx; return r; }

struct PInst {
  DInst d;
  PArg f[8];
};

struct VR {
  int width;
  int start = INT_MAX, end = -1, phys = -1;
};

class Planner {
 public:
  Planner(const Tape& t, bool grad, bool spill) : T(t), grad_(grad), spill_(spill) {}
  Plan build();

 private:
  const Tape& T;
  bool grad_, spill_;
  int N = 0;
  std::vector<uint8_t> active_, region_body_;
  std::vector<char> need_val_, need_aux_;
  std::vector<int> twin_inv_;  // DET/LOGDET node -> an INV node of the same matrix (or -1)
  // shared per-point values: pdep_ = depends on a parameter; derived_ = a region body
  // node computed by a derive plan instead; der_col_ = its column when the replay reads it
  std::vector<char> pdep_, derived_;
  std::vector<int> der_col_;
  std::vector<int> der_of_;       // DSUM node -> index of its derive plan (or -1)
  int emit_r_ = -1;               // DSUM node whose body is being emitted (forward or reverse)
  std::vector<DeriveInfo> der_info_;
  std::vector<int> der_region_;   // DSUM node of each derive plan
  int64_t der_elems_ = 0;
  void plan_derived();
  Plan build_derive(int r, const DeriveInfo& info) const;
  std::vector<int> val_vr_, aux_vr_, adj_vr_;
  std::vector<int64_t> save_, aux_save_;
  std::vector<VR> vrs_;
  std::vector<PInst> code_;
  std::vector<PArg> args_;
  int64_t S_ = 0;
  double work_fwd_ = 0, work_rev_ = 0, nops_ = 0;
  // data-axis regions
  int cur_region_ = -1;          // DSUM node whose body is being emitted
  std::vector<int> partial_of_;  // node -> offset of its partial in the block (current region)
  int block_vr_ = -1;            // current region: [sum, partials...]
  std::vector<int> body_adj_;    // node -> adjoint VR inside the current region body
  std::vector<std::vector<std::pair<int, int>>> region_inputs_;  // DSUM node -> (input, offset)
  std::vector<int> region_block_;                                // DSUM node -> block VR
  int one_const_ = -1;
  double mult_ = 1.0;  // executions per lane of the instruction being emitted
  std::vector<double> extra_consts_;
  int n_slots_ = 0;

  int width(int v) const { return T.nodes[v].rows * T.nodes[v].cols; }
  bool is_leaf(int v) const {
    uint16_t op = T.nodes[v].op;
    return op == OP_CONST || op == OP_PARAM || op == OP_OBS || op == OP_DOBS;
  }
  int new_vr(int w) { vrs_.push_back(VR{w}); return (int)vrs_.size() - 1; }
  int emit(const PInst& p) { code_.push_back(p); return (int)code_.size() - 1; }

  std::vector<int> inputs(int v) const;
  void analyze();
  PRef ref(int v);          // primal reference for forward use
  PRef rref(int v);         // primal reference for reverse use
  PRef rauxref(int v);
  PArg save_of(int v) { return I(spill_ && save_[v] >= 0 ? (int32_t)save_[v] : -1); }
  void emit_forward(int v);
  void emit_region(int v);
  // adjoint target of input x during reverse: returns (slot ref, first-contribution flag)
  std::pair<PRef, bool> target(int x);
  void emit_reverse(int v);
  void allocate();
  void prefetch_workspace();
  void normalize_operands();
  void hoist_seeds();
  void coalesce_copies();
  void lower_fma();
  int const_index(double v);
  int32_t encode(const PArg& a) const;
  int rev_begin_ = -1;  // first instruction of the reverse sweep
};

std::vector<int> Planner::inputs(int v) const {
  const Node& n = T.nodes[v];
  std::vector<int> r;
  switch (n.op) {
    case OP_CONST: case OP_PARAM: case OP_OBS: case OP_DOBS: break;
    case OP_MATFROM: for (int k = 0; k < n.rows * n.cols; k++) r.push_back(T.args[n.imm + k]); break;
    case OP_SELECT: r = {n.a, n.b, n.c}; break;
    case OP_DSUM: r = {n.c}; break;
    default:
      if (n.a >= 0) r.push_back(n.a);
      if (n.b >= 0) r.push_back(n.b);
      break;
  }
  return r;
}

void Planner::analyze() {
  N = (int)T.nodes.size();
  active_.assign(N, 0);
  region_body_.assign(N, 0);
  for (int v = 0; v < N; v++) {
    const Node& n = T.nodes[v];
    if (n.op == OP_DSUM) {
      // Only nodes that depend on the data point run per point; a node traced
      // inside the body but independent of the point is hoisted: it runs once per
      // lane, and its adjoint arrives through the region's partial sums.
      if (n.a < 0 || n.b > v || n.a > n.b) unsupported("malformed data-sum");
      for (int u = n.a; u < n.b; u++) {
        const Node& m = T.nodes[u];
        if (m.op == OP_DOBS) { region_body_[u] = 1; continue; }
        if (m.op == OP_CONST || m.op == OP_PARAM || m.op == OP_OBS) continue;
        for (int x : inputs(u))
          if (x >= n.a && x < u && region_body_[x]) { region_body_[u] = 1; break; }
      }
      if (n.c >= v) unsupported("malformed data-sum");
    }
  }
  for (int v = 0; v < N; v++) {
    const Node& n = T.nodes[v];
    switch (n.op) {
      case OP_PARAM: active_[v] = 1; break;
      case OP_CONST: case OP_OBS: case OP_DOBS: break;
      case OP_LT: case OP_LE: case OP_GT: case OP_GE: case OP_EQ: break;  // no gradient through a test
      case OP_SELECT: active_[v] = active_[n.b] || active_[n.c]; break;
      default:
        for (int x : inputs(v)) {
          if (x < 0 || x >= v) unsupported("tape is not in SSA order");
          if (active_[x]) active_[v] = 1;
        }
    }
    // body values must not escape their region (leaves are shared)
    if (!region_body_[v] || n.op == OP_DSUM) {
      for (int x : inputs(v))
        if (region_body_[x] && !is_leaf(x) && n.op != OP_DSUM) unsupported("a data-sum body value escapes its region");
    }
  }
  need_val_.assign(N, 0);
  need_aux_.assign(N, 0);
  twin_inv_.assign(N, -1);
  if (grad_) {
    for (int v = 0; v < N; v++) {
      if (!active_[v]) continue;
      const Node& n = T.nodes[v];
      auto need = [&](int x) { need_val_[x] = 1; };
      switch (n.op) {
        case OP_MUL: if (active_[n.a]) need(n.b); if (active_[n.b]) need(n.a); break;
        case OP_DIV:
          // the reverse rule reads b and, inside a data-axis body (where it stays in a slot
          // for the point's reverse sweep), the forward sweep's reciprocal of b; a lane-level
          // division divides again (a workspace round trip for the reciprocal measured no
          // faster on a serial chain)
          need(n.b); if (active_[n.b]) need(v);
          if (region_body_[v]) need_aux_[v] = 1;
          break;
        case OP_POW: need(n.a); need(n.b); need(v); break;
        case OP_EXP: case OP_TANH: case OP_INV: need(v); break;
        case OP_LOG: case OP_ABS: case OP_POWI: need(n.a); break;
        case OP_SQRT: need(n.a); need(v); break;
        case OP_SIN: case OP_COS: need_aux_[v] = 1; break;
        case OP_SELECT: need(n.a); break;
        case OP_MSCALE: if (active_[n.a]) need(n.b); if (active_[n.b]) need(n.a); break;
        case OP_MATMUL: if (active_[n.a]) need(n.b); if (active_[n.b]) need(n.a); break;
        case OP_DET: need(v); need_aux_[v] = 1; break;
        case OP_LOGDET: need_aux_[v] = 1; break;
        default: break;
      }
    }
    // a determinant whose matrix is also inverted by the program (a Kalman filter
    // takes both of its innovation covariance) reads that inverse in the reverse sweep
    // instead of computing its own: the forward sweep then finds the determinant only
    std::map<int, int> inv_of;
    for (int v = 0; v < N; v++)
      if (T.nodes[v].op == OP_INV && active_[v] && !region_body_[v]) inv_of.emplace(T.nodes[v].a, v);
    for (int v = 0; v < N; v++) {
      const Node& n = T.nodes[v];
      if ((n.op != OP_DET && n.op != OP_LOGDET) || !need_aux_[v] || region_body_[v]) continue;
      auto it = inv_of.find(n.a);
      if (it == inv_of.end()) continue;
      twin_inv_[v] = it->second;
      need_aux_[v] = 0;
      need_val_[it->second] = 1;
    }
  }
  val_vr_.assign(N, -1);
  aux_vr_.assign(N, -1);
  adj_vr_.assign(N, -1);
  save_.assign(N, -1);
  aux_save_.assign(N, -1);
  body_adj_.assign(N, -1);
  partial_of_.assign(N, -1);
  region_inputs_.assign(N, {});
  region_block_.assign(N, -1);
  for (int v = 0; v < N; v++) {
    if (is_leaf(v) || T.nodes[v].op == OP_DSUM) continue;
    val_vr_[v] = new_vr(width(v));
    bool lane_level = !region_body_[v];
    if (need_aux_[v]) {
      int aw = (T.nodes[v].op == OP_DET || T.nodes[v].op == OP_LOGDET) ? width(T.nodes[v].a) : 1;
      if (spill_ && lane_level) { aux_save_[v] = S_; S_ += aw; }
      else aux_vr_[v] = new_vr(aw);
    }
    if (spill_ && lane_level && need_val_[v]) { save_[v] = S_; S_ += width(v); }
  }
}

PRef Planner::ref(int v) {
  const Node& n = T.nodes[v];
  if (emit_r_ >= 0 && der_of_[emit_r_] >= 0) {
    // a region with shared per-point values reads its point's observations and derived
    // values from the region's block of the extended observations, column-major
    const DeriveInfo& di = der_info_[der_of_[emit_r_]];
    if (n.op == OP_DOBS) return kref(RK_DOBS, (int32_t)(n.imm * di.n_points));
    if (der_col_[v] >= 0) return kref(RK_DOBS, (int32_t)((di.obs_cols + der_col_[v]) * di.n_points));
  }
  switch (n.op) {
    case OP_CONST: return kref(RK_CONST, n.imm);
    case OP_PARAM: return kref(RK_PARAM, n.imm);
    case OP_OBS: return kref(RK_OBS, n.imm);
    case OP_DOBS: return kref(RK_DOBS, n.imm);
    case OP_DSUM: return slotref(val_vr_[v], 0);
    default: return slotref(val_vr_[v]);
  }
}

PRef Planner::rref(int v) {
  if (!is_leaf(v) && T.nodes[v].op != OP_DSUM && spill_ && !region_body_[v]) {
    if (save_[v] < 0) unsupported("internal: reverse reads an unsaved value");
    return kref(RK_SAVE, (int32_t)save_[v]);
  }
  return ref(v);
}

PRef Planner::rauxref(int v) {
  if (spill_ && !region_body_[v]) return kref(RK_SAVE, (int32_t)aux_save_[v]);
  return slotref(aux_vr_[v]);
}

void Planner::emit_forward(int v) {
  const Node& n = T.nodes[v];
  PInst p;
  p.d.r = n.rows; p.d.c = n.cols;
  PRef out = slotref(val_vr_[v]);
  p.f[0] = R(out);
  // (with_aux: the auxiliary output is kept; for a division, that it runs in a data-axis body)
  work_fwd_ += mult_ * cost::fwd(n.op, n.rows, n.cols, n.imm, T.nodes[n.a >= 0 ? n.a : v].rows,
                                 n.op == OP_DIV ? region_body_[v] != 0 : grad_ && need_aux_[v]);
  nops_ += mult_;
  switch (n.op) {
    case OP_ADD: case OP_SUB: case OP_MUL: case OP_DIV: case OP_POW:
      p.d.op = n.op == OP_ADD ? D_ADD : n.op == OP_SUB ? D_SUB : n.op == OP_MUL ? D_MUL : n.op == OP_DIV ? D_DIV : D_POW;
      p.f[1] = R(ref(n.a)); p.f[2] = R(ref(n.b)); p.f[3] = save_of(v);
      if (n.op == OP_DIV && region_body_[v]) {
        // through the correctly rounded reciprocal of b (flags bit 4), kept for the reverse rule
        p.d.flags |= 16;
        if (need_aux_[v]) {
          if (aux_vr_[v] >= 0) p.f[4] = R(slotref(aux_vr_[v]));
          else p.f[5] = I((int32_t)aux_save_[v]);
        }
      }
      break;
    case OP_NEG: case OP_EXP: case OP_LOG: case OP_TANH: case OP_SQRT: case OP_ABS:
      p.d.op = n.op == OP_NEG ? D_NEG : n.op == OP_EXP ? D_EXP : n.op == OP_LOG ? D_LOG : n.op == OP_TANH ? D_TANH
             : n.op == OP_SQRT ? D_SQRT : D_ABS;
      p.f[1] = R(ref(n.a)); p.f[3] = save_of(v);
      break;
    case OP_SIN: case OP_COS:
      p.d.op = n.op == OP_SIN ? D_SIN : D_COS;
      p.f[1] = R(ref(n.a)); p.f[3] = save_of(v);
      if (need_aux_[v]) {
        if (aux_vr_[v] >= 0) p.f[4] = R(slotref(aux_vr_[v]));
        else p.f[5] = I((int32_t)aux_save_[v]);
      }
      break;
    case OP_POWI:
      p.d.op = D_POWI; p.f[1] = R(ref(n.a)); p.f[3] = save_of(v); p.f[7] = I(n.imm);
      break;
    case OP_LT: case OP_LE: case OP_GT: case OP_GE: case OP_EQ:
      p.d.op = D_CMP;
      p.d.k = n.op == OP_LT ? 0 : n.op == OP_LE ? 1 : n.op == OP_GT ? 2 : n.op == OP_GE ? 3 : 4;
      p.f[1] = R(ref(n.a)); p.f[2] = R(ref(n.b)); p.f[3] = save_of(v);
      break;
    case OP_SELECT:
      p.d.op = D_SELECT; p.f[1] = R(ref(n.a)); p.f[2] = R(ref(n.b)); p.f[4] = R(ref(n.c)); p.f[3] = save_of(v);
      break;
    case OP_MATFROM: {
      p.d.op = D_GATHER;
      p.f[1] = I((int32_t)args_.size()); p.f[2] = I(n.rows * n.cols); p.f[3] = save_of(v);
      for (int k = 0; k < n.rows * n.cols; k++) args_.push_back(R(ref(T.args[n.imm + k])));
      break;
    }
    case OP_MREF: case OP_SUBMAT: case OP_TRANSPOSE: {
      // pure data movement: a gather of input elements
      p.d.op = D_GATHER;
      const Node& in = T.nodes[n.a];
      PRef base = ref(n.a);
      p.f[1] = I((int32_t)args_.size()); p.f[2] = I(n.rows * n.cols); p.f[3] = save_of(v);
      for (int i = 0; i < n.rows; i++)
        for (int j = 0; j < n.cols; j++) {
          int e;
          if (n.op == OP_MREF) e = n.imm;
          else if (n.op == OP_SUBMAT) e = (n.imm + i) * in.cols + n.imm2 + j;
          else e = j * in.cols + i;  // transpose: out(i,j) = in(j,i)
          PRef r = base; r.off += e;
          args_.push_back(R(r));
        }
      break;
    }
    case OP_MADD: case OP_MSUB:
      p.d.op = n.op == OP_MADD ? D_MADD : D_MSUB;
      p.f[1] = R(ref(n.a)); p.f[2] = R(ref(n.b)); p.f[3] = save_of(v);
      break;
    case OP_MSCALE:
      p.d.op = D_MSCALE; p.f[1] = R(ref(n.a)); p.f[2] = R(ref(n.b)); p.f[3] = save_of(v);
      break;
    case OP_MATMUL:
      p.d.op = D_MATMUL; p.d.k = (uint8_t)n.imm;
      p.f[1] = R(ref(n.a)); p.f[2] = R(ref(n.b)); p.f[3] = save_of(v);
      break;
    case OP_INV:
      p.d.op = D_INV; p.d.r = T.nodes[n.a].rows; p.f[1] = R(ref(n.a)); p.f[3] = save_of(v);
      break;
    case OP_DET: case OP_LOGDET:
      p.d.op = n.op == OP_DET ? D_DET : D_LOGDET; p.d.r = T.nodes[n.a].rows; p.d.c = 1;
      p.f[1] = R(ref(n.a)); p.f[3] = save_of(v);
      if (need_aux_[v]) {
        if (aux_vr_[v] >= 0) p.f[4] = R(slotref(aux_vr_[v]));
        else p.f[5] = I((int32_t)aux_save_[v]);
      }
      break;
    case OP_TRACE:
      p.d.op = D_TRACE; p.d.r = T.nodes[n.a].rows; p.d.c = 1; p.f[1] = R(ref(n.a));
      break;
    default:
      unsupported(std::string("no forward lowering for ") + op_name(n.op));
  }
  emit(p);
}

std::pair<PRef, bool> Planner::target(int x) {
  // inside a region body: body values get body adjoints, lane values get partial slots
  if (cur_region_ >= 0) {
    if (region_body_[x] && !is_leaf(x)) {
      if (body_adj_[x] < 0) { body_adj_[x] = new_vr(width(x)); return {slotref(body_adj_[x]), true}; }
      return {slotref(body_adj_[x]), false};
    }
    if (partial_of_[x] < 0) unsupported("internal: region input without a partial slot");
    return {slotref(block_vr_, partial_of_[x]), false};
  }
  if (adj_vr_[x] < 0) { adj_vr_[x] = new_vr(width(x)); return {slotref(adj_vr_[x]), true}; }
  return {slotref(adj_vr_[x]), false};
}

void Planner::emit_reverse(int v) {
  const Node& n = T.nodes[v];
  int gz_vr = cur_region_ >= 0 ? body_adj_[v] : adj_vr_[v];
  if (gz_vr < 0) return;  // no contribution reached this node: its adjoint is zero
  PInst p;
  p.d.r = n.rows; p.d.c = n.cols;
  p.f[0] = R(slotref(gz_vr));
  uint8_t flags = 0;
  auto tgt = [&](int x, int field, int bit) {
    if (!active_[x]) return;
    auto t = target(x);
    p.f[field] = R(t.first);
    if (t.second) flags |= (uint8_t)(1u << bit);
  };
  switch (n.op) {
    case OP_ADD: case OP_SUB:
      p.d.op = n.op == OP_ADD ? B_ADD : B_SUB; tgt(n.a, 1, 0); tgt(n.b, 2, 1);
      break;
    case OP_MUL:
      p.d.op = B_MUL; tgt(n.a, 1, 0); tgt(n.b, 2, 1);
      if (active_[n.a]) p.f[4] = R(rref(n.b));
      if (active_[n.b]) p.f[3] = R(rref(n.a));
      break;
    case OP_DIV:
      p.d.op = B_DIV; tgt(n.a, 1, 0); tgt(n.b, 2, 1);
      p.f[4] = R(rref(n.b));
      if (active_[n.b]) p.f[5] = R(rref(v));
      if (need_aux_[v]) p.f[6] = R(rauxref(v));
      break;
    case OP_POW:
      p.d.op = B_POW; tgt(n.a, 1, 0); tgt(n.b, 2, 1);
      p.f[3] = R(rref(n.a)); p.f[4] = R(rref(n.b)); p.f[5] = R(rref(v));
      break;
    case OP_NEG: p.d.op = B_NEG; tgt(n.a, 1, 0); break;
    case OP_EXP: case OP_TANH: p.d.op = n.op == OP_EXP ? B_EXP : B_TANH; tgt(n.a, 1, 0); p.f[5] = R(rref(v)); break;
    case OP_LOG: case OP_ABS: p.d.op = n.op == OP_LOG ? B_LOG : B_ABS; tgt(n.a, 1, 0); p.f[3] = R(rref(n.a)); break;
    case OP_SQRT: p.d.op = B_SQRT; tgt(n.a, 1, 0); p.f[3] = R(rref(n.a)); p.f[5] = R(rref(v)); break;
    case OP_SIN: case OP_COS: p.d.op = n.op == OP_SIN ? B_SIN : B_COS; tgt(n.a, 1, 0); p.f[6] = R(rauxref(v)); break;
    case OP_POWI: p.d.op = B_POWI; tgt(n.a, 1, 0); p.f[3] = R(rref(n.a)); p.f[7] = I(n.imm); break;
    case OP_SELECT:
      p.d.op = B_SELECT; tgt(n.b, 1, 0); tgt(n.c, 2, 1); p.f[3] = R(rref(n.a));
      break;
    case OP_MATFROM: {
      p.d.op = B_GATHER;
      int cnt = n.rows * n.cols;
      p.f[1] = I((int32_t)args_.size()); p.f[2] = I(cnt);
      for (int k = 0; k < cnt; k++) {
        int x = T.args[n.imm + k];
        if (!active_[x]) { args_.push_back(I(-1)); args_.push_back(I(0)); continue; }
        auto t = target(x);
        args_.push_back(R(t.first));
        args_.push_back(I(t.second ? 1 : 0));
      }
      break;
    }
    case OP_MREF: case OP_SUBMAT: case OP_TRANSPOSE: {
      p.d.op = B_SCATTER;
      const Node& in = T.nodes[n.a];
      tgt(n.a, 1, 0);
      p.f[2] = I(n.rows * n.cols); p.f[3] = I((int32_t)args_.size()); p.f[4] = I(in.rows * in.cols);
      for (int i = 0; i < n.rows; i++)
        for (int j = 0; j < n.cols; j++) {
          int e;
          if (n.op == OP_MREF) e = n.imm;
          else if (n.op == OP_SUBMAT) e = (n.imm + i) * in.cols + n.imm2 + j;
          else e = j * in.cols + i;
          args_.push_back(I(e));
        }
      break;
    }
    case OP_MADD: case OP_MSUB: p.d.op = n.op == OP_MADD ? B_MADD : B_MSUB; tgt(n.a, 1, 0); tgt(n.b, 2, 1); break;
    case OP_MSCALE:
      p.d.op = B_MSCALE; tgt(n.a, 1, 0); tgt(n.b, 2, 1);
      if (active_[n.a]) p.f[4] = R(rref(n.b));
      if (active_[n.b]) p.f[3] = R(rref(n.a));
      break;
    case OP_MATMUL:
      p.d.op = B_MATMUL; p.d.k = (uint8_t)n.imm; tgt(n.a, 1, 0); tgt(n.b, 2, 1);
      if (active_[n.a]) p.f[4] = R(rref(n.b));
      if (active_[n.b]) p.f[3] = R(rref(n.a));
      break;
    case OP_INV: p.d.op = B_INV; p.d.r = T.nodes[n.a].rows; tgt(n.a, 1, 0); p.f[5] = R(rref(v)); break;
    case OP_DET:
      p.d.op = B_DET; p.d.r = T.nodes[n.a].rows; p.d.c = 1; tgt(n.a, 1, 0);
      p.f[5] = R(rref(v)); p.f[6] = R(twin_inv_[v] >= 0 ? rref(twin_inv_[v]) : rauxref(v));
      break;
    case OP_LOGDET:
      p.d.op = B_LOGDET; p.d.r = T.nodes[n.a].rows; p.d.c = 1; tgt(n.a, 1, 0);
      p.f[6] = R(twin_inv_[v] >= 0 ? rref(twin_inv_[v]) : rauxref(v));
      break;
    case OP_TRACE: p.d.op = B_TRACE; p.d.r = T.nodes[n.a].rows; p.d.c = 1; tgt(n.a, 1, 0); break;
    case OP_DSUM: {
      p.d.op = B_DSUM;
      const auto& ins = region_inputs_[v];
      p.f[1] = I((int32_t)args_.size()); p.f[2] = I((int32_t)ins.size());
      for (auto& io : ins) {
        auto t = target(io.first);
        args_.push_back(R(t.first));
        args_.push_back(I(t.second ? 1 : 0));
        args_.push_back(R(slotref(region_block_[v], io.second)));
      }
      break;
    }
    default:
      return;  // leaves and comparisons carry no adjoint
  }
  p.d.flags = flags;
  {
    int in_rows = T.nodes[n.a >= 0 ? n.a : v].rows;
    bool aa = false, ba = false;
    if (n.op == OP_SELECT) { aa = active_[n.b]; ba = active_[n.c]; }
    else if (n.op != OP_MATFROM && n.op != OP_DSUM) { aa = n.a >= 0 && active_[n.a]; ba = n.b >= 0 && active_[n.b]; }
    int extra = 0;
    if (n.op == OP_MATFROM) for (int k = 0; k < n.rows * n.cols; k++) extra += active_[T.args[n.imm + k]] ? 1 : 0;
    if (n.op == OP_DSUM) extra = (int)region_inputs_[v].size();
    if (n.op == OP_DIV) extra = need_aux_[v] ? 1 : 0;  // the reverse rule has the reciprocal
    work_rev_ += mult_ * cost::rev(n.op, n.rows, n.cols, n.imm, in_rows, aa, ba, (flags & 1) != 0, (flags & 2) != 0, extra);
  }
  emit(p);
}

void Planner::emit_region(int v) {
  const Node& n = T.nodes[v];
  const int b0 = n.a, b1 = n.b, res = n.c;
  auto body_value = [&](int x) { return x >= b0 && x < b1 && region_body_[x] && !is_leaf(x); };
  // lane-level inputs whose partials the body reverse accumulates
  std::vector<std::pair<int, int>> ins;
  std::vector<char> seen(N, 0);
  auto add_input = [&](int x) {
    if (!grad_ || !active_[x] || body_value(x) || seen[x]) return;
    seen[x] = 1;
    ins.push_back({x, 1 + (int)ins.size()});
  };
  if (grad_) {
    for (int u = b0; u < b1; u++) {
      if (!body_value(u) || !active_[u]) continue;
      const Node& m = T.nodes[u];
      if (m.op == OP_SELECT) { add_input(m.b); add_input(m.c); continue; }
      for (int x : inputs(u)) add_input(x);
    }
    add_input(res);
  }
  int block = new_vr(1 + (int)ins.size());
  region_inputs_[v] = ins;
  region_block_[v] = block;
  val_vr_[v] = block;  // the sum is element 0 of the block
  const int32_t stride = T.args[n.imm2], base = T.args[n.imm2 + 1];

  PInst z; z.d.op = D_ZERO; z.f[0] = R(slotref(block)); z.f[1] = I(1 + (int)ins.size());
  emit(z);
  PInst lp; lp.d.op = D_LOOP; lp.f[0] = I(n.imm); lp.f[1] = I(stride); lp.f[2] = I(base);
  if (der_of_[v] >= 0) {  // the region's block of the extended observations
    lp.f[1] = I(1);
    lp.f[2] = I((int32_t)(T.n_obs_min + der_info_[der_of_[v]].offset));
  }
  emit_r_ = v;
  int loop_pc = emit(lp);
  mult_ = (double)n.imm;
  work_fwd_ += mult_;  // accumulation of the body value
  for (int u = b0; u < b1; u++) {
    if (!body_value(u)) continue;
    if (T.nodes[u].op == OP_DSUM) unsupported("nested data-sum");
    if (!derived_.empty() && derived_[u]) continue;  // a shared per-point value
    emit_forward(u);
  }
  PInst acc; acc.d.op = D_ACC; acc.f[0] = R(slotref(block, 0)); acc.f[1] = R(ref(res));
  emit(acc);
  if (grad_ && active_[res]) {
    cur_region_ = v;
    block_vr_ = block;
    for (auto& io : ins) partial_of_[io.first] = io.second;
    if (body_value(res)) {
      body_adj_[res] = new_vr(1);
      PInst sd; sd.d.op = D_SEED; sd.f[0] = R(slotref(body_adj_[res]));
      emit(sd);
    } else {
      // the body result is a lane-level value: d(body)/d(res) = 1 at every point
      PInst a1; a1.d.op = D_ACC; a1.f[0] = R(slotref(block, partial_of_[res]));
      a1.f[1] = R(kref(RK_CONST, one_const_));
      emit(a1);
    }
    for (int u = b1 - 1; u >= b0; u--) {
      if (!body_value(u) || !active_[u]) continue;
      emit_reverse(u);
    }
    for (auto& io : ins) partial_of_[io.first] = -1;
    for (int u = b0; u < b1; u++) body_adj_[u] = -1;
    cur_region_ = -1;
    block_vr_ = -1;
  }
  mult_ = 1.0;
  PInst el; el.d.op = D_ENDLOOP; el.f[0] = I(loop_pc);
  int end_pc = emit(el);
  code_[loop_pc].f[3] = I(end_pc);
  PInst gr; gr.d.op = D_GREDUCE; gr.f[0] = R(slotref(block)); gr.f[1] = I(1 + (int)ins.size());
  emit(gr);
  emit_r_ = -1;
}

// Shared per-point values.  Inside a data-axis region, a body node that depends on the
// data point but on no parameter has the same value on every lane.  When every such
// node of a region is a scalar primitive, they move to a derive plan (run once per call,
// one lane per point); the replay reads the ones that parameter-dependent nodes (or the
// region's sum) use from the derived buffer.  The values are the same IEEE results in
// the same order, computed once instead of once per lane.
void Planner::plan_derived() {
  pdep_.assign(N, 0);
  for (int v = 0; v < N; v++) {
    if (T.nodes[v].op == OP_PARAM) { pdep_[v] = 1; continue; }
    for (int x : inputs(v)) if (x >= 0 && x < v && pdep_[x]) { pdep_[v] = 1; break; }
  }
  derived_.assign(N, 0);
  der_col_.assign(N, -1);
  der_of_.assign(N, -1);
  if (!grad_ || !derive_enabled()) return;
  auto scalar_prim = [&](int u) {
    const Node& m = T.nodes[u];
    if (m.rows != 1 || m.cols != 1) return false;
    switch (m.op) {
      case OP_ADD: case OP_SUB: case OP_MUL: case OP_DIV: case OP_POW: case OP_NEG: case OP_EXP: case OP_LOG:
      case OP_SIN: case OP_COS: case OP_TANH: case OP_SQRT: case OP_ABS: case OP_POWI: case OP_LT: case OP_LE:
      case OP_GT: case OP_GE: case OP_EQ: case OP_SELECT:
        return true;
      default:
        return false;
    }
  };
  for (int r = 0; r < N; r++) {
    const Node& n = T.nodes[r];
    if (n.op != OP_DSUM) continue;
    std::vector<int> cand;
    bool ok = true;
    for (int u = n.a; u < n.b && ok; u++) {
      if (!region_body_[u] || is_leaf(u) || pdep_[u]) continue;
      if (!scalar_prim(u)) ok = false;
      else cand.push_back(u);
    }
    if (!ok || cand.empty()) continue;
    // inputs of the candidates that are neither leaves nor candidates are lane-level
    // values without parameters (constant subexpressions hoisted out of the body): the
    // derive plan recomputes them, so they too must be scalar primitives
    std::vector<char> incand(N, 0), seen(N, 0);
    for (int u : cand) incand[u] = 1;
    std::vector<int> stack;
    for (int u : cand)
      for (int x : inputs(u)) stack.push_back(x);
    while (!stack.empty() && ok) {
      const int x = stack.back();
      stack.pop_back();
      if (x < 0 || seen[x] || incand[x] || is_leaf(x)) continue;
      seen[x] = 1;
      if (pdep_[x] || !scalar_prim(x)) { ok = false; break; }
      for (int y : inputs(x)) stack.push_back(y);
    }
    if (!ok) continue;
    for (int u : cand) derived_[u] = 1;
    // columns: derived values that the replay reads
    std::vector<char> used(N, 0);
    for (int w = n.a; w < n.b; w++)
      if (region_body_[w] && !is_leaf(w) && !derived_[w])
        for (int x : inputs(w)) if (x >= 0 && derived_[x]) used[x] = 1;
    if (derived_[n.c]) used[n.c] = 1;
    DeriveInfo info;
    info.n_points = n.imm;
    info.stride = T.args[n.imm2];
    info.base = T.args[n.imm2 + 1];
    info.offset = der_elems_;
    // observation columns the region reads (copied into its block)
    int maxk = -1;
    for (int w = n.a; w < n.b; w++) {
      if (!region_body_[w] || is_leaf(w)) continue;
      for (int x : inputs(w))
        if (x >= 0 && T.nodes[x].op == OP_DOBS) maxk = std::max(maxk, T.nodes[x].imm);
    }
    if (T.nodes[n.c].op == OP_DOBS) maxk = std::max(maxk, T.nodes[n.c].imm);
    info.obs_cols = maxk + 1;
    int ncols = 0;
    for (int u : cand) {
      if (used[u]) der_col_[u] = ncols++;
      const Node& m = T.nodes[u];
      info.work += cost::fwd(m.op, 1, 1, m.imm, 1, m.op == OP_DIV);  // a derived division runs as a body division
    }
    info.n_cols = info.obs_cols + ncols;
    if ((int64_t)info.n_cols * info.n_points >= ((int64_t)1 << 27) ||
        T.n_obs_min + der_elems_ + (int64_t)info.n_cols * info.n_points >= ((int64_t)1 << 30)) {
      for (int u : cand) { derived_[u] = 0; der_col_[u] = -1; }  // outside the index range: keep per lane
      continue;
    }
    der_of_[r] = (int)der_info_.size();
    der_elems_ += info.n_points * info.n_cols;
    der_info_.push_back(info);
    der_region_.push_back(r);
  }
}

// The derive plan of region r: one slot per value, leaves loaded first, the region's
// derived nodes in tape order, each read value stored to its column (lanes = points).
Plan Planner::build_derive(int r, const DeriveInfo& info) const {
  const Node& n = T.nodes[r];
  Plan pl;
  // the point's observation record is the lane's parameter vector (params = obs + base,
  // P = stride), so observation column k of point d is parameter k of lane d
  pl.n_params = info.obs_cols;
  for (int u = n.a; u < n.b; u++)
    if (derived_[u])
      for (int x : inputs(u))
        if (x >= 0 && T.nodes[x].op == OP_DOBS) pl.n_params = std::max(pl.n_params, T.nodes[x].imm + 1);
  pl.n_obs_min = T.n_obs_min;
  pl.n_save = info.n_cols;
  pl.extra_consts = {1.0, -0.0};
  const int32_t k_one = (int32_t)T.consts.size(), k_mzero = k_one + 1;
  std::vector<int> slot(N, -1);
  int next = 0;
  auto load = [&](uint32_t kind, int32_t idx) {
    DInst d;
    d.op = D_LOAD;
    d.f[0] = mkref(RK_SLOT, next);
    d.f[1] = mkref(kind, idx);
    pl.code.push_back(d);
    return next++;
  };
  auto leaf_slot = [&](int x) {
    if (slot[x] >= 0) return slot[x];
    const Node& m = T.nodes[x];
    const uint32_t kind = m.op == OP_CONST ? RK_CONST : m.op == OP_OBS ? RK_OBS : RK_PARAM;
    return slot[x] = load(kind, m.imm);
  };
  // copies of the observation columns into the block (exact: x * 1 + (-0) = x)
  const int one = load(RK_CONST, k_one), mzero = load(RK_CONST, k_mzero);
  for (int k = 0; k < info.obs_cols; k++) {
    const int xk = load(RK_PARAM, k);
    DInst d;
    d.op = D_FMA;
    d.f[0] = mkref(RK_SLOT, next++);
    d.f[1] = mkref(RK_SLOT, xk);
    d.f[2] = mkref(RK_SLOT, one);
    d.f[3] = mkref(RK_SLOT, mzero);
    d.f[4] = mkref(RK_SLOT, one);
    d.f[5] = k;
    pl.code.push_back(d);
  }
  // a value of the plan: a leaf is loaded, a derived node was computed in tape order, and
  // a hoisted parameter-free lane-level node is computed on first use
  std::function<int32_t(int)> sref;
  auto emit_node = [&](int u, int32_t save_col) {
    const Node& m = T.nodes[u];
    int32_t ins[3] = {-1, -1, -1};
    if (m.op == OP_SELECT) { ins[0] = sref(m.a); ins[1] = sref(m.b); ins[2] = sref(m.c); }
    else { if (m.a >= 0) ins[0] = sref(m.a); if (m.b >= 0) ins[1] = sref(m.b); }
    DInst d;
    d.f[3] = save_col;
    switch (m.op) {
      case OP_ADD: d.op = D_ADD; break;
      case OP_SUB: d.op = D_SUB; break;
      case OP_MUL: d.op = D_MUL; break;
      case OP_DIV: d.op = D_DIV; d.flags = 16; break;  // a body division: through 1/b, as in the replay
      case OP_POW: d.op = D_POW; break;
      case OP_NEG: d.op = D_NEG; break;
      case OP_EXP: d.op = D_EXP; break;
      case OP_LOG: d.op = D_LOG; break;
      case OP_SIN: d.op = D_SIN; break;
      case OP_COS: d.op = D_COS; break;
      case OP_TANH: d.op = D_TANH; break;
      case OP_SQRT: d.op = D_SQRT; break;
      case OP_ABS: d.op = D_ABS; break;
      case OP_POWI: d.op = D_POWI; d.f[7] = m.imm; break;
      case OP_SELECT: d.op = D_SELECT; break;
      default:
        d.op = D_CMP;
        d.k = m.op == OP_LT ? 0 : m.op == OP_LE ? 1 : m.op == OP_GT ? 2 : m.op == OP_GE ? 3 : 4;
        break;
    }
    if (m.op == OP_SELECT) { d.f[1] = ins[0]; d.f[2] = ins[1]; d.f[4] = ins[2]; }
    else { d.f[1] = ins[0]; d.f[2] = ins[1]; }
    d.f[0] = mkref(RK_SLOT, next);
    pl.code.push_back(d);
    slot[u] = next++;
  };
  sref = [&](int x) -> int32_t {
    if (is_leaf(x)) return mkref(RK_SLOT, leaf_slot(x));
    if (slot[x] < 0) emit_node(x, -1);  // a hoisted constant subexpression
    return mkref(RK_SLOT, slot[x]);
  };
  for (int u = n.a; u < n.b; u++)
    if (derived_[u]) emit_node(u, der_col_[u] >= 0 ? info.obs_cols + der_col_[u] : -1);
  pl.n_slots = next;
  pl.work_fwd = info.work;
  return pl;
}

// The constant pool index holding exactly the bits of v (appended when absent).
int Planner::const_index(double v) {
  for (size_t k = 0; k < T.consts.size(); k++)
    if (std::memcmp(&T.consts[k], &v, 8) == 0) return (int)k;
  for (size_t k = 0; k < extra_consts_.size(); k++)
    if (std::memcmp(&extra_consts_[k], &v, 8) == 0) return (int)(T.consts.size() + k);
  extra_consts_.push_back(v);
  return (int)(T.consts.size() + extra_consts_.size() - 1);
}

// Fused multiply-add form.  The scalar rules whose arithmetic is one product and
// one sum become D_FMA, which the kernel executes without opcode dispatch:
//   forward   a + b = fma(a, 1, b)      a - b = fma(-b, 1, a)
//             a * b = fma(a, b, -0)     -a = fma(-a, 1, -0)     acc += x: fma(x, 1, acc)
// (all exact: the product by 1 is exact, and adding -0 leaves every value,
// including the sign of zero, unchanged), and
//   reverse   target += g * d = fma(g, d, target) -- or fma(g, d, -0) for the first
//             contribution -- for add, sub, neg, mul, exp, sin and cos, where the
//             local derivative d is 1, -1, the other factor, exp(x), cos x or -sin x.
// A reverse update is skipped when g is exactly zero (the first contribution then
// stores -0, an exact zero), as in the general rules.  Fusing the product into the
// accumulation rounds once where the general rules round twice.
void Planner::lower_fma() {
  const PArg one = R(kref(RK_CONST, one_const_));
  const PArg mzero = R(kref(RK_CONST, const_index(-0.0)));
  const int n = (int)code_.size();
  std::vector<PInst> out;
  out.reserve(n + n / 2);
  std::vector<int> newpc(n, -1);
  auto fma = [&](PArg dst, PArg a, bool neg, PArg b, PArg c, PArg zs, PArg save) {
    PInst q;
    q.d.op = D_FMA;
    q.d.flags = neg ? 1 : 0;
    q.f[0] = dst; q.f[1] = a; q.f[2] = b; q.f[3] = c; q.f[4] = zs; q.f[5] = save;
    out.push_back(q);
  };
  for (int pc = 0; pc < n; pc++) {
    newpc[pc] = (int)out.size();
    const PInst& p = code_[pc];
    const PArg* f = p.f;
    const bool fa = p.d.flags & 1, fb = p.d.flags & 2;
    auto upd = [&](const PArg& tgt, bool first, const PArg& g, bool neg, const PArg& d) {
      if (tgt.isref) fma(tgt, g, neg, d, first ? mzero : tgt, g, I(-1));
    };
    switch (p.d.op) {
      case D_ADD: fma(f[0], f[1], false, one, f[2], one, f[3]); break;
      case D_SUB: fma(f[0], f[2], true, one, f[1], one, f[3]); break;
      case D_MUL: fma(f[0], f[1], false, f[2], mzero, one, f[3]); break;
      case D_NEG: fma(f[0], f[1], true, one, mzero, one, f[3]); break;
      case D_ACC: fma(f[0], f[1], false, one, f[0], one, I(-1)); break;
      case B_ADD: case B_SUB:
        upd(f[1], fa, f[0], false, one);
        upd(f[2], fb, f[0], p.d.op == B_SUB, one);
        break;
      case B_NEG: upd(f[1], fa, f[0], true, one); break;
      case B_MUL:
        upd(f[1], fa, f[0], false, f[4]);
        upd(f[2], fb, f[0], false, f[3]);
        break;
      case B_EXP: upd(f[1], fa, f[0], false, f[5]); break;
      case B_SIN: upd(f[1], fa, f[0], false, f[6]); break;
      case B_COS: upd(f[1], fa, f[0], true, f[6]); break;
      default: out.push_back(p); break;
    }
  }
  for (PInst& p : out) {
    if (p.d.op == D_LOOP) p.f[3] = I(newpc[p.f[3].v]);
    if (p.d.op == D_ENDLOOP) p.f[0] = I(newpc[p.f[0].v]);
  }
  code_.swap(out);
  if (rev_begin_ >= 0 && rev_begin_ < n) rev_begin_ = newpc[rev_begin_];
}

// Load-store form: every operand that slot_operand() marks is made a slot.  A
// constant, parameter or observation is loaded once into a slot before its first
// use -- before the enclosing data-axis loop when the use is inside one -- and the
// slot stays live to its last use; a per-point observation is loaded at the start of
// the loop body; a workspace value not covered by the prefetch is loaded right before
// its use.
void Planner::normalize_operands() {
  const int n = (int)code_.size();
  std::vector<int> loop_of(n, -1);  // enclosing D_LOOP pc
  for (int pc = 0, open = -1; pc < n; pc++) {
    if (code_[pc].d.op == D_LOOP) { open = pc; continue; }
    if (code_[pc].d.op == D_ENDLOOP) { open = -1; continue; }
    loop_of[pc] = open;
  }
  std::vector<std::vector<PInst>> before(n + 1);
  std::map<std::pair<uint32_t, int32_t>, int> uni;  // (kind, index) -> slot VR
  std::map<int32_t, int> dob;                       // point column -> slot VR (current loop)
  int cur_loop = -2;
  auto load = [&](int vr, const PArg& src) {
    PInst l;
    l.d.op = D_LOAD;
    l.f[0] = R(slotref(vr));
    l.f[1] = src;
    return l;
  };
  for (int pc = 0; pc < n; pc++) {
    PInst& p = code_[pc];
    if (loop_of[pc] != cur_loop) { dob.clear(); cur_loop = loop_of[pc]; }
    for (int fld = 0; fld < 8; fld++) {
      if (!slot_operand(p.d.op, fld)) continue;
      PArg& a = p.f[fld];
      if (!a.isref || a.r.kind == RK_SLOT) continue;
      const uint32_t kind = a.r.kind;
      const int32_t idx = a.r.id + a.r.off;
      PArg src = a;
      if (kind == RK_CONST || kind == RK_PARAM || kind == RK_OBS) {
        auto key = std::make_pair(kind, idx);
        auto it = uni.find(key);
        if (it == uni.end()) {
          int vr = new_vr(1);
          it = uni.emplace(key, vr).first;
          before[loop_of[pc] >= 0 ? loop_of[pc] : pc].push_back(load(vr, src));
        }
        a = R(slotref(it->second));
      } else if (kind == RK_DOBS) {
        // the point's observations load at the start of the loop body, next to each
        // other, where merge_obs_loads packs them into fetch records
        auto it = dob.find(idx);
        if (it == dob.end()) {
          int vr = new_vr(1);
          it = dob.emplace(idx, vr).first;
          before[loop_of[pc] >= 0 ? loop_of[pc] + 1 : pc].push_back(load(vr, src));
        }
        a = R(slotref(it->second));
      } else {  // workspace value outside the prefetch
        int vr = new_vr(1);
        before[pc].push_back(load(vr, src));
        a = R(slotref(vr));
      }
    }
  }
  // rebuild with the loads in place and renumber the loop links
  std::vector<PInst> out;
  std::vector<int> newpc(n, -1);
  for (int pc = 0; pc < n; pc++) {
    for (PInst& l : before[pc]) out.push_back(l);
    newpc[pc] = (int)out.size();
    out.push_back(code_[pc]);
  }
  for (PInst& p : out) {
    if (p.d.op == D_LOOP) p.f[3] = I(newpc[p.f[3].v]);
    if (p.d.op == D_ENDLOOP) p.f[0] = I(newpc[p.f[0].v]);
  }
  code_.swap(out);
  // (a plan without a reverse sweep starts it one past its last instruction)
  if (rev_begin_ >= 0) rev_begin_ = rev_begin_ < n ? newpc[rev_begin_] : (int)code_.size();
}

// A first adjoint contribution that is a plain copy needs no work when the new adjoint
// d can share the slots of the copied adjoint g: a sum's scalar rule (d = g * 1 + (-0)),
// and the first target of a matrix sum's or difference's rule (d = gZ; also the second
// target of a sum).  Conditions: g is written no more after the copy, every later read
// of g comes no later than the first later write of d, that first writer reads every
// element it needs before it stores any if it also reads g, d is not referenced before
// the copy, both have the same width, neither appears in an argument list, and both
// live in the same place (the same data-axis loop body, or outside every loop, so that
// no loop repeats a read after a write).  The copy is then dropped (a matrix rule keeps
// its other target) and d renamed to g.  A zero is the one value whose bits can
// differ: the copy gives -0 (or +0), the shared slot keeps g's sign of zero.
namespace {
// whether field `fld` of an instruction with opcode `op` only reads its slot reference
// (a conservative answer: false for every field that may be written)
bool reads_only(int op, int fld) {
  if (op >= B_ADD && op <= B_GRAD) return fld == 0 || fld >= 3;  // gz and primal inputs; f1, f2 targets
  if (op == D_FETCH || fld == 0) return false;                    // destinations
  if ((op == D_SIN || op == D_COS || op == D_DET || op == D_LOGDET || op == D_DIV) && fld == 4) return false;  // aux outputs
  return true;
}
}  // namespace

void Planner::coalesce_copies() {
  if (!coalesce_enabled()) return;
  const int n = (int)code_.size();
  const int mzero = const_index(-0.0);
  std::vector<int> loop_of(n, -1);
  for (int pc = 0, open = -1; pc < n; pc++) {
    if (code_[pc].d.op == D_LOOP) { open = pc; continue; }
    if (code_[pc].d.op == D_ENDLOOP) { open = -1; continue; }
    loop_of[pc] = open;
  }
  struct Use { int pc, fld; bool read; };
  const int nv = (int)vrs_.size();
  std::vector<std::vector<Use>> uses(nv);
  std::vector<char> in_args(nv, 0);
  auto vr_of = [](const PArg& a) { return (a.isref && a.r.kind == RK_SLOT) ? a.r.id : -1; };
  for (const PArg& a : args_) if (vr_of(a) >= 0) in_args[vr_of(a)] = 1;
  for (int pc = 0; pc < n; pc++) {
    const PInst& p = code_[pc];
    for (int fld = 0; fld < 8; fld++) {
      const int v = vr_of(p.f[fld]);
      if (v >= 0) uses[v].push_back({pc, fld, reads_only(p.d.op, fld)});
    }
  }
  std::vector<int> rename(nv, -1);
  auto root = [&](int v) {
    if (v < 0) return v;
    while (rename[v] >= 0) v = rename[v];
    return v;
  };
  // whether an instruction may read g and write d when the two share slots: it must
  // read every element it needs before it stores any (the fused form loads all its
  // operands first; the scalar rules read their adjoint once; the matrix sum's rule
  // reads and writes the same element), which a product's or a scatter's rule does not
  auto reads_before_writes = [](int op) {
    return op == D_FMA || op == B_MADD || op == B_MSUB || (op >= B_ADD && op <= B_POWI) || op == B_SELECT;
  };
  // try to let the adjoint in field tf of instruction pc share the slots of the one in
  // field sf (the instruction's other references to g: the fields in also_g)
  auto try_merge = [&](int pc, int tf, int sf, int also_g) -> bool {
    const PInst& c = code_[pc];
    const int d = root(vr_of(c.f[tf])), g = root(vr_of(c.f[sf]));
    if (d < 0 || g < 0 || d == g || vrs_[d].width != vrs_[g].width || in_args[d] || in_args[g]) return false;
    if (c.f[tf].r.off != 0 || c.f[sf].r.off != 0) return false;
    const int here = loop_of[pc];
    int first_write_d = INT_MAX;
    for (const Use& u : uses[d]) {
      if (u.pc == pc && u.fld == tf) continue;
      if (u.pc <= pc || loop_of[u.pc] != here) return false;
      if (!u.read) first_write_d = std::min(first_write_d, u.pc);
    }
    // the instruction that first writes d after the copy may also read g (the slot
    // then holds g's value, which is d's); only one that reads before it writes may
    if (first_write_d != INT_MAX && !reads_before_writes(code_[first_write_d].d.op))
      for (int fld = 0; fld < 8; fld++)
        if (root(vr_of(code_[first_write_d].f[fld])) == g) return false;
    for (const Use& u : uses[g]) {
      if (u.pc == pc) {
        if (u.fld == sf || u.fld == also_g) continue;
        return false;
      }
      if (loop_of[u.pc] != here) return false;
      if (u.pc > pc && (!u.read || u.pc > first_write_d)) return false;
    }
    rename[d] = g;
    for (const Use& u : uses[d])
      if (!(u.pc == pc && u.fld == tf)) uses[g].push_back(u);
    uses[d].clear();
    return true;
  };
  auto is_const = [](const PArg& a, int idx) { return a.isref && a.r.kind == RK_CONST && a.r.id + a.r.off == idx; };
  std::vector<char> drop(n, 0);
  for (int pc = 0; pc < n; pc++) {
    PInst& c = code_[pc];
    if (c.d.op == D_FMA) {
      if (c.d.flags != 0 || !is_const(c.f[2], one_const_) || !is_const(c.f[3], mzero)) continue;
      if (c.f[5].isref || c.f[5].v != -1 || root(vr_of(c.f[4])) != root(vr_of(c.f[1]))) continue;
      if (try_merge(pc, 0, 1, 4)) drop[pc] = 1;
    } else if (c.d.op == B_MADD || c.d.op == B_MSUB) {
      if ((c.d.flags & 1) && try_merge(pc, 1, 0, -1)) {
        c.f[1] = I(-1);
        c.d.flags &= (uint8_t)~1u;
      }
      if (c.d.op == B_MADD && (c.d.flags & 2) && try_merge(pc, 2, 0, -1)) {
        c.f[2] = I(-1);
        c.d.flags &= (uint8_t)~2u;
      }
      if (vr_of(c.f[1]) < 0 && vr_of(c.f[2]) < 0) drop[pc] = 1;
    }
  }
  std::vector<PInst> out;
  std::vector<int> newpc(n, -1);
  for (int pc = 0; pc < n; pc++) {
    newpc[pc] = (int)out.size();
    if (drop[pc]) continue;
    PInst p = code_[pc];
    for (int fld = 0; fld < 8; fld++)
      if (vr_of(p.f[fld]) >= 0) p.f[fld].r.id = root(p.f[fld].r.id);
    out.push_back(p);
  }
  for (PInst& p : out) {
    if (p.d.op == D_LOOP) p.f[3] = I(newpc[p.f[3].v]);
    if (p.d.op == D_ENDLOOP) p.f[0] = I(newpc[p.f[0].v]);
  }
  if (rev_begin_ >= 0 && rev_begin_ < n) rev_begin_ = newpc[rev_begin_];
  code_.swap(out);
}

// The reverse sweep of a data-axis body starts from the seed d(body)/d(body) = 1 at every
// point.  When nothing in the loop writes the seed's slot (the body result feeds no
// other body node), the seed is set once before the loop instead of once per point;
// the allocator then keeps its slot live through the loop.  A reference other than as
// an operand of a scalar rule, a fused update or as a reverse rule's output adjoint
// keeps the seed in place.
void Planner::hoist_seeds() {
  if (!hoist_enabled()) return;
  const int n = (int)code_.size();
  std::vector<int> loop_of(n, -1);
  for (int pc = 0, open = -1; pc < n; pc++) {
    if (code_[pc].d.op == D_LOOP) { open = pc; continue; }
    if (code_[pc].d.op == D_ENDLOOP) { open = -1; continue; }
    loop_of[pc] = open;
  }
  std::vector<int> moved_to(n, -1);  // seed pc -> its loop's D_LOOP pc
  for (int pc = 0; pc < n; pc++) {
    const PInst& sd = code_[pc];
    if (sd.d.op != D_SEED || loop_of[pc] < 0 || !sd.f[0].isref || sd.f[0].r.kind != RK_SLOT) continue;
    const int vr = sd.f[0].r.id, lp = loop_of[pc];
    auto is_vr = [&](const PArg& a) { return a.isref && a.r.kind == RK_SLOT && a.r.id == vr; };
    bool ok = true;
    for (const PArg& a : args_) ok = ok && !is_vr(a);
    for (int q = lp + 1; ok && q < n && code_[q].d.op != D_ENDLOOP; q++) {
      if (q == pc) continue;
      const PInst& p = code_[q];
      for (int fld = 0; ok && fld < 8; fld++) {
        if (!is_vr(p.f[fld])) continue;
        const bool read = slot_operand(p.d.op, fld) || (p.d.op >= B_ADD && p.d.op <= B_GRAD && fld == 0);
        ok = read;
      }
    }
    if (ok) moved_to[pc] = lp;
  }
  std::vector<PInst> out;
  std::vector<int> newpc(n, -1);
  for (int pc = 0; pc < n; pc++) {
    if (code_[pc].d.op == D_LOOP)
      for (int q = pc + 1; q < n && code_[q].d.op != D_ENDLOOP; q++)
        if (moved_to[q] == pc) out.push_back(code_[q]);
    if (moved_to[pc] >= 0) continue;
    newpc[pc] = (int)out.size();
    out.push_back(code_[pc]);
  }
  for (PInst& p : out) {
    if (p.d.op == D_LOOP) p.f[3] = I(newpc[p.f[3].v]);
    if (p.d.op == D_ENDLOOP) p.f[0] = I(newpc[p.f[0].v]);
  }
  if (rev_begin_ >= 0) {
    int r = rev_begin_;
    while (r < n && newpc[r] < 0) r++;
    rev_begin_ = r < n ? newpc[r] : (int)out.size();
  }
  code_.swap(out);
}

// Software pipeline for the reverse sweep of a spill tape.  The reverse sweep is
// cut into windows of kFetchStride instructions; the workspace values that window k
// reads as scalar operands are copied into a ring of slots (asynchronous copies,
// committed as one group per window) by fetch instructions placed at the start of
// window k - kFetchWindows; before window k starts, a wait lets only the groups
// committed after window k's stay pending, so its values have landed.  The ring holds
// the values of any kFetchWindows + 2 consecutive windows.
void Planner::prefetch_workspace() {
  if (rev_begin_ < 0) return;
  const int n = (int)code_.size();
  const int nins = n - rev_begin_;
  const int stride = fetch_stride();
  const int nwin = (nins + stride - 1) / stride;
  std::vector<std::vector<std::pair<int, int>>> uses(nwin);  // window -> (pc, field)
  size_t total = 0;
  for (int pc = rev_begin_; pc < n; pc++) {
    const PInst& p = code_[pc];
    for (int fld = 0; fld < 8; fld++)
      if (slot_operand(p.d.op, fld) && p.f[fld].isref && p.f[fld].r.kind == RK_SAVE) {
        uses[(pc - rev_begin_) / stride].push_back({pc, fld});
        total++;
      }
  }
  if (total == 0) return;
  int ring = 1;
  for (int k = 0, run = 0; k < nwin; k++) {
    run += (int)uses[k].size();
    if (k >= kFetchWindows + 2) run -= (int)uses[k - kFetchWindows - 2].size();
    ring = std::max(ring, run);
  }
  const int ring_vr = new_vr(ring);
  std::vector<std::vector<std::pair<PArg, PArg>>> pairs(nwin);
  int counter = 0;
  for (int k = 0; k < nwin; k++)
    for (auto& u : uses[k]) {
      PArg slot = R(slotref(ring_vr, counter++ % ring));
      PArg& fld = code_[u.first].f[u.second];
      pairs[k].push_back({fld, slot});
      fld = slot;
    }
  // The fetch instructions before window j issue the copies of window k = j + kFetchWindows
  // (kFetchPairs per record) and commit them as one group, then wait for window j's
  // group: at most n groups may stay pending, n = the groups committed after it (those
  // of the windows j+1 .. j+kFetchWindows that fetch anything).  A window that fetches
  // nothing commits no group, and one that reads nothing fetched waits for nothing; when
  // both hold, no record is emitted (NDVM_FETCHTRIM=0 keeps one commit and a wait for
  // kFetchWindows groups per window, empty ones included).
  const bool trim = fetch_trim_enabled();
  auto has = [&](int k) { return k >= 0 && k < nwin && !pairs[k].empty(); };
  auto fetches = [&](int k, int j, std::vector<PInst>& out) {
    const int cnt = k < nwin ? (int)pairs[k].size() : 0;
    bool wait = j >= 0;
    int pending = kFetchWindows;
    if (trim && wait) {
      wait = has(j);
      pending = 0;
      for (int q = j + 1; q <= j + kFetchWindows; q++) pending += has(q) ? 1 : 0;
    }
    if (trim && cnt == 0 && !wait) return;
    int e = 0;
    do {
      PInst f;
      f.d.op = D_FETCH;
      const int m = std::min(kFetchPairs, cnt - e);
      for (int q = 0; q < m; q++) { f.f[2 * q] = pairs[k][e + q].first; f.f[2 * q + 1] = pairs[k][e + q].second; }
      f.d.k = (uint8_t)m;
      e += m;
      if (e >= cnt) f.d.flags = (uint8_t)(((cnt > 0 || !trim) ? 2 : 0) | (wait ? 1 | (pending << 2) : 0));
      out.push_back(f);
    } while (e < cnt);
  };
  std::vector<PInst> out(code_.begin(), code_.begin() + rev_begin_);
  std::vector<int> newpc(n, -1);
  for (int pc = 0; pc < rev_begin_; pc++) newpc[pc] = pc;
  for (int k = 0; k < kFetchWindows; k++) fetches(k, -1, out);  // prologue
  for (int k = 0; k < nwin; k++) {
    fetches(k + kFetchWindows, k, out);
    for (int pc = rev_begin_ + k * stride; pc < std::min(n, rev_begin_ + (k + 1) * stride); pc++) {
      newpc[pc] = (int)out.size();
      out.push_back(code_[pc]);
    }
  }
  for (PInst& p : out) {
    if (p.d.op == D_LOOP) p.f[3] = I(newpc[p.f[3].v]);
    if (p.d.op == D_ENDLOOP) p.f[0] = I(newpc[p.f[0].v]);
  }
  code_.swap(out);
}

int32_t Planner::encode(const PArg& a) const {
  if (!a.isref) return a.v;
  if (a.r.kind == RK_SLOT) {
    const VR& vr = vrs_[a.r.id];
    if (vr.phys < 0) unsupported("internal: unallocated slot");
    return mkref(RK_SLOT, vr.phys + a.r.off);
  }
  return mkref(a.r.kind, a.r.id + a.r.off);
}

// Liveness over the linear instruction stream and first-fit allocation of
// contiguous slot ranges (closed intervals: an output never aliases an input).
void Planner::allocate() {
  auto touch = [&](const PArg& a, int pos) {
    if (!a.isref || a.r.kind != RK_SLOT) return;
    VR& vr = vrs_[a.r.id];
    vr.start = std::min(vr.start, pos);
    vr.end = std::max(vr.end, pos);
  };
  for (int pc = 0; pc < (int)code_.size(); pc++) {
    const PInst& p = code_[pc];
    for (int k = 0; k < 8; k++) touch(p.f[k], pc);
    int off = -1, cnt = 0, stride = 1;
    switch (p.d.op) {
      case D_GATHER: off = p.f[1].v; cnt = p.f[2].v; stride = 1; break;
      case B_GATHER: off = p.f[1].v; cnt = p.f[2].v; stride = 2; break;
      case B_DSUM: off = p.f[1].v; cnt = p.f[2].v; stride = 3; break;
      default: break;
    }
    if (off >= 0)
      for (int e = 0; e < cnt * stride; e++) touch(args_[off + e], pc);
  }
  // values live across a data-axis loop stay live to its end
  for (int pc = 0; pc < (int)code_.size(); pc++) {
    if (code_[pc].d.op != D_LOOP) continue;
    int end = code_[pc].f[3].v;
    for (VR& vr : vrs_)
      if (vr.start < pc && vr.end >= pc && vr.end < end) vr.end = end;
  }
  std::vector<int> order;
  for (int i = 0; i < (int)vrs_.size(); i++) if (vrs_[i].end >= 0) order.push_back(i);
  std::sort(order.begin(), order.end(), [&](int a, int b) {
    if (vrs_[a].start != vrs_[b].start) return vrs_[a].start < vrs_[b].start;
    return a < b;
  });
  std::vector<int> busy_until;  // per physical slot: last position it is occupied
  for (int id : order) {
    VR& vr = vrs_[id];
    int w = vr.width, run = 0, base = -1;
    for (int s = 0; s < (int)busy_until.size(); s++) {
      if (busy_until[s] < vr.start) { if (++run == w) { base = s - w + 1; break; } }
      else run = 0;
    }
    if (base < 0) {
      base = (int)busy_until.size() - run;
      busy_until.resize(base + w, -1);
    }
    for (int s = base; s < base + w; s++) busy_until[s] = vr.end;
    vr.phys = base;
  }
  n_slots_ = (int)busy_until.size();
}

Plan Planner::build() {
  // a shared constant 1.0 for seeds of lane-level region results
  one_const_ = -1;
  for (size_t k = 0; k < T.consts.size(); k++) {
    double one = 1.0;
    if (std::memcmp(&T.consts[k], &one, 8) == 0) { one_const_ = (int)k; break; }
  }
  if (one_const_ < 0) { extra_consts_.push_back(1.0); one_const_ = (int)T.consts.size(); }
  if (T.loss < 0 || T.loss >= (int)T.nodes.size()) unsupported("tape has no loss");
  analyze();
  plan_derived();
  Plan pl;
  pl.grad = grad_;
  pl.spill = spill_;
  // forward sweep
  for (int v = 0; v < N; v++) {
    if (is_leaf(v) || region_body_[v]) continue;
    if (T.nodes[v].op == OP_DSUM) { pl.has_regions = true; emit_region(v); continue; }
    emit_forward(v);
  }
  PInst ls; ls.d.op = D_LOSS; ls.f[0] = R(ref(T.loss));
  emit(ls);
  rev_begin_ = (int)code_.size();
  if (grad_) {
    if (active_[T.loss]) {
      if (is_leaf(T.loss)) {
        adj_vr_[T.loss] = new_vr(1);
      } else {
        adj_vr_[T.loss] = new_vr(1);
      }
      PInst sd; sd.d.op = D_SEED; sd.f[0] = R(slotref(adj_vr_[T.loss]));
      emit(sd);
      for (int v = N - 1; v >= 0; v--) {
        if (is_leaf(v) || region_body_[v] || !active_[v]) continue;
        emit_reverse(v);
      }
    }
    // parameter gradients: a PARAM leaf's adjoint is the gradient
    std::vector<int> pnode(T.n_params, -1);
    for (int v = 0; v < N; v++) if (T.nodes[v].op == OP_PARAM) pnode[T.nodes[v].imm] = v;
    for (int k = 0; k < T.n_params; k++) {
      PInst g; g.d.op = B_GRAD;
      int v = pnode[k];
      if (v >= 0 && adj_vr_[v] >= 0) g.f[0] = R(slotref(adj_vr_[v]));
      g.f[1] = I(k);
      emit(g);
    }
  }
  if (fma_enabled()) lower_fma();
  if (grad_ && spill_ && prefetch_enabled()) prefetch_workspace();
  if (fma_enabled()) coalesce_copies();
  normalize_operands();
  hoist_seeds();
  allocate();
  pl.n_slots = n_slots_;
  pl.n_save = S_;
  pl.n_params = T.n_params;
  pl.n_obs_min = T.n_obs_min;
  for (const Node& nd : T.nodes) if (nd.op == OP_DOBS && nd.imm > pl.max_dobs) pl.max_dobs = nd.imm;
  for (const DeriveInfo& di : der_info_)  // column-major block reads: up to the last column's start
    pl.max_dobs = std::max<int32_t>(pl.max_dobs, (int32_t)((di.n_cols - 1) * di.n_points));
  for (const PInst& p : code_) {
    DInst d = p.d;
    for (int k = 0; k < 8; k++) d.f[k] = encode(p.f[k]);
    pl.code.push_back(d);
  }
  for (const PArg& a : args_) pl.args.push_back(encode(a));
  // one scratch area at the end of the slot file for the instructions that need working
  // space beyond their operands (scratch_elems); each uses it only while it runs
  int scratch = 0;
  for (const DInst& d : pl.code) scratch = std::max(scratch, scratch_elems(d));
  if (scratch > 0) {
    for (DInst& d : pl.code)
      if (scratch_elems(d) > 0) d.f[2] = mkref(RK_SLOT, pl.n_slots);
    pl.n_slots += scratch;
  }
  if (merge_loads_enabled()) pl.code = merge_obs_loads(pl.code);
  if (fma_enabled() && pair_enabled()) pl.code_paired = pair_fma(pl.code);
  for (const DInst& d : pl.code)
    if (d.op == D_MATMUL || d.op == D_MADD || d.op == D_MSUB || d.op == D_MSCALE || d.op == D_INV ||
        ((d.op == D_DET || d.op == D_LOGDET) && d.r > 1) || (d.op == D_GATHER && d.f[2] > 1))
      pl.has_matrix = true;
  for (size_t k = 0; k < der_info_.size(); k++) pl.derive.push_back(build_derive(der_region_[k], der_info_[k]));
  pl.derive_info = der_info_;
  pl.derived_elems = der_elems_;
  pl.extra_consts = extra_consts_;
  pl.work_fwd = work_fwd_;
  pl.work_rev = work_rev_;
  pl.n_ops_per_lane = nops_;
  return pl;
}

}  // namespace

int scratch_elems(const DInst& d) {
  const int n = d.r;
  if (d.op == B_INV) return n * n;
  if (d.op == D_INV && n >= 4) return 2 * n * n;
  if ((d.op == D_DET || d.op == D_LOGDET) && n >= 4) return (d.f[4] != -1 || d.f[5] >= 0) ? 2 * n * n : n * n;
  return 0;
}

bool slot_operand(int op, int field) {
  switch (op) {
    case D_ADD: case D_SUB: case D_MUL: case D_DIV: case D_POW: case D_CMP: return field == 1 || field == 2;
    case D_NEG: case D_EXP: case D_LOG: case D_TANH: case D_SQRT: case D_ABS: case D_SIN: case D_COS: case D_POWI:
    case D_ACC:
      return field == 1;
    case D_SELECT: return field == 1 || field == 2 || field == 4;
    case B_MUL: return field == 3 || field == 4;
    case B_DIV: return field == 4 || field == 5 || field == 6;
    case B_POW: return field == 3 || field == 4 || field == 5;
    case B_EXP: case B_TANH: return field == 5;
    case B_LOG: case B_ABS: case B_POWI: case B_SELECT: return field == 3;
    case B_SQRT: return field == 3 || field == 5;
    case B_SIN: case B_COS: return field == 6;
    case D_FMA: return field >= 1 && field <= 4;
    default: return false;
  }
}

Plan make_plan(const Tape& t, bool grad, int force_mode) {
  if (force_mode == 0 || force_mode == 1) return Planner(t, grad, force_mode == 1).build();
  Plan keep = Planner(t, grad, false).build();
  if (!grad || keep.n_slots <= 192) return keep;
  return Planner(t, grad, true).build();
}

bool validate_code(const Plan& p, const std::vector<DInst>& code, size_t n_consts, std::string& why);

bool validate_plan(const Plan& p, size_t n_consts, std::string& why) {
  if (p.derive.size() != p.derive_info.size()) { why = "derive plans"; return false; }
  for (const Plan& d : p.derive)
    if (!d.derive.empty() || !validate_code(d, d.code, n_consts, why)) return false;
  return validate_code(p, p.code, n_consts, why) &&
         (p.code_paired.empty() || validate_code(p, p.code_paired, n_consts, why));
}

bool validate_code(const Plan& p, const std::vector<DInst>& code, size_t n_consts, std::string& why) {
  const size_t nconst = n_consts + p.extra_consts.size();
  // ref: any readable operand; slot: a writable slot reference
  auto ref_ok = [&](int32_t r, int64_t width, bool must_slot) -> bool {
    if (r == -1) return true;
    if (width < 1) width = 1;
    uint32_t kind = ref_kind(r);
    int64_t idx = ref_index(r);
    if (must_slot && kind != RK_SLOT) return false;
    switch (kind) {
      case RK_SLOT: return idx + width <= p.n_slots;
      case RK_CONST: return (size_t)(idx + width) <= nconst;
      case RK_OBS: return idx + width <= p.n_obs_min;
      case RK_DOBS: return idx + width - 1 <= p.max_dobs;
      case RK_SAVE: return idx + width <= p.n_save;
      case RK_PARAM: return idx + width <= p.n_params;
      default: return false;
    }
  };
  auto save_ok = [&](int32_t s, int64_t width) { return s == -1 || (s >= 0 && s + width <= p.n_save); };
  // an instruction with working space names a slot area of its size (and none otherwise)
  auto scratch_ok = [&](const DInst& d) {
    const int need = scratch_elems(d);
    return need == 0 ? d.f[2] == -1 : (d.f[2] != -1 && ref_ok(d.f[2], need, true));
  };
  auto args_ok = [&](int32_t off, int64_t cnt, int stride) {
    return off >= 0 && cnt >= 0 && (size_t)off + (size_t)cnt * stride <= p.args.size();
  };
  int open_loop = -1;
  for (size_t pc = 0; pc < code.size(); pc++) {
    const DInst& d = code[pc];
    const int32_t* f = d.f;
    const int r = d.r, c = d.c, k = d.k, w = r * c, n = d.r;
    bool ok = true;
    // (a paired update's r, c and k bytes hold a save index, not a shape)
    if ((d.op != D_FMA2 && (r < 1 || c < 1 || r > kMaxDim || c > kMaxDim)) ||
        ((d.op == D_MATMUL || d.op == B_MATMUL) && (k < 1 || k > kMaxDim)) || (d.op == D_CMP && k > 4)) {
      why = "bad shape";
      return false;
    }
    switch (d.op) {
      case D_ADD: case D_SUB: case D_MUL: case D_DIV: case D_POW: case D_CMP:
        ok = ref_ok(f[0], 1, true) && ref_ok(f[1], 1, false) && ref_ok(f[2], 1, false) && save_ok(f[3], 1);
        if (d.op == D_DIV) ok = ok && ref_ok(f[4], 1, true) && save_ok(f[5], 1);  // the reciprocal of b
        break;
      case D_NEG: case D_EXP: case D_LOG: case D_TANH: case D_SQRT: case D_ABS: case D_POWI:
        ok = ref_ok(f[0], 1, true) && ref_ok(f[1], 1, false) && save_ok(f[3], 1) && (d.op != D_POWI || (f[7] >= 0 && f[7] <= 64));
        break;
      case D_SIN: case D_COS:
        ok = ref_ok(f[0], 1, true) && ref_ok(f[1], 1, false) && save_ok(f[3], 1) && ref_ok(f[4], 1, true) && save_ok(f[5], 1);
        break;
      case D_SELECT:
        ok = ref_ok(f[0], 1, true) && ref_ok(f[1], 1, false) && ref_ok(f[2], 1, false) && ref_ok(f[4], 1, false) && save_ok(f[3], 1);
        break;
      case D_GATHER:
        ok = ref_ok(f[0], f[2], true) && args_ok(f[1], f[2], 1) && save_ok(f[3], f[2]);
        if (ok) for (int e = 0; e < f[2]; e++) ok = ok && ref_ok(p.args[f[1] + e], 1, false);
        break;
      case D_MADD: case D_MSUB:
        ok = ref_ok(f[0], w, true) && ref_ok(f[1], w, false) && ref_ok(f[2], w, false) && save_ok(f[3], w);
        break;
      case D_MSCALE:
        ok = ref_ok(f[0], w, true) && ref_ok(f[1], 1, false) && ref_ok(f[2], w, false) && save_ok(f[3], w);
        break;
      case D_MATMUL:
        ok = ref_ok(f[0], w, true) && ref_ok(f[1], r * k, false) && ref_ok(f[2], k * c, false) && save_ok(f[3], w);
        break;
      case D_INV:
        ok = n <= 8 && ref_ok(f[0], n * n, true) && ref_ok(f[1], n * n, false) && save_ok(f[3], n * n) &&
             scratch_ok(d);
        break;
      case D_DET: case D_LOGDET:
        ok = n <= 8 && ref_ok(f[0], 1, true) && ref_ok(f[1], n * n, false) && save_ok(f[3], 1) &&
             ref_ok(f[4], n * n, true) && save_ok(f[5], n * n) && scratch_ok(d);
        break;
      case D_TRACE: ok = ref_ok(f[0], 1, true) && ref_ok(f[1], n * n, false); break;
      case D_ZERO: case D_GREDUCE: ok = f[1] >= 0 && ref_ok(f[0], f[1], true); break;
      case D_LOOP:
        ok = open_loop < 0 && f[3] > (int)pc && f[3] < (int)code.size() && code[f[3]].op == D_ENDLOOP &&
             f[0] >= 0 && f[1] >= 0 && f[2] >= 0;
        // a region reading a block of the extended observations stays inside it
        for (const DeriveInfo& di : p.derive_info)
          if (ok && f[2] == p.n_obs_min + di.offset && f[1] == 1)
            ok = f[0] == di.n_points && di.offset + di.n_points * di.n_cols <= p.derived_elems;
        open_loop = (int)pc;
        break;
      case D_ENDLOOP: ok = f[0] == open_loop && code[f[0]].f[3] == (int)pc; open_loop = -1; break;
      case D_ACC: ok = ref_ok(f[0], 1, true) && ref_ok(f[1], 1, false); break;
      case D_SEED: ok = ref_ok(f[0], 1, true); break;
      case D_LOAD: ok = ref_ok(f[0], 1, true) && f[1] != -1 && ref_ok(f[1], 1, false); break;
      case D_FMA2:
        ok = f[0] != -1 && f[5] != -1 && ref_ok(f[0], 1, true) && ref_ok(f[5], 1, true);
        if (d.flags & 8) {
          const int32_t s1 = d.r | (d.c << 8) | (d.k << 16), s2 = d.pad0 | (d.pad1 << 8) | (d.pad2 << 16);
          ok = ok && (s1 == kNoSave24 || save_ok(s1, 1)) && (s2 == kNoSave24 || save_ok(s2, 1));
        }
        for (int q = 1; q <= 4; q++) ok = ok && f[q] != -1 && ref_ok(f[q], 1, true);
        ok = ok && f[6] != -1 && f[7] != -1 && d.pad3 != -1 && d.pad4 != -1 && ref_ok(f[6], 1, true) &&
             ref_ok(f[7], 1, true) && ref_ok(d.pad3, 1, true) && ref_ok(d.pad4, 1, true);
        break;
      case D_FMA:
        ok = ref_ok(f[0], 1, true) && f[0] != -1 && save_ok(f[5], 1);
        for (int q = 1; q <= 4; q++) ok = ok && f[q] != -1 && ref_ok(f[q], 1, true);
        break;
      case D_LOSS: ok = ref_ok(f[0], 1, false); break;
      case B_ADD: case B_SUB: ok = ref_ok(f[0], 1, true) && ref_ok(f[1], 1, true) && ref_ok(f[2], 1, true); break;
      case B_NEG: ok = ref_ok(f[0], 1, true) && ref_ok(f[1], 1, true); break;
      case B_MUL: case B_DIV: case B_POW:
        ok = ref_ok(f[0], 1, true) && ref_ok(f[1], 1, true) && ref_ok(f[2], 1, true) && ref_ok(f[3], 1, false) &&
             ref_ok(f[4], 1, false) && ref_ok(f[5], 1, false) && (d.op != B_DIV || ref_ok(f[6], 1, false));
        break;
      case B_EXP: case B_TANH: case B_LOG: case B_ABS: case B_SQRT: case B_SIN: case B_COS: case B_POWI:
        ok = ref_ok(f[0], 1, true) && ref_ok(f[1], 1, true) && ref_ok(f[3], 1, false) && ref_ok(f[5], 1, false) &&
             ref_ok(f[6], 1, false) && (d.op != B_POWI || (f[7] >= 0 && f[7] <= 64));
        break;
      case B_SELECT: ok = ref_ok(f[0], 1, true) && ref_ok(f[1], 1, true) && ref_ok(f[2], 1, true) && ref_ok(f[3], 1, false); break;
      case B_GATHER:
        ok = ref_ok(f[0], f[2], true) && args_ok(f[1], f[2], 2);
        if (ok) for (int e = 0; e < f[2]; e++) ok = ok && ref_ok(p.args[f[1] + 2 * e], 1, true);
        break;
      case B_SCATTER:
        ok = ref_ok(f[0], f[2], true) && ref_ok(f[1], f[4], true) && args_ok(f[3], f[2], 1) && f[4] >= 1 && f[4] <= kMaxDim * kMaxDim;
        if (ok) for (int e = 0; e < f[2]; e++) ok = ok && p.args[f[3] + e] >= 0 && p.args[f[3] + e] < f[4];
        break;
      case B_MADD: case B_MSUB: ok = ref_ok(f[0], w, true) && ref_ok(f[1], w, true) && ref_ok(f[2], w, true); break;
      case B_MSCALE:
        ok = ref_ok(f[0], w, true) && ref_ok(f[1], 1, true) && ref_ok(f[2], w, true) && ref_ok(f[3], 1, false) && ref_ok(f[4], w, false);
        break;
      case B_MATMUL:
        ok = ref_ok(f[0], w, true) && ref_ok(f[1], r * k, true) && ref_ok(f[2], k * c, true) && ref_ok(f[3], r * k, false) &&
             ref_ok(f[4], k * c, false);
        break;
      case B_INV:
        ok = n <= 8 && ref_ok(f[0], n * n, true) && ref_ok(f[1], n * n, true) && ref_ok(f[5], n * n, false) && scratch_ok(d);
        break;
      case B_DET: case B_LOGDET:
        ok = n <= 8 && ref_ok(f[0], 1, true) && ref_ok(f[1], n * n, true) && ref_ok(f[5], 1, false) && ref_ok(f[6], n * n, false);
        break;
      case B_TRACE: ok = ref_ok(f[0], 1, true) && ref_ok(f[1], n * n, true); break;
      case B_DSUM:
        ok = ref_ok(f[0], 1, true) && args_ok(f[1], f[2], 3);
        if (ok)
          for (int e = 0; e < f[2]; e++)
            ok = ok && ref_ok(p.args[f[1] + 3 * e], 1, true) && p.args[f[1] + 3 * e] != -1 && ref_ok(p.args[f[1] + 3 * e + 2], 1, true);
        break;
      case B_GRAD: ok = ref_ok(f[0], 1, true) && f[1] >= 0 && f[1] < p.n_params; break;
      case D_FETCH: {
        const bool from_obs = d.flags & 32;
        ok = k <= kFetchPairs && ((d.flags >> 2) & 7) <= kFetchWindows && (!from_obs || open_loop >= 0);
        for (int e = 0; ok && e < k; e++)
          ok = ref_kind(f[2 * e]) == (from_obs ? RK_DOBS : RK_SAVE) && ref_ok(f[2 * e], 1, false) &&
               f[2 * e + 1] != -1 && ref_ok(f[2 * e + 1], 1, true);
        break;
      }
      default: why = "bad opcode"; return false;
    }
    const bool forward_scalar = (d.op >= D_ADD && d.op <= D_SELECT) || d.op == D_ACC;
    for (int fld = 0; ok && fld < 8; fld++)
      if (slot_operand(d.op, fld) && (f[fld] == -1 ? forward_scalar : ref_kind(f[fld]) != RK_SLOT)) ok = false;
    if (!ok) { why = "operand out of range at instruction " + std::to_string(pc) + " (op " + std::to_string(d.op) + ")"; return false; }
  }
  if (open_loop >= 0) { why = "unterminated loop"; return false; }
  return true;
}

}  // namespace ndvm
