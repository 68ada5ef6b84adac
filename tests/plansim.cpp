// Test infrastructure: a CPU executor of the replay plans for scalar and data-axis
// tapes (one lane at a time, one thread per lane), used to check the planner's stream
// rewrites on a machine without a GPU.  It follows the device interpreter's documented
// instruction semantics (plan.h): slot files, the fused multiply-add form and its
// paired record, data-axis loops, shared per-point values, workspace saves and
// fetches (a fetch copies at once; the device's later wait then has nothing to wait
// for), first-contribution stores and exact-zero adjoint skips.  Matrix instructions
// are not simulated (exit status 3).
//
// Input on stdin:  frontend B P n_obs stream(0 plain, 1 paired) / B*P params / n_obs obs /
//                  the program text up to end of input.
// Output: one line per lane: the loss and the P gradient components as C hex floats.
#include <cmath>
#include <cstdio>
#include <cstdlib>
#include <iostream>
#include <sstream>
#include <string>
#include <vector>

#include "plan.h"
#include "tape.h"

using namespace ndvm;

namespace {

bool is_zero(double x) { return x == 0.0; }
bool gt_eps(double x) { return x > 1e-8; }
double powi_rep(double a, int n) {
  if (n == 0) return 1.0;
  double z = a;
  for (int i = 1; i < n; i++) z = z * a;
  return z;
}

struct Unsupported {};

// one lane's execution of one plan
struct Run {
  const Plan& p;
  const std::vector<DInst>& code;
  const std::vector<double>& consts;
  const double* obs;     // observations (extended when the tape has shared values)
  const double* params;  // this lane's P parameters
  double* save;          // workspace: element e of this lane at save[e * save_ld + col]
  int64_t save_ld, col;
  double* loss = nullptr;
  double* grad = nullptr;
  std::vector<double> s;
  int64_t dbase = 0;

  Run(const Plan& p_, const std::vector<DInst>& c, const std::vector<double>& k, const double* o, const double* pa,
      double* sv, int64_t ld, int64_t cl)
      : p(p_), code(c), consts(k), obs(o), params(pa), save(sv), save_ld(ld), col(cl), s((size_t)p_.n_slots, 0.0) {}

  double& slot(int32_t ref) { return s[(size_t)ref_index(ref)]; }
  double ld(int32_t ref) {
    const int32_t i = ref_index(ref);
    switch (ref_kind(ref)) {
      case RK_SLOT: return s[(size_t)i];
      case RK_CONST: return consts[(size_t)i];
      case RK_OBS: return obs[i];
      case RK_DOBS: return obs[dbase + i];
      case RK_SAVE: return save[(int64_t)i * save_ld + col];
      default: return params[i];
    }
  }
  void save_out(int32_t sidx, double v) {
    if (sidx >= 0) save[(int64_t)sidx * save_ld + col] = v;
  }
  void upd(int32_t ref, double v, bool first) {
    double& q = slot(ref);
    q = first ? v : q + v;
  }
  void zero_if_first(int32_t ref, bool first) {
    if (first && ref != -1) slot(ref) = 0.0;
  }

  void exec() {
    int64_t d = 0, dN = 0, dstride = 0, dbase0 = 0;
    int loop_pc = -1;
    const int n = (int)code.size();
    for (int pc = 0; pc < n; pc++) {
      const DInst& in = code[(size_t)pc];
      const int32_t* f = in.f;
      switch (in.op) {
        case D_FMA: {
          const double x = (in.flags & 1) ? -ld(f[1]) : ld(f[1]);
          const double c = ld(f[3]);
          const double z = is_zero(ld(f[4])) ? c : std::fma(x, ld(f[2]), c);
          slot(f[0]) = z;
          save_out(f[5], z);
          break;
        }
        case D_FMA2: {
          const double x1 = (in.flags & 1) ? -ld(f[1]) : ld(f[1]), y1 = ld(f[2]), c1 = ld(f[3]), g1 = ld(f[4]);
          double x2 = ld(f[6]), y2 = ld(f[7]), c2 = ld(in.pad3), g2 = ld(in.pad4);
          const double z1 = is_zero(g1) ? c1 : std::fma(x1, y1, c1);
          if (in.flags & 4) {
            if (f[6] == f[0]) x2 = z1;
            if (f[7] == f[0]) y2 = z1;
            if (in.pad3 == f[0]) c2 = z1;
            if (in.pad4 == f[0]) g2 = z1;
          }
          if (in.flags & 2) x2 = -x2;
          const double z2 = is_zero(g2) ? c2 : std::fma(x2, y2, c2);
          slot(f[0]) = z1;
          slot(f[5]) = z2;
          if (in.flags & 8) {
            const int32_t s1 = in.r | (in.c << 8) | (in.k << 16), s2 = in.pad0 | (in.pad1 << 8) | (in.pad2 << 16);
            if (s1 != kNoSave24) save_out(s1, z1);
            if (s2 != kNoSave24) save_out(s2, z2);
          }
          break;
        }
        case D_FETCH:
          for (int e = 0; e < in.k; e++) {
            const int32_t src = f[2 * e], dst = f[2 * e + 1];
            slot(dst) = (in.flags & 32) ? obs[dbase + ref_index(src)] : save[(int64_t)ref_index(src) * save_ld + col];
          }
          break;
        case D_ADD: case D_SUB: case D_MUL: case D_DIV: case D_POW: {
          const double x = ld(f[1]), y = ld(f[2]);
          const double z = in.op == D_ADD ? x + y : in.op == D_SUB ? x - y : in.op == D_MUL ? x * y
                           : in.op == D_DIV ? x / y : std::pow(x, y);
          slot(f[0]) = z;
          save_out(f[3], z);
          break;
        }
        case D_NEG: case D_EXP: case D_LOG: case D_TANH: case D_SQRT: case D_ABS: {
          const double x = ld(f[1]);
          const double z = in.op == D_NEG ? -x : in.op == D_EXP ? std::exp(x)
                           : in.op == D_LOG ? std::log(gt_eps(x) ? x : 1e-8) : in.op == D_TANH ? std::tanh(x)
                           : in.op == D_SQRT ? std::sqrt(gt_eps(x) ? x : 1e-8) : std::fabs(x);
          slot(f[0]) = z;
          save_out(f[3], z);
          break;
        }
        case D_SIN: case D_COS: {
          const double x = ld(f[1]);
          const double sv = std::sin(x), cv = std::cos(x);
          if (f[4] != -1 || f[5] >= 0) {
            const double aux = in.op == D_SIN ? cv : sv;
            if (f[4] != -1) slot(f[4]) = aux;
            save_out(f[5], aux);
          }
          const double z = in.op == D_SIN ? sv : cv;
          slot(f[0]) = z;
          save_out(f[3], z);
          break;
        }
        case D_POWI: {
          const double z = powi_rep(ld(f[1]), f[7]);
          slot(f[0]) = z;
          save_out(f[3], z);
          break;
        }
        case D_CMP: {
          const double x = ld(f[1]), y = ld(f[2]);
          const bool r = in.k == 0 ? x < y : in.k == 1 ? x <= y : in.k == 2 ? x > y : in.k == 3 ? x >= y : x == y;
          slot(f[0]) = r ? 1.0 : 0.0;
          save_out(f[3], r ? 1.0 : 0.0);
          break;
        }
        case D_SELECT: {
          const double z = !is_zero(ld(f[1])) ? ld(f[2]) : ld(f[4]);
          slot(f[0]) = z;
          save_out(f[3], z);
          break;
        }
        case D_ZERO:
          for (int e = 0; e < f[1]; e++) s[(size_t)(ref_index(f[0]) + e)] = 0.0;
          break;
        case D_LOOP:
          dN = f[0]; dstride = f[1]; dbase0 = f[2];
          d = 0;
          loop_pc = pc;
          if (d >= dN) { pc = f[3]; break; }
          dbase = dbase0 + d * dstride;
          break;
        case D_ENDLOOP:
          d += 1;
          if (d < dN) { dbase = dbase0 + d * dstride; pc = loop_pc; }
          break;
        case D_ACC: slot(f[0]) = slot(f[0]) + ld(f[1]); break;
        case D_LOAD: slot(f[0]) = ld(f[1]); break;
        case D_SEED: slot(f[0]) = 1.0; break;
        case D_GREDUCE: break;  // one thread per lane: nothing to reduce
        case D_LOSS: if (loss) *loss = ld(f[0]); break;
        case B_ADD: case B_SUB: case B_MUL: case B_DIV: case B_POW: {
          const double g = slot(f[0]);
          const bool fa = in.flags & 1, fb = in.flags & 2;
          if (is_zero(g)) { zero_if_first(f[1], fa); zero_if_first(f[2], fb); break; }
          // each operand is read only for the target that needs it (the others may be absent)
          if (in.op == B_ADD || in.op == B_SUB) {
            if (f[1] != -1) upd(f[1], g, fa);
            if (f[2] != -1) upd(f[2], in.op == B_ADD ? g : -g, fb);
          } else if (in.op == B_MUL) {
            if (f[1] != -1) upd(f[1], g * ld(f[4]), fa);
            if (f[2] != -1) upd(f[2], g * ld(f[3]), fb);
          } else if (in.op == B_DIV) {
            const double q = g / ld(f[4]);
            if (f[1] != -1) upd(f[1], q, fa);
            if (f[2] != -1) upd(f[2], -(q * ld(f[5])), fb);
          } else {
            const double x = ld(f[3]), e = ld(f[4]), z = ld(f[5]);
            if (f[1] != -1) upd(f[1], g * e * z / x, fa);
            if (f[2] != -1) upd(f[2], g * z * std::log(x), fb);
          }
          break;
        }
        case B_NEG: case B_EXP: case B_TANH: case B_LOG: case B_ABS: case B_SQRT: case B_SIN: case B_COS:
        case B_POWI: {
          const double g = slot(f[0]);
          const bool fa = in.flags & 1;
          if (f[1] == -1) break;
          if (is_zero(g)) { zero_if_first(f[1], fa); break; }
          double v = 0;
          switch (in.op) {
            case B_NEG: v = -g; break;
            case B_EXP: v = g * ld(f[5]); break;
            case B_TANH: v = g * (1.0 - ld(f[5]) * ld(f[5])); break;
            case B_LOG: v = gt_eps(ld(f[3])) ? g / ld(f[3]) : 0.0; break;
            case B_ABS: v = ld(f[3]) > 0 ? g : (ld(f[3]) < 0 ? -g : g * 0.0); break;
            case B_SQRT: v = gt_eps(ld(f[3])) ? g / (2.0 * ld(f[5])) : 0.0; break;
            case B_SIN: v = g * ld(f[6]); break;
            case B_COS: v = -(g * ld(f[6])); break;
            default: v = f[7] > 0 ? g * ((double)f[7] * powi_rep(ld(f[3]), f[7] - 1)) : 0.0; break;
          }
          upd(f[1], v, fa);
          break;
        }
        case B_SELECT: {
          const double g = slot(f[0]);
          const bool fa = in.flags & 1, fb = in.flags & 2;
          const bool taken = !is_zero(ld(f[3]));
          if (f[1] != -1) { if (taken && !is_zero(g)) upd(f[1], g, fa); else zero_if_first(f[1], fa); }
          if (f[2] != -1) { if (!taken && !is_zero(g)) upd(f[2], g, fb); else zero_if_first(f[2], fb); }
          break;
        }
        case B_DSUM: {
          const double g = slot(f[0]);
          const int32_t* q = p.args.data() + f[1];
          for (int e = 0; e < f[2]; e++) {
            const int32_t t = q[3 * e];
            const bool first = q[3 * e + 1] != 0;
            if (is_zero(g)) zero_if_first(t, first);
            else upd(t, g * slot(q[3 * e + 2]), first);
          }
          break;
        }
        case B_GRAD:
          if (grad) grad[f[1]] = f[0] == -1 ? 0.0 : slot(f[0]);
          break;
        default:
          throw Unsupported{};
      }
    }
  }
};

}  // namespace

int main() {
  int fe = 0, stream = 0;
  int64_t B = 0, P = 0, n_obs = 0;
  std::cin >> fe >> B >> P >> n_obs >> stream;
  std::vector<double> params((size_t)(B * P)), obs((size_t)n_obs);
  for (auto& v : params) std::cin >> v;
  for (auto& v : obs) std::cin >> v;
  std::stringstream rest;
  rest << std::cin.rdbuf();
  const std::string text = rest.str();
  try {
    Builder b;
    std::string err;
    if (fe == 0) trace_scheme(text.data(), text.size(), b, err);
    else trace_bytecode(text.data(), text.size(), b, err);
    if (b.t.loss < 0) { std::fprintf(stderr, "no result: %s\n", err.c_str()); return 2; }
    const Plan p = make_plan(b.t, true);
    std::string why;
    if (!validate_plan(p, b.t.consts.size(), why)) { std::fprintf(stderr, "plan check: %s\n", why.c_str()); return 4; }
    std::vector<double> consts = b.t.consts;
    consts.insert(consts.end(), p.extra_consts.begin(), p.extra_consts.end());
    // extended observations: the observations the program reads, then each region's
    // block (its points' observation records run through the derive plan, one lane per point)
    std::vector<double> ext;
    const double* obs_used = obs.data();
    if (!p.derive.empty()) {
      ext.assign((size_t)(p.n_obs_min + p.derived_elems), 0.0);
      for (int64_t i = 0; i < p.n_obs_min; i++) ext[(size_t)i] = obs[(size_t)i];
      for (size_t k = 0; k < p.derive.size(); k++) {
        const Plan& q = p.derive[k];
        const DeriveInfo& di = p.derive_info[k];
        std::vector<double> qc = b.t.consts;
        qc.insert(qc.end(), q.extra_consts.begin(), q.extra_consts.end());
        double* block = ext.data() + p.n_obs_min + di.offset;
        for (int64_t pt = 0; pt < di.n_points; pt++) {
          Run r(q, q.code, qc, obs.data(), obs.data() + di.base + pt * di.stride, block, di.n_points, pt);
          r.exec();
        }
      }
      obs_used = ext.data();
    }
    const std::vector<DInst>& code = (stream == 1 && !p.code_paired.empty()) ? p.code_paired : p.code;
    std::vector<double> ws((size_t)std::max<int64_t>(p.n_save, 1));
    std::vector<double> g((size_t)P);
    for (int64_t lane = 0; lane < B; lane++) {
      double loss = 0;
      std::fill(g.begin(), g.end(), 0.0);
      Run r(p, code, consts, obs_used, params.data() + lane * P, ws.data(), 1, 0);
      r.loss = &loss;
      r.grad = g.data();
      r.exec();
      std::printf("%a", loss);
      for (double v : g) std::printf(" %a", v);
      std::printf("\n");
    }
  } catch (const Unsupported&) {
    return 3;
  } catch (const BuildError& e) {
    std::fprintf(stderr, "build error: %s\n", e.msg.c_str());
    return 2;
  }
  return 0;
}
