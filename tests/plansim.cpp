// Test infrastructure: a CPU executor of the replay plans for scalar and data-axis
// tapes (one lane at a time, one thread per lane), used to check the planner's stream
// rewrites on a machine without a GPU.  It follows the device interpreter's documented
// instruction semantics (plan.h): slot files, the fused multiply-add form and its
// paired record, data-axis loops, shared per-point values, workspace saves and
// fetches (a fetch copies at once; the device's later wait then has nothing to wait
// for), first-contribution stores and exact-zero adjoint skips, and the matrix
// instructions (element e of a matrix operand is element ref + e; products accumulate
// left to right with fused multiply-adds; inverses and determinants by closed forms to
// 3 x 3, Gauss-Jordan elimination with partial pivoting above).  An instruction the
// executor does not know ends the run with exit status 3.
//
// Input on stdin:  frontend B P n_obs stream(0 plain, 1 paired, 2 the value-only plan) / B*P params /
//                  n_obs obs /
//                  the program text up to end of input.
// Output: one line per lane: the loss and the P gradient components as C hex floats.
// (The executor takes G = 1: one thread owns every element of its lane.)
#include <cmath>
#include <cstdio>
#include <cstdlib>
#include <iostream>
#include <utility>
#include <sstream>
#include <string>
#include <vector>

#include "plan.h"
#include "tape.h"

using namespace ndvm;

namespace {

bool is_zero(double x) { return x == 0.0; }
bool gt_eps(double x) { return x > 1e-8; }
// a / b from r = the correctly rounded 1 / b by one correction step where a and b have
// exponents within +-500 (zeros, infinities and NaNs excluded), else the division
double div_by_rcp(double a, double b, double r) {
  int ea = 0, eb = 0;
  std::frexp(a, &ea);
  std::frexp(b, &eb);
  const bool ok = std::isnormal(a) && std::isnormal(b) && ea - 1 >= -500 && ea - 1 <= 500 && eb - 1 >= -500 &&
                  eb - 1 <= 500;
  if (!ok) return a / b;
  const double q = a * r;
  return std::fma(r, std::fma(-b, q, a), q);
}
double powi_rep(double a, int n) {
  if (n == 0) return 1.0;
  double z = a;
  for (int i = 1; i < n; i++) z = z * a;
  return z;
}

// determinant and (optionally) inverse of the n x n matrix a (row-major)
double det_inv(const std::vector<double>& a, int n, std::vector<double>* inv) {
  if (n == 1) {
    if (inv) (*inv)[0] = 1.0 / a[0];
    return a[0];
  }
  if (n == 2) {
    const double d = a[0] * a[3] - a[1] * a[2];
    if (inv) {
      const double r = 1.0 / d;
      (*inv)[0] = a[3] * r; (*inv)[1] = -a[1] * r; (*inv)[2] = -a[2] * r; (*inv)[3] = a[0] * r;
    }
    return d;
  }
  if (n == 3) {
    const double c00 = a[4] * a[8] - a[5] * a[7], c01 = a[5] * a[6] - a[3] * a[8], c02 = a[3] * a[7] - a[4] * a[6];
    const double d = a[0] * c00 + a[1] * c01 + a[2] * c02;
    if (inv) {
      const double c10 = a[2] * a[7] - a[1] * a[8], c11 = a[0] * a[8] - a[2] * a[6], c12 = a[1] * a[6] - a[0] * a[7];
      const double c20 = a[1] * a[5] - a[2] * a[4], c21 = a[2] * a[3] - a[0] * a[5], c22 = a[0] * a[4] - a[1] * a[3];
      const double r = 1.0 / d;
      const double cof[9] = {c00, c10, c20, c01, c11, c21, c02, c12, c22};
      for (int e = 0; e < 9; e++) (*inv)[e] = cof[e] * r;
    }
    return d;
  }
  std::vector<std::vector<double>> w(n, std::vector<double>(2 * n));
  for (int i = 0; i < n; i++)
    for (int j = 0; j < 2 * n; j++) w[i][j] = j < n ? a[i * n + j] : (j - n == i ? 1.0 : 0.0);
  double d = 1.0;
  for (int col = 0; col < n; col++) {
    int piv = col;
    for (int i = col + 1; i < n; i++)
      if (std::fabs(w[i][col]) > std::fabs(w[piv][col])) piv = i;
    if (piv != col) { std::swap(w[piv], w[col]); d = -d; }
    const double pv = w[col][col];
    d = d * pv;
    const double r = 1.0 / pv;
    for (int j = 0; j < 2 * n; j++) w[col][j] = w[col][j] * r;
    for (int i = 0; i < n; i++) {
      if (i == col) continue;
      const double fct = w[i][col];
      if (fct != 0.0)
        for (int j = 0; j < 2 * n; j++) w[i][j] = w[i][j] - fct * w[col][j];
    }
  }
  if (inv)
    for (int i = 0; i < n; i++)
      for (int j = 0; j < n; j++) (*inv)[i * n + j] = w[i][n + j];
  return d;
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
  // element e of a (matrix) operand, and of a slot range
  double el(int32_t ref, int e) {
    const int32_t i = ref_index(ref) + e;
    switch (ref_kind(ref)) {
      case RK_SLOT: return s[(size_t)i];
      case RK_CONST: return consts[(size_t)i];
      case RK_OBS: return obs[i];
      case RK_DOBS: return obs[dbase + i];
      case RK_SAVE: return save[(int64_t)i * save_ld + col];
      default: return params[i];
    }
  }
  double& sel(int32_t ref, int e) { return s[(size_t)(ref_index(ref) + e)]; }
  void upd_el(int32_t ref, int e, double v, bool first) {
    double& q = sel(ref, e);
    q = first ? v : q + v;
  }
  void zero_first(int32_t ref, int w, bool first) {
    if (first && ref != -1)
      for (int e = 0; e < w; e++) sel(ref, e) = 0.0;
  }
  bool all_zero(int32_t gz, int w) {
    for (int e = 0; e < w; e++)
      if (!is_zero(sel(gz, e))) return false;
    return true;
  }
  // a[0] b[0] + a[sa] b[sb] + ... over n terms, left to right, fused after the first
  double dot(int32_t ra, int ea, int sa, int32_t rb, int eb, int sb, int n) {
    double acc = el(ra, ea) * el(rb, eb);
    for (int q = 1; q < n; q++) acc = std::fma(el(ra, ea + q * sa), el(rb, eb + q * sb), acc);
    return acc;
  }
  std::vector<double> mat(int32_t ref, int w) {
    std::vector<double> m((size_t)w);
    for (int e = 0; e < w; e++) m[(size_t)e] = el(ref, e);
    return m;
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
          const double r = 1.0 / y;  // a body division (flags bit 4) keeps y's reciprocal
          const bool via_rcp = in.op == D_DIV && (in.flags & 16);
          const double z = in.op == D_ADD ? x + y : in.op == D_SUB ? x - y : in.op == D_MUL ? x * y
                           : in.op == D_DIV ? (via_rcp ? div_by_rcp(x, y, r) : x / y) : std::pow(x, y);
          slot(f[0]) = z;
          save_out(f[3], z);
          if (via_rcp) {
            if (f[4] != -1) slot(f[4]) = r;
            save_out(f[5], r);
          }
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
        case D_GATHER: {
          const int32_t* g = p.args.data() + f[1];
          for (int e = 0; e < f[2]; e++) {
            const double v = ld(g[e]);
            sel(f[0], e) = v;
            save_out(f[3] < 0 ? -1 : f[3] + e, v);
          }
          break;
        }
        case D_MADD: case D_MSUB: case D_MSCALE: {
          const int w = in.r * in.c;
          const double sc = in.op == D_MSCALE ? ld(f[1]) : 0.0;
          for (int e = 0; e < w; e++) {
            const double z = in.op == D_MADD ? el(f[1], e) + el(f[2], e)
                             : in.op == D_MSUB ? el(f[1], e) - el(f[2], e) : sc * el(f[2], e);
            sel(f[0], e) = z;
            save_out(f[3] < 0 ? -1 : f[3] + e, z);
          }
          break;
        }
        case D_MATMUL: {
          const int r = in.r, c = in.c, kk = in.k;
          std::vector<double> z((size_t)(r * c));
          for (int i = 0; i < r; i++)
            for (int j = 0; j < c; j++) z[(size_t)(i * c + j)] = dot(f[1], i * kk, 1, f[2], j, c, kk);
          for (int e = 0; e < r * c; e++) {
            sel(f[0], e) = z[(size_t)e];
            save_out(f[3] < 0 ? -1 : f[3] + e, z[(size_t)e]);
          }
          break;
        }
        case D_INV: {
          const int n = in.r;
          std::vector<double> inv((size_t)(n * n));
          det_inv(mat(f[1], n * n), n, &inv);
          for (int e = 0; e < n * n; e++) {
            sel(f[0], e) = inv[(size_t)e];
            save_out(f[3] < 0 ? -1 : f[3] + e, inv[(size_t)e]);
          }
          break;
        }
        case D_DET: case D_LOGDET: {
          const int n = in.r;
          const bool aux = f[4] != -1 || f[5] >= 0;
          std::vector<double> inv((size_t)(n * n));
          const double dt = det_inv(mat(f[1], n * n), n, aux ? &inv : nullptr);
          const double z = in.op == D_DET ? dt : std::log(dt);
          slot(f[0]) = z;
          save_out(f[3], z);
          if (aux)
            for (int e = 0; e < n * n; e++) {
              if (f[4] != -1) sel(f[4], e) = inv[(size_t)e];
              save_out(f[5] < 0 ? -1 : f[5] + e, inv[(size_t)e]);
            }
          break;
        }
        case D_TRACE: {
          const int n = in.r;
          double t = el(f[1], 0);
          for (int i = 1; i < n; i++) t = t + el(f[1], i * n + i);
          slot(f[0]) = t;
          break;
        }
        case B_GATHER: {
          const int32_t* g = p.args.data() + f[1];
          const bool z = all_zero(f[0], f[2]);
          for (int e = 0; e < f[2]; e++) {
            const int32_t t = g[2 * e];
            if (t == -1) continue;
            const bool first = g[2 * e + 1] != 0;
            if (z) zero_if_first(t, first);
            else upd(t, sel(f[0], e), first);
          }
          break;
        }
        case B_SCATTER: {
          if (f[1] == -1) break;
          zero_first(f[1], f[4], in.flags & 1);
          if (all_zero(f[0], f[2])) break;
          const int32_t* m = p.args.data() + f[3];
          for (int e = 0; e < f[2]; e++) sel(f[1], m[e]) = sel(f[1], m[e]) + sel(f[0], e);
          break;
        }
        case B_MADD: case B_MSUB: {
          const int w = in.r * in.c;
          const bool fa = in.flags & 1, fb = in.flags & 2;
          if (all_zero(f[0], w)) { zero_first(f[1], w, fa); zero_first(f[2], w, fb); break; }
          for (int e = 0; e < w; e++) {
            const double g = sel(f[0], e);
            if (f[1] != -1) upd_el(f[1], e, g, fa);
            if (f[2] != -1) upd_el(f[2], e, in.op == B_MADD ? g : -g, fb);
          }
          break;
        }
        case B_MSCALE: {
          const int w = in.r * in.c;
          const bool fa = in.flags & 1, fb = in.flags & 2;
          if (all_zero(f[0], w)) { zero_first(f[1], 1, fa); zero_first(f[2], w, fb); break; }
          if (f[1] != -1) {
            double acc = sel(f[0], 0) * el(f[4], 0);
            for (int e = 1; e < w; e++) acc = std::fma(sel(f[0], e), el(f[4], e), acc);
            upd(f[1], acc, fa);
          }
          if (f[2] != -1) {
            const double sc = ld(f[3]);
            for (int e = 0; e < w; e++) upd_el(f[2], e, sc * sel(f[0], e), fb);
          }
          break;
        }
        case B_MATMUL: {
          const int r = in.r, c = in.c, kk = in.k;
          const bool fa = in.flags & 1, fb = in.flags & 2;
          if (all_zero(f[0], r * c)) { zero_first(f[1], r * kk, fa); zero_first(f[2], kk * c, fb); break; }
          // element by element, each update stored before the next element is computed
          // (the device's order)
          if (f[1] != -1)  // gA (r x k) += gZ (r x c) B^T
            for (int i = 0; i < r; i++)
              for (int q = 0; q < kk; q++) upd_el(f[1], i * kk + q, dot(f[0], i * c, 1, f[4], q * c, 1, c), fa);
          if (f[2] != -1)  // gB (k x c) += A^T gZ
            for (int q = 0; q < kk; q++)
              for (int j = 0; j < c; j++) upd_el(f[2], q * c + j, dot(f[3], q, kk, f[0], j, c, r), fb);
          break;
        }
        case B_INV: {
          const int n = in.r;
          const bool fa = in.flags & 1;
          if (f[1] == -1) break;
          if (all_zero(f[0], n * n)) { zero_first(f[1], n * n, fa); break; }
          std::vector<double> m((size_t)(n * n));  // M = gZ B^T, B the saved inverse
          for (int pp = 0; pp < n; pp++)
            for (int j = 0; j < n; j++) m[(size_t)(pp * n + j)] = dot(f[0], pp * n, 1, f[5], j * n, 1, n);
          for (int e = 0; e < n * n; e++) {  // gA -= B^T M
            const int i = e / n, j = e - i * n;
            double acc = el(f[5], i) * m[(size_t)j];
            for (int pp = 1; pp < n; pp++) acc = std::fma(el(f[5], pp * n + i), m[(size_t)(pp * n + j)], acc);
            upd_el(f[1], e, -acc, fa);
          }
          break;
        }
        case B_DET: case B_LOGDET: {
          const int n = in.r;
          const bool fa = in.flags & 1;
          if (f[1] == -1) break;
          const double g = slot(f[0]);
          if (is_zero(g)) { zero_first(f[1], n * n, fa); break; }
          const double fac = in.op == B_DET ? g * ld(f[5]) : g;
          for (int e = 0; e < n * n; e++) {
            const int i = e / n, j = e - i * n;
            upd_el(f[1], e, fac * el(f[6], j * n + i), fa);
          }
          break;
        }
        case B_TRACE: {
          const int n = in.r;
          if (f[1] == -1) break;
          const double g = slot(f[0]);
          zero_first(f[1], n * n, in.flags & 1);
          if (is_zero(g)) break;
          for (int i = 0; i < n; i++) sel(f[1], i * n + i) = sel(f[1], i * n + i) + g;
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
            const double q = f[6] != -1 ? div_by_rcp(g, ld(f[4]), ld(f[6])) : g / ld(f[4]);
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
    const Plan p = make_plan(b.t, stream != 2);  // stream 2: the value-only plan
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
