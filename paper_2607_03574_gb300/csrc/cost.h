// Algorithmic FP64 work per tape primitive, in DFMA-equivalents (one FP64
// instruction issue = 1).  Arithmetic counts one per add, multiply or fused
// multiply-add; a first adjoint contribution that is a copy or a sign flip counts
// zero.  A function counts the FP64 instructions one call executes on GB300, counted
// by ncu (smsp__inst_executed_pipe_fp64 per call) on the cost probe
// (ndvm_measure_op_cost: four independent chains per thread on every SM, finite
// ordinary arguments), less the chain's one add or multiply: the replay's own exp 10
// and log 13 (fmath.cuh; the same counts in the source, and in ncu counts of
// single-function programs through the replay), and CUDA's tanh 24, sqrt 8, division 8,
// reciprocal 5, log 29.75 (inside pow's adjoint) and pow 84.  Each call's device time on the probe agrees with its
// instruction count within 5 %.  The replay's own sin (or cos) and sincos (fmath.cuh)
// execute 16 and 19 FP64 instructions (counted in the source; the probe's device time
// per call, 16.7 and 19.5 DFMA with the chain's add, agrees).  The roofline divides
// this work by the FP64 pipe's peak issue rate.
#pragma once
#include "tape.h"

namespace ndvm {
namespace cost {

constexpr double kExp = 10, kLog = 13, kSin = 16, kSinCos = 19, kTanh = 24, kSqrt = 8,
                 kRcp = 5, kPow = 84, kDiv = 8, kLogLib = 29.75;
// A division in a data-axis body takes 1/b from the hardware estimate and two Newton
// steps (kRcpNewton: four fused multiply-adds) and one correction step (a product and
// two fused multiply-adds, kDivStep); its reverse rule divides the adjoint by b with the
// forward sweep's reciprocal (kDivStep).  A lane-level division is the IEEE division
// (kDiv) in both sweeps.  The log's adjoint divides the same way as a body division.
constexpr double kDivStep = 3, kRcpNewton = 4;

// (the reciprocal of a determinant or pivot is the correctly rounded rcp)
inline double inv_cost(int n) {
  if (n == 1) return kRcp;
  if (n == 2) return 2 + kRcp + 4;           // det, 1/det, four scaled cofactors
  if (n == 3) return 18 + 3 + kRcp + 9;      // nine cofactors, det, 1/det, nine scalings
  return 2.0 * n * n * n + n * kRcp;        // elimination
}
inline double det_cost(int n) {
  if (n == 1) return 0;
  if (n == 2) return 2;
  if (n == 3) return 9;
  return (2.0 * n * n * n) / 3.0 + n * kRcp;
}

inline double fwd(int op, int r, int c, int imm, int n, bool with_aux) {
  const double e = (double)r * c;
  switch (op) {
    case OP_ADD: case OP_SUB: case OP_MUL: return 1;
    case OP_DIV: return with_aux ? kRcpNewton + kDivStep : kDiv;  // with_aux: a data-axis body
    case OP_POW: return kPow;
    case OP_NEG: case OP_ABS: case OP_SELECT: return 0;
    case OP_EXP: return kExp;
    case OP_LOG: return kLog;
    case OP_SIN: case OP_COS: return with_aux ? kSinCos : kSin;
    case OP_TANH: return kTanh;
    case OP_SQRT: return kSqrt;
    case OP_POWI: return imm > 1 ? imm - 1 : 0;
    case OP_LT: case OP_LE: case OP_GT: case OP_GE: case OP_EQ: return 1;
    case OP_MADD: case OP_MSUB: case OP_MSCALE: return e;
    case OP_MATMUL: return e * imm;
    case OP_INV: return inv_cost(n);
    case OP_DET: return with_aux ? inv_cost(n) : det_cost(n);
    case OP_LOGDET: return (with_aux ? inv_cost(n) : det_cost(n)) + kLog;
    case OP_TRACE: return n - 1;
    default: return 0;
  }
}

// a_init / b_init: the contribution is the first one to that input's adjoint
inline double rev(int op, int r, int c, int imm, int n, bool aa, bool ba, bool a_init, bool b_init, int extra) {
  const double e = (double)r * c;
  auto acc = [](bool active, bool init) { return active && !init ? 1.0 : 0.0; };
  switch (op) {
    case OP_ADD: case OP_SUB: return acc(aa, a_init) + acc(ba, b_init);
    case OP_NEG: return acc(aa, a_init);
    case OP_MUL: return (aa ? 1 : 0) + (ba ? 1 : 0);
    case OP_DIV: return (extra ? kDivStep : kDiv) + acc(aa, a_init) + (ba ? 1 : 0);  // extra: 1/b kept
    case OP_POW: return (aa ? kDiv + 2 : 0) + (ba ? kLogLib + 2 : 0);
    case OP_EXP: case OP_SIN: case OP_COS: case OP_ABS: return 1;
    case OP_TANH: return 2;
    case OP_LOG: return kRcpNewton + kDivStep + acc(aa, a_init);  // g / x
    case OP_SQRT: return kDiv + 1 + acc(aa, a_init);             // g / (2 z)
    case OP_POWI: return imm > 0 ? imm : 0;
    case OP_SELECT: return acc(aa, a_init) + acc(ba, b_init);
    case OP_MATFROM: return 0.0 + extra * 0.5;  // scattered copies and adds
    case OP_MREF: case OP_SUBMAT: case OP_TRANSPOSE: return a_init ? 0 : e;
    case OP_MADD: case OP_MSUB: return (aa && !a_init ? e : 0) + (ba && !b_init ? e : 0);
    case OP_MSCALE: return (aa ? e : 0) + (ba ? e : 0);
    case OP_MATMUL: return (aa ? e * imm : 0) + (ba ? e * imm : 0);
    case OP_INV: return 2.0 * n * n * n;
    case OP_DET: return 2.0 * n * n;
    case OP_LOGDET: return 1.0 * n * n;
    case OP_TRACE: return a_init ? 0 : n;
    case OP_DSUM: return 2.0 * extra;
    default: return 0;
  }
}

}  // namespace cost
}  // namespace ndvm
