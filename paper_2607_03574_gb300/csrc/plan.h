// Device program ("plan") for tape replay, produced on the host from a Tape.
//
// The kernel interprets a linear instruction stream.  Every lane runs the same
// stream (the tape is shared by the population, section 3.5), so dispatch is
// uniform across a warp.  Per-lane values live in a slot file in shared memory,
// laid out [slot][thread]; the planner register-allocates slots by liveness.
// Values that the reverse sweep reads are either kept in slots until then (short
// tapes) or stored to an HBM workspace laid out [element][lane] (lane-contiguous,
// coalesced) and read back in the reverse sweep (long tapes).
#pragma once
#include <cstdint>
#include <string>
#include <vector>

#include "tape.h"

namespace ndvm {

// Operand reference: kind in bits 28..30, index in bits 0..27; element e of a
// matrix operand is ref + e.  -1 means "none".
enum RefKind : uint32_t { RK_SLOT = 0, RK_CONST = 1, RK_OBS = 2, RK_DOBS = 3, RK_SAVE = 4, RK_PARAM = 5 };
constexpr int32_t kRefIndexMask = 0x0fffffff;
inline int32_t mkref(uint32_t kind, int32_t idx) { return (int32_t)((kind << 28) | (uint32_t)idx); }
inline uint32_t ref_kind(int32_t r) { return ((uint32_t)r >> 28) & 7u; }
inline int32_t ref_index(int32_t r) { return r & kRefIndexMask; }

enum DOp : uint8_t {
  // ---- forward ----
  D_ADD = 1, D_SUB, D_MUL, D_DIV, D_POW,  // f0 out, f1 a, f2 b, f3 save; D_DIV with flags bit 4 (a
                    // division in a data-axis body): a / b by one correction step from 1/b correctly
                    // rounded (the IEEE division outside the safe exponent range), 1/b kept in f4
                    // aux slot / f5 aux save; without the bit, the IEEE division
  D_NEG, D_EXP, D_LOG, D_TANH, D_SQRT, D_ABS,  // f0 out, f1 a, f3 save
  D_SIN, D_COS,     // f0 out, f1 a, f3 save, f4 aux slot (the other trig value), f5 aux save
  D_POWI,           // f0 out, f1 a, f3 save, f7 n
  D_CMP,            // f0 out, f1 a, f2 b, k = comparison (0 lt, 1 le, 2 gt, 3 ge, 4 eq)
  D_SELECT,         // f0 out, f1 predicate, f2 a, f3 save, f4 b
  D_GATHER,         // f0 out, f1 args offset, f2 count (args: element refs), f3 save
  D_MADD, D_MSUB,   // f0 out, f1 a, f2 b, f3 save; r x c
  D_MSCALE,         // f0 out, f1 s, f2 A, f3 save; r x c
  D_MATMUL,         // f0 out, f1 A, f2 B, f3 save; r x c, inner k
  D_INV,            // f0 out, f1 A, f2 scratch (n >= 4), f3 save; n = r
  D_DET, D_LOGDET,  // f0 out, f1 A, f2 scratch (n >= 4), f3 save, f4 aux slot (inverse), f5 aux save; n = r
  D_TRACE,          // f0 out, f1 A; n = r
  // ---- data-axis regions ----
  D_ZERO,           // f0 slot, f1 count
  D_LOOP,           // f0 N, f1 stride, f2 base, f3 pc of the matching D_ENDLOOP
  D_ENDLOOP,        // f0 pc of the matching D_LOOP
  D_ACC,            // slot f0 += ref f1
  D_SEED,           // slot f0 = 1
  D_GREDUCE,        // f0 slot, f1 count: sum over the lane's thread group
  D_LOSS,           // loss[lane] = ref f0
  // ---- reverse ----  (f0 = adjoint of the output "gz"; targets f1/f2; flags bit0/bit1 = first
  //                     contribution to target 1/2, which stores instead of accumulating)
  B_ADD, B_SUB,     // f1 ga, f2 gb
  B_MUL,            // f1 ga, f2 gb, f3 pa, f4 pb
  B_DIV,            // f1 ga, f2 gb, f4 pb, f5 pz, f6 p(1/b): g / b by one correction step from 1/b
  B_POW,            // f1 ga, f2 gb, f3 pa, f4 pb, f5 pz
  B_NEG,            // f1 ga
  B_EXP, B_TANH,    // f1 ga, f5 pz
  B_LOG, B_ABS,     // f1 ga, f3 pa
  B_SQRT,           // f1 ga, f3 pa, f5 pz
  B_SIN, B_COS,     // f1 ga, f6 paux (cos x for sin, sin x for cos)
  B_POWI,           // f1 ga, f3 pa, f7 n
  B_SELECT,         // f1 ga, f2 gb, f3 pp
  B_GATHER,         // f1 args offset, f2 count (args: pairs target slot|-1, first flag)
  B_SCATTER,        // f1 ga, f2 count, f3 args offset (input element per output), f4 input width
  B_MADD, B_MSUB,   // f1 ga, f2 gb; r x c
  B_MSCALE,         // f1 gs, f2 gA, f3 ps, f4 pA; r x c
  B_MATMUL,         // f1 gA, f2 gB, f3 pA, f4 pB; r x c, inner k
  B_INV,            // f1 gA, f2 scratch, f5 pz; n = r
  B_DET,            // f1 gA, f5 pz, f6 pinv; n = r
  B_LOGDET,         // f1 gA, f6 pinv; n = r
  B_TRACE,          // f1 gA; n = r
  B_DSUM,           // f1 args offset, f2 count (args: triples target slot, first flag, partial slot)
  B_GRAD,           // grad[lane, f1] = slot f0 (or 0 if f0 < 0)
  // ---- workspace prefetch (reverse sweep of long tapes) ----
  D_LOAD,           // slot f0 = ref f1 (a constant, parameter, observation or workspace value)
  D_FETCH,          // k = count <= kFetchPairs; pairs (f0 workspace ref, f1 slot), (f2, f3), ...:
                    // asynchronous copies into slots; flags bit1: then commit the copies issued
                    // since the last commit as one group; bit0: then wait until at most n groups
                    // are pending, n = flags bits 2..4 (<= kFetchWindows); bit5: the sources are
                    // observations of the current data point (DOBS refs, inside a data-axis loop)
  // ---- fused multiply-add form of the cheap scalar rules ----
  D_FMA,            // slot f0 = (is_zero(slot f4) ? slot f3 : fma(+-slot f1, slot f2, slot f3)), f5 save;
                    // flags bit0 negates the first factor.  f4 is the zero-skip test (an adjoint
                    // whose contribution vanishes when it is exactly zero; the slot holding 1.0
                    // when there is none)
  D_FMA2,           // two D_FMA without saves in one record: (f0 dst, f1, f2, f3, f4 zero-skip)
                    // and (f5 dst, f6, f7, pad3, pad4 zero-skip); flags bit0 / bit1 negate the first
                    // factor of the first / second; bit2: the second's operands that name f0 read
                    // the first's result; bit3: saves, the first's workspace index in bytes
                    // (r, c, k) and the second's in (pad0, pad1, pad2), 24 bits little-endian,
                    // kNoSave24 for none
  D_NOPS
};

// Scalar instructions take slot operands only (constants, parameters, observations
// and workspace values reach them through D_LOAD or D_FETCH); true for the operand
// field `field` of opcode `op` whose value the kernel reads without decoding its kind.
bool slot_operand(int op, int field);

// Reverse instructions read their workspace values from slots that D_FETCH fills
// ahead of use: the reverse sweep is cut into windows of kFetchStride instructions,
// whose values are fetched kFetchWindows windows ahead, kFetchPairs per instruction.
constexpr int kFetchPairs = 4;
constexpr int kFetchStride = 16;
constexpr int kFetchWindows = 4;

// "no save" in the 24-bit save fields of D_FMA2
constexpr int32_t kNoSave24 = 0xFFFFFF;

// 48 bytes, 16-byte aligned (three 128-bit words; staged copies move 16-byte pieces).
struct alignas(16) DInst {
  uint8_t op = 0, r = 1, c = 1, k = 1;
  uint8_t flags = 0, pad0 = 0, pad1 = 0, pad2 = 0;
  int32_t f[8] = {-1, -1, -1, -1, -1, -1, -1, -1};
  int32_t pad3 = 0, pad4 = 0;
};
static_assert(sizeof(DInst) == 48, "DInst layout");

// Shared per-point values of a data-axis region.  The body nodes that depend on the data
// point but on no parameter are the same on every lane, so a derive plan computes them
// once per call (one lane per point) into an extended observation buffer:
//   [ obs[0 .. n_obs_min) | region blocks ],
// where region r's block, at n_obs_min + offset, holds columns [col][point] of N values:
// first copies of the point's observation columns 0 .. obs_cols-1, then the derived
// values.  The replay's loop over the region then reads column c of point d as
// observation (n_obs_min + offset) + c * N + d: base n_obs_min + offset, stride 1, and
// DOBS index c * N.
struct DeriveInfo {
  int64_t n_points = 0, stride = 0, base = 0;  // the region's points: obs[base + d*stride + k]
  int64_t offset = 0;                          // block offset after the copied observations
  int32_t obs_cols = 0;                        // observation columns copied into the block
  int32_t n_cols = 0;                          // all columns of the block
  double work = 0;                             // DFMA-equivalents per point
};

struct Plan {
  bool grad = false;          // has a reverse sweep
  bool spill = false;         // reverse reads primals from the HBM workspace
  bool has_regions = false;   // contains data-axis loops
  bool has_matrix = false;    // contains instructions over matrices
  int32_t n_slots = 0;        // per-lane slot file size (elements)
  int64_t n_save = 0;         // per-lane workspace elements
  int32_t n_params = 0;
  int64_t n_obs_min = 0;
  int32_t max_dobs = -1;      // largest DOBS column read (for validation)
  std::vector<DInst> code;
  // the same stream with adjacent independent D_FMA paired into D_FMA2 (for the staged
  // and element-split kernel variants; the plain variant runs `code`)
  std::vector<DInst> code_paired;
  std::vector<int32_t> args;
  std::vector<double> extra_consts;  // appended after the tape's constant pool
  // algorithmic cost per lane (for the roofline): DFMA-equivalents and saved bytes
  double work_fwd = 0, work_rev = 0;
  double n_ops_per_lane = 0;
  // shared per-point values (gradient plans of data-axis tapes): one forward-only plan
  // per region, whose lanes are the points (its parameters are the point's observation
  // record: params = obs + base, P = stride); derived_elems = size of the region blocks
  std::vector<Plan> derive;
  std::vector<DeriveInfo> derive_info;
  int64_t derived_elems = 0;
};

// Per-lane working space (slot elements) that an instruction needs beyond its operands,
// named by its field f2: the inverse's adjoint keeps M = gZ B^T there (n^2); Gauss-Jordan
// elimination (n >= 4) keeps [A | I] (2 n^2) or, for a determinant alone, A (n^2).
int scratch_elems(const DInst& d);

// Build the plan; throws BuildError on unsupported tapes.
Plan make_plan(const Tape& t, bool grad, int force_mode = -1 /* -1 auto, 0 keep, 1 spill */);

// Check every reference against the plan's own sizes (host-side, before upload).
bool validate_plan(const Plan& p, size_t n_consts, std::string& why);

}  // namespace ndvm
