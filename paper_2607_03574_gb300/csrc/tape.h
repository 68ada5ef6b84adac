// Tape IR shared by the host front ends, the planner and the C ABI.
//
// A tape is the realized numeric trace of one structural walk (paper section 3.4:
// one node per differentiable numeric primitive, nothing for structural work).
// Nodes are in SSA form: node i defines value i.  Leaves (constants, parameters,
// observations) carry no arithmetic; every other node is one primitive of the
// Appendix C table (plus tanh, neg, select, compare, matrix add/sub/scale).
//
// A data-axis region (section 3.5: data points as one of the batch axes) is a contiguous run of
// body nodes [a, b) followed by a DSUM node that sums the body result over N data
// points; inside the body, DOBS k reads obs[base + d*stride + k] for point d.
#pragma once
#include <cstddef>
#include <cstdint>
#include <string>
#include <unordered_map>
#include <vector>

namespace ndvm {

enum Op : uint16_t {
  OP_NONE = 0,
  // leaves
  OP_CONST, OP_PARAM, OP_OBS, OP_DOBS,
  // scalar arithmetic
  OP_ADD, OP_SUB, OP_MUL, OP_DIV, OP_NEG,
  OP_EXP, OP_LOG, OP_SIN, OP_COS, OP_TANH, OP_SQRT, OP_ABS, OP_POW, OP_POWI,
  // per-lane control (lane masks, section 3.5)
  OP_LT, OP_LE, OP_GT, OP_GE, OP_EQ, OP_SELECT,
  // small fixed-size matrices
  OP_MATFROM, OP_MREF, OP_SUBMAT, OP_TRANSPOSE,
  OP_MADD, OP_MSUB, OP_MSCALE, OP_MATMUL,
  OP_INV, OP_DET, OP_LOGDET, OP_TRACE,
  // data-axis sum
  OP_DSUM,
  OP_COUNT
};

const char* op_name(int op);

// Largest matrix dimension (rows, columns, inner size of a product); inverse and
// determinant take n <= 8.
constexpr int kMaxDim = 64;

// 24 bytes, serialized field by field in little-endian order.
struct Node {
  uint16_t op = 0;
  uint8_t rows = 1, cols = 1;  // output shape
  int32_t a = -1, b = -1, c = -1;  // input node ids (or region bounds)
  int32_t imm = 0, imm2 = 0;       // immediates (see below)
};
// Immediates by op:
//   CONST    imm = offset into consts (rows*cols values, row-major)
//   PARAM    imm = parameter index
//   OBS      imm = first observation index (rows x 1 for a vector)
//   DOBS     imm = column k within the data point
//   POWI     imm = integer exponent (0..64)
//   MATFROM  imm = offset into args, rows*cols element node ids
//   MREF     imm = element index in the input
//   SUBMAT   imm = first row, imm2 = first column
//   MATMUL   imm = inner dimension
//   SELECT   a = predicate, b = value if true, c = value if false
//   DSUM     a = first body node, b = one past the last body node, c = body result,
//            imm = N points, imm2 = offset into args: (stride, base)

struct Tape {
  int32_t n_params = 0;
  int64_t n_obs_min = 0;       // observations the program reads (highest index + 1)
  int32_t loss = -1;           // node id of the loss (a scalar)
  std::vector<Node> nodes;
  std::vector<double> consts;  // constant pool
  std::vector<int32_t> args;   // operand lists

  std::vector<uint8_t> serialize() const;
  uint64_t hash() const;       // FNV-1a 64 of serialize()
};

// Tape construction with interning of leaves.  All shape checks happen here.
class Builder {
 public:
  Tape t;
  std::string err;

  int konst(double v);
  int konst_matrix(int r, int c, const double* v);
  int param(int k);
  int obs(int64_t k, int n);  // n == 1: scalar; n > 1: n x 1 column
  int dobs(int k);
  int unary(Op op, int a);
  int binary(Op op, int a, int b);
  int powi(int a, int n);
  int compare(Op op, int a, int b);
  int select(int p, int a, int b);
  int matfrom(int r, int c, const std::vector<int>& el);
  int mref(int a, int i, int j);
  int submat(int a, int r0, int nr, int c0, int nc);
  int transpose(int a);
  int madd(Op op, int a, int b);
  int mscale(int s, int a);
  int matmul(int a, int b);
  int matfun(Op op, int a);  // INV, DET, LOGDET, TRACE

  // data-axis regions
  bool region_open() const { return region_begin_ >= 0; }
  void begin_region();
  int end_region(int result, int64_t n, int64_t stride, int64_t base);

  int rows(int v) const { return t.nodes[v].rows; }
  int cols(int v) const { return t.nodes[v].cols; }
  bool is_scalar(int v) const { return rows(v) == 1 && cols(v) == 1; }
  bool is_const(int v) const { return t.nodes[v].op == OP_CONST; }
  double const_value(int v, int e = 0) const { return t.consts[t.nodes[v].imm + e]; }

  size_t max_nodes = 50u * 1000u * 1000u;  // trace budget

 private:
  int push(const Node& n);
  int64_t region_begin_ = -1;
  std::unordered_map<uint64_t, int> const_ids_;
  std::unordered_map<int, int> param_ids_;
  std::unordered_map<int64_t, int> obs_ids_;
  std::unordered_map<int, int> dobs_ids_;
};

// Front ends: return 0 on success, else fill err.
int trace_scheme(const char* text, size_t len, Builder& b, std::string& err);
int trace_bytecode(const char* text, size_t len, Builder& b, std::string& err);

struct BuildError {
  int code;
  std::string msg;
};

}  // namespace ndvm
