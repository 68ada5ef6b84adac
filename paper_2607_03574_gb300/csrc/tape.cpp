// Tape construction, serialization and hashing (host side).
#include "tape.h"

#include <cstring>

#include "status.h"

namespace ndvm {

const char* op_name(int op) {
  static const char* names[OP_COUNT] = {
      "none", "const", "param", "obs", "dobs", "add", "sub", "mul", "div", "neg",
      "exp", "log", "sin", "cos", "tanh", "sqrt", "abs", "pow", "powi",
      "lt", "le", "gt", "ge", "eq", "select",
      "matfrom", "mref", "submat", "transpose", "madd", "msub", "mscale", "matmul",
      "inv", "det", "logdet", "trace", "dsum"};
  return (op >= 0 && op < OP_COUNT) ? names[op] : "?";
}

[[noreturn]] static void shape_error(const std::string& m) { throw BuildError{NDVM_E_SHAPE, m}; }

static void put_u16(std::vector<uint8_t>& o, uint16_t v) { o.push_back(v & 0xff); o.push_back(v >> 8); }
static void put_u32(std::vector<uint8_t>& o, uint32_t v) { for (int i = 0; i < 4; i++) o.push_back((v >> (8 * i)) & 0xff); }
static void put_u64(std::vector<uint8_t>& o, uint64_t v) { for (int i = 0; i < 8; i++) o.push_back((v >> (8 * i)) & 0xff); }

// Layout: "NDVMTAP1", u32 version(1), i32 n_params, i64 n_obs_min, i32 loss,
// u32 n_nodes, u32 n_consts, u32 n_args, nodes (op u16, rows u8, cols u8,
// a b c imm imm2 i32), consts (IEEE-754 bits u64), args (i32).
std::vector<uint8_t> Tape::serialize() const {
  std::vector<uint8_t> o;
  o.reserve(48 + nodes.size() * 24 + consts.size() * 8 + args.size() * 4);
  const char magic[8] = {'N', 'D', 'V', 'M', 'T', 'A', 'P', '1'};
  o.insert(o.end(), magic, magic + 8);
  put_u32(o, 1);
  put_u32(o, (uint32_t)n_params);
  put_u64(o, (uint64_t)n_obs_min);
  put_u32(o, (uint32_t)loss);
  put_u32(o, (uint32_t)nodes.size());
  put_u32(o, (uint32_t)consts.size());
  put_u32(o, (uint32_t)args.size());
  for (const Node& n : nodes) {
    put_u16(o, n.op);
    o.push_back(n.rows);
    o.push_back(n.cols);
    put_u32(o, (uint32_t)n.a);
    put_u32(o, (uint32_t)n.b);
    put_u32(o, (uint32_t)n.c);
    put_u32(o, (uint32_t)n.imm);
    put_u32(o, (uint32_t)n.imm2);
  }
  for (double d : consts) {
    uint64_t bits;
    std::memcpy(&bits, &d, 8);
    put_u64(o, bits);
  }
  for (int32_t a : args) put_u32(o, (uint32_t)a);
  return o;
}

uint64_t Tape::hash() const {
  std::vector<uint8_t> s = serialize();
  uint64_t h = 1469598103934665603ull;  // FNV-1a 64 offset basis
  for (uint8_t c : s) {
    h ^= c;
    h *= 1099511628211ull;  // FNV prime
  }
  return h;
}

int Builder::push(const Node& n) {
  if (t.nodes.size() >= max_nodes) throw BuildError{NDVM_E_UNSUPPORTED, "trace exceeds the node budget"};
  t.nodes.push_back(n);
  return (int)t.nodes.size() - 1;
}

static uint64_t const_key(int r, int c, const double* v) {
  // FNV over shape and bits; collisions are resolved by comparing values
  uint64_t h = 1469598103934665603ull;
  auto mix = [&](uint64_t x) { for (int i = 0; i < 8; i++) { h ^= (x >> (8 * i)) & 0xff; h *= 1099511628211ull; } };
  mix((uint64_t)r); mix((uint64_t)c);
  for (int i = 0; i < r * c; i++) { uint64_t b; std::memcpy(&b, v + i, 8); mix(b); }
  return h;
}

int Builder::konst_matrix(int r, int c, const double* v) {
  if (r < 1 || c < 1 || r > kMaxDim || c > kMaxDim) shape_error("constant matrix shape outside 1..64");
  uint64_t key = const_key(r, c, v);
  auto it = const_ids_.find(key);
  if (it != const_ids_.end()) {
    const Node& n = t.nodes[it->second];
    if (n.rows == r && n.cols == c && std::memcmp(&t.consts[n.imm], v, sizeof(double) * r * c) == 0) return it->second;
  }
  Node n;
  n.op = OP_CONST; n.rows = (uint8_t)r; n.cols = (uint8_t)c; n.imm = (int32_t)t.consts.size();
  t.consts.insert(t.consts.end(), v, v + r * c);
  int id = push(n);
  const_ids_[key] = id;
  return id;
}

int Builder::konst(double v) { return konst_matrix(1, 1, &v); }

int Builder::param(int k) {
  if (k < 0 || k >= t.n_params) throw BuildError{NDVM_E_INVALID_ARG, "parameter index out of range"};
  auto it = param_ids_.find(k);
  if (it != param_ids_.end()) return it->second;
  Node n;
  n.op = OP_PARAM; n.imm = k;
  int id = push(n);
  param_ids_[k] = id;
  return id;
}

int Builder::obs(int64_t k, int n) {
  if (k < 0 || n < 1 || n > kMaxDim || k > (int64_t)0x7fffffff - n) throw BuildError{NDVM_E_INVALID_ARG, "observation index out of range"};
  int64_t key = k * 32 + n;
  auto it = obs_ids_.find(key);
  if (it != obs_ids_.end()) return it->second;
  Node nd;
  nd.op = OP_OBS; nd.rows = (uint8_t)n; nd.cols = 1; nd.imm = (int32_t)k;
  if (k + n > t.n_obs_min) t.n_obs_min = k + n;
  int id = push(nd);
  obs_ids_[key] = id;
  return id;
}

int Builder::dobs(int k) {
  if (!region_open()) throw BuildError{NDVM_E_PARSE, "dobs outside data-sum"};
  if (k < 0) throw BuildError{NDVM_E_INVALID_ARG, "dobs column must be >= 0"};
  auto it = dobs_ids_.find(k);
  if (it != dobs_ids_.end()) return it->second;
  Node n;
  n.op = OP_DOBS; n.imm = k;
  int id = push(n);
  dobs_ids_[k] = id;
  return id;
}

int Builder::unary(Op op, int a) {
  if (!is_scalar(a)) shape_error(std::string(op_name(op)) + " of a matrix");
  Node n;
  n.op = op; n.a = a;
  return push(n);
}

int Builder::binary(Op op, int a, int b) {
  if (!is_scalar(a) || !is_scalar(b)) shape_error(std::string(op_name(op)) + " of a matrix");
  Node n;
  n.op = op; n.a = a; n.b = b;
  return push(n);
}

int Builder::powi(int a, int e) {
  if (!is_scalar(a)) shape_error("pow of a matrix");
  if (e < 0 || e > 64) throw BuildError{NDVM_E_UNSUPPORTED, "integer exponent outside 0..64"};
  Node n;
  n.op = OP_POWI; n.a = a; n.imm = e;
  return push(n);
}

int Builder::compare(Op op, int a, int b) { return binary(op, a, b); }

int Builder::select(int p, int a, int b) {
  if (!is_scalar(a) || !is_scalar(b)) shape_error("a branch on a numeric test must produce a scalar");
  Node n;
  n.op = OP_SELECT; n.a = p; n.b = a; n.c = b;
  return push(n);
}

int Builder::matfrom(int r, int c, const std::vector<int>& el) {
  if (r < 1 || c < 1 || r > kMaxDim || c > kMaxDim) shape_error("matrix shape outside 1..64");
  if ((int)el.size() != r * c) shape_error("matrix element count mismatch");
  bool allc = true;
  for (int e : el) {
    if (!is_scalar(e)) shape_error("matrix element is not a scalar");
    if (!is_const(e)) allc = false;
  }
  if (allc) {  // pure data movement of constants: fold
    std::vector<double> v(r * c);
    for (int i = 0; i < r * c; i++) v[i] = const_value(el[i]);
    return konst_matrix(r, c, v.data());
  }
  Node n;
  n.op = OP_MATFROM; n.rows = (uint8_t)r; n.cols = (uint8_t)c; n.imm = (int32_t)t.args.size();
  t.args.insert(t.args.end(), el.begin(), el.end());
  return push(n);
}

int Builder::mref(int a, int i, int j) {
  if (i < 0 || j < 0 || i >= rows(a) || j >= cols(a)) shape_error("mref index outside the matrix");
  int e = i * cols(a) + j;
  if (is_const(a)) return konst(const_value(a, e));
  if (rows(a) == 1 && cols(a) == 1) return a;
  Node n;
  n.op = OP_MREF; n.a = a; n.imm = e;
  return push(n);
}

int Builder::submat(int a, int r0, int nr, int c0, int nc) {
  if (r0 < 0 || c0 < 0 || nr < 1 || nc < 1 || r0 + nr > rows(a) || c0 + nc > cols(a)) shape_error("submatrix outside the matrix");
  if (is_const(a)) {
    std::vector<double> v(nr * nc);
    for (int i = 0; i < nr; i++)
      for (int j = 0; j < nc; j++) v[i * nc + j] = const_value(a, (r0 + i) * cols(a) + c0 + j);
    return konst_matrix(nr, nc, v.data());
  }
  Node n;
  n.op = OP_SUBMAT; n.a = a; n.rows = (uint8_t)nr; n.cols = (uint8_t)nc; n.imm = r0; n.imm2 = c0;
  return push(n);
}

int Builder::transpose(int a) {
  int r = rows(a), c = cols(a);
  if (is_const(a)) {
    std::vector<double> v(r * c);
    for (int i = 0; i < r; i++)
      for (int j = 0; j < c; j++) v[j * r + i] = const_value(a, i * c + j);
    return konst_matrix(c, r, v.data());
  }
  Node n;
  n.op = OP_TRANSPOSE; n.a = a; n.rows = (uint8_t)c; n.cols = (uint8_t)r;
  return push(n);
}

int Builder::madd(Op op, int a, int b) {
  if (rows(a) != rows(b) || cols(a) != cols(b)) shape_error("m+/m- shape mismatch");
  Node n;
  n.op = op; n.a = a; n.b = b; n.rows = (uint8_t)rows(a); n.cols = (uint8_t)cols(a);
  return push(n);
}

int Builder::mscale(int s, int a) {
  if (!is_scalar(s)) shape_error("mscale needs a scalar first argument");
  Node n;
  n.op = OP_MSCALE; n.a = s; n.b = a; n.rows = (uint8_t)rows(a); n.cols = (uint8_t)cols(a);
  return push(n);
}

int Builder::matmul(int a, int b) {
  if (cols(a) != rows(b)) shape_error("matmul shape mismatch");
  Node n;
  n.op = OP_MATMUL; n.a = a; n.b = b; n.rows = (uint8_t)rows(a); n.cols = (uint8_t)cols(b); n.imm = cols(a);
  return push(n);
}

int Builder::matfun(Op op, int a) {
  if (rows(a) != cols(a)) shape_error("square matrix required");
  if ((op == OP_INV || op == OP_DET || op == OP_LOGDET) && rows(a) > 8)
    throw BuildError{NDVM_E_UNSUPPORTED, "inverse/determinant above 8x8"};
  Node n;
  n.op = op; n.a = a;
  if (op == OP_INV) { n.rows = (uint8_t)rows(a); n.cols = (uint8_t)rows(a); }
  return push(n);
}

void Builder::begin_region() {
  if (region_open()) throw BuildError{NDVM_E_UNSUPPORTED, "nested data-sum"};
  region_begin_ = (int64_t)t.nodes.size();
  dobs_ids_.clear();
}

int Builder::end_region(int result, int64_t npts, int64_t stride, int64_t base) {
  if (!region_open()) throw BuildError{NDVM_E_PARSE, "data-sum end without begin"};
  if (!is_scalar(result)) shape_error("data-sum body must produce a scalar");
  if (npts < 0 || stride < 0 || base < 0 || npts > 0x7fffffff || stride > 0x7fffffff || base > 0x7fffffff)
    throw BuildError{NDVM_E_INVALID_ARG, "data-sum sizes out of range"};
  Node n;
  n.op = OP_DSUM;
  n.a = (int32_t)region_begin_;
  n.b = (int32_t)t.nodes.size();
  n.c = result;
  n.imm = (int32_t)npts;
  n.imm2 = (int32_t)t.args.size();
  t.args.push_back((int32_t)stride);
  t.args.push_back((int32_t)base);
  // observations the region reads
  int maxk = -1;
  for (int i = n.a; i < n.b; i++)
    if (t.nodes[i].op == OP_DOBS && t.nodes[i].imm > maxk) maxk = t.nodes[i].imm;
  if (maxk >= 0 && npts > 0) {
    int64_t need = base + (npts - 1) * stride + maxk + 1;
    if (need > t.n_obs_min) t.n_obs_min = need;
  }
  // body values other than leaves may not escape the region; leaves are interned
  // process-wide, so drop region-local observation leaves from the intern table
  region_begin_ = -1;
  dobs_ids_.clear();
  return push(n);
}

}  // namespace ndvm
