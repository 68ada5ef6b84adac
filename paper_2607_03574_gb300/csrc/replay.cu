// Tape replay on the GPU (sm_103a): forward sweep, reverse adjoint sweep and
// per-lane loss for a population of parameter lanes (paper sections 3.4-3.5,
// Appendix C).
//
// Execution model.  Every lane runs the same instruction stream (the tape is
// shared by the population), so instruction fetch and dispatch are uniform across
// a warp; the stream is read through L1 or, for long loop-free streams, staged in
// shared memory in double-buffered chunks.  A group of G consecutive threads serves
// one lane: for tapes with data-axis regions the group splits the lane's data points
// (each thread has its own slot column; partial sums are reduced with warp
// shuffles); for matrix tapes the group shares the lane's slot column and splits
// each matrix instruction's elements.  Slot files live in shared memory, laid out
// [slot][thread] (or [slot][lane]) so a warp touches consecutive elements.  Forward
// values read by the reverse sweep are either kept in slots (short tapes) or stored
// to the workspace as [element][lane] -- each warp store/load is one contiguous,
// coalesced run -- and copied back into slots ahead of use in the reverse sweep.
//
// GB300 note: FP64 issues at about 1/73 of the FP32 rate (one warp instruction per
// 64 cycles per scheduler by the unit count, one per 76 in a saturated stream), and a
// dependent FP64 operation waits about 64 cycles.  A warp instruction with lanes
// predicated off still takes its full slot.
// With enough warps the FP64 pipe binds; with few lanes (one warp per scheduler)
// each lane's serial chain and the interpreter's own instructions set the time.
// The cheap scalar rules therefore take a dispatch-free fused multiply-add path.
#include <cuda_runtime.h>

#include <cmath>
#include <cstdint>
#include <map>
#include <mutex>

#include "ndvm.h"
#include "plan.h"
#include "replay.h"
#include "fmath.cuh"

namespace ndvm {
namespace {

// operand view: element e is p[e * s] (the host keeps e * s within 32 bits)
template <typename T>
struct Opnd {
  const T* p;
  int s;
  __device__ __forceinline__ T operator[](int e) const { return p[e * s]; }
  __device__ __forceinline__ const T* at(int e) const { return p + e * s; }
};

template <typename T> __device__ __forceinline__ T neg_zero() { return -(T)0; }

// s + a[0] b[0] + a[sa] b[sb] + ... over n terms, accumulated left to right with fma;
// unrolled for n <= 8 so that all operand loads issue before the chain starts.  Started
// from s = -0 it is the plain dot product (fma(a, b, -0) rounds a * b exactly as a
// multiplication does, signed zeros included); started from an adjoint, the update
// folds into the chain instead of costing a separate addition.
template <typename T, int K>
__device__ __forceinline__ T dot_fixed(const T* a, int sa, const T* b, int sb, T s) {
  T av[K], bv[K];
#pragma unroll
  for (int q = 0; q < K; q++) { av[q] = a[q * sa]; bv[q] = b[q * sb]; }
#pragma unroll
  for (int q = 0; q < K; q++) s = fma(av[q], bv[q], s);
  return s;
}
// WIDE: the long products' eight-term blocks (the element-split variants, whose matrices
// reach 64 x 64); the other variants keep the two-term loop and its smaller register
// footprint.  Both sum the same terms in the same chains.
template <typename T, bool WIDE = true>
__device__ __forceinline__ T dot(const T* a, int sa, const T* b, int sb, int n, T s) {
  switch (n) {
    case 1: return fma(a[0], b[0], s);
    case 2: return dot_fixed<T, 2>(a, sa, b, sb, s);
    case 3: return dot_fixed<T, 3>(a, sa, b, sb, s);
    case 4: return dot_fixed<T, 4>(a, sa, b, sb, s);
    case 5: return dot_fixed<T, 5>(a, sa, b, sb, s);
    case 6: return dot_fixed<T, 6>(a, sa, b, sb, s);
    case 7: return dot_fixed<T, 7>(a, sa, b, sb, s);
    case 8: return dot_fixed<T, 8>(a, sa, b, sb, s);
    default: {
      // long products (n > 8): even and odd terms in two chains, joined at the end, so
      // that each chain's dependent latency is half the product's
      // (eight terms at a time with every load issued first; the even and odd terms keep
      // their chains, so the sums are the same to the last bit)
      T s1 = neg_zero<T>();
      int q = 0;
      for (; WIDE && q + 8 <= n; q += 8) {
        T av[8], bv[8];
#pragma unroll
        for (int u = 0; u < 8; u++) { av[u] = a[(q + u) * sa]; bv[u] = b[(q + u) * sb]; }
#pragma unroll
        for (int u = 0; u < 8; u += 2) {
          s = fma(av[u], bv[u], s);
          s1 = fma(av[u + 1], bv[u + 1], s1);
        }
      }
      for (; q + 1 < n; q += 2) {
        s = fma(a[q * sa], b[q * sb], s);
        s1 = fma(a[(q + 1) * sa], b[(q + 1) * sb], s1);
      }
      if (q < n) s = fma(a[q * sa], b[q * sb], s);
      return s + s1;
    }
  }
}

// n / c for 0 <= n < 4096 and 1 <= c <= 255 without a division instruction (an integer
// division by a run-time value compiles to a reciprocal sequence on the conversion and
// special-function units): q = (n m) >> 20 with m = ceil(2^20 / c).  With
// m c = 2^20 + d, 0 <= d < c, n m / 2^20 = n/c + n d / (c 2^20), and the excess stays
// below 1/c, the least distance from n/c up to the next integer, while n c < 2^20.
// Matrices are at most 64 x 64 (kMaxDim), so element indices stay below 4096, and
// n m < 2^32.
struct DivTable {
  uint32_t m[256];
  constexpr DivTable() : m() {
    for (uint32_t c = 1; c < 256; c++) m[c] = ((1u << 20) + c - 1) / c;
  }
};
__constant__ DivTable kDivTable = DivTable();
__device__ __forceinline__ uint32_t div_magic(int c) { return kDivTable.m[c]; }
__device__ __forceinline__ int divq(int n, uint32_t m) { return (int)(((uint32_t)n * m) >> 20); }

// walks a thread's elements e = first, first + step, ... of a matrix with c columns
// as (row, column) pairs without a division per element
struct RowCol {
  int i, j;
  uint32_t m;  // div_magic(c)
  __device__ __forceinline__ RowCol(int first, int c) : m(div_magic(c)) {
    i = divq(first, m);
    j = first - i * c;
  }
  __device__ __forceinline__ void next(int step, int c) {
    j += step;
    const int q = divq(j, m);
    i += q;
    j -= q * c;
  }
};

template <typename T> __device__ __noinline__ void add_to(T* q, T v) { *q = *q + v; }

// BRANCH_ADD: accumulate through a call behind a real branch (see upd)
template <typename T, bool SHARED, bool BRANCH_ADD>
struct Lane {
  T* sbase;           // this thread's slot column: element s of the slot file is sbase[s * ss]
  int ss;             // slot row stride in elements
  int eg, emask;      // SHARED: this thread writes the elements e with (e & emask) == eg
  const T* consts;
  const T* obs;
  const T* params;
  T* save;
  int64_t lane, col, save_ld, dbase;
  int P;

  __device__ __forceinline__ Opnd<T> rd(int32_t ref) const {
    const uint32_t kind = ((uint32_t)ref >> 28) & 7u;
    const int32_t idx = ref & kRefIndexMask;
    if (kind == RK_SLOT) return {sbase + idx * ss, ss};
    switch (kind) {
      case RK_CONST: return {consts + idx, 1};
      case RK_OBS: return {obs + idx, 1};
      case RK_DOBS: return {obs + dbase + idx, 1};
      case RK_SAVE: return {save + (int64_t)idx * save_ld + col, (int)save_ld};
      default: return {params + lane * P + idx, 1};
    }
  }
  __device__ __forceinline__ T ld(int32_t ref) const {
    if (((uint32_t)ref >> 28) == RK_SLOT) return sbase[ref * ss];
    return rd(ref)[0];
  }
  // workspace element of this lane (a reference of kind RK_SAVE)
  __device__ __forceinline__ const T* savep(int32_t ref) const { return save + (int64_t)(ref & kRefIndexMask) * save_ld + col; }
  // operand of a scalar instruction: always a slot (the planner's load-store form)
  __device__ __forceinline__ T lds(int32_t ref) const { return sbase[ref * ss]; }
  __device__ __forceinline__ bool own(int e) const { return SHARED ? ((e & emask) == eg) : true; }
  __device__ __forceinline__ int step() const { return SHARED ? emask + 1 : 1; }
  __device__ __forceinline__ int first() const { return SHARED ? eg : 0; }
  // slot references only
  __device__ __forceinline__ T* wp(int32_t ref) const { return sbase + (ref & kRefIndexMask) * ss; }
  __device__ __forceinline__ T sl(int32_t ref, int e) const { return wp(ref)[e * ss]; }
  __device__ __forceinline__ void st(int32_t ref, int e, T v) const {
    if (own(e)) wp(ref)[e * ss] = v;
  }
  // adjoint update: the first contribution stores, later ones accumulate.  In the plain
  // variant (BRANCH_ADD, the FP64-bound data-axis tapes) the accumulation is a call
  // behind a real branch: inlined, the add is predicated and issues (all lanes off) on
  // every first contribution, a full FP64 slot on GB300, and most targets of an
  // expression tree get one contribution only; on a serial chain (the staged variant)
  // the call's latency costs more than the slot
  __device__ __forceinline__ void upd(int32_t ref, int e, T v, bool first) const {
    if (own(e)) upd_mine(ref, e, v, first);
  }
  // adjoint update by a product a * b: the first contribution stores it (rounded as a
  // multiplication); later ones fold it into the sum with one fused multiply-add
  __device__ __forceinline__ void upd_fma(int32_t ref, int e, T a, T b, bool first) const {
    if (own(e)) upd_fma_mine(ref, e, a, b, first);
  }
  __device__ __forceinline__ void save_out(int32_t sidx, int e, T v) const {
    if (sidx >= 0 && own(e)) save[(int64_t)(sidx + e) * save_ld + col] = v;
  }
  // The element loops (e = first(), first() + step(), ...) visit only the thread's own
  // elements: their writes skip the ownership test.
  __device__ __forceinline__ void st_mine(int32_t ref, int e, T v) const { wp(ref)[e * ss] = v; }
  __device__ __forceinline__ void save_mine(int32_t sidx, int e, T v) const {
    if (sidx >= 0) save[(int64_t)(sidx + e) * save_ld + col] = v;
  }
  __device__ __forceinline__ void upd_mine(int32_t ref, int e, T v, bool first) const {
    T* q = wp(ref) + e * ss;
    if (!BRANCH_ADD) *q = first ? v : *q + v;
    else if (first) *q = v;
    else add_to(q, v);
  }
  __device__ __forceinline__ void upd_fma_mine(int32_t ref, int e, T a, T b, bool first) const {
    T* q = wp(ref) + e * ss;
    *q = fma(a, b, first ? -(T)0 : *q);
  }
};

template <typename T> __device__ __forceinline__ T clamp_eps() { return (T)1e-8; }

// Tests on IEEE bit patterns run on the integer pipes, leaving the FP64 pipe to
// arithmetic (fbits keeps the compiler from turning them into FP64 compares).
// is_zero: +0 or -0.  gt_eps: x > 1e-8 with NaN false (IEEE order).
__device__ __forceinline__ bool is_zero(double x) { return (fbits(x) << 1) == 0; }
__device__ __forceinline__ bool is_zero(float x) { return (__float_as_uint(x) << 1) == 0u; }
__device__ __forceinline__ bool gt_eps(double x) {
  const long long b = fbits(x);
  return b > __double_as_longlong(1e-8) && (b & 0x7fffffffffffffffLL) <= 0x7ff0000000000000LL;
}
__device__ __forceinline__ bool gt_eps(float x) {
  const int b = __float_as_int(x);
  return b > __float_as_int(1e-8f) && (b & 0x7fffffff) <= 0x7f800000;
}

// x with its sign bit flipped when neg is set (IEEE negation, exact for every value)
__device__ __forceinline__ double flip_sign(double x, unsigned neg) {
  return __longlong_as_double(fbits(x) ^ ((long long)neg << 63));
}
__device__ __forceinline__ float flip_sign(float x, unsigned neg) {
  return __int_as_float(__float_as_int(x) ^ (int)(neg << 31));
}

// a^n by left-to-right repeated multiplication, and n a^(n-1) (the base adjoint of an
// integer power): small n take straight-line code with literal factors (a loop with a
// run-time trip count compiles to predicated multiplies, and converting n to a float
// costs an FP64 slot); the same operations in the same order either way
template <typename T> __device__ __forceinline__ T powi_loop(T a, int n) {
  T z = a;
#pragma unroll 1
  for (int i = 1; i < n; i++) z = z * a;
  return z;
}
template <typename T> __device__ __forceinline__ T powi_rep(T a, int n) {
  switch (n) {
    case 0: return (T)1;
    case 1: return a;
    case 2: return a * a;
    case 3: return (a * a) * a;
    case 4: return ((a * a) * a) * a;
    default: return powi_loop(a, n);
  }
}
template <typename T> __device__ __forceinline__ T powi_deriv(T a, int n) {  // n >= 1
  switch (n) {
    case 1: return (T)1 * (T)1;
    case 2: return (T)2 * a;
    case 3: return (T)3 * (a * a);
    case 4: return (T)4 * ((a * a) * a);
    default: return (T)n * powi_loop(a, n - 1);
  }
}

// correctly rounded reciprocal: the value of the IEEE division 1 / x, at lower cost
__device__ __forceinline__ double rcp_rn(double x) { return __drcp_rn(x); }
__device__ __forceinline__ float rcp_rn(float x) { return __frcp_rn(x); }

// a / b from r, the correctly rounded reciprocal of b, by one correction step
// (Markstein): q = a r, e = a - b q (exact by fma), q + r e.  The step is taken where a,
// b and the quotient lie well inside the normal range (exponents within +-500 for double,
// +-60 for float, zeros, infinities and NaNs excluded); elsewhere the IEEE division.
__device__ __forceinline__ bool div_step_ok(double a, double b) {
  const unsigned ea = (unsigned)(fbits(a) >> 52) & 0x7ffu;
  const unsigned eb = (unsigned)(fbits(b) >> 52) & 0x7ffu;
  return ea - 523u <= 1000u && eb - 523u <= 1000u;
}
__device__ __forceinline__ bool div_step_ok(float a, float b) {
  const unsigned ea = (__float_as_uint(a) >> 23) & 0xffu, eb = (__float_as_uint(b) >> 23) & 0xffu;
  return ea - 67u <= 120u && eb - 67u <= 120u;
}
// the IEEE division and the correctly rounded reciprocal as calls (rarely taken paths;
// see fmath.cuh's slow paths)
template <typename T> __device__ __noinline__ T slow_div(T a, T b) { return a / b; }
template <typename T> __device__ __noinline__ T slow_rcp(T b) { return rcp_rn(b); }

// 1/b for b with an exponent within +-500 (div_step_ok): the hardware estimate
// (rcp.approx.ftz.f64, off the FP64 pipe) refined by two Newton-Raphson steps
// y <- y + y (1 - b y), each doubling its correct bits; 4 FP64 instructions and no
// special-case code.  The result is within a hair of half an ulp, which is what the
// correction step of a division needs.
__device__ __forceinline__ double rcp_newton(double b) {
  double y;
  asm("rcp.approx.ftz.f64 %0, %1;" : "=d"(y) : "d"(b));
  double e = fma(-b, y, 1.0);
  y = fma(y, e, y);
  e = fma(-b, y, 1.0);
  return fma(y, e, y);
}
__device__ __forceinline__ float rcp_newton(float b) { return __frcp_rn(b); }

// a / b and 1/b (into *r): in the safe range by the Newton reciprocal and one correction
// step, else the IEEE division and the correctly rounded reciprocal
template <typename T>
__device__ __forceinline__ T div_rcp(T a, T b, T* r);
template <typename T>
__device__ __forceinline__ T div_rcp_q(T a, T b) {  // a / b alone
  T r;
  return div_rcp(a, b, &r);
}
template <typename T>
__device__ __forceinline__ T div_rcp(T a, T b, T* r) {
  if (!div_step_ok(a, b)) {
    *r = slow_rcp(b);
    return slow_div(a, b);
  }
  const T y = rcp_newton(b);
  *r = y;
  const T q = a * y;
  return fma(y, fma(-b, q, a), q);
}
template <typename T>
__device__ __forceinline__ T div_by_rcp(T a, T b, T r) {
  if (!div_step_ok(a, b)) return slow_div(a, b);
  const T q = a * r;
  return fma(r, fma(-b, q, a), q);
}

// Determinants and inverses to 3 x 3 in closed form, element by element: a lane's
// thread group splits an inverse's elements like those of any other matrix result,
// and every element has the same arithmetic whichever thread computes it.
// cofactor of element (r, s) of a 3 x 3 matrix (the cyclic form carries the sign)
template <typename T>
__device__ __forceinline__ T cof3(const Opnd<T>& A, int r, int s) {
  const int r1 = r == 2 ? 0 : r + 1, r2 = r == 0 ? 2 : r - 1;
  const int s1 = s == 2 ? 0 : s + 1, s2 = s == 0 ? 2 : s - 1;
  return fma(A[r1 * 3 + s1], A[r2 * 3 + s2], -(A[r1 * 3 + s2] * A[r2 * 3 + s1]));
}
// determinant, n <= 3 (expansion along the first row)
template <typename T>
__device__ __forceinline__ T det_small(const Opnd<T>& A, int n) {
  if (n == 1) return A[0];
  if (n == 2) return fma(A[0], A[3], -(A[1] * A[2]));
  return fma(A[2], cof3(A, 0, 2), fma(A[1], cof3(A, 0, 1), A[0] * cof3(A, 0, 0)));
}
// element e of the inverse, n <= 3, given r = 1 / det: the adjugate's element times r
template <typename T>
__device__ __forceinline__ T inv_small(const Opnd<T>& A, int n, int e, T r) {
  if (n == 1) return r;
  if (n == 2) return flip_sign(A[(e == 0 || e == 3) ? 3 - e : e], (unsigned)(e == 1 || e == 2)) * r;
  const int i = e / 3, j = e - 3 * i;
  return cof3(A, j, i) * r;
}

// IEEE bits of |x| as an integer: ordered like |x| for every value that is not a NaN
__device__ __forceinline__ unsigned long long abs_key(double x) {
  return (unsigned long long)fbits(x) & 0x7fffffffffffffffULL;
}
__device__ __forceinline__ unsigned long long abs_key(float x) { return __float_as_uint(x) & 0x7fffffffu; }
__device__ __forceinline__ bool nan_key(unsigned long long k, double) { return k > 0x7ff0000000000000ULL; }
__device__ __forceinline__ bool nan_key(unsigned long long k, float) { return k > 0x7f800000ULL; }

// Gauss-Jordan elimination with partial pivoting (n = 4..8) on [A | I] (want_inv) or on
// A alone, in the lane's scratch slots at sref: n rows of wc = 2n (or n) elements,
// row-major.  Rows are never moved: the exchanges are kept as a permutation in a
// register, four bits per logical row, logical row i being physical row perm(i).  The
// lane's threads split the columns: in a column step a thread normalizes the pivot row
// in its own columns and eliminates the other rows there, so the only values the
// threads share within a step are the pivot column's, which every thread reads before
// any is written.  The pivot is the first logical row at or below the diagonal of
// largest magnitude (a strict comparison; a NaN never wins), a row whose factor is
// exactly zero is left alone, and every element takes the same operations as in the
// sequential elimination.  Returns the determinant (the product of the pivots, negated
// per exchange); the inverse's row i is physical row perm(i), columns n .. 2n-1.
template <typename T, bool SYNC, typename LaneT>
__device__ T gauss_jordan(const LaneT& L, const Opnd<T>& A, int n, int32_t sref, bool want_inv, uint32_t& perm) {
  T* W = L.wp(sref);
  const int ss = L.ss, wc = want_inv ? 2 * n : n;
  const int first = L.first(), es = L.step();
  for (int j = first; j < wc; j += es)
    for (int i = 0; i < n; i++) W[(i * wc + j) * ss] = j < n ? A[i * n + j] : (T)(j - n == i ? 1 : 0);
  perm = 0x76543210u;
  if (SYNC) __syncwarp();
  T d = (T)1;
  for (int col = 0; col < n; col++) {
    int piv = col;
    unsigned long long best = abs_key(W[((int)((perm >> (4 * col)) & 15u) * wc + col) * ss]);
    for (int i = col + 1; i < n; i++) {
      const unsigned long long k = abs_key(W[((int)((perm >> (4 * i)) & 15u) * wc + col) * ss]);
      if (!nan_key(k, T()) && !nan_key(best, T()) && k > best) { best = k; piv = i; }
    }
    if (piv != col) {
      const uint32_t a = (perm >> (4 * col)) & 15u, b = (perm >> (4 * piv)) & 15u;
      perm = (perm & ~((15u << (4 * col)) | (15u << (4 * piv)))) | (b << (4 * col)) | (a << (4 * piv));
      d = -d;
    }
    const int pr = (int)((perm >> (4 * col)) & 15u);
    const T pv = W[(pr * wc + col) * ss];
    d = d * pv;
    const T r = rcp_rn(pv);
    T fct[8];  // the pivot column in the other rows, by physical row
#pragma unroll
    for (int i = 0; i < 8; i++) fct[i] = (i < n && i != pr) ? W[(i * wc + col) * ss] : (T)0;
    if (SYNC) __syncwarp();
    for (int j = first; j < wc; j += es) {
      const T p = W[(pr * wc + j) * ss] * r;
      W[(pr * wc + j) * ss] = p;
#pragma unroll
      for (int i = 0; i < 8; i++)
        if (i < n && i != pr && !is_zero(fct[i])) W[(i * wc + j) * ss] = fma(-fct[i], p, W[(i * wc + j) * ss]);
    }
    if (SYNC) __syncwarp();
  }
  return d;
}
// element e = (i, j) of the inverse left by gauss_jordan in the scratch slots
template <typename T, typename LaneT>
__device__ __forceinline__ T gj_inverse(const LaneT& L, int32_t sref, int n, uint32_t perm, int e) {
  const int i = divq(e, div_magic(n)), j = e - i * n;
  return L.wp(sref)[((int)((perm >> (4 * i)) & 15u) * 2 * n + n + j) * L.ss];
}

template <typename LaneT>
__device__ __forceinline__ bool all_zero(const LaneT& L, int32_t gz, int w) {
  for (int e = 0; e < w; e++)
    if (!is_zero(L.sl(gz, e))) return false;
  return true;
}
template <typename LaneT>
__device__ __forceinline__ void zero_if_first(const LaneT& L, int32_t ref, int w, bool first) {
  if (first && ref != -1)
    for (int e = L.first(); e < w; e += L.step()) L.wp(ref)[e * L.ss] = 0;
}

// Two layouts of the slot file.  Per-thread (shared_lane = 0): every thread owns a
// lane -- or, for data-axis tapes, a share of a lane's data points -- and its own
// column of slots.  Per-lane (shared_lane = 1): the G threads of a lane share one
// column; each matrix instruction's output elements are split over them (element e
// belongs to thread e mod G), scalar instructions are computed by all G and written
// by the owner of element 0, and a warp barrier after every instruction publishes
// the writes.  FP64 time is per warp instruction, so splitting matrix work keeps its
// cost while G times more warps cover the lanes.
template <typename T, bool SHARED, bool STAGED, bool BLOCK>
__device__ __forceinline__ void replay_body(const ReplayArgs& a, const int block) {
  static_assert(!BLOCK || SHARED, "a block-cooperative lane is an element-split group");
  extern __shared__ __align__(16) unsigned char smem_raw[];
  const int tid = threadIdx.x;
  const int tpb = blockDim.x;
  const int G = 1 << a.log2g;
  const int lane_in_block = tid >> a.log2g;
  const int64_t lane_raw = a.lane0 + (int64_t)block * (tpb >> a.log2g) + lane_in_block;
  const int grank = tid & (G - 1);
  const bool live = lane_raw < a.lane_end;
  if (G == 1 && !live && !STAGED) return;  // staged blocks keep every thread for the block barriers

  Lane<T, SHARED, !SHARED && !STAGED> L;
  if (SHARED) {
    L.ss = a.sstride;
    L.sbase = reinterpret_cast<T*>(smem_raw) + lane_in_block;
    L.eg = grank;
    L.emask = G - 1;
  } else {
    L.ss = tpb;
    L.sbase = reinterpret_cast<T*>(smem_raw) + tid;
    L.eg = 0;
    L.emask = 0;
  }
  L.consts = static_cast<const T*>(a.consts);
  L.obs = static_cast<const T*>(a.obs);
  L.params = static_cast<const T*>(a.params);
  L.save = static_cast<T*>(a.save);
  L.lane = live ? lane_raw : a.lane_end - 1;
  L.col = L.lane - a.lane0;
  L.save_ld = a.save_ld;
  L.P = a.P;
  L.dbase = 0;
  T* loss = static_cast<T*>(a.loss);
  T* grad = static_cast<T*>(a.grad);
  const bool writer = live && grank == 0;
  // element-split groups publish each instruction's writes: a warp barrier when the
  // group lies within a warp, a block barrier when one lane spans the whole block
  // (BLOCK: one lane per block, G = the block; a separate variant, so that the
  // in-warp groups do not carry the block-mode paths)
  const bool sync_each = SHARED && G > 1;
  const bool sync_block = BLOCK;
  auto group_sync = [&]() {
    if (sync_block) __syncthreads();
    else __syncwarp();
  };
  int es = L.step();

  int64_t d = 0, dN = 0, dstride = 0, dbase0 = 0;
  int loop_pc = -1;
  const DInst* __restrict__ code = a.code;
  const int32_t* __restrict__ args = a.args;

  // Staged instruction stream: chunk k of kStageChunk instructions sits in buffer
  // k % 2; the copy of chunk k + 1 is in flight while chunk k executes.  Every
  // thread of the block runs the same instruction sequence (staged plans have no
  // data-axis loops), so the block barrier at each chunk boundary is uniform.
  DInst* stage = reinterpret_cast<DInst*>(smem_raw + a.stage_off);
  auto stage_copy = [&](int chunk) {
    const int first = chunk * kStageChunk;
    if (first >= a.n_code) return;
    const int n = min(kStageChunk, a.n_code - first);
    const char* src = reinterpret_cast<const char*>(code + first);
    char* dst = reinterpret_cast<char*>(stage + (chunk & 1) * kStageChunk);
    const int pieces = (n * (int)sizeof(DInst) + 15) / 16;  // the device copy is padded to 16 bytes
    for (int i = tid; i < pieces; i += tpb) {
      const unsigned d = (unsigned)__cvta_generic_to_shared(dst + 16 * i);
      asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(d), "l"(src + 16 * i) : "memory");
    }
  };
  if (STAGED) {
    stage_copy(0);
    asm volatile("cp.async.commit_group;\n" ::: "memory");
    stage_copy(1);
    asm volatile("cp.async.commit_group;\n" ::: "memory");
    asm volatile("cp.async.wait_group 1;\n" ::: "memory");
    __syncthreads();
  }
  // non-staged streams: the record of the next instruction is loaded before the
  // current one executes, so its latency overlaps the current instruction (the same
  // look-ahead on the staged stream measured slower: it holds a second record in
  // registers, and a shared-memory record is close at hand anyway)
  DInst nxt;
  if (!STAGED && a.n_code > 0) nxt = code[0];
  int chunk_end = kStageChunk;  // staged: first instruction of the next chunk
  for (int pc = 0; pc < a.n_code; pc++) {
    if (STAGED && pc == chunk_end) {
      const int k = pc / kStageChunk;
      __syncthreads();  // every warp has left chunk k - 1: its buffer is free
      stage_copy(k + 1);
      asm volatile("cp.async.commit_group;\n" ::: "memory");
      asm volatile("cp.async.wait_group 1;\n" ::: "memory");  // chunk k has landed
      __syncthreads();
      chunk_end += kStageChunk;
    }
    const DInst in = STAGED ? stage[(unsigned)pc & (2 * kStageChunk - 1)] : nxt;
    if (!STAGED && pc + 1 < a.n_code) nxt = code[pc + 1];

    const int32_t* f = in.f;
    if (BLOCK && (in.op == 0 || in.op >= D_NOPS)) {  // not an opcode: every thread stops together
      if (a.err && tid == 0) atomicExch(a.err, 1);
      return;
    }
    if (sync_block) {
      // a lane spread over the whole block: instructions over many elements use every
      // thread; the rest (scalars, small inverses and determinants, fetches) run in
      // warp 0 alone, with ownership narrowed to its 32 threads, while the other warps
      // wait at the barrier that ends the instruction
      const bool wide = in.op == D_GATHER || in.op == D_MADD || in.op == D_MSUB || in.op == D_MSCALE ||
                        in.op == D_MATMUL || in.op == D_ZERO || in.op == B_MADD || in.op == B_MSUB ||
                        in.op == B_MSCALE || in.op == B_MATMUL || in.op == B_SCATTER;
      if (!wide && (tid >> 5) != 0) {
        group_sync();
        continue;
      }
      L.emask = wide ? G - 1 : 31;
      es = L.step();
    }
    // The fused scalar records and the fetches: ahead of the opcode switch where they make
    // up most of the stream (scalar tapes), as switch cases in the element-split variants,
    // whose streams are mostly matrix instructions
    constexpr bool kFastFirst = !SHARED;
    auto op_fma = [&]() {
      // the fused form of the cheap scalar rules: no opcode dispatch.  A zero gate (f4
      // is +-0: a zero adjoint contributes nothing, even against an infinite factor)
      // leaves c; it selects the inputs, fma(+0, -0, c) == c exactly for every c
      // (signed zeros included), so no select waits on the multiply-add's result
      const T x = flip_sign(L.lds(f[1]), in.flags & 1);
      const T c = L.lds(f[3]);
      const bool off = is_zero(L.lds(f[4]));
      const T z = fma(off ? (T)0 : x, off ? neg_zero<T>() : L.lds(f[2]), c);
      L.st(f[0], 0, z);
      L.save_out(f[5], 0, z);
    };
    auto op_fma2 = [&]() {
      // two fused updates in one record: every operand is loaded before either store;
      // when the second reads the first's result (flags bit 2), the operands that name
      // the first's destination take its value from the register instead
      // (the plain variant is given the unpaired stream and does not carry this path)
      const T x1 = flip_sign(L.lds(f[1]), in.flags & 1), y1 = L.lds(f[2]), c1 = L.lds(f[3]), g1 = L.lds(f[4]);
      T x2 = L.lds(f[6]), y2 = L.lds(f[7]), c2 = L.lds(in.pad3), g2 = L.lds(in.pad4);
      const bool off1 = is_zero(g1);
      const T z1 = fma(off1 ? (T)0 : x1, off1 ? neg_zero<T>() : y1, c1);
      if (in.flags & 4) {
        if (f[6] == f[0]) x2 = z1;
        if (f[7] == f[0]) y2 = z1;
        if (in.pad3 == f[0]) c2 = z1;
        if (in.pad4 == f[0]) g2 = z1;
      }
      x2 = flip_sign(x2, (in.flags >> 1) & 1);
      const bool off2 = is_zero(g2);
      const T z2 = fma(off2 ? (T)0 : x2, off2 ? neg_zero<T>() : y2, c2);
      L.st(f[0], 0, z1);
      L.st(f[5], 0, z2);
      if (in.flags & 8) {  // saves: 24-bit workspace indices in (r, c, k) and (pad0, pad1, pad2)
        const int32_t s1 = in.r | (in.c << 8) | (in.k << 16), s2 = in.pad0 | (in.pad1 << 8) | (in.pad2 << 16);
        if (s1 != kNoSave24) L.save_out(s1, 0, z1);
        if (s2 != kNoSave24) L.save_out(s2, 0, z2);
      }
    };
    auto op_fetch = [&]() {
      // asynchronous copies of workspace values into slots (the owner of element 0
      // copies; the warp barrier after the wait publishes them to the group)
      // (unrolled: the record's fields stay in registers only when indexed by constants)
      // (flags bit 5: the sources are observations of the current data point)
      if (L.own(0))
#pragma unroll
        for (int e = 0; e < kFetchPairs; e++) {
          if (e >= in.k) break;
          const T* src = (in.flags & 32) ? L.obs + L.dbase + (f[2 * e] & kRefIndexMask) : L.savep(f[2 * e]);
          const unsigned dst = (unsigned)__cvta_generic_to_shared(L.wp(f[2 * e + 1]));
          if (sizeof(T) == 8)
            asm volatile("cp.async.ca.shared.global [%0], [%1], 8;\n" ::"r"(dst), "l"(src) : "memory");
          else
            asm volatile("cp.async.ca.shared.global [%0], [%1], 4;\n" ::"r"(dst), "l"(src) : "memory");
        }
      if (in.flags & 2) asm volatile("cp.async.commit_group;\n" ::: "memory");
      if (in.flags & 1) {  // wait until at most n = flags bits 2..4 groups are pending
        switch ((in.flags >> 2) & 7) {
          case 0: asm volatile("cp.async.wait_group 0;\n" ::: "memory"); break;
          case 1: asm volatile("cp.async.wait_group 1;\n" ::: "memory"); break;
          case 2: asm volatile("cp.async.wait_group 2;\n" ::: "memory"); break;
          case 3: asm volatile("cp.async.wait_group 3;\n" ::: "memory"); break;
          default: asm volatile("cp.async.wait_group %0;\n" ::"n"(kFetchWindows) : "memory"); break;
        }
      }
    };
    if (kFastFirst) {
      if (in.op == D_FMA) {
        op_fma();
        if (sync_each) group_sync();
        continue;
      }
      if (STAGED && in.op == D_FMA2) {
        op_fma2();
        if (sync_each) group_sync();
        continue;
      }
      if (in.op == D_FETCH) {
        op_fetch();
        if (sync_each) group_sync();
        continue;
      }
    }
    const int w = in.r * in.c;
    switch (in.op) {
      // ------------------------------------------------------------ forward
      // one case per opcode: the switch's jump is the only dispatch branch
#define NDVM_FWD1(OPC, EXPR)                 \
  case OPC: {                                \
    const T x = L.lds(f[1]);                 \
    const T z = (EXPR);                      \
    L.st(f[0], 0, z);                        \
    L.save_out(f[3], 0, z);                  \
    break;                                   \
  }
#define NDVM_FWD2(OPC, EXPR)                 \
  case OPC: {                                \
    const T x = L.lds(f[1]), y = L.lds(f[2]); \
    const T z = (EXPR);                      \
    L.st(f[0], 0, z);                        \
    L.save_out(f[3], 0, z);                  \
    break;                                   \
  }
      NDVM_FWD2(D_ADD, x + y)
      NDVM_FWD2(D_SUB, x - y)
      NDVM_FWD2(D_MUL, x * y)
      NDVM_FWD2(D_POW, pow(x, y))
      NDVM_FWD1(D_NEG, -x)
      NDVM_FWD1(D_EXP, fast_exp(x))
      NDVM_FWD1(D_LOG, fast_log(gt_eps(x) ? x : clamp_eps<T>()))
      NDVM_FWD1(D_TANH, tanh(x))
      NDVM_FWD1(D_SQRT, sqrt(gt_eps(x) ? x : clamp_eps<T>()))
      NDVM_FWD1(D_ABS, fabs(x))
#undef NDVM_FWD1
#undef NDVM_FWD2
      case D_DIV: {
        // flags bit 4 (a division in a data-axis body): x / y through y's correctly rounded
        // reciprocal, kept (f4 slot, f5 save) for the reverse rule, which divides its
        // adjoint by y with it; else the IEEE division (staged streams have no data-axis
        // bodies, so the staged variants carry the IEEE division alone)
        const T x = L.lds(f[1]), y = L.lds(f[2]);
        T z;
        if (!STAGED && (in.flags & 16)) {
          T r;
          z = div_rcp(x, y, &r);
          if (f[4] != -1) L.st(f[4], 0, r);
          L.save_out(f[5], 0, r);
        } else {
          z = STAGED ? x / y : slow_div(x, y);  // a call where the other path is inlined
        }
        L.st(f[0], 0, z);
        L.save_out(f[3], 0, z);
        break;
      }
      case D_SIN: case D_COS: {
        T x = L.lds(f[1]);
        T s = 0, c = 0;
        if (f[4] != -1 || f[5] >= 0) {
          fast_sincos(x, &s, &c);
          T aux = in.op == D_SIN ? c : s;
          if (f[4] != -1) L.st(f[4], 0, aux);
          L.save_out(f[5], 0, aux);
        } else if (in.op == D_SIN) {
          s = fast_sin(x);
        } else {
          c = fast_cos(x);
        }
        T z = in.op == D_SIN ? s : c;
        L.st(f[0], 0, z);
        L.save_out(f[3], 0, z);
        break;
      }
      case D_POWI: {
        T z = powi_rep(L.lds(f[1]), f[7]);
        L.st(f[0], 0, z);
        L.save_out(f[3], 0, z);
        break;
      }
      case D_CMP: {
        T x = L.lds(f[1]), y = L.lds(f[2]);
        bool r = in.k == 0 ? x < y : in.k == 1 ? x <= y : in.k == 2 ? x > y : in.k == 3 ? x >= y : x == y;
        T z = r ? (T)1 : (T)0;
        L.st(f[0], 0, z);
        L.save_out(f[3], 0, z);
        break;
      }
      case D_SELECT: {
        T p = L.lds(f[1]);
        T z = !is_zero(p) ? L.lds(f[2]) : L.lds(f[4]);
        L.st(f[0], 0, z);
        L.save_out(f[3], 0, z);
        break;
      }
      case D_GATHER: {
        const int32_t* g = args + f[1];
        for (int e = L.first(); e < f[2]; e += es) {
          T v = L.ld(g[e]);
          L.st_mine(f[0], e, v);
          L.save_mine(f[3], e, v);
        }
        break;
      }
      case D_MADD: case D_MSUB: {
        Opnd<T> A = L.rd(f[1]), Bm = L.rd(f[2]);
        for (int e = L.first(); e < w; e += es) {
          T z = in.op == D_MADD ? A[e] + Bm[e] : A[e] - Bm[e];
          L.st_mine(f[0], e, z);
          L.save_mine(f[3], e, z);
        }
        break;
      }
      case D_MSCALE: {
        T s = L.ld(f[1]);
        Opnd<T> A = L.rd(f[2]);
        for (int e = L.first(); e < w; e += es) {
          T z = s * A[e];
          L.st_mine(f[0], e, z);
          L.save_mine(f[3], e, z);
        }
        break;
      }
      case D_MATMUL: {
        Opnd<T> A = L.rd(f[1]), Bm = L.rd(f[2]);
        const int c = in.c, kk = in.k;
        RowCol rc(L.first(), c);
        for (int e = L.first(); e < w; e += es, rc.next(es, c)) {
          const T s = dot<T, SHARED>(A.at(rc.i * kk), A.s, Bm.at(rc.j), c * Bm.s, kk, neg_zero<T>());
          L.st_mine(f[0], e, s);
          L.save_mine(f[3], e, s);
        }
        break;
      }
      case D_INV: {
        // each thread its own elements: closed forms to 3 x 3, else Gauss-Jordan
        // elimination in the scratch slots (f2) shared by the lane's threads
        const int n = in.r;
        Opnd<T> A = L.rd(f[1]);
        uint32_t perm = 0;
        T r = (T)0;
        if (n <= 3) r = rcp_rn(det_small(A, n));
        else gauss_jordan<T, SHARED>(L, A, n, f[2], true, perm);
        for (int e = L.first(); e < n * n; e += es) {
          const T v = n <= 3 ? inv_small(A, n, e, r) : gj_inverse<T>(L, f[2], n, perm, e);
          L.st_mine(f[0], e, v);
          L.save_mine(f[3], e, v);
        }
        break;
      }
      case D_DET: case D_LOGDET: {
        // with an auxiliary output (f4 slot / f5 save) the inverse comes too, for the
        // reverse rule
        const int n = in.r;
        const bool aux = f[4] != -1 || f[5] >= 0;
        Opnd<T> A = L.rd(f[1]);
        uint32_t perm = 0;
        const T dt = n <= 3 ? det_small(A, n) : gauss_jordan<T, SHARED>(L, A, n, f[2], aux, perm);
        const T z = in.op == D_DET ? dt : fast_log(dt);
        L.st(f[0], 0, z);
        L.save_out(f[3], 0, z);
        if (aux) {
          const T r = n <= 3 ? rcp_rn(dt) : (T)0;
          for (int e = L.first(); e < n * n; e += es) {
            const T v = n <= 3 ? inv_small(A, n, e, r) : gj_inverse<T>(L, f[2], n, perm, e);
            if (f[4] != -1) L.st_mine(f[4], e, v);
            L.save_mine(f[5], e, v);
          }
        }
        break;
      }
      case D_TRACE: {
        const int n = in.r;
        Opnd<T> A = L.rd(f[1]);
        T s = A[0];
        for (int i = 1; i < n; i++) s = s + A[i * n + i];
        L.st(f[0], 0, s);
        break;
      }
      // ------------------------------------------------------------ data axis
      case D_ZERO:
        for (int e = L.first(); e < f[1]; e += es) L.st_mine(f[0], e, (T)0);
        break;
      case D_LOOP:
        dN = f[0]; dstride = f[1]; dbase0 = f[2];
        d = grank;
        loop_pc = pc;
        if (d >= dN) {  // no point for this thread: resume after the loop end
          pc = f[3];
          if (!STAGED && pc + 1 < a.n_code) nxt = code[pc + 1];
          break;
        }
        L.dbase = dbase0 + d * dstride;
        break;
      case D_ENDLOOP:
        d += G;
        if (d < dN) {
          L.dbase = dbase0 + d * dstride;
          pc = loop_pc;
          if (!STAGED) nxt = code[pc + 1];
        }
        break;
      case D_ACC: L.st(f[0], 0, L.sl(f[0], 0) + L.lds(f[1])); break;
      case D_LOAD: L.st(f[0], 0, L.ld(f[1])); break;
      case D_SEED: L.st(f[0], 0, (T)1); break;
      case D_GREDUCE:
        if (G > 1) {
          __syncwarp();
          for (int e = 0; e < f[1]; e++) {
            T v = L.sl(f[0], e);
            for (int o = G >> 1; o >= 1; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
            L.st(f[0], e, v);
          }
        }
        break;
      case D_LOSS:
        if (writer) loss[L.lane] = L.ld(f[0]);
        break;
      // ------------------------------------------------------------ reverse
      case B_ADD: case B_SUB: {
        const T g = L.sl(f[0], 0);
        const bool fa = in.flags & 1, fb = in.flags & 2;
        if (is_zero(g)) { zero_if_first(L, f[1], 1, fa); zero_if_first(L, f[2], 1, fb); break; }
        if (f[1] != -1) L.upd(f[1], 0, g, fa);
        if (f[2] != -1) L.upd(f[2], 0, in.op == B_ADD ? g : -g, fb);
        break;
      }
      case B_NEG: {
        const T g = L.sl(f[0], 0);
        const bool fa = in.flags & 1;
        if (is_zero(g)) { zero_if_first(L, f[1], 1, fa); break; }
        if (f[1] != -1) L.upd(f[1], 0, -g, fa);
        break;
      }
      case B_MUL: {
        T g = L.sl(f[0], 0);
        bool fa = in.flags & 1, fb = in.flags & 2;
        if (is_zero(g)) { zero_if_first(L, f[1], 1, fa); zero_if_first(L, f[2], 1, fb); break; }
        if (f[1] != -1) L.upd(f[1], 0, g * L.lds(f[4]), fa);
        if (f[2] != -1) L.upd(f[2], 0, g * L.lds(f[3]), fb);
        break;
      }
      case B_DIV: {
        T g = L.sl(f[0], 0);
        bool fa = in.flags & 1, fb = in.flags & 2;
        if (is_zero(g)) { zero_if_first(L, f[1], 1, fa); zero_if_first(L, f[2], 1, fb); break; }
        const T b = L.lds(f[4]);
        const T q = f[6] != -1 ? div_by_rcp(g, b, L.lds(f[6])) : (STAGED ? g / b : slow_div(g, b));
        if (f[1] != -1) L.upd(f[1], 0, q, fa);
        if (f[2] != -1) L.upd(f[2], 0, -(q * L.lds(f[5])), fb);
        break;
      }
      case B_POW: {
        T g = L.sl(f[0], 0);
        bool fa = in.flags & 1, fb = in.flags & 2;
        if (is_zero(g)) { zero_if_first(L, f[1], 1, fa); zero_if_first(L, f[2], 1, fb); break; }
        T x = L.lds(f[3]), e = L.lds(f[4]), z = L.lds(f[5]);
        if (f[1] != -1) L.upd(f[1], 0, g * e * z / x, fa);
        if (f[2] != -1) L.upd(f[2], 0, g * z * log(x), fb);
        break;
      }
      // unary adjoints: g times the local derivative (one case per opcode)
#define NDVM_REV1(OPC, EXPR)                             \
  case OPC: {                                            \
    const T g = L.sl(f[0], 0);                           \
    const bool fa = in.flags & 1;                        \
    if (f[1] == -1) break;                               \
    if (is_zero(g)) { zero_if_first(L, f[1], 1, fa); break; } \
    L.upd(f[1], 0, (EXPR), fa);                          \
    break;                                               \
  }
      NDVM_REV1(B_EXP, g * L.lds(f[5]))
      NDVM_REV1(B_TANH, g * ((T)1 - L.lds(f[5]) * L.lds(f[5])))
      NDVM_REV1(B_LOG, gt_eps(L.lds(f[3])) ? div_rcp_q(g, L.lds(f[3])) : (T)0)
      NDVM_REV1(B_ABS, L.lds(f[3]) > (T)0 ? g : (L.lds(f[3]) < (T)0 ? -g : g * (T)0))
      NDVM_REV1(B_SQRT, gt_eps(L.lds(f[3])) ? g / ((T)2 * L.lds(f[5])) : (T)0)
      NDVM_REV1(B_SIN, g * L.lds(f[6]))
      NDVM_REV1(B_COS, -(g * L.lds(f[6])))
      NDVM_REV1(B_POWI, f[7] > 0 ? g * powi_deriv(L.lds(f[3]), f[7]) : (T)0)
#undef NDVM_REV1
      case B_SELECT: {
        T g = L.sl(f[0], 0);
        bool fa = in.flags & 1, fb = in.flags & 2;
        bool taken = !is_zero(L.lds(f[3]));
        if (f[1] != -1) { if (taken && !is_zero(g)) L.upd(f[1], 0, g, fa); else zero_if_first(L, f[1], 1, fa); }
        if (f[2] != -1) { if (!taken && !is_zero(g)) L.upd(f[2], 0, g, fb); else zero_if_first(L, f[2], 1, fb); }
        break;
      }
      case B_GATHER: {
        // every target is a scalar (element 0 of its own value)
        const int32_t* g = args + f[1];
        const bool z = all_zero(L, f[0], f[2]);
        for (int e = 0; e < f[2]; e++) {
          int32_t t = g[2 * e];
          if (t == -1) continue;
          bool first = g[2 * e + 1] != 0;
          if (z) zero_if_first(L, t, 1, first);
          else L.upd(t, 0, L.sl(f[0], e), first);
        }
        break;
      }
      case B_SCATTER: {
        if (f[1] == -1) break;
        const bool first = in.flags & 1;
        zero_if_first(L, f[1], f[4], first);
        if (all_zero(L, f[0], f[2])) break;
        const int32_t* m = args + f[3];
        for (int e = 0; e < f[2]; e++)
          if (L.own(m[e])) L.st(f[1], m[e], L.sl(f[1], m[e]) + L.sl(f[0], e));
        break;
      }
      case B_MADD: case B_MSUB: {
        bool fa = in.flags & 1, fb = in.flags & 2;
        if (all_zero(L, f[0], w)) { zero_if_first(L, f[1], w, fa); zero_if_first(L, f[2], w, fb); break; }
        for (int e = L.first(); e < w; e += es) {
          T g = L.sl(f[0], e);
          if (f[1] != -1) L.upd_mine(f[1], e, g, fa);
          if (f[2] != -1) L.upd_mine(f[2], e, in.op == B_MADD ? g : -g, fb);
        }
        break;
      }
      case B_MSCALE: {
        bool fa = in.flags & 1, fb = in.flags & 2;
        if (all_zero(L, f[0], w)) { zero_if_first(L, f[1], 1, fa); zero_if_first(L, f[2], w, fb); break; }
        if (f[1] != -1) {
          Opnd<T> A = L.rd(f[4]);
          T s = fa ? neg_zero<T>() : L.sl(f[1], 0);
          for (int e = 0; e < w; e++) s = fma(L.sl(f[0], e), A[e], s);
          L.st(f[1], 0, s);
        }
        if (f[2] != -1) {
          T s = L.ld(f[3]);
          for (int e = L.first(); e < w; e += es) L.upd_fma_mine(f[2], e, s, L.sl(f[0], e), fb);
        }
        break;
      }
      case B_MATMUL: {
        // the running adjoint of each target element starts its dot product's chain
        const int r = in.r, c = in.c, kk = in.k;
        bool fa = in.flags & 1, fb = in.flags & 2;
        if (all_zero(L, f[0], w)) { zero_if_first(L, f[1], r * kk, fa); zero_if_first(L, f[2], kk * c, fb); break; }
        Opnd<T> G_ = {L.wp(f[0]), L.ss};
        if (f[1] != -1) {  // gA (r x k) += gZ (r x c) * B^T (B is k x c)
          Opnd<T> Bm = L.rd(f[4]);
          RowCol rq(L.first(), kk);
          for (int e = L.first(); e < r * kk; e += es, rq.next(es, kk)) {
            T* q = L.wp(f[1]) + e * L.ss;
            *q = dot<T, SHARED>(G_.at(rq.i * c), G_.s, Bm.at(rq.j * c), Bm.s, c, fa ? neg_zero<T>() : *q);
          }
        }
        if (f[2] != -1) {  // gB (k x c) += A^T (A is r x k) * gZ
          Opnd<T> A = L.rd(f[3]);
          RowCol qj(L.first(), c);
          for (int e = L.first(); e < kk * c; e += es, qj.next(es, c)) {
            T* q = L.wp(f[2]) + e * L.ss;
            *q = dot<T, SHARED>(A.at(qj.i), kk * A.s, G_.at(qj.j), c * G_.s, r, fb ? neg_zero<T>() : *q);
          }
        }
        break;
      }
      case B_INV: {
        // gA -= B^T gZ B^T (B the inverse): M = gZ B^T into the scratch slots (f2), each
        // thread its own elements, then each thread its own elements of gA from M
        const int n = in.r;
        bool fa = in.flags & 1;
        if (f[1] == -1) break;
        if (all_zero(L, f[0], n * n)) { zero_if_first(L, f[1], n * n, fa); break; }
        Opnd<T> Bv = L.rd(f[5]);
        Opnd<T> G_ = {L.wp(f[0]), L.ss};
        Opnd<T> M = {L.wp(f[2]), L.ss};
        const uint32_t mn = div_magic(n);
        for (int e = L.first(); e < n * n; e += es) {
          const int p = divq(e, mn), j = e - p * n;
          L.wp(f[2])[e * L.ss] = dot<T, SHARED>(G_.at(p * n), G_.s, Bv.at(j * n), Bv.s, n, neg_zero<T>());
        }
        if (SHARED) __syncwarp();
        for (int e = L.first(); e < n * n; e += es) {
          const int i = divq(e, mn), j = e - i * n;
          T* q = L.wp(f[1]) + e * L.ss;
          *q = -dot<T, SHARED>(Bv.at(i), n * Bv.s, M.at(j), n * M.s, n, fa ? neg_zero<T>() : -*q);
        }
        break;
      }
      case B_DET: case B_LOGDET: {
        const int n = in.r;
        bool fa = in.flags & 1;
        if (f[1] == -1) break;
        T g = L.sl(f[0], 0);
        if (is_zero(g)) { zero_if_first(L, f[1], n * n, fa); break; }
        T fac = in.op == B_DET ? g * L.ld(f[5]) : g;
        Opnd<T> Iv = L.rd(f[6]);
        const uint32_t mn = div_magic(n);
        for (int e = L.first(); e < n * n; e += es) {
          const int i = divq(e, mn), j = e - i * n;
          L.upd_fma_mine(f[1], e, fac, Iv[j * n + i], fa);
        }
        break;
      }
      case B_TRACE: {
        const int n = in.r;
        bool fa = in.flags & 1;
        if (f[1] == -1) break;
        T g = L.sl(f[0], 0);
        zero_if_first(L, f[1], n * n, fa);
        if (is_zero(g)) break;
        for (int i = 0; i < n; i++)
          if (L.own(i * n + i)) L.st(f[1], i * n + i, L.sl(f[1], i * n + i) + g);
        break;
      }
      case B_DSUM: {
        T g = L.sl(f[0], 0);
        const int32_t* q = args + f[1];
        for (int e = 0; e < f[2]; e++) {
          int32_t t = q[3 * e];
          bool first = q[3 * e + 1] != 0;
          if (is_zero(g)) zero_if_first(L, t, 1, first);
          else L.upd_fma(t, 0, g, L.sl(q[3 * e + 2], 0), first);
        }
        break;
      }
      case B_GRAD:
        if (writer) grad[L.lane * L.P + f[1]] = f[0] == -1 ? (T)0 : L.sl(f[0], 0);
        break;
      case D_FMA:
        if (!kFastFirst) op_fma();
        break;
      case D_FMA2:
        if (!kFastFirst) {
          op_fma2();
          break;
        }
        if (a.err) atomicExch(a.err, 1);  // the plain variant carries no paired records
        return;
      case D_FETCH:
        if (!kFastFirst) op_fetch();
        break;
      default:  // not an opcode of this variant: every thread stops
        if (a.err) atomicExch(a.err, 1);
        if (sync_block) break;  // warp 0 alone may be here: keep the barrier count, stop nothing
        return;
    }
    if (sync_each) group_sync();
  }
}

template <typename T, bool SHARED, bool STAGED, bool BLOCK>
__global__ void __launch_bounds__(256, (SHARED || STAGED) ? 2 : 4) k_replay(ReplayArgs a) {
  replay_body<T, SHARED, STAGED, BLOCK>(a, blockIdx.x);
}

// Several replays in one launch (one per tape of a batch, all of one kernel variant and
// block size): block b serves the member m with start[m] <= b < start[m + 1], as its
// block b - start[m].  The member table travels as the kernel's parameter.
template <typename T, bool SHARED, bool STAGED, bool BLOCK>
__global__ void __launch_bounds__(256, (SHARED || STAGED) ? 2 : 4) k_replay_multi(const __grid_constant__ MultiArgs ma) {
  const int b = blockIdx.x;
  int lo = 0, hi = ma.n - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (ma.start[mid] <= b) lo = mid;
    else hi = mid - 1;
  }
  replay_body<T, SHARED, STAGED, BLOCK>(ma.a[lo], b - ma.start[lo]);
}

template <typename T, bool SHARED, bool STAGED, bool BLOCK>
cudaError_t launch_multi_v(const MultiArgs& m, int blocks, int tpb, size_t smem, cudaStream_t s) {
  static int configured_dev = -1;
  static size_t configured_smem = 0;
  int dev = 0;
  cudaGetDevice(&dev);
  if (configured_dev != dev || smem > configured_smem) {
    cudaError_t e = cudaFuncSetAttribute(k_replay_multi<T, SHARED, STAGED, BLOCK>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    configured_dev = dev;
    configured_smem = smem;
  }
  k_replay_multi<T, SHARED, STAGED, BLOCK><<<blocks, tpb, smem, s>>>(m);
  return cudaGetLastError();
}

template <typename T>
cudaError_t launch_multi_t(const MultiArgs& m, int blocks, int tpb, size_t smem, cudaStream_t s) {
  const ReplayArgs& a = m.a[0];  // every member has the same variant
  if (a.shared_lane && (1 << a.log2g) > 32)
    return a.staged ? launch_multi_v<T, true, true, true>(m, blocks, tpb, smem, s)
                    : launch_multi_v<T, true, false, true>(m, blocks, tpb, smem, s);
  if (a.shared_lane)
    return a.staged ? launch_multi_v<T, true, true, false>(m, blocks, tpb, smem, s)
                    : launch_multi_v<T, true, false, false>(m, blocks, tpb, smem, s);
  return a.staged ? launch_multi_v<T, false, true, false>(m, blocks, tpb, smem, s)
                  : launch_multi_v<T, false, false, false>(m, blocks, tpb, smem, s);
}

// Copies of n_copy runs of values (src[i] -> dst[i], len[i] elements of elem bytes, in
// 4-byte words: every run's addresses and length are multiples of 4 bytes), one block
// per run: the observations of a batch's tapes into their extended observation buffers.
__global__ void __launch_bounds__(256) k_copy_runs(const __grid_constant__ CopyRuns c) {
  const int r = blockIdx.x;
  if (r >= c.n) return;
  const uint32_t* src = static_cast<const uint32_t*>(c.src[r]);
  uint32_t* dst = static_cast<uint32_t*>(c.dst[r]);
  for (int64_t i = threadIdx.x; i < c.words[r]; i += blockDim.x) dst[i] = src[i];
}

template <typename T, bool SHARED, bool STAGED, bool BLOCK>
cudaError_t launch_v(const ReplayArgs& a, int blocks, int tpb, size_t smem, cudaStream_t s) {
  static int configured_dev = -1;
  static size_t configured_smem = 0;
  int dev = 0;
  cudaGetDevice(&dev);
  if (configured_dev != dev || smem > configured_smem) {
    cudaError_t e =
        cudaFuncSetAttribute(k_replay<T, SHARED, STAGED, BLOCK>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    configured_dev = dev;
    configured_smem = smem;
  }
  k_replay<T, SHARED, STAGED, BLOCK><<<blocks, tpb, smem, s>>>(a);
  return cudaGetLastError();
}

template <typename T>
cudaError_t launch_t(const ReplayArgs& a, int blocks, int tpb, size_t smem, cudaStream_t s) {
  if (a.shared_lane && (1 << a.log2g) > 32)  // one lane per block
    return a.staged ? launch_v<T, true, true, true>(a, blocks, tpb, smem, s)
                    : launch_v<T, true, false, true>(a, blocks, tpb, smem, s);
  if (a.shared_lane)
    return a.staged ? launch_v<T, true, true, false>(a, blocks, tpb, smem, s)
                    : launch_v<T, true, false, false>(a, blocks, tpb, smem, s);
  return a.staged ? launch_v<T, false, true, false>(a, blocks, tpb, smem, s)
                  : launch_v<T, false, false, false>(a, blocks, tpb, smem, s);
}

}  // namespace

cudaError_t launch_replay(const ReplayArgs& a, bool f32, int blocks, int tpb, size_t smem, cudaStream_t s) {
  return f32 ? launch_t<float>(a, blocks, tpb, smem, s) : launch_t<double>(a, blocks, tpb, smem, s);
}

cudaError_t launch_replay_multi(const MultiArgs& m, bool f32, int blocks, int tpb, size_t smem, cudaStream_t s) {
  if (m.n < 1 || m.n > kMultiMax || blocks < 1) return cudaErrorInvalidValue;
  return f32 ? launch_multi_t<float>(m, blocks, tpb, smem, s) : launch_multi_t<double>(m, blocks, tpb, smem, s);
}

cudaError_t launch_copy_runs(const CopyRuns& c, cudaStream_t s) {
  if (c.n < 1 || c.n > kCopyRunsMax) return cudaErrorInvalidValue;
  k_copy_runs<<<c.n, 256, 0, s>>>(c);
  return cudaGetLastError();
}

}  // namespace ndvm

// ---------------------------------------------------------------------------
// FP64 peak probe: the roofline denominator of this FP64-bound path, measured on
// the device in the same process as the replay.  Eight independent fused
// multiply-add chains per thread, four 256-thread blocks per SM.
namespace ndvm {
namespace {
__global__ void __launch_bounds__(256) k_dfma_peak(double* out, int iters) {
  double a[8];
  const double y = 0.999999999, c = 1e-9;
#pragma unroll
  for (int k = 0; k < 8; k++) a[k] = 1.0 + 1e-3 * k + 1e-7 * threadIdx.x;
  for (int i = 0; i < iters; i++) {
#pragma unroll
    for (int k = 0; k < 8; k++) a[k] = fma(a[k], y, c);
  }
  double s = 0;
#pragma unroll
  for (int k = 0; k < 8; k++) s += a[k];
  out[(size_t)blockIdx.x * blockDim.x + threadIdx.x] = s;
}
}  // namespace

cudaError_t measure_fp64_peak(double* flops_per_s, cudaStream_t s) {
  int dev = 0, sms = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return e;
  const int blocks = sms * 4, threads = 256, iters = 20000;
  double* out = nullptr;
  if ((e = cudaMalloc(&out, sizeof(double) * blocks * threads)) != cudaSuccess) return e;
  cudaEvent_t e0, e1;
  cudaEventCreate(&e0);
  cudaEventCreate(&e1);
  k_dfma_peak<<<blocks, threads, 0, s>>>(out, 200);  // warm-up
  float best = 1e30f;
  for (int rep = 0; rep < 3; rep++) {
    cudaEventRecord(e0, s);
    k_dfma_peak<<<blocks, threads, 0, s>>>(out, iters);
    cudaEventRecord(e1, s);
    e = cudaEventSynchronize(e1);
    if (e != cudaSuccess) break;
    float ms = 0;
    cudaEventElapsedTime(&ms, e0, e1);
    if (ms < best) best = ms;
  }
  if (e == cudaSuccess) e = cudaGetLastError();
  cudaEventDestroy(e0);
  cudaEventDestroy(e1);
  cudaFree(out);
  if (e == cudaSuccess) *flops_per_s = 2.0 * 8.0 * iters * (double)blocks * threads / (best * 1e-3);
  return e;
}
}  // namespace ndvm

// ---------------------------------------------------------------------------
// Per-function cost probe: the throughput of one library function (or of the
// replay's own exp and log) relative to DFMA, for the roofline's cost table.  Every
// thread runs four independent chains x <- f(x) + c (or f(x) c; c keeps x in the
// function's ordinary domain); one FP64 add or multiply per call is part of the chain
// and is counted in the measured time.  Launch shape and iteration count match the FP64 peak probe's
// per-thread work, so an ncu capture of a probe launch gives the function's FP64-pipe
// instructions per call (calls = blocks x threads x iters x 4).
namespace ndvm {
namespace {
template <int FN>
__device__ __forceinline__ double probe_f(double x) {
  switch (FN) {
    case NDVM_PROBE_DFMA: return fma(x, 0.999999999, 1e-9);
    case NDVM_PROBE_EXP: return fast_exp(x) * 0.25;  // x settles near 0.357
    case NDVM_PROBE_LOG: return fast_log(x) + 2.0;
    case NDVM_PROBE_SIN: return fast_sin(x) + 1.0;
    case NDVM_PROBE_COS: return fast_cos(x) + 1.0;
    case NDVM_PROBE_SINCOS: { double s, c; fast_sincos(x, &s, &c); return s + c; }
    case NDVM_PROBE_SINLIB: return sin(x) + 1.0;
    case NDVM_PROBE_SINCOSLIB: { double s, c; sincos(x, &s, &c); return s + c; }
    case NDVM_PROBE_TANH: return tanh(x) + 0.5;
    case NDVM_PROBE_SQRT: return sqrt(x) + 1.0;
    case NDVM_PROBE_DIV: return 3.0 / (x + 1.0);
    case NDVM_PROBE_RCP: return 1.0 / x + 0.5;
    case NDVM_PROBE_POW: return pow(x, 0.75) + 1.0;
    case NDVM_PROBE_LOGLIB: return log(x) + 2.0;
    case NDVM_PROBE_EXPLIB: return exp(x) * 0.25;
    default: return x;
  }
}
template <int FN>
__global__ void __launch_bounds__(256) k_op_probe(double* out, int iters) {
  double a[4];
#pragma unroll
  for (int k = 0; k < 4; k++) a[k] = 1.0 + 0.125 * k + 1e-7 * threadIdx.x;
  for (int i = 0; i < iters; i++) {
#pragma unroll
    for (int k = 0; k < 4; k++) a[k] = probe_f<FN>(a[k]);
  }
  out[(size_t)blockIdx.x * blockDim.x + threadIdx.x] = a[0] + a[1] + a[2] + a[3];
}
template <int FN>
void launch_probe(double* out, int blocks, int iters, cudaStream_t s) {
  k_op_probe<FN><<<blocks, 256, 0, s>>>(out, iters);
}
using ProbeFn = void (*)(double*, int, int, cudaStream_t);
constexpr ProbeFn kProbes[NDVM_PROBE_COUNT] = {
    launch_probe<0>, launch_probe<1>, launch_probe<2>, launch_probe<3>, launch_probe<4>,
    launch_probe<5>, launch_probe<6>, launch_probe<7>, launch_probe<8>, launch_probe<9>,
    launch_probe<10>, launch_probe<11>, launch_probe<12>, launch_probe<13>, launch_probe<14>};
}  // namespace

cudaError_t measure_op_cost(int fn, int iters, double* ns_per_call, cudaStream_t s) {
  if (fn < 0 || fn >= NDVM_PROBE_COUNT || iters < 1) return cudaErrorInvalidValue;
  int dev = 0, sms = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return e;
  const int blocks = sms * 4, threads = 256;
  double* out = nullptr;
  if ((e = cudaMalloc(&out, sizeof(double) * blocks * threads)) != cudaSuccess) return e;
  cudaEvent_t e0, e1;
  cudaEventCreate(&e0);
  cudaEventCreate(&e1);
  kProbes[fn](out, blocks, 16, s);  // warm-up
  float best = 1e30f;
  for (int rep = 0; rep < 3; rep++) {
    cudaEventRecord(e0, s);
    kProbes[fn](out, blocks, iters, s);
    cudaEventRecord(e1, s);
    e = cudaEventSynchronize(e1);
    if (e != cudaSuccess) break;
    float ms = 0;
    cudaEventElapsedTime(&ms, e0, e1);
    if (ms < best) best = ms;
  }
  if (e == cudaSuccess) e = cudaGetLastError();
  cudaEventDestroy(e0);
  cudaEventDestroy(e1);
  cudaFree(out);
  // device time per call, all SMs busy: total time / calls
  if (e == cudaSuccess) *ns_per_call = best * 1e6 / (4.0 * iters * (double)blocks * threads);
  return e;
}
}  // namespace ndvm

// ---------------------------------------------------------------------------
// Fixed scratch for the no-allocation entry point (ndvm_value_and_grad_noalloc).
// Some callers may not allocate device memory while they run -- their device
// memory is planned up front and must not grow.  For them the workspace of the
// replay lives in this file-scope array, held by every GPU that loads the
// library until the process exits.  Every call uses the same array, so calls
// whose work overlaps on the GPU race; the replay writes each saved element
// before it reads it, so nothing in it needs clearing between calls.
namespace ndvm {
namespace {
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];
}  // namespace

cudaError_t noalloc_scratch(void** ptr) {
  // The array's name is a host-side stand-in; its device address is looked up
  // once per device, with that device current.
  static std::mutex mu;
  static std::map<int, void*> addr;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  std::lock_guard<std::mutex> lk(mu);
  auto it = addr.find(dev);
  if (it == addr.end()) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess) return e;
    it = addr.emplace(dev, p).first;
  }
  *ptr = it->second;
  return cudaSuccess;
}
}  // namespace ndvm
