/*
 * ndvm_oracle.c -- the reference ("oracle") evaluator for the NDVM tape-replay path.
 *
 * TEST INFRASTRUCTURE ONLY.  Only the test suite, the smoke check and the
 * benchmark's CPU-baseline leg may load this library.  The product path never
 * links, imports or calls it, and it shares no code, header, table or helper
 * with the product (the host tracer, the tape planner or the CUDA kernels).
 *
 * What it computes (paper section 2, the problem statement): for every lane b
 * independently, y_b = E(P, theta_b) -- the value of the program text P run
 * with the parameter vector theta_b -- and the exact gradient dy_b/dtheta_b
 * along the realized trace (Property 1, section 4).  It does this the plain way:
 *
 *   - it reads the PROGRAM TEXT itself (never a tape), with its own reader and
 *     its own tree-walking evaluator (environments, closures, named let with
 *     proper tail calls, structural integers and lists);
 *   - it evaluates one lane at a time, scalar by scalar, in IEEE double with
 *     round-to-nearest; it is compiled with -ffp-contract=off so no multiply-add
 *     is fused and results are identical on every host;
 *   - per-lane numeric control (`if` on a comparison of numbers) simply takes
 *     the branch this lane takes -- no masks, no select;
 *   - reverse mode: every numeric value is a heap node holding pointers to its
 *     input nodes; the backward pass orders the reachable graph by a depth-first
 *     search from the loss and propagates adjoints with the rules of Appendix C
 *     (table "Numeric primitives implemented by NDVM and their reverse-mode
 *     adjoints") -- there is no flat tape;
 *   - forward mode (cross-check): every numeric value carries its P partial
 *     derivatives (dual numbers, the method section 6 uses for its hand-compiled
 *     Kalman ceiling).
 *
 * Readings of points the paper leaves open (the GPU path takes the same ones):
 *   R1  tanh, neg, select, compare, param/obs loads and matrix add/sub/scale are
 *       not in Appendix C: tanh' = 1 - z^2, neg' = -1, select passes the adjoint
 *       to the branch the lane took (section 6: only lanes that took a side send
 *       adjoints into it), comparisons carry no gradient.
 *   R2  sqrt/log clamp (Appendix C): forward on max(x, 1e-8); zero gradient
 *       unless x > 1e-8 strictly.  abs'(x) = sign(x) with sign(0) = 0.
 *   R3  integer powers (pow with a structural integer exponent n >= 0): forward by
 *       left-to-right repeated multiplication; base adjoint g * (n * a^(n-1)),
 *       a^(n-1) again by repeated multiplication; no exponent gradient.
 *       General pow (numeric exponent) follows Appendix C literally.
 *   R4  det / logdet / inv: closed-form adjugate for 1x1, 2x2 and 3x3; Gauss-Jordan
 *       elimination with partial pivoting above that.  logdet = ln(det A).
 *   R5  a node whose whole adjoint is exactly zero propagates nothing (so an
 *       untaken or zero-weight path never turns 0 * inf into NaN).
 *   R6  n-ary + - * / follow Appendix C: z = x0 - (x1 + ... + xn) for sub and
 *       z = x0 / (x1 * ... * xn) for div, sums and products left to right;
 *       single-argument - and / are negation and reciprocal.
 *   R7  (data-sum N S [BASE] body) sums body over the data axis (section 3.5,
 *       data points as a batch axis) left to right; (dobs k) inside body reads
 *       obs[BASE + d*S + k] for data point d.
 */
#define _GNU_SOURCE
#include <math.h>
#include <pthread.h>
#include <setjmp.h>
#include <stdarg.h>
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#define OR_OK 0
#define OR_ERR 1

/* evaluation modes */
#define MODE_VALUE 0   /* loss only */
#define MODE_REVERSE 1 /* loss + gradient by the pointer-graph reverse mode */
#define MODE_DUAL 2    /* loss + gradient by forward-mode dual numbers */

/* ------------------------------------------------------------------------- */
/* Arena: bump allocator, one per worker thread, reset between lanes.        */
/* ------------------------------------------------------------------------- */
typedef struct Chunk { struct Chunk* next; size_t used, cap; unsigned char data[]; } Chunk;
typedef struct { Chunk* head; size_t total; } Arena;

static void* arena_alloc(Arena* a, size_t n) {
  n = (n + 15) & ~(size_t)15;
  if (!a->head || a->head->used + n > a->head->cap) {
    size_t cap = n > (1u << 22) ? n : (1u << 22);
    Chunk* c = (Chunk*)malloc(sizeof(Chunk) + cap);
    if (!c) return NULL;
    c->next = a->head; c->used = 0; c->cap = cap; a->head = c;
    a->total += cap;
  }
  void* p = a->head->data + a->head->used;
  a->head->used += n;
  return p;
}
static void arena_free_all(Arena* a) {
  Chunk* c = a->head;
  while (c) { Chunk* n = c->next; free(c); c = n; }
  a->head = NULL; a->total = 0;
}

/* ------------------------------------------------------------------------- */
/* Values.  Structural values are plain data (section 3.1, Definition 1);     */
/* numbers are Num nodes (payloads) that also form the reverse-mode graph.    */
/* ------------------------------------------------------------------------- */
typedef enum { V_NIL, V_BOOL, V_PBOOL, V_INT, V_FLT, V_NUM, V_PAIR, V_CLOS, V_PRIM, V_SYM } VTag;
struct Num; struct Pair; struct Clos;
typedef struct Val {
  VTag t;
  union { long long i; double f; struct Num* n; struct Pair* p; struct Clos* c; int prim; int sym; } u;
} Val;
typedef struct Pair { Val car, cdr; } Pair;

/* numeric node kinds */
enum {
  N_CONST, N_PARAM, N_ADD, N_SUB, N_MUL, N_DIV, N_NEG, N_EXP, N_LOG, N_SIN, N_COS, N_TANH,
  N_SQRT, N_ABS, N_POW, N_POWI, N_DOT, N_SELECTED, N_MAT, N_MREF, N_MADD, N_MSUB, N_MSCALE,
  N_MATMUL, N_TRANSPOSE, N_INV, N_DET, N_LOGDET, N_TRACE, N_SUBMAT
};

typedef struct Num {
  int kind;
  int r, c;           /* shape (rows, cols); scalars are 1x1 */
  int nin;
  struct Num** in;    /* input nodes */
  int ia, ib, ic, id; /* immediates: param index, exponent, element/submatrix offsets */
  int dep;            /* 1 if the value depends on a parameter */
  int mark;           /* depth-first-search state for the backward ordering */
  double* v;          /* primal values, row-major r*c */
  double* g;          /* adjoint, allocated in the backward pass */
  double* d;          /* dual partials: d[e*P + k] = d v[e] / d theta_k (NULL = all zero) */
} Num;

typedef struct Clos {
  int nparams; int* params; /* interned parameter names */
  Val body;                 /* list of body expressions */
  struct Frame* env;
} Clos;

typedef struct Frame { int n; int* syms; Val* vals; struct Frame* parent; } Frame;

/* ------------------------------------------------------------------------- */
/* Program (parsed once, shared read-only by every lane and thread).          */
/* ------------------------------------------------------------------------- */
typedef struct {
  int nsyms, capsyms; char** names;
  Arena ast;      /* AST nodes live here */
  Val forms;      /* list of top-level forms */
  /* bytecode */
  int nins; int* bc_op; double* bc_f; long long* bc_i;
} Program;

/* per-lane evaluation context */
typedef struct {
  const Program* prog;
  Arena* ar;
  int mode, P, f32;  /* f32: round every arithmetic result to binary32 */
  const double* theta;     /* this lane's parameters */
  const double* obs; long long nobs;
  /* data-axis context for (dobs k) */
  int in_data; long long dbase;
  Frame* globals;
  jmp_buf jb;
  char* err; size_t errcap;
  int depth;
} Ctx;

/* fp32 mode: a result computed in double and rounded once to float is the correctly
 * rounded float result for + - * / and sqrt (53 >= 2*24 + 2 bits). */
#define RF(cx, x) ((cx)->f32 ? (double)(float)(x) : (x))

static void fail(Ctx* cx, const char* fmt, ...) {
  va_list ap; va_start(ap, fmt);
  vsnprintf(cx->err, cx->errcap, fmt, ap);
  va_end(ap);
  longjmp(cx->jb, 1);
}

/* ------------------------------------------------------------------------- */
/* Reader (section 3.2: symbols are interned to integers).                    */
/* ------------------------------------------------------------------------- */
static int intern(Program* pg, const char* s, size_t n) {
  for (int i = 0; i < pg->nsyms; i++)
    if (strlen(pg->names[i]) == n && memcmp(pg->names[i], s, n) == 0) return i;
  if (pg->nsyms == pg->capsyms) {
    pg->capsyms = pg->capsyms ? 2 * pg->capsyms : 64;
    pg->names = (char**)realloc(pg->names, sizeof(char*) * pg->capsyms);
  }
  char* c = (char*)malloc(n + 1); memcpy(c, s, n); c[n] = 0;
  pg->names[pg->nsyms] = c;
  return pg->nsyms++;
}

typedef struct { const char* s; size_t n, i; Program* pg; char* err; size_t errcap; int bad; } Reader;

static Val mkpair_ast(Program* pg, Val a, Val d) {
  Pair* p = (Pair*)arena_alloc(&pg->ast, sizeof(Pair));
  p->car = a; p->cdr = d;
  Val v; v.t = V_PAIR; v.u.p = p; return v;
}
static Val nil(void) { Val v; v.t = V_NIL; v.u.i = 0; return v; }

static void skip_ws(Reader* r) {
  while (r->i < r->n) {
    char ch = r->s[r->i];
    if (ch == ';') { while (r->i < r->n && r->s[r->i] != '\n') r->i++; }
    else if (ch == ' ' || ch == '\t' || ch == '\n' || ch == '\r') r->i++;
    else break;
  }
}

static Val read_form(Reader* r);

static Val read_atom(Reader* r) {
  size_t st = r->i;
  while (r->i < r->n) {
    char ch = r->s[r->i];
    if (ch == '(' || ch == ')' || ch == ' ' || ch == '\t' || ch == '\n' || ch == '\r' || ch == ';') break;
    r->i++;
  }
  size_t len = r->i - st;
  const char* t = r->s + st;
  char buf[128];
  Val v;
  if (len == 2 && t[0] == '#' && (t[1] == 't' || t[1] == 'f')) { v.t = V_BOOL; v.u.i = (t[1] == 't'); return v; }
  /* integer literal: optional sign then digits only -> structural integer */
  size_t k = 0; int isint = 1, isnum = 0;
  if (k < len && (t[k] == '+' || t[k] == '-')) k++;
  if (k == len) isint = 0;
  for (size_t j = k; j < len; j++) if (t[j] < '0' || t[j] > '9') { isint = 0; break; }
  if (!isint && len < sizeof(buf)) {
    memcpy(buf, t, len); buf[len] = 0;
    char* end = NULL;
    if ((buf[0] >= '0' && buf[0] <= '9') || buf[0] == '.' ||
        ((buf[0] == '-' || buf[0] == '+') && len > 1 && ((buf[1] >= '0' && buf[1] <= '9') || buf[1] == '.'))) {
      double f = strtod(buf, &end);
      if (end == buf + len) { isnum = 1; v.t = V_FLT; v.u.f = f; }
    }
  }
  if (isint) {
    if (len >= sizeof(buf)) { r->bad = 1; snprintf(r->err, r->errcap, "integer literal too long"); return nil(); }
    memcpy(buf, t, len); buf[len] = 0;
    v.t = V_INT; v.u.i = strtoll(buf, NULL, 10); return v;
  }
  if (isnum) return v;
  v.t = V_SYM; v.u.sym = intern(r->pg, t, len); return v;
}

static Val read_form(Reader* r) {
  skip_ws(r);
  if (r->i >= r->n) { r->bad = 1; snprintf(r->err, r->errcap, "unexpected end of program text"); return nil(); }
  char ch = r->s[r->i];
  if (ch == ')') { r->bad = 1; snprintf(r->err, r->errcap, "unexpected ')' at offset %zu", r->i); return nil(); }
  if (ch == '(') {
    r->i++;
    Val head = nil(); Pair* tail = NULL;
    for (;;) {
      skip_ws(r);
      if (r->i >= r->n) { r->bad = 1; snprintf(r->err, r->errcap, "missing ')'"); return nil(); }
      if (r->s[r->i] == ')') { r->i++; break; }
      Val x = read_form(r);
      if (r->bad) return nil();
      Val cell = mkpair_ast(r->pg, x, nil());
      if (tail) tail->cdr = cell; else head = cell;
      tail = cell.u.p;
    }
    return head;
  }
  return read_atom(r);
}

/* ------------------------------------------------------------------------- */
/* Bytecode reader (section 7, second client: a linear instruction stream).   */
/* ------------------------------------------------------------------------- */
enum {
  B_PUSH, B_PARAM, B_OBS, B_OBSN, B_LOAD, B_STORE, B_DUP, B_SWAP, B_POP, B_ADD, B_SUB, B_MUL,
  B_DIV, B_NEG, B_EXP, B_LOG, B_SIN, B_COS, B_TANH, B_SQRT, B_ABS, B_POW, B_POWI, B_LT, B_GT,
  B_LE, B_GE, B_SEL, B_LOOP, B_END, B_DOT, B_NOPS
};
static const char* bc_names[B_NOPS] = {
  "PUSH", "PARAM", "OBS", "OBSN", "LOAD", "STORE", "DUP", "SWAP", "POP", "ADD", "SUB", "MUL",
  "DIV", "NEG", "EXP", "LOG", "SIN", "COS", "TANH", "SQRT", "ABS", "POW", "POWI", "LT", "GT",
  "LE", "GE", "SEL", "LOOP", "END", "DOT"};

static int parse_bytecode(Program* pg, const char* s, size_t n, char* err, size_t errcap) {
  int cap = 64; pg->nins = 0;
  pg->bc_op = (int*)malloc(sizeof(int) * cap);
  pg->bc_f = (double*)malloc(sizeof(double) * cap);
  pg->bc_i = (long long*)malloc(sizeof(long long) * cap);
  size_t i = 0; int line = 1; int depth = 0;
  while (i < n) {
    /* one line */
    size_t st = i; while (i < n && s[i] != '\n') i++;
    size_t en = i; if (i < n) i++;
    char buf[256]; size_t len = en - st;
    if (len >= sizeof(buf)) { snprintf(err, errcap, "line %d too long", line); return OR_ERR; }
    memcpy(buf, s + st, len); buf[len] = 0;
    char* semi = strchr(buf, ';'); if (semi) *semi = 0;
    char op[32] = {0}, arg[200] = {0};
    int got = sscanf(buf, "%31s %199s", op, arg);
    if (got <= 0) { line++; continue; }
    int code = -1;
    for (int k = 0; k < B_NOPS; k++) if (strcmp(op, bc_names[k]) == 0) code = k;
    if (code < 0) { snprintf(err, errcap, "line %d: unknown instruction '%s'", line, op); return OR_ERR; }
    int needs = (code == B_PUSH || code == B_PARAM || code == B_OBS || code == B_LOAD || code == B_STORE ||
                 code == B_POWI || code == B_LOOP || code == B_DOT);
    if (needs && got < 2) { snprintf(err, errcap, "line %d: %s needs an operand", line, op); return OR_ERR; }
    if (!needs && got >= 2) { snprintf(err, errcap, "line %d: %s takes no operand", line, op); return OR_ERR; }
    if (pg->nins == cap) {
      cap *= 2;
      pg->bc_op = (int*)realloc(pg->bc_op, sizeof(int) * cap);
      pg->bc_f = (double*)realloc(pg->bc_f, sizeof(double) * cap);
      pg->bc_i = (long long*)realloc(pg->bc_i, sizeof(long long) * cap);
    }
    pg->bc_op[pg->nins] = code; pg->bc_f[pg->nins] = 0; pg->bc_i[pg->nins] = 0;
    if (needs) {
      char* end = NULL;
      if (code == B_PUSH) {
        pg->bc_f[pg->nins] = strtod(arg, &end);
      } else {
        pg->bc_i[pg->nins] = strtoll(arg, &end, 10);
      }
      if (!end || *end) { snprintf(err, errcap, "line %d: bad operand '%s'", line, arg); return OR_ERR; }
    }
    if (code == B_LOOP) depth++;
    if (code == B_END) { if (--depth < 0) { snprintf(err, errcap, "line %d: END without LOOP", line); return OR_ERR; } }
    pg->nins++; line++;
  }
  if (depth != 0) { snprintf(err, errcap, "LOOP without END"); return OR_ERR; }
  return OR_OK;
}

/* ------------------------------------------------------------------------- */
/* Numeric node construction.  Each constructor computes the primal (and, in */
/* dual mode, the partials) following Appendix C and readings R1-R7.          */
/* ------------------------------------------------------------------------- */
static Num* new_num(Ctx* cx, int kind, int r, int c, int nin) {
  Num* n = (Num*)arena_alloc(cx->ar, sizeof(Num));
  if (!n) fail(cx, "out of memory");
  memset(n, 0, sizeof(Num));
  n->kind = kind; n->r = r; n->c = c; n->nin = nin;
  n->in = nin ? (Num**)arena_alloc(cx->ar, sizeof(Num*) * nin) : NULL;
  n->v = (double*)arena_alloc(cx->ar, sizeof(double) * (size_t)r * c);
  if ((nin && !n->in) || !n->v) fail(cx, "out of memory");
  return n;
}
static double* dual_alloc(Ctx* cx, Num* n) {
  size_t m = (size_t)n->r * n->c * cx->P;
  n->d = (double*)arena_alloc(cx->ar, sizeof(double) * (m ? m : 1));
  if (!n->d) fail(cx, "out of memory");
  memset(n->d, 0, sizeof(double) * m);
  return n->d;
}
static int any_dep(Num* n) {
  for (int i = 0; i < n->nin; i++) if (n->in[i]->dep) return 1;
  return 0;
}
static Num* const_num(Ctx* cx, double x) {
  Num* n = new_num(cx, N_CONST, 1, 1, 0);
  n->v[0] = RF(cx, x); return n;
}
static int is_scalar(Num* n) { return n->r == 1 && n->c == 1; }

/* dual helper: partial of input i element e, or 0 */
static inline double dpart(Ctx* cx, Num* x, int e, int k) { return x->d ? x->d[(size_t)e * cx->P + k] : 0.0; }

/* unary scalar op: z = f(x), dz = f'(x) dx (dual mode only) */
static Num* unary(Ctx* cx, int kind, Num* x) {
  if (!is_scalar(x)) fail(cx, "scalar function applied to a %dx%d matrix", x->r, x->c);
  Num* z = new_num(cx, kind, 1, 1, 1);
  z->in[0] = x; z->dep = x->dep;
  double a = x->v[0], v = 0, dv = 0; /* dv = dz/dx */
  switch (kind) {
    case N_NEG: v = -a; dv = -1.0; break;
    case N_EXP: v = exp(a); dv = v; break;
    case N_LOG: v = log(a > 1e-8 ? a : 1e-8); dv = (a > 1e-8) ? 1.0 / a : 0.0; break;
    case N_SIN: v = sin(a); dv = cos(a); break;
    case N_COS: v = cos(a); dv = -sin(a); break;
    case N_TANH: v = tanh(a); dv = 1.0 - v * v; break;
    case N_SQRT: v = sqrt(a > 1e-8 ? a : 1e-8); dv = (a > 1e-8) ? 1.0 / (2.0 * v) : 0.0; break;
    case N_ABS: v = fabs(a); dv = (a > 0) ? 1.0 : (a < 0 ? -1.0 : 0.0); break;
    default: fail(cx, "internal: bad unary kind");
  }
  z->v[0] = RF(cx, v);
  if (cx->mode == MODE_DUAL && x->d) {
    dual_alloc(cx, z);
    for (int k = 0; k < cx->P; k++) z->d[k] = dv * x->d[k];
  }
  return z;
}

/* n-ary scalar arithmetic (R6) */
static Num* nary(Ctx* cx, int kind, int n, Num** xs) {
  for (int i = 0; i < n; i++) if (!is_scalar(xs[i])) fail(cx, "scalar arithmetic on a %dx%d matrix", xs[i]->r, xs[i]->c);
  Num* z = new_num(cx, kind, 1, 1, n);
  for (int i = 0; i < n; i++) z->in[i] = xs[i];
  z->dep = any_dep(z);
  double v = 0;
  if (kind == N_ADD) { v = xs[0]->v[0]; for (int i = 1; i < n; i++) v = RF(cx, v + xs[i]->v[0]); }
  else if (kind == N_SUB) {
    if (n == 1) v = -xs[0]->v[0];
    else { double s = xs[1]->v[0]; for (int i = 2; i < n; i++) s = RF(cx, s + xs[i]->v[0]); v = xs[0]->v[0] - s; }
  } else if (kind == N_MUL) { v = xs[0]->v[0]; for (int i = 1; i < n; i++) v = RF(cx, v * xs[i]->v[0]); }
  else if (kind == N_DIV) {
    if (n == 1) v = 1.0 / xs[0]->v[0];
    else { double p = xs[1]->v[0]; for (int i = 2; i < n; i++) p = RF(cx, p * xs[i]->v[0]); v = xs[0]->v[0] / p; }
  }
  z->v[0] = RF(cx, v);
  if (cx->mode == MODE_DUAL && z->dep) {
    dual_alloc(cx, z);
    for (int k = 0; k < cx->P; k++) {
      double s = 0;
      if (kind == N_ADD) { for (int i = 0; i < n; i++) s += dpart(cx, xs[i], 0, k); }
      else if (kind == N_SUB) {
        if (n == 1) s = -dpart(cx, xs[0], 0, k);
        else { s = dpart(cx, xs[0], 0, k); for (int i = 1; i < n; i++) s -= dpart(cx, xs[i], 0, k); }
      } else if (kind == N_MUL) {
        for (int i = 0; i < n; i++) {
          double di = dpart(cx, xs[i], 0, k);
          if (di == 0) continue;
          double p = 1.0;
          for (int j = 0; j < n; j++) if (j != i) p *= xs[j]->v[0];
          s += di * p;
        }
      } else { /* DIV */
        if (n == 1) { double x = xs[0]->v[0]; s = -dpart(cx, xs[0], 0, k) / (x * x); }
        else {
          double p = 1.0; for (int i = 1; i < n; i++) p *= xs[i]->v[0];
          s = dpart(cx, xs[0], 0, k) / p;
          for (int i = 1; i < n; i++) { double di = dpart(cx, xs[i], 0, k); if (di != 0) s -= v / xs[i]->v[0] * di; }
        }
      }
      z->d[k] = s;
    }
  }
  return z;
}

/* z = a^n by left-to-right repeated multiplication (R3) */
static double powi_rep(double a, long long n) {
  if (n == 0) return 1.0;
  double z = a;
  for (long long i = 1; i < n; i++) z = z * a;
  return z;
}
static Num* powi_num(Ctx* cx, Num* a, long long e) {
  if (!is_scalar(a)) fail(cx, "pow on a matrix");
  if (e < 0 || e > 64) fail(cx, "integer exponent %lld outside 0..64", e);
  Num* z = new_num(cx, N_POWI, 1, 1, 1);
  z->in[0] = a; z->ia = (int)e; z->dep = a->dep;
  z->v[0] = powi_rep(a->v[0], e);
  if (cx->mode == MODE_DUAL && a->d) {
    dual_alloc(cx, z);
    double dv = e == 0 ? 0.0 : (double)e * powi_rep(a->v[0], e - 1);
    for (int k = 0; k < cx->P; k++) z->d[k] = a->d[k] * dv;
  }
  return z;
}
/* general pow, Appendix C: a += g e z / a, e += g z ln a */
static Num* pow_num(Ctx* cx, Num* a, Num* e) {
  if (!is_scalar(a) || !is_scalar(e)) fail(cx, "pow on a matrix");
  Num* z = new_num(cx, N_POW, 1, 1, 2);
  z->in[0] = a; z->in[1] = e; z->dep = any_dep(z);
  double av = a->v[0], ev = e->v[0], zv = pow(av, ev);
  z->v[0] = zv;
  if (cx->mode == MODE_DUAL && z->dep) {
    dual_alloc(cx, z);
    for (int k = 0; k < cx->P; k++) {
      double s = 0, da = dpart(cx, a, 0, k), de = dpart(cx, e, 0, k);
      if (da != 0) s += da * ev * zv / av;
      if (de != 0) s += de * zv * log(av);
      z->d[k] = s;
    }
  }
  return z;
}
/* dot product, Appendix C "dot": a += g b, b += g a; sum left to right */
static Num* dot_num(Ctx* cx, int n, Num** a, Num** b) {
  Num* z = new_num(cx, N_DOT, 1, 1, 2 * n);
  for (int i = 0; i < n; i++) { z->in[i] = a[i]; z->in[n + i] = b[i]; }
  z->ia = n; z->dep = any_dep(z);
  double s = 0;
  for (int i = 0; i < n; i++) { double t = RF(cx, a[i]->v[0] * b[i]->v[0]); s = (i == 0) ? t : RF(cx, s + t); }
  z->v[0] = s;
  if (cx->mode == MODE_DUAL && z->dep) {
    dual_alloc(cx, z);
    for (int k = 0; k < cx->P; k++) {
      double d = 0;
      for (int i = 0; i < n; i++) d += dpart(cx, a[i], 0, k) * b[i]->v[0] + a[i]->v[0] * dpart(cx, b[i], 0, k);
      z->d[k] = d;
    }
  }
  return z;
}

/* ---- matrices (Appendix C "Matrix operations") ---- */
static Num* mat_from(Ctx* cx, int r, int c, Num** el) {
  Num* z = new_num(cx, N_MAT, r, c, r * c);
  for (int i = 0; i < r * c; i++) {
    if (!is_scalar(el[i])) fail(cx, "matrix element is not a scalar");
    z->in[i] = el[i]; z->v[i] = el[i]->v[0];
  }
  z->dep = any_dep(z);
  if (cx->mode == MODE_DUAL && z->dep) {
    dual_alloc(cx, z);
    for (int i = 0; i < r * c; i++) for (int k = 0; k < cx->P; k++) z->d[(size_t)i * cx->P + k] = dpart(cx, el[i], 0, k);
  }
  return z;
}
static Num* const_mat(Ctx* cx, int r, int c, const double* v) {
  Num* z = new_num(cx, N_CONST, r, c, 0);
  for (int i = 0; i < r * c; i++) z->v[i] = RF(cx, v[i]);
  return z;
}
static Num* mref_num(Ctx* cx, Num* a, long long i, long long j) {
  if (i < 0 || j < 0 || i >= a->r || j >= a->c) fail(cx, "mref (%lld,%lld) outside %dx%d", i, j, a->r, a->c);
  Num* z = new_num(cx, N_MREF, 1, 1, 1);
  z->in[0] = a; z->ia = (int)(i * a->c + j); z->dep = a->dep;
  z->v[0] = a->v[z->ia];
  if (cx->mode == MODE_DUAL && a->d) {
    dual_alloc(cx, z);
    for (int k = 0; k < cx->P; k++) z->d[k] = a->d[(size_t)z->ia * cx->P + k];
  }
  return z;
}
static Num* submat_num(Ctx* cx, Num* a, long long r0, long long nr, long long c0, long long nc) {
  if (r0 < 0 || c0 < 0 || nr < 1 || nc < 1 || r0 + nr > a->r || c0 + nc > a->c)
    fail(cx, "submatrix outside %dx%d", a->r, a->c);
  Num* z = new_num(cx, N_SUBMAT, (int)nr, (int)nc, 1);
  z->in[0] = a; z->ia = (int)r0; z->ib = (int)c0; z->dep = a->dep;
  for (int i = 0; i < nr; i++) for (int j = 0; j < nc; j++) z->v[i * nc + j] = a->v[(r0 + i) * a->c + c0 + j];
  if (cx->mode == MODE_DUAL && a->d) {
    dual_alloc(cx, z);
    for (int i = 0; i < nr; i++) for (int j = 0; j < nc; j++) for (int k = 0; k < cx->P; k++)
      z->d[(size_t)(i * nc + j) * cx->P + k] = a->d[(size_t)((r0 + i) * a->c + c0 + j) * cx->P + k];
  }
  return z;
}
static Num* madd_num(Ctx* cx, int kind, Num* a, Num* b) {
  if (a->r != b->r || a->c != b->c) fail(cx, "m+/m- shape mismatch %dx%d vs %dx%d", a->r, a->c, b->r, b->c);
  Num* z = new_num(cx, kind, a->r, a->c, 2);
  z->in[0] = a; z->in[1] = b; z->dep = any_dep(z);
  int m = a->r * a->c;
  for (int i = 0; i < m; i++) z->v[i] = RF(cx, kind == N_MADD ? a->v[i] + b->v[i] : a->v[i] - b->v[i]);
  if (cx->mode == MODE_DUAL && z->dep) {
    dual_alloc(cx, z);
    for (int i = 0; i < m; i++) for (int k = 0; k < cx->P; k++) {
      double da = dpart(cx, a, i, k), db = dpart(cx, b, i, k);
      z->d[(size_t)i * cx->P + k] = kind == N_MADD ? da + db : da - db;
    }
  }
  return z;
}
static Num* mscale_num(Ctx* cx, Num* s, Num* a) {
  if (!is_scalar(s)) fail(cx, "mscale needs a scalar first argument");
  Num* z = new_num(cx, N_MSCALE, a->r, a->c, 2);
  z->in[0] = s; z->in[1] = a; z->dep = any_dep(z);
  int m = a->r * a->c;
  for (int i = 0; i < m; i++) z->v[i] = RF(cx, s->v[0] * a->v[i]);
  if (cx->mode == MODE_DUAL && z->dep) {
    dual_alloc(cx, z);
    for (int i = 0; i < m; i++) for (int k = 0; k < cx->P; k++)
      z->d[(size_t)i * cx->P + k] = dpart(cx, s, 0, k) * a->v[i] + s->v[0] * dpart(cx, a, i, k);
  }
  return z;
}
static Num* matmul_num(Ctx* cx, Num* a, Num* b) {
  if (a->c != b->r) fail(cx, "matmul shape mismatch %dx%d * %dx%d", a->r, a->c, b->r, b->c);
  Num* z = new_num(cx, N_MATMUL, a->r, b->c, 2);
  z->in[0] = a; z->in[1] = b; z->dep = any_dep(z);
  int n = a->r, K = a->c, m = b->c;
  for (int i = 0; i < n; i++) for (int j = 0; j < m; j++) {
    double s = 0;
    for (int k = 0; k < K; k++) { double t = RF(cx, a->v[i * K + k] * b->v[k * m + j]); s = (k == 0) ? t : RF(cx, s + t); }
    z->v[i * m + j] = s;
  }
  if (cx->mode == MODE_DUAL && z->dep) {
    dual_alloc(cx, z);
    for (int i = 0; i < n; i++) for (int j = 0; j < m; j++) for (int p = 0; p < cx->P; p++) {
      double s = 0;
      for (int k = 0; k < K; k++) s += dpart(cx, a, i * K + k, p) * b->v[k * m + j] + a->v[i * K + k] * dpart(cx, b, k * m + j, p);
      z->d[(size_t)(i * m + j) * cx->P + p] = s;
    }
  }
  return z;
}
static Num* transpose_num(Ctx* cx, Num* a) {
  Num* z = new_num(cx, N_TRANSPOSE, a->c, a->r, 1);
  z->in[0] = a; z->dep = a->dep;
  for (int i = 0; i < a->r; i++) for (int j = 0; j < a->c; j++) z->v[j * a->r + i] = a->v[i * a->c + j];
  if (cx->mode == MODE_DUAL && a->d) {
    dual_alloc(cx, z);
    for (int i = 0; i < a->r; i++) for (int j = 0; j < a->c; j++) for (int k = 0; k < cx->P; k++)
      z->d[(size_t)(j * a->r + i) * cx->P + k] = a->d[(size_t)(i * a->c + j) * cx->P + k];
  }
  return z;
}

/* Inverse and determinant of an n x n matrix (R4): closed-form adjugate for n <= 3,
 * Gauss-Jordan elimination with partial pivoting otherwise. */
static void inv_det(Ctx* cx, int n, const double* a, double* inv, double* det) {
#define R(x) RF(cx, (x))
  if (n == 1) { *det = a[0]; inv[0] = R(1.0 / a[0]); return; }
  if (n == 2) {
    double d = R(R(a[0] * a[3]) - R(a[1] * a[2]));
    *det = d;
    inv[0] = R(a[3] / d); inv[1] = R(-a[1] / d); inv[2] = R(-a[2] / d); inv[3] = R(a[0] / d);
    return;
  }
  if (n == 3) {
    /* cofactors C_ij of A */
    double c00 = R(R(a[4] * a[8]) - R(a[5] * a[7]));
    double c01 = R(R(a[5] * a[6]) - R(a[3] * a[8]));
    double c02 = R(R(a[3] * a[7]) - R(a[4] * a[6]));
    double c10 = R(R(a[2] * a[7]) - R(a[1] * a[8]));
    double c11 = R(R(a[0] * a[8]) - R(a[2] * a[6]));
    double c12 = R(R(a[1] * a[6]) - R(a[0] * a[7]));
    double c20 = R(R(a[1] * a[5]) - R(a[2] * a[4]));
    double c21 = R(R(a[2] * a[3]) - R(a[0] * a[5]));
    double c22 = R(R(a[0] * a[4]) - R(a[1] * a[3]));
    double d = R(R(R(a[0] * c00) + R(a[1] * c01)) + R(a[2] * c02));
    *det = d;
    /* inverse = transpose of the cofactor matrix / det */
    inv[0] = R(c00 / d); inv[1] = R(c10 / d); inv[2] = R(c20 / d);
    inv[3] = R(c01 / d); inv[4] = R(c11 / d); inv[5] = R(c21 / d);
    inv[6] = R(c02 / d); inv[7] = R(c12 / d); inv[8] = R(c22 / d);
    return;
  }
  /* Gauss-Jordan on [A | I] */
  double* w = (double*)malloc(sizeof(double) * n * 2 * n);
  for (int i = 0; i < n; i++) for (int j = 0; j < 2 * n; j++)
    w[i * 2 * n + j] = j < n ? a[i * n + j] : (j - n == i ? 1.0 : 0.0);
  double d = 1.0;
  for (int col = 0; col < n; col++) {
    int piv = col; double best = fabs(w[col * 2 * n + col]);
    for (int i = col + 1; i < n; i++) if (fabs(w[i * 2 * n + col]) > best) { best = fabs(w[i * 2 * n + col]); piv = i; }
    if (piv != col) {
      for (int j = 0; j < 2 * n; j++) { double t = w[col * 2 * n + j]; w[col * 2 * n + j] = w[piv * 2 * n + j]; w[piv * 2 * n + j] = t; }
      d = -d;
    }
    double p = w[col * 2 * n + col];
    d = R(d * p);
    for (int j = 0; j < 2 * n; j++) w[col * 2 * n + j] = R(w[col * 2 * n + j] / p);
    for (int i = 0; i < n; i++) if (i != col) {
      double f = w[i * 2 * n + col];
      if (f != 0) for (int j = 0; j < 2 * n; j++) w[i * 2 * n + j] = R(w[i * 2 * n + j] - R(f * w[col * 2 * n + j]));
    }
  }
  for (int i = 0; i < n; i++) for (int j = 0; j < n; j++) inv[i * n + j] = w[i * 2 * n + n + j];
  *det = d;
  free(w);
#undef R
}

static Num* matfun_num(Ctx* cx, int kind, Num* a) {
  if (a->r != a->c) fail(cx, "square matrix required, got %dx%d", a->r, a->c);
  int n = a->r;
  if (kind == N_TRACE) {
    Num* z = new_num(cx, N_TRACE, 1, 1, 1);
    z->in[0] = a; z->dep = a->dep;
    double s = 0; for (int i = 0; i < n; i++) s = (i == 0) ? a->v[0] : RF(cx, s + a->v[i * n + i]);
    z->v[0] = s;
    if (cx->mode == MODE_DUAL && a->d) {
      dual_alloc(cx, z);
      for (int k = 0; k < cx->P; k++) { double t = 0; for (int i = 0; i < n; i++) t += a->d[(size_t)(i * n + i) * cx->P + k]; z->d[k] = t; }
    }
    return z;
  }
  double* inv = (double*)arena_alloc(cx->ar, sizeof(double) * n * n);
  double det;
  inv_det(cx, n, a->v, inv, &det);
  Num* z;
  if (kind == N_INV) {
    z = new_num(cx, N_INV, n, n, 1);
    memcpy(z->v, inv, sizeof(double) * n * n);
  } else {
    z = new_num(cx, kind, 1, 1, 1);
    z->v[0] = kind == N_DET ? det : RF(cx, log(det));
  }
  z->in[0] = a; z->dep = a->dep;
  if (cx->mode == MODE_DUAL && a->d) {
    dual_alloc(cx, z);
    for (int p = 0; p < cx->P; p++) {
      /* dA for this parameter */
      if (kind == N_INV) {
        /* d(A^-1) = -A^-1 dA A^-1 */
        for (int i = 0; i < n; i++) for (int j = 0; j < n; j++) {
          double s = 0;
          for (int k = 0; k < n; k++) for (int l = 0; l < n; l++)
            s += inv[i * n + k] * a->d[(size_t)(k * n + l) * cx->P + p] * inv[l * n + j];
          z->d[(size_t)(i * n + j) * cx->P + p] = -s;
        }
      } else {
        /* d ln det A = tr(A^-1 dA); d det A = det * tr(A^-1 dA) */
        double t = 0;
        for (int i = 0; i < n; i++) for (int k = 0; k < n; k++) t += inv[i * n + k] * a->d[(size_t)(k * n + i) * cx->P + p];
        z->d[p] = kind == N_DET ? det * t : t;
      }
    }
  }
  return z;
}

/* ------------------------------------------------------------------------- */
/* Backward pass (section 3.4 semantics, Appendix C rules; R5 zero skip).     */
/* The reachable graph is ordered by an explicit-stack depth-first search     */
/* from the loss; adjoints flow from the loss towards the parameters.         */
/* ------------------------------------------------------------------------- */
static double* gbuf(Ctx* cx, Num* n) {
  if (!n->g) {
    size_t m = (size_t)n->r * n->c;
    n->g = (double*)arena_alloc(cx->ar, sizeof(double) * m);
    if (!n->g) fail(cx, "out of memory");
    memset(n->g, 0, sizeof(double) * m);
  }
  return n->g;
}

static void backward(Ctx* cx, Num* loss, double* grad) {
  /* post-order over dependent nodes */
  size_t cap = 1024, cnt = 0, sp = 0;
  Num** order = (Num**)malloc(sizeof(Num*) * cap);
  size_t scap = 1024;
  Num** stk = (Num**)malloc(sizeof(Num*) * scap);
  int* sidx = (int*)malloc(sizeof(int) * scap);
  if (!loss->dep) { free(order); free(stk); free(sidx); return; }
  stk[0] = loss; sidx[0] = 0; sp = 1; loss->mark = 1;
  while (sp) {
    Num* n = stk[sp - 1];
    int i = sidx[sp - 1];
    if (i < n->nin) {
      sidx[sp - 1] = i + 1;
      Num* m = n->in[i];
      if (m->dep && m->mark != 1) {
        m->mark = 1;
        if (sp == scap) { scap *= 2; stk = (Num**)realloc(stk, sizeof(Num*) * scap); sidx = (int*)realloc(sidx, sizeof(int) * scap); }
        stk[sp] = m; sidx[sp] = 0; sp++;
      }
    } else {
      if (cnt == cap) { cap *= 2; order = (Num**)realloc(order, sizeof(Num*) * cap); }
      order[cnt++] = n; sp--;
    }
  }
  free(stk); free(sidx);
  gbuf(cx, loss)[0] = 1.0;
#define ADD(dst, v) ((dst) = RF(cx, (dst) + RF(cx, (v))))
#define SUB(dst, v) ((dst) = RF(cx, (dst) + -RF(cx, (v))))
  for (size_t q = cnt; q-- > 0;) {
    Num* n = order[q];
    size_t m = (size_t)n->r * n->c;
    double* g = n->g;
    if (!g) continue;
    int nz = 0;
    for (size_t e = 0; e < m; e++) if (g[e] != 0.0) { nz = 1; break; }
    if (!nz) continue; /* R5 */
    Num** x = n->in;
    switch (n->kind) {
      case N_CONST: break;
      case N_PARAM: ADD(grad[n->ia], g[0]); break;
      case N_ADD:
        for (int i = 0; i < n->nin; i++) if (x[i]->dep) ADD(gbuf(cx, x[i])[0], g[0]);
        break;
      case N_SUB:
        if (n->nin == 1) { if (x[0]->dep) SUB(gbuf(cx, x[0])[0], g[0]); }
        else {
          if (x[0]->dep) ADD(gbuf(cx, x[0])[0], g[0]);
          for (int i = 1; i < n->nin; i++) if (x[i]->dep) SUB(gbuf(cx, x[i])[0], g[0]);
        }
        break;
      case N_MUL:
        for (int i = 0; i < n->nin; i++) if (x[i]->dep) {
          double p = 1.0;
          for (int j = 0; j < n->nin; j++) if (j != i) p *= x[j]->v[0];
          ADD(gbuf(cx, x[i])[0], g[0] * p);
        }
        break;
      case N_DIV:
        if (n->nin == 1) {
          /* reciprocal: x -= g / x^2 */
          double a = x[0]->v[0];
          if (x[0]->dep) SUB(gbuf(cx, x[0])[0], g[0] / (a * a));
        } else {
          double p = 1.0; for (int i = 1; i < n->nin; i++) p *= x[i]->v[0];
          if (x[0]->dep) ADD(gbuf(cx, x[0])[0], g[0] / p);
          for (int i = 1; i < n->nin; i++) if (x[i]->dep) SUB(gbuf(cx, x[i])[0], g[0] * n->v[0] / x[i]->v[0]);
        }
        break;
      case N_NEG: SUB(gbuf(cx, x[0])[0], g[0]); break;
      case N_EXP: ADD(gbuf(cx, x[0])[0], g[0] * n->v[0]); break;
      case N_LOG: if (x[0]->v[0] > 1e-8) ADD(gbuf(cx, x[0])[0], g[0] / x[0]->v[0]); break;
      case N_SIN: ADD(gbuf(cx, x[0])[0], g[0] * cos(x[0]->v[0])); break;
      case N_COS: SUB(gbuf(cx, x[0])[0], g[0] * sin(x[0]->v[0])); break;
      case N_TANH: ADD(gbuf(cx, x[0])[0], g[0] * (1.0 - n->v[0] * n->v[0])); break;
      case N_SQRT: if (x[0]->v[0] > 1e-8) ADD(gbuf(cx, x[0])[0], g[0] / (2.0 * n->v[0])); break;
      case N_ABS: {
        double a = x[0]->v[0];
        double s = a > 0 ? 1.0 : (a < 0 ? -1.0 : 0.0);
        ADD(gbuf(cx, x[0])[0], g[0] * s);
        break;
      }
      case N_POWI: {
        long long e = n->ia;
        if (e > 0) ADD(gbuf(cx, x[0])[0], g[0] * ((double)e * powi_rep(x[0]->v[0], e - 1)));
        break;
      }
      case N_POW: {
        double a = x[0]->v[0], e = x[1]->v[0], z = n->v[0];
        if (x[0]->dep) ADD(gbuf(cx, x[0])[0], g[0] * e * z / a);
        if (x[1]->dep) ADD(gbuf(cx, x[1])[0], g[0] * z * log(a));
        break;
      }
      case N_DOT: {
        int k = n->ia;
        for (int i = 0; i < k; i++) {
          if (x[i]->dep) ADD(gbuf(cx, x[i])[0], g[0] * x[k + i]->v[0]);
          if (x[k + i]->dep) ADD(gbuf(cx, x[k + i])[0], g[0] * x[i]->v[0]);
        }
        break;
      }
      case N_SELECTED: ADD(gbuf(cx, x[0])[0], g[0]); break;
      case N_MAT:
        for (int i = 0; i < n->nin; i++) if (x[i]->dep) ADD(gbuf(cx, x[i])[0], g[i]);
        break;
      case N_MREF: ADD(gbuf(cx, x[0])[n->ia], g[0]); break;
      case N_SUBMAT: {
        double* ga = gbuf(cx, x[0]);
        for (int i = 0; i < n->r; i++) for (int j = 0; j < n->c; j++) ADD(ga[(n->ia + i) * x[0]->c + n->ib + j], g[i * n->c + j]);
        break;
      }
      case N_MADD: case N_MSUB:
        if (x[0]->dep) { double* ga = gbuf(cx, x[0]); for (size_t e = 0; e < m; e++) ADD(ga[e], g[e]); }
        if (x[1]->dep) {
          double* gb = gbuf(cx, x[1]);
          for (size_t e = 0; e < m; e++) ADD(gb[e], n->kind == N_MADD ? g[e] : -g[e]);
        }
        break;
      case N_MSCALE: {
        Num* s = x[0]; Num* a = x[1];
        if (s->dep) { double t = 0; for (size_t e = 0; e < m; e++) t = RF(cx, t + RF(cx, g[e] * a->v[e])); ADD(gbuf(cx, s)[0], t); }
        if (a->dep) { double* ga = gbuf(cx, a); for (size_t e = 0; e < m; e++) ADD(ga[e], s->v[0] * g[e]); }
        break;
      }
      case N_MATMUL: {
        /* Z = A B:  A += g B^T,  B += A^T g */
        Num* A = x[0]; Num* B = x[1];
        int nr = A->r, K = A->c, nc = B->c;
        if (A->dep) {
          double* ga = gbuf(cx, A);
          for (int i = 0; i < nr; i++) for (int k = 0; k < K; k++) {
            double s = 0; for (int j = 0; j < nc; j++) s = RF(cx, s + RF(cx, g[i * nc + j] * B->v[k * nc + j]));
            ADD(ga[i * K + k], s);
          }
        }
        if (B->dep) {
          double* gb = gbuf(cx, B);
          for (int k = 0; k < K; k++) for (int j = 0; j < nc; j++) {
            double s = 0; for (int i = 0; i < nr; i++) s = RF(cx, s + RF(cx, A->v[i * K + k] * g[i * nc + j]));
            ADD(gb[k * nc + j], s);
          }
        }
        break;
      }
      case N_TRANSPOSE: {
        double* ga = gbuf(cx, x[0]);
        int r = x[0]->r, c = x[0]->c;
        for (int i = 0; i < r; i++) for (int j = 0; j < c; j++) ADD(ga[i * c + j], g[j * r + i]);
        break;
      }
      case N_TRACE: {
        double* ga = gbuf(cx, x[0]);
        for (int i = 0; i < x[0]->r; i++) ADD(ga[i * x[0]->r + i], g[0]);
        break;
      }
      case N_INV: {
        /* B = A^-1:  A -= B^T g B^T */
        int k = n->r; double* Bv = n->v; double* ga = gbuf(cx, x[0]);
        for (int i = 0; i < k; i++) for (int j = 0; j < k; j++) {
          double s = 0;
          for (int p = 0; p < k; p++) for (int q2 = 0; q2 < k; q2++)
            s = RF(cx, s + RF(cx, RF(cx, Bv[p * k + i] * g[p * k + q2]) * Bv[j * k + q2]));
          SUB(ga[i * k + j], s);
        }
        break;
      }
      case N_DET: case N_LOGDET: {
        /* det: A += g z A^-T ; logdet: A += g A^-T */
        int k = x[0]->r;
        double* inv = (double*)malloc(sizeof(double) * k * k);
        double det;
        inv_det(cx, k, x[0]->v, inv, &det);
        double f = n->kind == N_DET ? RF(cx, g[0] * n->v[0]) : g[0];
        double* ga = gbuf(cx, x[0]);
        for (int i = 0; i < k; i++) for (int j = 0; j < k; j++) ADD(ga[i * k + j], f * inv[j * k + i]);
        free(inv);
        break;
      }
      default: free(order); fail(cx, "internal: no adjoint rule for node kind %d", n->kind);
    }
  }
#undef ADD
#undef SUB
  free(order);
}

/* ------------------------------------------------------------------------- */
/* Evaluator (section 3.3: exact realized trace, proper tail calls).         */
/* ------------------------------------------------------------------------- */
static Val mkint(long long i) { Val v; v.t = V_INT; v.u.i = i; return v; }
static Val mkbool(int b) { Val v; v.t = V_BOOL; v.u.i = b; return v; }
static Val mkpbool(int b) { Val v; v.t = V_PBOOL; v.u.i = b; return v; }
static Val mknum(Num* n) { Val v; v.t = V_NUM; v.u.n = n; return v; }
static Val cons(Ctx* cx, Val a, Val d) {
  Pair* p = (Pair*)arena_alloc(cx->ar, sizeof(Pair));
  if (!p) fail(cx, "out of memory");
  p->car = a; p->cdr = d;
  Val v; v.t = V_PAIR; v.u.p = p; return v;
}

static const char* symname(Ctx* cx, int s) { return cx->prog->names[s]; }
static int symeq(Ctx* cx, Val x, const char* s) { return x.t == V_SYM && strcmp(symname(cx, x.u.sym), s) == 0; }

static int list_len(Val x) { int n = 0; while (x.t == V_PAIR) { n++; x = x.u.p->cdr; } return n; }
static Val nth(Val x, int i) { while (i-- > 0) x = x.u.p->cdr; return x.u.p->car; }

static Frame* new_frame(Ctx* cx, int n, Frame* parent) {
  Frame* f = (Frame*)arena_alloc(cx->ar, sizeof(Frame));
  f->n = n; f->parent = parent;
  f->syms = (int*)arena_alloc(cx->ar, sizeof(int) * (n ? n : 1));
  f->vals = (Val*)arena_alloc(cx->ar, sizeof(Val) * (n ? n : 1));
  return f;
}
static Val lookup(Ctx* cx, Frame* env, int sym) {
  for (Frame* f = env; f; f = f->parent)
    for (int i = f->n - 1; i >= 0; i--) if (f->syms[i] == sym) return f->vals[i];
  fail(cx, "unbound variable '%s'", symname(cx, sym));
  return nil();
}
static void global_define(Ctx* cx, int sym, Val v) {
  Frame* g = cx->globals;
  for (int i = 0; i < g->n; i++) if (g->syms[i] == sym) { g->vals[i] = v; return; }
  /* grow the global frame */
  int n = g->n + 1;
  int* s = (int*)arena_alloc(cx->ar, sizeof(int) * n);
  Val* vv = (Val*)arena_alloc(cx->ar, sizeof(Val) * n);
  memcpy(s, g->syms, sizeof(int) * g->n); memcpy(vv, g->vals, sizeof(Val) * g->n);
  s[g->n] = sym; vv[g->n] = v;
  g->syms = s; g->vals = vv; g->n = n;
}

/* primitive procedures */
enum {
  P_ADD, P_SUB, P_MUL, P_DIV, P_EXP, P_LOG, P_SIN, P_COS, P_TANH, P_SQRT, P_ABS, P_POW, P_EXPT,
  P_LT, P_LE, P_GT, P_GE, P_EQ, P_NOT, P_QUOT, P_REM, P_PARAM, P_OBS, P_DOBS, P_OBSVEC,
  P_CONS, P_CAR, P_CDR, P_LIST, P_NULLP, P_PAIRP, P_LENGTH, P_LISTREF,
  P_MATRIX, P_MREF, P_MADD, P_MSUB, P_MSCALE, P_MATMUL, P_TRANSPOSE, P_INV, P_DET, P_LOGDET,
  P_TRACE, P_IDENTITY, P_ZEROS, P_SUBMAT, P_ROWS, P_COLS, P_EXACT2INEXACT, P_DOT, P_NPRIMS
};
static const char* prim_names[P_NPRIMS] = {
  "+", "-", "*", "/", "exp", "log", "sin", "cos", "tanh", "sqrt", "abs", "pow", "expt",
  "<", "<=", ">", ">=", "=", "not", "quotient", "remainder", "param", "obs", "dobs", "obs-vec",
  "cons", "car", "cdr", "list", "null?", "pair?", "length", "list-ref",
  "matrix", "mref", "m+", "m-", "mscale", "matmul", "transpose", "inv", "det", "logdet",
  "trace", "identity", "zeros", "submatrix", "rows", "cols", "exact->inexact", "dot"};

static Num* to_num(Ctx* cx, Val v) {
  if (v.t == V_NUM) return v.u.n;
  if (v.t == V_INT) return const_num(cx, (double)v.u.i);
  fail(cx, "number expected");
  return NULL;
}
static long long to_int(Ctx* cx, Val v, const char* what) {
  if (v.t != V_INT) fail(cx, "%s: structural integer expected", what);
  return v.u.i;
}

static Val apply_prim(Ctx* cx, int p, int argc, Val* av) {
#define NEED(k) do { if (argc != (k)) fail(cx, "%s expects %d argument(s), got %d", prim_names[p], (k), argc); } while (0)
  switch (p) {
    case P_ADD: case P_SUB: case P_MUL: case P_DIV: {
      if (argc < 1) fail(cx, "%s needs at least one argument", prim_names[p]);
      int allint = 1;
      for (int i = 0; i < argc; i++) {
        if (av[i].t != V_INT && av[i].t != V_NUM) fail(cx, "%s: number expected", prim_names[p]);
        if (av[i].t != V_INT) allint = 0;
      }
      if (allint && p != P_DIV) {
        long long v = av[0].u.i;
        if (p == P_SUB && argc == 1) return mkint(-v);
        for (int i = 1; i < argc; i++) v = p == P_ADD ? v + av[i].u.i : p == P_SUB ? v - av[i].u.i : v * av[i].u.i;
        return mkint(v);
      }
      Num** xs = (Num**)arena_alloc(cx->ar, sizeof(Num*) * argc);
      for (int i = 0; i < argc; i++) xs[i] = to_num(cx, av[i]);
      if (p == P_SUB && argc == 1) return mknum(unary(cx, N_NEG, xs[0]));
      int kind = p == P_ADD ? N_ADD : p == P_SUB ? N_SUB : p == P_MUL ? N_MUL : N_DIV;
      return mknum(nary(cx, kind, argc, xs));
    }
    case P_EXP: case P_LOG: case P_SIN: case P_COS: case P_TANH: case P_SQRT: case P_ABS: {
      NEED(1);
      int kind = p == P_EXP ? N_EXP : p == P_LOG ? N_LOG : p == P_SIN ? N_SIN : p == P_COS ? N_COS
               : p == P_TANH ? N_TANH : p == P_SQRT ? N_SQRT : N_ABS;
      return mknum(unary(cx, kind, to_num(cx, av[0])));
    }
    case P_POW: case P_EXPT: {
      NEED(2);
      if (av[1].t == V_INT) return mknum(powi_num(cx, to_num(cx, av[0]), av[1].u.i));
      return mknum(pow_num(cx, to_num(cx, av[0]), to_num(cx, av[1])));
    }
    case P_LT: case P_LE: case P_GT: case P_GE: case P_EQ: {
      NEED(2);
      if (av[0].t == V_INT && av[1].t == V_INT) {
        long long a = av[0].u.i, b = av[1].u.i;
        int r = p == P_LT ? a < b : p == P_LE ? a <= b : p == P_GT ? a > b : p == P_GE ? a >= b : a == b;
        return mkbool(r);
      }
      Num* a = to_num(cx, av[0]); Num* b = to_num(cx, av[1]);
      if (!is_scalar(a) || !is_scalar(b)) fail(cx, "comparison of matrices");
      double x = a->v[0], y = b->v[0];
      int r = p == P_LT ? x < y : p == P_LE ? x <= y : p == P_GT ? x > y : p == P_GE ? x >= y : x == y;
      return mkpbool(r);
    }
    case P_NOT: NEED(1); if (av[0].t != V_BOOL) fail(cx, "not: structural boolean expected"); return mkbool(!av[0].u.i);
    case P_QUOT: case P_REM: {
      NEED(2);
      long long a = to_int(cx, av[0], prim_names[p]), b = to_int(cx, av[1], prim_names[p]);
      if (b == 0) fail(cx, "%s by zero", prim_names[p]);
      return mkint(p == P_QUOT ? a / b : a % b);
    }
    case P_PARAM: {
      NEED(1);
      long long k = to_int(cx, av[0], "param");
      if (k < 0 || k >= cx->P) fail(cx, "param index %lld outside 0..%d", k, cx->P - 1);
      Num* z = new_num(cx, N_PARAM, 1, 1, 0);
      z->ia = (int)k; z->dep = 1; z->v[0] = cx->theta[k];
      if (cx->mode == MODE_DUAL) { dual_alloc(cx, z); z->d[k] = 1.0; }
      return mknum(z);
    }
    case P_OBS: {
      NEED(1);
      long long k = to_int(cx, av[0], "obs");
      if (k < 0 || k >= cx->nobs) fail(cx, "obs index %lld outside 0..%lld", k, cx->nobs - 1);
      return mknum(const_num(cx, cx->obs[k]));
    }
    case P_DOBS: {
      NEED(1);
      if (!cx->in_data) fail(cx, "dobs outside data-sum");
      long long k = to_int(cx, av[0], "dobs");
      long long idx = cx->dbase + k;
      if (k < 0 || idx < 0 || idx >= cx->nobs) fail(cx, "dobs index %lld outside the observations", idx);
      return mknum(const_num(cx, cx->obs[idx]));
    }
    case P_OBSVEC: {
      NEED(2);
      long long k = to_int(cx, av[0], "obs-vec"), n = to_int(cx, av[1], "obs-vec");
      if (n < 1 || k < 0 || k + n > cx->nobs) fail(cx, "obs-vec range outside the observations");
      return mknum(const_mat(cx, (int)n, 1, cx->obs + k));
    }
    case P_CONS: NEED(2); return cons(cx, av[0], av[1]);
    case P_CAR: NEED(1); if (av[0].t != V_PAIR) fail(cx, "car of a non-pair"); return av[0].u.p->car;
    case P_CDR: NEED(1); if (av[0].t != V_PAIR) fail(cx, "cdr of a non-pair"); return av[0].u.p->cdr;
    case P_LIST: { Val r = nil(); for (int i = argc - 1; i >= 0; i--) r = cons(cx, av[i], r); return r; }
    case P_NULLP: NEED(1); return mkbool(av[0].t == V_NIL);
    case P_PAIRP: NEED(1); return mkbool(av[0].t == V_PAIR);
    case P_LENGTH: NEED(1); return mkint(list_len(av[0]));
    case P_LISTREF: {
      NEED(2);
      long long k = to_int(cx, av[1], "list-ref");
      if (k < 0 || k >= list_len(av[0])) fail(cx, "list-ref index out of range");
      return nth(av[0], (int)k);
    }
    case P_MATRIX: {
      if (argc < 2) fail(cx, "matrix needs rows and cols");
      long long r = to_int(cx, av[0], "matrix"), c = to_int(cx, av[1], "matrix");
      if (r < 1 || c < 1 || r > 64 || c > 64) fail(cx, "matrix shape %lldx%lld outside 1..64", r, c);
      if (argc != 2 + r * c) fail(cx, "matrix %lldx%lld needs %lld elements, got %d", r, c, r * c, argc - 2);
      int allconst = 1;
      for (int i = 0; i < r * c; i++) {
        Val e = av[2 + i];
        if (e.t == V_NUM && (e.u.n->dep || !is_scalar(e.u.n))) allconst = 0;
        else if (e.t != V_NUM && e.t != V_INT) fail(cx, "matrix element must be a number");
      }
      if (allconst) {
        double* v = (double*)arena_alloc(cx->ar, sizeof(double) * r * c);
        for (int i = 0; i < r * c; i++) v[i] = av[2 + i].t == V_INT ? (double)av[2 + i].u.i : av[2 + i].u.n->v[0];
        return mknum(const_mat(cx, (int)r, (int)c, v));
      }
      Num** el = (Num**)arena_alloc(cx->ar, sizeof(Num*) * r * c);
      for (int i = 0; i < r * c; i++) el[i] = to_num(cx, av[2 + i]);
      return mknum(mat_from(cx, (int)r, (int)c, el));
    }
    case P_MREF: NEED(3); return mknum(mref_num(cx, to_num(cx, av[0]), to_int(cx, av[1], "mref"), to_int(cx, av[2], "mref")));
    case P_MADD: NEED(2); return mknum(madd_num(cx, N_MADD, to_num(cx, av[0]), to_num(cx, av[1])));
    case P_MSUB: NEED(2); return mknum(madd_num(cx, N_MSUB, to_num(cx, av[0]), to_num(cx, av[1])));
    case P_MSCALE: NEED(2); return mknum(mscale_num(cx, to_num(cx, av[0]), to_num(cx, av[1])));
    case P_MATMUL: NEED(2); return mknum(matmul_num(cx, to_num(cx, av[0]), to_num(cx, av[1])));
    case P_TRANSPOSE: NEED(1); return mknum(transpose_num(cx, to_num(cx, av[0])));
    case P_INV: NEED(1); return mknum(matfun_num(cx, N_INV, to_num(cx, av[0])));
    case P_DET: NEED(1); return mknum(matfun_num(cx, N_DET, to_num(cx, av[0])));
    case P_LOGDET: NEED(1); return mknum(matfun_num(cx, N_LOGDET, to_num(cx, av[0])));
    case P_TRACE: NEED(1); return mknum(matfun_num(cx, N_TRACE, to_num(cx, av[0])));
    case P_IDENTITY: case P_ZEROS: {
      long long r, c;
      if (p == P_IDENTITY) { NEED(1); r = c = to_int(cx, av[0], "identity"); }
      else { NEED(2); r = to_int(cx, av[0], "zeros"); c = to_int(cx, av[1], "zeros"); }
      if (r < 1 || c < 1 || r > 64 || c > 64) fail(cx, "matrix shape outside 1..64");
      double* v = (double*)arena_alloc(cx->ar, sizeof(double) * r * c);
      for (int i = 0; i < r; i++) for (int j = 0; j < c; j++) v[i * c + j] = (p == P_IDENTITY && i == j) ? 1.0 : 0.0;
      return mknum(const_mat(cx, (int)r, (int)c, v));
    }
    case P_SUBMAT: NEED(5);
      return mknum(submat_num(cx, to_num(cx, av[0]), to_int(cx, av[1], "submatrix"), to_int(cx, av[2], "submatrix"),
                              to_int(cx, av[3], "submatrix"), to_int(cx, av[4], "submatrix")));
    case P_ROWS: NEED(1); return mkint(to_num(cx, av[0])->r);
    case P_COLS: NEED(1); return mkint(to_num(cx, av[0])->c);
    case P_EXACT2INEXACT: NEED(1); return mknum(const_num(cx, (double)to_int(cx, av[0], "exact->inexact")));
    case P_DOT: {
      NEED(2);
      Num* a = to_num(cx, av[0]); Num* b = to_num(cx, av[1]);
      if (a->c != 1 || b->c != 1 || a->r != b->r) fail(cx, "dot needs two column vectors of equal length");
      int n = a->r;
      Num** ae = (Num**)arena_alloc(cx->ar, sizeof(Num*) * n);
      Num** be = (Num**)arena_alloc(cx->ar, sizeof(Num*) * n);
      for (int i = 0; i < n; i++) { ae[i] = mref_num(cx, a, i, 0); be[i] = mref_num(cx, b, i, 0); }
      return mknum(dot_num(cx, n, ae, be));
    }
  }
  fail(cx, "internal: unknown primitive");
  return nil();
#undef NEED
}

static Val eval(Ctx* cx, Val x, Frame* env);

static Val eval_body(Ctx* cx, Val body, Frame* env, Val* last) {
  /* evaluate all but the last expression; return the last unevaluated (for the tail loop) */
  if (body.t != V_PAIR) fail(cx, "empty body");
  while (body.u.p->cdr.t == V_PAIR) { eval(cx, body.u.p->car, env); body = body.u.p->cdr; }
  *last = body.u.p->car;
  return nil();
}

static Val make_closure(Ctx* cx, Val params, Val body, Frame* env) {
  Clos* c = (Clos*)arena_alloc(cx->ar, sizeof(Clos));
  int n = list_len(params);
  c->nparams = n; c->params = (int*)arena_alloc(cx->ar, sizeof(int) * (n ? n : 1));
  for (int i = 0; i < n; i++) {
    Val s = nth(params, i);
    if (s.t != V_SYM) fail(cx, "lambda parameter must be a symbol");
    c->params[i] = s.u.sym;
  }
  c->body = body; c->env = env;
  Val v; v.t = V_CLOS; v.u.c = c; return v;
}

/* select for a per-lane branch: the oracle simply evaluates the branch taken (R1) */
static Val eval(Ctx* cx, Val x, Frame* env) {
  if (++cx->depth > 10000) fail(cx, "evaluation nested too deeply");
  for (;;) {
    switch (x.t) {
      case V_SYM: cx->depth--; return lookup(cx, env, x.u.sym);
      case V_INT: case V_BOOL: cx->depth--; return x;
      case V_FLT: cx->depth--; return mknum(const_num(cx, x.u.f));
      case V_PAIR: break;
      default: fail(cx, "cannot evaluate this form");
    }
    Val head = x.u.p->car;
    Val rest = x.u.p->cdr;
    if (head.t == V_SYM) {
      const char* h = symname(cx, head.u.sym);
      if (strcmp(h, "quote") == 0) { cx->depth--; return rest.u.p->car; }
      if (strcmp(h, "if") == 0) {
        int n = list_len(rest);
        if (n != 3) fail(cx, "if needs exactly a test, a consequent and an alternative");
        Val c = eval(cx, nth(rest, 0), env);
        int take;
        if (c.t == V_BOOL || c.t == V_PBOOL) take = (int)c.u.i;
        else fail(cx, "if: test must be a boolean");
        x = nth(rest, take ? 1 : 2);
        if (c.t == V_PBOOL) {
          /* per-lane branch: the value must be numeric; mark it so gradient flows only here */
          Val r = eval(cx, x, env);
          if (r.t == V_INT) r = mknum(const_num(cx, (double)r.u.i));
          if (r.t != V_NUM) fail(cx, "a branch on a numeric test must produce a number");
          if (!is_scalar(r.u.n)) fail(cx, "a branch on a numeric test must produce a scalar");
          Num* z = new_num(cx, N_SELECTED, 1, 1, 1);
          z->in[0] = r.u.n; z->dep = r.u.n->dep; z->v[0] = r.u.n->v[0];
          if (cx->mode == MODE_DUAL && r.u.n->d) { dual_alloc(cx, z); memcpy(z->d, r.u.n->d, sizeof(double) * cx->P); }
          cx->depth--;
          return mknum(z);
        }
        continue;
      }
      if (strcmp(h, "and") == 0 || strcmp(h, "or") == 0) {
        int isand = h[0] == 'a';
        Val r = mkbool(isand);
        for (Val e = rest; e.t == V_PAIR; e = e.u.p->cdr) {
          r = eval(cx, e.u.p->car, env);
          if (r.t != V_BOOL) fail(cx, "%s: structural boolean expected", h);
          if (isand ? !r.u.i : r.u.i) break;
        }
        cx->depth--;
        return r;
      }
      if (strcmp(h, "begin") == 0) { Val last; eval_body(cx, rest, env, &last); x = last; continue; }
      if (strcmp(h, "lambda") == 0) { cx->depth--; return make_closure(cx, rest.u.p->car, rest.u.p->cdr, env); }
      if (strcmp(h, "let") == 0 || strcmp(h, "let*") == 0) {
        int star = h[3] == '*';
        Val b = rest.u.p->car;
        if (!star && b.t == V_SYM) {
          /* named let: (let name ((v init) ...) body...) */
          int name = b.u.sym;
          Val binds = nth(rest, 1);
          Val body = rest.u.p->cdr.u.p->cdr;
          int n = list_len(binds);
          Frame* lf = new_frame(cx, 1, env);
          Val params = nil();
          for (int i = n - 1; i >= 0; i--) params = cons(cx, nth(nth(binds, i), 0), params);
          Val clo = make_closure(cx, params, body, lf);
          lf->syms[0] = name; lf->vals[0] = clo;
          Frame* f = new_frame(cx, n, lf);
          for (int i = 0; i < n; i++) { f->syms[i] = nth(nth(binds, i), 0).u.sym; f->vals[i] = eval(cx, nth(nth(binds, i), 1), env); }
          Val last; eval_body(cx, body, f, &last); x = last; env = f; continue;
        }
        int n = list_len(b);
        Frame* f;
        if (star) {
          f = env;
          for (int i = 0; i < n; i++) {
            Val bi = nth(b, i);
            if (bi.t != V_PAIR || list_len(bi) != 2 || nth(bi, 0).t != V_SYM) fail(cx, "bad let* binding");
            Val v = eval(cx, nth(bi, 1), f);
            Frame* nf = new_frame(cx, 1, f);
            nf->syms[0] = nth(bi, 0).u.sym; nf->vals[0] = v; f = nf;
          }
        } else {
          f = new_frame(cx, n, env);
          for (int i = 0; i < n; i++) {
            Val bi = nth(b, i);
            if (bi.t != V_PAIR || list_len(bi) != 2 || nth(bi, 0).t != V_SYM) fail(cx, "bad let binding");
            f->syms[i] = nth(bi, 0).u.sym; f->vals[i] = eval(cx, nth(bi, 1), env);
          }
        }
        Val last; eval_body(cx, rest.u.p->cdr, f, &last); x = last; env = f; continue;
      }
      if (strcmp(h, "data-sum") == 0) {
        /* (data-sum N S [BASE] body), R7 */
        int n = list_len(rest);
        if (n != 3 && n != 4) fail(cx, "data-sum needs N S [BASE] body");
        long long N = to_int(cx, eval(cx, nth(rest, 0), env), "data-sum N");
        long long S = to_int(cx, eval(cx, nth(rest, 1), env), "data-sum S");
        long long base = n == 4 ? to_int(cx, eval(cx, nth(rest, 2), env), "data-sum BASE") : 0;
        Val body = nth(rest, n - 1);
        if (cx->in_data) fail(cx, "nested data-sum");
        if (N < 0 || S < 0) fail(cx, "data-sum N and S must be >= 0");
        Num* acc = NULL;
        for (long long d = 0; d < N; d++) {
          cx->in_data = 1; cx->dbase = base + d * S;
          Val r = eval(cx, body, env);
          cx->in_data = 0;
          if (r.t == V_INT) r = mknum(const_num(cx, (double)r.u.i));
          if (r.t != V_NUM || !is_scalar(r.u.n)) fail(cx, "data-sum body must produce a scalar number");
          if (!acc) acc = r.u.n;
          else { Num* two[2] = {acc, r.u.n}; acc = nary(cx, N_ADD, 2, two); }
        }
        if (!acc) acc = const_num(cx, 0.0);
        cx->depth--;
        return mknum(acc);
      }
      if (strcmp(h, "define") == 0 || strcmp(h, "model") == 0) fail(cx, "%s is only allowed at top level", h);
    }
    /* application */
    Val f = eval(cx, head, env);
    int argc = list_len(rest);
    Val* av = (Val*)arena_alloc(cx->ar, sizeof(Val) * (argc ? argc : 1));
    int i = 0;
    for (Val e = rest; e.t == V_PAIR; e = e.u.p->cdr) av[i++] = eval(cx, e.u.p->car, env);
    if (f.t == V_PRIM) { cx->depth--; return apply_prim(cx, f.u.prim, argc, av); }
    if (f.t != V_CLOS) fail(cx, "application of a non-procedure");
    Clos* c = f.u.c;
    if (c->nparams != argc) fail(cx, "procedure expects %d argument(s), got %d", c->nparams, argc);
    Frame* nf = new_frame(cx, argc, c->env);
    for (int k = 0; k < argc; k++) { nf->syms[k] = c->params[k]; nf->vals[k] = av[k]; }
    Val last; eval_body(cx, c->body, nf, &last);
    x = last; env = nf; /* proper tail call */
  }
}

/* Run the top-level forms; the (model (params ...) body...) form gives the loss. */
static Num* run_scheme(Ctx* cx) {
  cx->globals = new_frame(cx, 0, NULL);
  /* primitives */
  for (int p = 0; p < P_NPRIMS; p++) {
    int s = -1;
    for (int i = 0; i < cx->prog->nsyms; i++) if (strcmp(cx->prog->names[i], prim_names[p]) == 0) { s = i; break; }
    if (s < 0) continue; /* not used by this program */
    Val v; v.t = V_PRIM; v.u.prim = p;
    global_define(cx, s, v);
  }
  Num* loss = NULL; int nmodel = 0;
  for (Val fs = cx->prog->forms; fs.t == V_PAIR; fs = fs.u.p->cdr) {
    Val f = fs.u.p->car;
    if (f.t == V_PAIR && symeq(cx, f.u.p->car, "define")) {
      Val t = nth(f, 1);
      if (t.t == V_SYM) global_define(cx, t.u.sym, eval(cx, nth(f, 2), cx->globals));
      else if (t.t == V_PAIR && t.u.p->car.t == V_SYM)
        global_define(cx, t.u.p->car.u.sym, make_closure(cx, t.u.p->cdr, f.u.p->cdr.u.p->cdr, cx->globals));
      else fail(cx, "bad define");
      continue;
    }
    if (f.t == V_PAIR && symeq(cx, f.u.p->car, "model")) {
      if (nmodel++) fail(cx, "more than one model form");
      Val ps = nth(f, 1);
      if (ps.t != V_PAIR || !symeq(cx, ps.u.p->car, "params")) fail(cx, "model needs (params name...)");
      int np = list_len(ps) - 1;
      if (np != cx->P) fail(cx, "model declares %d parameter(s) but %d were given", np, cx->P);
      Frame* fr = new_frame(cx, np, cx->globals);
      for (int k = 0; k < np; k++) {
        Val s = nth(ps, k + 1);
        if (s.t != V_SYM) fail(cx, "parameter name must be a symbol");
        Num* z = new_num(cx, N_PARAM, 1, 1, 0);
        z->ia = k; z->dep = 1; z->v[0] = cx->theta[k];
        if (cx->mode == MODE_DUAL) { dual_alloc(cx, z); z->d[k] = 1.0; }
        fr->syms[k] = s.u.sym; fr->vals[k] = mknum(z);
      }
      Val body = f.u.p->cdr.u.p->cdr, last;
      eval_body(cx, body, fr, &last);
      Val r = eval(cx, last, fr);
      if (r.t == V_INT) r = mknum(const_num(cx, (double)r.u.i));
      if (r.t != V_NUM || !is_scalar(r.u.n)) fail(cx, "the model must produce a scalar number");
      loss = r.u.n;
      continue;
    }
    eval(cx, f, cx->globals);
  }
  if (!loss) fail(cx, "no model form");
  return loss;
}

/* Stack machine (section 7): the second front end, interpreted directly per lane. */
typedef struct { Val* v; int n, cap; } Stack;
static void spush(Ctx* cx, Stack* s, Val v) {
  if (s->n == s->cap) {
    int nc = s->cap ? 2 * s->cap : 64;
    Val* nv = (Val*)arena_alloc(cx->ar, sizeof(Val) * nc);
    if (s->n) memcpy(nv, s->v, sizeof(Val) * s->n);
    s->v = nv; s->cap = nc;
  }
  s->v[s->n++] = v;
}
static Val spop(Ctx* cx, Stack* s) { if (!s->n) fail(cx, "stack underflow"); return s->v[--s->n]; }
static Num* spopn(Ctx* cx, Stack* s) {
  Val v = spop(cx, s);
  if (v.t != V_NUM) fail(cx, "number expected on the stack");
  return v.u.n;
}

static Num* run_bytecode(Ctx* cx) {
  const Program* pg = cx->prog;
  Stack st = {0};
  Val regs[16]; int set[16] = {0};
  long long cursor = 0;
  int* loop_pc = (int*)arena_alloc(cx->ar, sizeof(int) * (pg->nins + 1));
  long long* loop_left = (long long*)arena_alloc(cx->ar, sizeof(long long) * (pg->nins + 1));
  int lsp = 0;
  for (int pc = 0; pc < pg->nins; pc++) {
    int op = pg->bc_op[pc];
    long long ia = pg->bc_i[pc];
    switch (op) {
      case B_PUSH: spush(cx, &st, mknum(const_num(cx, pg->bc_f[pc]))); break;
      case B_PARAM: {
        if (ia < 0 || ia >= cx->P) fail(cx, "PARAM %lld outside 0..%d", ia, cx->P - 1);
        Num* z = new_num(cx, N_PARAM, 1, 1, 0);
        z->ia = (int)ia; z->dep = 1; z->v[0] = cx->theta[ia];
        if (cx->mode == MODE_DUAL) { dual_alloc(cx, z); z->d[ia] = 1.0; }
        spush(cx, &st, mknum(z));
        break;
      }
      case B_OBS:
        if (ia < 0 || ia >= cx->nobs) fail(cx, "OBS %lld outside the observations", ia);
        spush(cx, &st, mknum(const_num(cx, cx->obs[ia])));
        break;
      case B_OBSN:
        if (cursor >= cx->nobs) fail(cx, "OBSN ran past the observations");
        spush(cx, &st, mknum(const_num(cx, cx->obs[cursor++])));
        break;
      case B_LOAD:
        if (ia < 0 || ia > 15 || !set[ia]) fail(cx, "LOAD of an unset register %lld", ia);
        spush(cx, &st, regs[ia]);
        break;
      case B_STORE:
        if (ia < 0 || ia > 15) fail(cx, "STORE register %lld outside 0..15", ia);
        regs[ia] = spop(cx, &st); set[ia] = 1;
        break;
      case B_DUP: { Val v = spop(cx, &st); spush(cx, &st, v); spush(cx, &st, v); break; }
      case B_SWAP: { Val b = spop(cx, &st), a = spop(cx, &st); spush(cx, &st, b); spush(cx, &st, a); break; }
      case B_POP: spop(cx, &st); break;
      case B_ADD: case B_SUB: case B_MUL: case B_DIV: {
        Num* b = spopn(cx, &st); Num* a = spopn(cx, &st);
        Num* two[2] = {a, b};
        int kind = op == B_ADD ? N_ADD : op == B_SUB ? N_SUB : op == B_MUL ? N_MUL : N_DIV;
        spush(cx, &st, mknum(nary(cx, kind, 2, two)));
        break;
      }
      case B_NEG: case B_EXP: case B_LOG: case B_SIN: case B_COS: case B_TANH: case B_SQRT: case B_ABS: {
        Num* a = spopn(cx, &st);
        int kind = op == B_NEG ? N_NEG : op == B_EXP ? N_EXP : op == B_LOG ? N_LOG : op == B_SIN ? N_SIN
                 : op == B_COS ? N_COS : op == B_TANH ? N_TANH : op == B_SQRT ? N_SQRT : N_ABS;
        spush(cx, &st, mknum(unary(cx, kind, a)));
        break;
      }
      case B_POW: { Num* e = spopn(cx, &st); Num* a = spopn(cx, &st); spush(cx, &st, mknum(pow_num(cx, a, e))); break; }
      case B_POWI: { Num* a = spopn(cx, &st); spush(cx, &st, mknum(powi_num(cx, a, ia))); break; }
      case B_LT: case B_GT: case B_LE: case B_GE: {
        Num* b = spopn(cx, &st); Num* a = spopn(cx, &st);
        double x = a->v[0], y = b->v[0];
        int r = op == B_LT ? x < y : op == B_GT ? x > y : op == B_LE ? x <= y : x >= y;
        spush(cx, &st, mkpbool(r));
        break;
      }
      case B_SEL: {
        Num* b = spopn(cx, &st); Num* a = spopn(cx, &st);
        Val p = spop(cx, &st);
        if (p.t != V_PBOOL) fail(cx, "SEL needs a predicate under its two values");
        Num* t = p.u.i ? a : b;
        Num* z = new_num(cx, N_SELECTED, 1, 1, 1);
        z->in[0] = t; z->dep = t->dep; z->v[0] = t->v[0];
        if (cx->mode == MODE_DUAL && t->d) { dual_alloc(cx, z); memcpy(z->d, t->d, sizeof(double) * cx->P); }
        spush(cx, &st, mknum(z));
        break;
      }
      case B_LOOP:
        if (ia < 0) fail(cx, "LOOP count must be >= 0");
        if (ia == 0) {
          /* skip to the matching END */
          int depth = 1;
          while (depth) { pc++; if (pg->bc_op[pc] == B_LOOP) depth++; else if (pg->bc_op[pc] == B_END) depth--; }
        } else { loop_pc[lsp] = pc; loop_left[lsp] = ia; lsp++; }
        break;
      case B_END:
        if (--loop_left[lsp - 1] > 0) pc = loop_pc[lsp - 1];
        else lsp--;
        break;
      case B_DOT: {
        if (ia < 1) fail(cx, "DOT length must be >= 1");
        Num** b = (Num**)arena_alloc(cx->ar, sizeof(Num*) * ia);
        Num** a = (Num**)arena_alloc(cx->ar, sizeof(Num*) * ia);
        for (long long i = ia - 1; i >= 0; i--) b[i] = spopn(cx, &st);
        for (long long i = ia - 1; i >= 0; i--) a[i] = spopn(cx, &st);
        spush(cx, &st, mknum(dot_num(cx, (int)ia, a, b)));
        break;
      }
    }
  }
  if (st.n != 1) fail(cx, "the program must leave exactly one value on the stack (found %d)", st.n);
  Val r = st.v[0];
  if (r.t != V_NUM) fail(cx, "the result must be a number");
  return r.u.n;
}

/* ------------------------------------------------------------------------- */
/* Lane loop and threading (section 6, multicore execution: one interpreter per  */
/* worker, results placed by lane index).                                     */
/* ------------------------------------------------------------------------- */
typedef struct {
  const Program* prog; int frontend, mode, P;
  const double* params; const double* obs; long long nobs;
  double* loss; double* grad;
  long long b0, b1;
  int status; char err[512];
  int f32;
} Job;

/* One lane: evaluate, then differentiate; errors unwind here. */
static int run_lane(Job* jb, Arena* ar, long long b, double* g) {
  Ctx cx;
  memset(&cx, 0, sizeof(cx));
  cx.prog = jb->prog; cx.ar = ar; cx.mode = jb->mode; cx.P = jb->P;
  cx.f32 = jb->f32;
  double theta32[64];
  cx.theta = jb->params + b * jb->P; cx.obs = jb->obs; cx.nobs = jb->nobs;
  if (jb->f32) {  /* parameters rounded to float (observations are rounded by the caller) */
    if (jb->P > 64) { snprintf(jb->err, sizeof(jb->err), "fp32 mode supports at most 64 parameters"); return OR_ERR; }
    for (int k = 0; k < jb->P; k++) theta32[k] = (double)(float)cx.theta[k];
    cx.theta = theta32;
  }
  cx.err = jb->err; cx.errcap = sizeof(jb->err);
  if (setjmp(cx.jb)) return OR_ERR;
  Num* loss = jb->frontend == 0 ? run_scheme(&cx) : run_bytecode(&cx);
  jb->loss[b] = loss->v[0];
  if (jb->grad && jb->mode != MODE_VALUE) {
    for (int k = 0; k < jb->P; k++) g[k] = 0.0;
    if (jb->mode == MODE_REVERSE) backward(&cx, loss, g);
    else if (loss->d) for (int k = 0; k < jb->P; k++) g[k] = loss->d[k];
    for (int k = 0; k < jb->P; k++) jb->grad[b * jb->P + k] = g[k];
  }
  return OR_OK;
}

static void* worker(void* arg) {
  Job* jb = (Job*)arg;
  Arena ar = {0};
  double* g = (double*)malloc(sizeof(double) * (jb->P ? jb->P : 1));
  for (long long b = jb->b0; b < jb->b1; b++) {
    if (run_lane(jb, &ar, b, g) != OR_OK) { jb->status = OR_ERR; break; }
    /* reset the arena but keep one chunk */
    while (ar.head && ar.head->next) { Chunk* n = ar.head->next; free(ar.head); ar.head = n; }
    if (ar.head) ar.head->used = 0;
  }
  free(g);
  arena_free_all(&ar);
  return NULL;
}

static void free_program(Program* pg) {
  for (int i = 0; i < pg->nsyms; i++) free(pg->names[i]);
  free(pg->names);
  arena_free_all(&pg->ast);
  free(pg->bc_op); free(pg->bc_f); free(pg->bc_i);
}

/*
 * ndvm_oracle_run: evaluate B lanes of a program.
 *   program/len : program text; frontend 0 = Scheme-style, 1 = stack bytecode
 *   params      : B x P row-major parameters (host)
 *   obs/nobs    : observations shared by every lane (host)
 *   loss        : B outputs; grad: B x P outputs or NULL
 *   mode        : 0 value only, 1 reverse mode, 2 dual numbers; + 4 = fp32 mode
 *                 (every arithmetic result rounded to binary32; obs must be
 *                 given already rounded to float)
 *   nthreads    : worker threads (lanes split into contiguous chunks)
 * Returns 0 on success; on error writes a message into err.
 */
int ndvm_oracle_run(const char* program, size_t len, int frontend, long long B, int P,
                    const double* params, long long nobs, const double* obs,
                    double* loss, double* grad, int mode, int nthreads, char* err, size_t errcap) {
  Program pg; memset(&pg, 0, sizeof(pg));
  if (err && errcap) err[0] = 0;
  const int f32 = (mode & 4) != 0;
  mode &= 3;
  if (B < 0 || P < 0 || (frontend != 0 && frontend != 1) || mode < 0 || mode > 2) {
    if (err) snprintf(err, errcap, "bad arguments");
    return OR_ERR;
  }
  if (frontend == 0) {
    Reader r = {program, len, 0, &pg, err, errcap, 0};
    Val head = nil(); Pair* tail = NULL;
    for (;;) {
      skip_ws(&r);
      if (r.i >= r.n) break;
      Val f = read_form(&r);
      if (r.bad) { free_program(&pg); return OR_ERR; }
      Val cell = mkpair_ast(&pg, f, nil());
      if (tail) tail->cdr = cell; else head = cell;
      tail = cell.u.p;
    }
    pg.forms = head;
  } else {
    if (parse_bytecode(&pg, program, len, err, errcap) != OR_OK) { free_program(&pg); return OR_ERR; }
  }
  if (nthreads < 1) nthreads = 1;
  if (nthreads > B) nthreads = B > 0 ? (int)B : 1;
  Job* jobs = (Job*)calloc(nthreads, sizeof(Job));
  pthread_t* th = (pthread_t*)calloc(nthreads, sizeof(pthread_t));
  long long per = (B + nthreads - 1) / (nthreads ? nthreads : 1);
  for (int t = 0; t < nthreads; t++) {
    Job* j = &jobs[t];
    j->prog = &pg; j->frontend = frontend; j->mode = mode; j->P = P; j->f32 = f32;
    j->params = params; j->obs = obs; j->nobs = nobs; j->loss = loss; j->grad = grad;
    j->b0 = t * per; j->b1 = (t + 1) * per < B ? (t + 1) * per : B;
    if (j->b0 > B) j->b0 = B;
  }
  if (nthreads == 1) worker(&jobs[0]);
  else {
    for (int t = 0; t < nthreads; t++) pthread_create(&th[t], NULL, worker, &jobs[t]);
    for (int t = 0; t < nthreads; t++) pthread_join(th[t], NULL);
  }
  int st = OR_OK;
  for (int t = 0; t < nthreads; t++) if (jobs[t].status != OR_OK) {
    st = OR_ERR;
    if (err) snprintf(err, errcap, "lane chunk %d: %s", t, jobs[t].err);
    break;
  }
  free(jobs); free(th);
  free_program(&pg);
  return st;
}
