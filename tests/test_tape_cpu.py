"""Host-side tests (no GPU): the C-ABI library's exports, the tape format, the
tracers' realized-trace semantics and their error paths.

Expected tapes are written here by hand from the format's definition (an encoder
independent of the library), so the byte layout and the bit-exactness of tracing
are pinned on every host.
"""
import os
import re
import struct

import numpy as np
import pytest

import workloads as W

HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include", "ndvm.h")

# opcode numbering of the tape format
OPS = ["none", "const", "param", "obs", "dobs", "add", "sub", "mul", "div", "neg", "exp", "log", "sin", "cos", "tanh",
       "sqrt", "abs", "pow", "powi", "lt", "le", "gt", "ge", "eq", "select", "matfrom", "mref", "submat", "transpose",
       "madd", "msub", "mscale", "matmul", "inv", "det", "logdet", "trace", "dsum"]
OP = {n: i for i, n in enumerate(OPS)}


def encode(n_params, n_obs_min, loss, nodes, consts=(), args=()):
    """Serialized tape: header, 24-byte nodes, constant bits, argument words (little-endian)."""
    out = b"NDVMTAP1" + struct.pack("<IiqiIII", 1, n_params, n_obs_min, loss, len(nodes), len(consts), len(args))
    for (op, rows, cols, a, b, c, imm, imm2) in nodes:
        out += struct.pack("<HBBiiiii", OP[op], rows, cols, a, b, c, imm, imm2)
    for x in consts:
        out += struct.pack("<d", x)
    for x in args:
        out += struct.pack("<i", x)
    return out


def fnv1a64(data: bytes) -> int:
    h = 1469598103934665603
    for byte in data:
        h ^= byte
        h = (h * 1099511628211) & 0xFFFFFFFFFFFFFFFF
    return h


def N(op, a=-1, b=-1, c=-1, imm=0, imm2=0, rows=1, cols=1):
    return (op, rows, cols, a, b, c, imm, imm2)


def test_library_exports_every_declared_symbol(ndvm):
    import ctypes
    text = open(HEADER).read()
    decl = r"^(?:ndvm_status|void|size_t|const char\*|unsigned long long)\s+\*?(ndvm_[a-z0-9_]+)\s*\("
    names = sorted(set(re.findall(decl, text, flags=re.M)))
    assert len(names) >= 14
    lib = ctypes.CDLL(ndvm.library_path())
    missing = [n for n in names if not hasattr(lib, n)]
    assert not missing, missing
    assert lib.ndvm_version


def test_scalar_tape_bytes(ndvm):
    t = ndvm.trace_build("(model (params a) (* a 2.0))")
    exp = encode(1, 0, 2, [N("param"), N("const"), N("mul", 0, 1)], [2.0])
    assert t.serialize() == exp
    assert t.info()["hash"] == fnv1a64(exp)


def test_bytecode_tape_bytes(ndvm):
    t = ndvm.trace_build("PARAM 0\nPUSH 3.0\nADD\nPARAM 1\nMUL\nOBSN\nSUB\n", ndvm.FE_BYTECODE)
    exp = encode(2, 1, 6, [N("param"), N("const"), N("add", 0, 1), N("param", imm=1), N("mul", 2, 3),
                           N("obs", imm=0), N("sub", 4, 5)], [3.0])
    assert t.serialize() == exp


def test_data_sum_tape_bytes(ndvm):
    t = ndvm.trace_build("(model (params a) (data-sum 3 2 (* a (dobs 1))))")
    exp = encode(1, 6, 3, [N("param"), N("dobs", imm=1), N("mul", 0, 1), N("dsum", 1, 3, 2, imm=3, imm2=0)],
                 [], [2, 0])
    assert t.serialize() == exp


def test_structural_work_records_nothing(ndvm):
    # integer arithmetic, structural tests, lists and closures emit no nodes (section 3.4)
    prog = """
    (define (twice f x) (f (f x)))
    (model (params a)
      (let* ((n (+ 1 2)) (xs (list 1 2 3)) (k (length xs)))
        (if (= n k) (twice (lambda (y) (* y a)) a) (exp a))))
    """
    t = ndvm.trace_build(prog)
    assert t.serialize() == encode(1, 0, 2, [N("param"), N("mul", 0, 0), N("mul", 1, 0)])


def test_loops_are_unrolled_into_the_trace(ndvm):
    prog = "(model (params a) (let loop ((i 0) (x 1.0)) (if (= i 5) x (loop (+ i 1) (* x a)))))"
    t = ndvm.trace_build(prog)
    nodes = [N("param"), N("const")]
    prev = 1
    for _ in range(5):
        nodes.append(N("mul", prev, 0))
        prev = len(nodes) - 1
    assert t.serialize() == encode(1, 0, prev, nodes, [1.0])
    bc = ndvm.trace_build("PUSH 1.0\nSTORE 0\nLOOP 5\nLOAD 0\nPARAM 0\nMUL\nSTORE 0\nEND\nLOAD 0\n", ndvm.FE_BYTECODE)
    assert bc.info()["n_nodes"] == 7


def test_constants_interned_and_data_movement_folded(ndvm):
    t = ndvm.trace_build("(model (params a) (+ (* a 2.0) (* a 2.0) (mref (transpose (matrix 2 2 1 2 3 4)) 0 1)))")
    # equal constants share one node (2.0 is reused by the matrix element 2); the 2x2
    # constant, its transpose and the extracted element fold to constants (element
    # (0,1) of the transpose is 3.0, the existing node 5); arithmetic is not merged
    exp = encode(1, 0, 10, [N("param"), N("const", imm=0), N("mul", 0, 1), N("mul", 0, 1),
                            N("const", imm=1), N("const", imm=2), N("const", imm=3),
                            N("const", rows=2, cols=2, imm=4), N("const", rows=2, cols=2, imm=8),
                            N("add", 2, 3), N("add", 9, 5)],
                 [2.0, 1.0, 3.0, 4.0, 1.0, 2.0, 3.0, 4.0, 1.0, 3.0, 2.0, 4.0])
    assert t.serialize() == exp


def test_numeric_branch_becomes_lane_mask(ndvm):
    t = ndvm.trace_build("(model (params a) (if (< a 0.0) (- a) a))")
    assert t.serialize() == encode(1, 0, 4, [N("param"), N("const", imm=0), N("lt", 0, 1), N("neg", 0),
                                             N("select", 2, 3, 0)], [0.0])


def test_tracing_is_deterministic_and_host_independent(ndvm):
    for cfg in (1, 3, 4):
        w = W.config(cfg, B=1)
        a = ndvm.trace_build(w.program, w.frontend).serialize()
        b = ndvm.trace_build(w.program, w.frontend).serialize()
        assert a == b
        assert ndvm.trace_build(w.program, w.frontend).info()["hash"] == fnv1a64(a)
    w = W.random_exprs(n_programs=3, B=1, n_points=16)[2]
    assert ndvm.trace_build(w.program).serialize() == ndvm.trace_build(w.program).serialize()


def test_tape_sizes_of_the_workloads(ndvm):
    info = ndvm.trace_build(W.logistic(B=1).program, ndvm.FE_BYTECODE).info()
    # 1000 Euler steps x 6 primitives + 100 observations x 4 + leaves and the final divide
    assert 6400 <= info["n_nodes"] <= 6420
    assert info["n_params"] == 2 and info["n_obs"] == 100
    k4 = ndvm.trace_build(W.kalman_cv4(B=1).program).info()
    assert k4["n_params"] == 4 and k4["n_obs"] == 400
    e = ndvm.trace_build(W.exp_decay(B=1).program).info()
    assert e["n_params"] == 3 and e["n_obs"] == 100


def test_cost_model_counts(ndvm):
    c = ndvm.trace_build("(model (params a) (* a 2.0))").cost()
    assert c["work_fwd"] == 1 and c["work_rev"] == 1 and c["save_elems"] == 0
    c = ndvm.trace_build("(model (params a b) (+ (* a b) a))").cost()
    # forward mul + add; reverse: add copies into its first targets, mul contributes two products
    assert c["work_fwd"] == 2 and c["work_rev"] == 2
    lg = ndvm.trace_build(W.logistic(B=1).program, ndvm.FE_BYTECODE)
    assert lg.cost()["spill"] and lg.workspace_bytes(10) == lg.cost()["save_elems"] * 8 * 10
    assert lg.workspace_bytes(10, ndvm.F32) == lg.cost()["save_elems"] * 4 * 10


@pytest.mark.parametrize("prog,fe,status", [
    ("(model (params a) (+ a", 0, "PARSE"),
    ("(model (params a) (+ a b))", 0, "PARSE"),
    ("(model (params a) (matmul (identity 2) (identity 3)))", 0, "SHAPE"),
    ("(model (params a) (exp (identity 2)))", 0, "SHAPE"),
    ("(model (params a) (dobs 0))", 0, "PARSE"),
    ("(model (params a) (data-sum 2 1 (data-sum 2 1 (* a (dobs 0)))))", 0, "UNSUPPORTED"),
    ("(define x 1)", 0, "PARSE"),
    ("(model (params a) a) (model (params b) b)", 0, "PARSE"),
    ("(model (params a) (let loop ((x a)) (if (< x 1.0) (loop (* x 2.0)) x)))", 0, "UNSUPPORTED"),
    ("(model (params a) (pow a 99))", 0, "UNSUPPORTED"),
    ("PARAM 0\nFROB\n", 1, "PARSE"),
    ("PARAM 0\nADD\n", 1, "PARSE"),
    ("PARAM 0\nLOOP 2\nDUP\n", 1, "PARSE"),
    ("PARAM 0\nPARAM 0\n", 1, "PARSE"),
    ("LOAD 3\n", 1, "PARSE"),
])
def test_errors_are_statuses_not_crashes(ndvm, prog, fe, status):
    with pytest.raises(ndvm.NdvmError) as ei:
        ndvm.trace_build(prog, fe)
    assert ndvm.STATUS[ei.value.status] == status, str(ei.value)
    assert len(str(ei.value)) > 10


def test_null_and_bad_arguments(ndvm):
    import ctypes
    lib = ndvm.load()
    h = ctypes.c_void_p()
    assert lib.ndvm_trace_build(None, 0, 0, ctypes.byref(h)) == 1
    assert lib.ndvm_trace_build(b"(model (params a) a)", 20, 7, ctypes.byref(h)) == 1
    assert lib.ndvm_tape_info(None, None, None, None, None, None) == 1
    assert lib.ndvm_workspace_bytes(None, 10, 0) == 0
    lib.ndvm_tape_free(None)
    t = ndvm.trace_build("(model (params a) a)")
    n = ctypes.c_size_t()
    buf = ctypes.create_string_buffer(4)
    assert lib.ndvm_tape_serialize(t.handle, buf, 4, ctypes.byref(n)) == 1
    assert n.value == len(t.serialize())


def test_structural_surface_records_only_numeric_primitives(ndvm):
    """Recursion depth, closures and list traffic leave no trace: the tape holds the
    leaves and one node per numeric primitive that ran."""
    rec = "(define (pw x n) (if (= n 0) 1.0 (* x (pw x (- n 1))))) (model (params a) (pw a 5))"
    assert ndvm.trace_build(rec).info()["n_nodes"] == 2 + 5          # 1.0, a, five products
    lst = ("(define (sum l) (if (null? l) 0.0 (+ (car l) (sum (cdr l))))) "
           "(model (params a b) (sum (list a b (* a b))))")
    assert ndvm.trace_build(lst).info()["n_nodes"] == 3 + 1 + 3       # 0.0, a, b; a*b; three sums


def test_integer_helpers_and_stack_ops_record_only_numbers(ndvm):
    """quotient, remainder, list-ref and exact->inexact are structural (one constant node
    for the number they produce); expt with an integer exponent is the integer power;
    the bytecode's SWAP moves stack entries and POWI n records one node."""
    t = ndvm.trace_build("(model (params a) (* a (exact->inexact (+ (quotient 7 2) (remainder 7 3) "
                         "(list-ref (list 4 5 6) 2)))))")
    assert t.serialize() == encode(1, 0, 2, [N("param"), N("const"), N("mul", 0, 1)], [10.0])
    t = ndvm.trace_build("(model (params a) (expt a 3))")
    assert t.serialize() == encode(1, 0, 1, [N("param"), N("powi", 0, imm=3)])
    t = ndvm.trace_build("PARAM 0\nPARAM 1\nSWAP\nSUB\nPOWI 2\n", ndvm.FE_BYTECODE)
    assert t.serialize() == encode(2, 0, 3, [N("param"), N("param", imm=1), N("sub", 1, 0), N("powi", 2, imm=2)])
