/*
 * ndvm.h -- C ABI of the NDVM tape-replay library (GB300, sm_103a).
 *
 * The library builds the realized numeric trace ("tape") of a program run by a
 * fixed evaluator and replays it on the GPU across a population of B parameter
 * lanes: a forward sweep over a lane-major value buffer, an exact reverse-mode
 * adjoint sweep back to per-lane parameter gradients, and the per-lane loss.
 *
 * Problem statement (paper section 2): a fixed evaluator E walks a program P given
 * as runtime data with numeric parameters theta, y = E(P, theta), and we want
 * dy/dtheta.  Section 3.4: the tape records one node per differentiable numeric
 * primitive of the realized trace and is replayed in reverse to accumulate
 * adjoints; section 3.5: one walk serves a batch axis of B lanes; Appendix C lists
 * the primitives and their adjoints.
 *
 * Conventions for every entry point:
 *   - No exception or C++ type crosses this boundary; every function returns an
 *     ndvm_status (or a plain value documented below).  On a non-OK status,
 *     ndvm_last_error() returns a message for the calling thread.
 *   - Pointers documented "device" are CUDA device pointers on the current device;
 *     "host" pointers are ordinary CPU memory.  The caller owns every buffer it
 *     passes; the library owns tapes and their cached device copies.
 *   - Argument errors are detected on the host and return a status before any
 *     launch.  Compute calls are asynchronous and ordered on the given CUDA stream
 *     (NULL = legacy default stream), except that the first call for a tape on a
 *     device uploads the tape synchronously (make that call before any stream
 *     capture).
 *   - Non-finite lane results are data, not errors.
 *   - dtype NDVM_F64 means every buffer holds double; NDVM_F32 means float.
 */
#ifndef NDVM_H
#define NDVM_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  NDVM_OK = 0,
  NDVM_E_INVALID_ARG = 1,  /* null pointer, bad size, too small a buffer */
  NDVM_E_PARSE = 2,        /* program text is not well formed */
  NDVM_E_UNSUPPORTED = 3,  /* well formed but outside the supported surface */
  NDVM_E_SHAPE = 4,        /* matrix shape mismatch in the program */
  NDVM_E_OOM = 5,          /* host or device allocation failed */
  NDVM_E_CUDA = 6,         /* a CUDA runtime call failed */
  NDVM_E_DEVICE_CHECK = 7  /* a device-side consistency check fired */
} ndvm_status;

typedef enum { NDVM_FE_SCHEME = 0, NDVM_FE_BYTECODE = 1 } ndvm_frontend;
typedef enum { NDVM_F64 = 0, NDVM_F32 = 1 } ndvm_dtype;

typedef struct ndvm_tape ndvm_tape; /* opaque; immutable once built */

/*
 * ndvm_trace_build -- walk the program once on the host and record its tape
 * (sections 3.3-3.4: control is the exact realized trace; only numeric
 * primitives are recorded; structural work records nothing).
 *   program, len : program text (host); not NUL-terminated necessarily
 *   fe           : NDVM_FE_SCHEME (Scheme-style evaluator) or NDVM_FE_BYTECODE
 *                  (stack-bytecode VM, section 7's second client)
 *   out          : receives a new tape; free it with ndvm_tape_free
 * The tape is a deterministic function of the text: byte-identical across runs,
 * threads and hosts (constants are parsed correctly rounded and stored as bits).
 * Errors: NDVM_E_INVALID_ARG, NDVM_E_PARSE, NDVM_E_UNSUPPORTED, NDVM_E_SHAPE, NDVM_E_OOM.
 */
ndvm_status ndvm_trace_build(const char* program, size_t len, ndvm_frontend fe, ndvm_tape** out);

/*
 * ndvm_tape_info -- sizes of a tape (any output pointer may be NULL).
 *   n_nodes : tape nodes; n_params : P (parameters per lane);
 *   n_obs   : observations the program reads (the obs buffer must hold at least this many);
 *   n_slots : per-lane value/adjoint slots of the gradient replay plan;
 *   hash    : FNV-1a 64 of the serialized tape.
 */
ndvm_status ndvm_tape_info(const ndvm_tape* tape, int64_t* n_nodes, int32_t* n_params, int64_t* n_obs,
                           int64_t* n_slots, uint64_t* hash);

/*
 * ndvm_tape_serialize -- write the tape's canonical byte form into buf (host).
 * *len receives the full size; if cap < size nothing is written and
 * NDVM_E_INVALID_ARG is returned (call with buf = NULL, cap = 0 to query).
 */
ndvm_status ndvm_tape_serialize(const ndvm_tape* tape, void* buf, size_t cap, size_t* len);

/* ndvm_tape_free -- release a tape and its device copies (NULL is ignored). */
void ndvm_tape_free(ndvm_tape* tape);

/*
 * ndvm_workspace_bytes -- device workspace needed by ndvm_value_and_grad to run all
 * B lanes in one launch (forward intermediates that the reverse sweep reads, stored
 * lane-contiguous).  A smaller workspace is accepted: lanes then run in chunks
 * sized to fit; 0 is returned when the tape needs no workspace.
 */
size_t ndvm_workspace_bytes(const ndvm_tape* tape, int64_t B, ndvm_dtype dtype);

/*
 * ndvm_forward -- per-lane loss only (no reverse sweep, no workspace).
 *   B      : lanes (0 is allowed and does nothing)
 *   params : device, B x P row-major (lane b's parameters at params[b*P .. b*P+P-1])
 *   obs    : device, n_obs values shared by every lane (may be NULL if the tape reads none)
 *   n_obs  : length of obs; must be >= the tape's n_obs
 *   loss   : device, B outputs
 *   stream : cudaStream_t or NULL
 */
ndvm_status ndvm_forward(const ndvm_tape* tape, ndvm_dtype dtype, int64_t B, const void* params,
                         const void* obs, int64_t n_obs, void* loss, void* stream);

/*
 * ndvm_value_and_grad -- per-lane loss and exact gradient along the realized trace
 * (Property 1, section 4; Appendix C adjoints).  Arguments as ndvm_forward, plus
 *   grad      : device, B x P row-major outputs
 *   workspace : device scratch of ws_bytes bytes (may be NULL when ws_bytes = 0);
 *               contents are overwritten; it must not be used concurrently by
 *               another call.
 * Returns NDVM_E_INVALID_ARG if the tape needs workspace and ws_bytes cannot hold
 * even one block of lanes.
 */
ndvm_status ndvm_value_and_grad(const ndvm_tape* tape, ndvm_dtype dtype, int64_t B, const void* params,
                                const void* obs, int64_t n_obs, void* loss, void* grad, void* workspace,
                                size_t ws_bytes, void* stream);

/*
 * ndvm_workspace_bytes_multi -- device workspace that ndvm_value_and_grad_multi needs
 * for the batch (tapes[k] with B[k] lanes): per tape, its shared per-point values and
 * all of its lanes' saved forward values, each tape's region 256-byte aligned.  0 when
 * the batch needs none (or an argument is invalid).
 */
size_t ndvm_workspace_bytes_multi(const ndvm_tape* const* tapes, int32_t n_tapes, const int64_t* B,
                                  ndvm_dtype dtype);

/*
 * ndvm_value_and_grad_multi -- ndvm_value_and_grad for a batch of tapes in as few
 * launches as possible (the optional multi-tape extension of the boundary; the paper's
 * setting of many candidate programs evaluated together, sections 5-6).  Tape k replays
 * B[k] lanes with its own params[k] (device, B[k] x P_k), obs[k] (device, n_obs[k]
 * values), loss[k] (device, B[k]) and grad[k] (device, B[k] x P_k); the results are
 * those of n_tapes separate ndvm_value_and_grad calls.  Replays of the same kernel
 * variant, block size, threads per lane and occupancy share one launch (up to 240
 * tapes each); a batch with shared per-point values adds one launch of observation
 * copies and one of derive plans in front.
 *   tapes, B, params, obs, n_obs, loss, grad : host arrays of n_tapes entries
 *   workspace : device, 256-byte aligned, at least ndvm_workspace_bytes_multi bytes
 *               (NULL if that is 0); overwritten; not to be shared with a concurrent call
 * Tapes with B[k] = 0 are skipped.  Returns NDVM_E_INVALID_ARG before any launch when an
 * entry is invalid (the message names the tape) or the workspace is too small; the
 * first call for a tape uploads it synchronously, as for ndvm_value_and_grad.
 */
ndvm_status ndvm_value_and_grad_multi(const ndvm_tape* const* tapes, int32_t n_tapes, ndvm_dtype dtype,
                                      const int64_t* B, const void* const* params, const void* const* obs,
                                      const int64_t* n_obs, void* const* loss, void* const* grad, void* workspace,
                                      size_t ws_bytes, void* stream);

/*
 * ndvm_value_and_grad_host -- the same computation through host buffers: copies
 * params and obs to the device, runs ndvm_value_and_grad, copies loss and grad
 * back, and synchronizes the stream.  Device buffers are cached per tape and
 * reused across calls.
 *   params, obs, loss, grad : host pointers (grad may be NULL for value only)
 */
ndvm_status ndvm_value_and_grad_host(const ndvm_tape* tape, ndvm_dtype dtype, int64_t B, const void* params,
                                     const void* obs, int64_t n_obs, void* loss, void* grad, void* stream);

/*
 * ndvm_value_and_grad_host_async -- ndvm_value_and_grad_host without the final
 * synchronization: the copies and the replay are queued on `stream` and the call
 * returns.  loss and grad hold the results once the caller has synchronized the
 * stream; params and obs must stay unchanged until then.  Host buffers should be
 * page-locked (cudaHostAlloc / pinned), else the copies are not asynchronous.
 * The tape's cached device buffers are shared by its calls, so two calls on the
 * same tape must be ordered (same stream, or a synchronization between them);
 * calls on different tapes may overlap on different streams.  The paper has no
 * counterpart; it lets a host-driven population of programs overlap its copies
 * and replays.
 */
ndvm_status ndvm_value_and_grad_host_async(const ndvm_tape* tape, ndvm_dtype dtype, int64_t B, const void* params,
                                           const void* obs, int64_t n_obs, void* loss, void* grad, void* stream);

/*
 * ndvm_value_and_grad_noalloc -- ndvm_value_and_grad for callers that may not
 * allocate device memory while they run (their device memory is planned up front
 * and must not grow).  The paper has no counterpart; this is a deployment variant.
 * Arguments as ndvm_value_and_grad, without a workspace: the forward values that
 * the reverse sweep reads go to a fixed scratch array of 32 MiB inside the
 * library, held by every GPU that loads the library until the process exits.
 * The call allocates nothing: it makes no cudaMalloc, cudaFree or other allocating
 * call.  Therefore:
 *   - the tape must already be resident on the current device: one earlier
 *     ndvm_forward or ndvm_value_and_grad call for this tape uploads it (that
 *     call allocates); otherwise NDVM_E_INVALID_ARG;
 *   - the first call on a device looks up the scratch array's device address
 *     (once per device); make that first call before any stream capture;
 *   - lanes run in chunks that fit the scratch; a tape whose workspace for one
 *     block of lanes exceeds 32 MiB is rejected with NDVM_E_INVALID_ARG;
 *   - every call shares the one array, so calls whose work overlaps on the GPU
 *     race; nothing in the array needs clearing (each saved value is written
 *     before it is read).
 */
ndvm_status ndvm_value_and_grad_noalloc(const ndvm_tape* tape, ndvm_dtype dtype, int64_t B, const void* params,
                                        const void* obs, int64_t n_obs, void* loss, void* grad, void* stream);

/*
 * ndvm_check_device -- synchronize and report whether any kernel of this tape
 * on the current device recorded a consistency failure (NDVM_E_DEVICE_CHECK);
 * clears the flag.
 */
ndvm_status ndvm_check_device(const ndvm_tape* tape);

/*
 * ndvm_tape_cost -- algorithmic cost of one lane's value-and-gradient replay (any
 * output may be NULL): FP64 work of the forward and reverse sweeps in
 * DFMA-equivalents, workspace elements per lane, and flags (bit 0: the tape has
 * data-axis regions; bit 1: the reverse sweep reads the workspace).
 */
ndvm_status ndvm_tape_cost(const ndvm_tape* tape, double* work_fwd, double* work_rev, int64_t* save_elems,
                           int32_t* flags);

/*
 * ndvm_tape_shared_work -- FP64 work (DFMA-equivalents) per value-and-gradient call
 * that does not scale with the lanes: the shared per-point values of data-axis regions
 * (section 3.5: values that depend on the data point but on no parameter are the same
 * on every lane, so they are computed once per call).  0 when there are none.
 */
ndvm_status ndvm_tape_shared_work(const ndvm_tape* tape, double* work_per_call);

/*
 * ndvm_measure_fp64_peak -- measure the device's FP64 fused multiply-add rate
 * (flop/s, two per FMA) with a dependent-chain microbenchmark on all SMs.  On GB300
 * a saturated DFMA stream issues one warp instruction per 19 cycles per SM, 84 % of
 * the FP64 pipe's unit-count peak (2 per clock per SM); the benchmark reports it
 * beside that peak.  The paper has no counterpart.  Synchronous.
 */
ndvm_status ndvm_measure_fp64_peak(double* flops_per_s, void* stream);

/* Functions that ndvm_measure_op_cost times (the replay's own exp, log, sin, cos and
 * sincos; CUDA's other functions, and CUDA's log, exp, sin and sincos for comparison;
 * DFMA as the unit). */
enum {
  NDVM_PROBE_DFMA = 0, NDVM_PROBE_EXP = 1, NDVM_PROBE_LOG = 2, NDVM_PROBE_SIN = 3, NDVM_PROBE_COS = 4,
  NDVM_PROBE_SINCOS = 5, NDVM_PROBE_TANH = 6, NDVM_PROBE_SQRT = 7, NDVM_PROBE_DIV = 8, NDVM_PROBE_RCP = 9,
  NDVM_PROBE_POW = 10, NDVM_PROBE_LOGLIB = 11, NDVM_PROBE_EXPLIB = 12, NDVM_PROBE_SINLIB = 13,
  NDVM_PROBE_SINCOSLIB = 14, NDVM_PROBE_COUNT = 15
};

/*
 * ndvm_measure_op_cost -- device time per call (ns, every SM busy with four
 * independent chains per thread, 1024 threads per SM) of the function `fn`
 * (NDVM_PROBE_*), each call followed by one FP64 add.  Dividing by the DFMA probe's
 * time gives the function's throughput cost in DFMA-equivalents; an ncu capture of
 * the probe launch gives its FP64-pipe instructions per call (calls = 4 x iters x
 * threads).  The paper has no counterpart: it measures the denominators of the
 * roofline.  Synchronous; NDVM_E_INVALID_ARG for an unknown fn or iters < 1.
 */
ndvm_status ndvm_measure_op_cost(int fn, int iters, double* ns_per_call, void* stream);

/* ndvm_launch_count -- replay kernels launched by this process so far. */
unsigned long long ndvm_launch_count(void);

/* ndvm_last_error -- message for the last non-OK status on this thread ("" if none). */
const char* ndvm_last_error(void);

/* ndvm_version -- library version string. */
const char* ndvm_version(void);

#ifdef __cplusplus
}
#endif

#endif /* NDVM_H */
