// Launch interface of the replay kernel (host side).
#pragma once
#include <cuda_runtime.h>

#include <cstdint>

#include "plan.h"

namespace ndvm {

struct ReplayArgs {
  const DInst* code;     // device instruction stream
  int n_code;
  const int32_t* args;   // device operand lists
  const void* consts;    // device constant pool in the compute type
  const void* obs;       // device observations
  const void* params;    // device B x P parameters
  void* loss;            // device B losses
  void* grad;            // device B x P gradients (gradient plans only)
  void* save;            // device workspace [element][lane in chunk]
  int64_t lane0;         // first lane of this launch
  int64_t lane_end;      // one past the last lane of this launch
  int64_t save_ld;       // workspace column count (lanes per chunk)
  int P;
  int log2g;             // threads per lane = 1 << log2g
  int shared_lane;       // 1: the lane's threads share one slot column and split matrix elements
  int sstride;           // slot row stride in elements (threads per block, or lanes per block + pad)
  int* err;              // device flag set on an invalid instruction
  int staged;            // 1: the instruction stream is staged through shared memory in chunks
  int stage_off;         // byte offset of the two chunk buffers in dynamic shared memory
};

cudaError_t launch_replay(const ReplayArgs& a, bool f32, int blocks, int tpb, size_t smem, cudaStream_t s);

// Replays of several tapes in one launch: member m takes blocks [start[m], start[m + 1]).
// Every member has the same kernel variant (shared_lane, staged, threads per lane) and
// block size; the launch's shared memory is the largest member's.  The table is the
// kernel's parameter (at most 32 KB), so a launch holds at most kMultiMax members.
constexpr int kMultiMax = 240;
struct MultiArgs {
  int n;
  int start[kMultiMax + 1];
  ReplayArgs a[kMultiMax];
};
static_assert(sizeof(MultiArgs) <= 32000, "kernel parameter space");
cudaError_t launch_replay_multi(const MultiArgs& m, bool f32, int blocks, int tpb, size_t smem, cudaStream_t s);

// Device-to-device copies of up to kCopyRunsMax runs of 4-byte words in one launch.
constexpr int kCopyRunsMax = 1000;
struct CopyRuns {
  int n;
  const void* src[kCopyRunsMax];
  void* dst[kCopyRunsMax];
  int64_t words[kCopyRunsMax];
};
static_assert(sizeof(CopyRuns) <= 32000, "kernel parameter space");
cudaError_t launch_copy_runs(const CopyRuns& c, cudaStream_t s);

// Instructions per staged chunk (two chunk buffers of 6 KB sit after the slot file).
constexpr int kStageChunk = 128;

// Size of the fixed scratch array of the no-allocation entry point (32 MiB).
constexpr size_t kNoAllocScratchBytes = size_t(32) << 20;

// Device address of that array on the current device (looked up once per device).
cudaError_t noalloc_scratch(void** ptr);

// Measured FP64 fused multiply-add throughput of the current device (flop/s, 2 per FMA).
cudaError_t measure_fp64_peak(double* flops_per_s, cudaStream_t s);

// Device time per call of one probed function (NDVM_PROBE_*), every SM busy.
cudaError_t measure_op_cost(int fn, int iters, double* ns_per_call, cudaStream_t s);

}  // namespace ndvm
