// C ABI implementation: tape objects, device caches, launch configuration.
#include <cuda_runtime.h>

#include <algorithm>
#include <atomic>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <map>
#include <memory>
#include <mutex>
#include <new>
#include <string>
#include <vector>

#include "plan.h"
#include "replay.h"
#include "status.h"
#include "tape.h"

using namespace ndvm;

namespace {

thread_local std::string g_last_error;
std::mutex g_launch_mu;
unsigned long long g_launches = 0;

ndvm_status fail(ndvm_status s, const std::string& m) {
  g_last_error = m;
  return s;
}
ndvm_status cuda_fail(cudaError_t e, const char* where) {
  return fail(NDVM_E_CUDA, std::string(where) + ": " + cudaGetErrorString(e));
}

struct DevPlan {
  std::vector<DevPlan> derive;  // derive plans of the shared per-point values
  DInst* code = nullptr;
  DInst* code_paired = nullptr;  // the paired stream (staged and element-split variants), or null
  int32_t* args = nullptr;
  double* consts_d = nullptr;
  float* consts_f = nullptr;
};

struct DevCache {
  DevPlan grad, value;
  int* err = nullptr;
  // buffers for the host-pointer entry point
  void* h_params = nullptr; size_t h_params_bytes = 0;
  void* h_obs = nullptr; size_t h_obs_bytes = 0;
  void* h_loss = nullptr; size_t h_loss_bytes = 0;
  void* h_grad = nullptr; size_t h_grad_bytes = 0;
  void* h_ws = nullptr; size_t h_ws_bytes = 0;
};

}  // namespace

struct ndvm_tape {
  Tape tape;
  Plan grad_plan, value_plan;
  std::mutex mu;       // guards dev (device copies)
  std::mutex host_mu;  // serializes the host-buffer entry point and its cached buffers
  std::map<int, DevCache> dev;
};

namespace {

void free_plan(DevPlan& p) {
  for (DevPlan& d : p.derive) free_plan(d);
  cudaFree(p.code); cudaFree(p.code_paired); cudaFree(p.args); cudaFree(p.consts_d); cudaFree(p.consts_f);
  p = DevPlan{};
}

ndvm_status upload_plan(const Tape& t, const Plan& p, DevPlan& d) {
  std::vector<double> c = t.consts;
  c.insert(c.end(), p.extra_consts.begin(), p.extra_consts.end());
  if (c.empty()) c.push_back(0.0);
  std::vector<float> cf(c.begin(), c.end());
  std::vector<int32_t> args = p.args;
  if (args.empty()) args.push_back(0);
  cudaError_t e;
  // one spare record: staged copies move 16-byte pieces and may read up to 15 bytes past the end
  if ((e = cudaMalloc(&d.code, sizeof(DInst) * (p.code.size() + 1))) != cudaSuccess) return cuda_fail(e, "cudaMalloc");
  if ((e = cudaMalloc(&d.args, sizeof(int32_t) * args.size())) != cudaSuccess) return cuda_fail(e, "cudaMalloc");
  if ((e = cudaMalloc(&d.consts_d, sizeof(double) * c.size())) != cudaSuccess) return cuda_fail(e, "cudaMalloc");
  if ((e = cudaMalloc(&d.consts_f, sizeof(float) * cf.size())) != cudaSuccess) return cuda_fail(e, "cudaMalloc");
  if (!p.code.empty() && (e = cudaMemcpy(d.code, p.code.data(), sizeof(DInst) * p.code.size(), cudaMemcpyHostToDevice)) != cudaSuccess)
    return cuda_fail(e, "cudaMemcpy");
  if (!p.code_paired.empty()) {
    if ((e = cudaMalloc(&d.code_paired, sizeof(DInst) * (p.code_paired.size() + 1))) != cudaSuccess) return cuda_fail(e, "cudaMalloc");
    if ((e = cudaMemcpy(d.code_paired, p.code_paired.data(), sizeof(DInst) * p.code_paired.size(), cudaMemcpyHostToDevice)) != cudaSuccess)
      return cuda_fail(e, "cudaMemcpy");
  }
  d.derive.resize(p.derive.size());
  for (size_t k = 0; k < p.derive.size(); k++) {
    ndvm_status s = upload_plan(t, p.derive[k], d.derive[k]);
    if (s != NDVM_OK) return s;
  }
  if ((e = cudaMemcpy(d.args, args.data(), sizeof(int32_t) * args.size(), cudaMemcpyHostToDevice)) != cudaSuccess) return cuda_fail(e, "cudaMemcpy");
  if ((e = cudaMemcpy(d.consts_d, c.data(), sizeof(double) * c.size(), cudaMemcpyHostToDevice)) != cudaSuccess) return cuda_fail(e, "cudaMemcpy");
  if ((e = cudaMemcpy(d.consts_f, cf.data(), sizeof(float) * cf.size(), cudaMemcpyHostToDevice)) != cudaSuccess) return cuda_fail(e, "cudaMemcpy");
  return NDVM_OK;
}

// device cache for the current device (uploads on first use)
ndvm_status device_cache(ndvm_tape* t, DevCache** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
  std::lock_guard<std::mutex> lk(t->mu);
  auto it = t->dev.find(dev);
  if (it == t->dev.end()) {
    DevCache c;
    ndvm_status s = upload_plan(t->tape, t->grad_plan, c.grad);
    if (s == NDVM_OK) s = upload_plan(t->tape, t->value_plan, c.value);
    if (s == NDVM_OK) {
      if ((e = cudaMalloc(&c.err, sizeof(int))) != cudaSuccess) s = cuda_fail(e, "cudaMalloc");
      else if ((e = cudaMemset(c.err, 0, sizeof(int))) != cudaSuccess) s = cuda_fail(e, "cudaMemset");
    }
    if (s != NDVM_OK) {
      free_plan(c.grad); free_plan(c.value); cudaFree(c.err);
      return s;
    }
    it = t->dev.emplace(dev, c).first;
  }
  *out = &it->second;
  return NDVM_OK;
}

constexpr size_t kSmemLimit = 227 * 1024;
// per-SM resources that bound resident blocks (sm_103a): shared memory and its
// per-block reservation, registers, and the kernel's register caps (its launch
// bounds: 128 per thread for the element-split and staged variants, 64 otherwise)
constexpr size_t kSmemPerSm = 228 * 1024, kSmemPerBlockReserved = 1024;
constexpr int kRegsPerSm = 65536, kMaxRegsStagedOrShared = 128, kMaxRegsPlain = 64;
// SMs of the current device, which the launch heuristics size grids by (152 on GB300,
// also the answer when no device responds); cached per device
int64_t num_sms() {
  static std::atomic<int> cache[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) {
    cudaGetLastError();
    return 152;
  }
  int n = cache[dev].load(std::memory_order_relaxed);
  if (n > 0) return n;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) {
    cudaGetLastError();
    return 152;
  }
  cache[dev].store(n, std::memory_order_relaxed);
  return n;
}
// threads of a block that serves a single lane (block-cooperative matrix tapes)
constexpr int kBlockLaneThreads = 256;
// lanes per launch when a workspace is used: the kernel indexes a lane's workspace
// elements of one matrix operand with 32-bit products (element * lanes per launch)
constexpr int64_t kMaxChunk = (int64_t)1 << 22;

// Threads per lane for data-axis tapes: NDVM_THREADS_PER_LANE (1..32, a power of two)
// overrides the default, which splits a lane's points over enough threads to give
// the launch about 192 threads per SM (more threads per lane replicate the lane-level
// instructions and lengthen the reductions: 4096-lane random-expression programs on 16
// streams run 2 % faster with 8 threads per lane than with 16; 64 lanes take 32).
int threads_per_lane_override() {
  static int v = [] {
    const char* e = std::getenv("NDVM_THREADS_PER_LANE");
    int g = e ? std::atoi(e) : 0;
    return (g >= 1 && g <= 32 && (g & (g - 1)) == 0) ? g : 0;
  }();
  return v;
}

// NDVM_STAGE=0 reads the instruction stream from global memory instead of staging
// it through shared memory (a tuning knob).
bool stage_enabled() {
  static bool v = [] {
    const char* e = std::getenv("NDVM_STAGE");
    return !(e && e[0] == '0');
  }();
  return v;
}

// Launch shape of a plan: threads per block, threads per lane (1 << log2g), slot-file
// layout and shared memory per block.
struct Shape {
  int tpb = 128, log2g = 0, shared = 0, sstride = 128;
  int staged = 0, stage_off = 0;
  size_t smem = 0;
};

int ilog2(int g) {
  int l = 0;
  while ((1 << l) < g) l++;
  return l;
}

Shape launch_shape(const Plan& p, size_t elem, int64_t B) {
  Shape s;
  const int64_t sms = num_sms();
  const int ov = threads_per_lane_override();
  if (p.has_regions && p.n_save == 0) {
    // data-axis tapes: a lane's points split over a thread group, one slot column per thread
    int g = ov;
    if (!g) {
      g = 1;
      while (g < 32 && B * g < sms * 192) g *= 2;
    }
    s.log2g = ilog2(g);
    while (s.tpb > 32 && (size_t)p.n_slots * s.tpb * elem > kSmemLimit) s.tpb /= 2;
    s.sstride = s.tpb;
  } else if (p.has_matrix) {
    // matrix tapes: G threads share a lane's slot column and split matrix elements;
    // G is large enough to give every SMSP two warps and to fit four 128-thread
    // blocks per SM in shared memory
    int g = ov > 16 ? 16 : ov;
    if (!g) {
      int gf = 1, gs = 1;
      while (gf < 16 && B * gf < sms * 4 * 64) gf *= 2;
      while (gs < 16 && (size_t)p.n_slots * (128 / gs + 1) * elem > kSmemLimit / 4) gs *= 2;
      g = gf > gs ? gf : gs;
    }
    while (g < 16 && (size_t)p.n_slots * (128 / g + 1) * elem > kSmemLimit) g *= 2;
    s.log2g = ilog2(g);
    s.shared = 1;
    // threads per block: the largest of 128, 64 and 32 whose grid spreads the lanes over
    // the SMs within 5 % of the average (the busiest SM holds ceil(blocks / SMs) blocks);
    // a 4-state filter's 8192 lanes in 16-lane blocks leave 56 SMs with 64 lanes and 96
    // with 48, in 8-lane blocks 112 SMs with 56 and 40 with 48
    auto spread = [&](int tpb) {
      const int64_t lpb = tpb >> s.log2g;
      const int64_t grid = (B + lpb - 1) / lpb;
      return (double)((grid + sms - 1) / sms * lpb) * (double)sms / (double)B;
    };
    for (int t = 128; t >= 32 && t >= g; t /= 2)
      if (spread(t) <= 1.05) { s.tpb = t; break; }
    s.sstride = (s.tpb >> s.log2g) + 1;
    if ((size_t)p.n_slots * s.sstride * elem > kSmemLimit) {
      // block-cooperative: one lane per block, whose threads split every matrix
      // instruction (large state dimensions: the lane's slot file alone fills the block)
      s.tpb = kBlockLaneThreads;
      s.log2g = ilog2(kBlockLaneThreads);
      s.sstride = 1;
    }
  } else {
    while (s.tpb > 32 && (size_t)p.n_slots * s.tpb * elem > kSmemLimit) s.tpb /= 2;
    s.sstride = s.tpb;
  }
  s.smem = (size_t)p.n_slots * s.sstride * elem;
  // long loop-free streams are staged through shared memory in double-buffered chunks,
  // unless the staging buffers would cost the launch resident blocks
  const size_t stage_bytes = 2 * kStageChunk * sizeof(DInst);
  auto blocks_per_sm = [&](size_t bytes, bool staged) {
    const int by_smem = (int)(kSmemPerSm / (bytes + kSmemPerBlockReserved));
    const int regs = (s.shared || staged) ? kMaxRegsStagedOrShared : kMaxRegsPlain;
    const int by_regs = kRegsPerSm / (regs * s.tpb);
    return by_smem < by_regs ? by_smem : by_regs;
  };
  // blocks an SM would hold at most: the grid's blocks spread over the SMs
  const int64_t lanes_per_block = s.tpb >> s.log2g;
  const int64_t grid = (B + lanes_per_block - 1) / lanes_per_block;
  const int want = (int)std::min<int64_t>((grid + sms - 1) / sms, 64);
  auto resident = [&](size_t bytes, bool staged) { return std::min(blocks_per_sm(bytes, staged), want); };
  const size_t staged_smem = (s.smem + 15) / 16 * 16 + stage_bytes;
  if (stage_enabled() && !p.has_regions && p.code.size() > 2 * (size_t)kStageChunk && staged_smem <= kSmemLimit &&
      resident(staged_smem, true) >= resident(s.smem, false)) {
    s.staged = 1;
    s.stage_off = (int)((s.smem + 15) / 16 * 16);
    s.smem = s.stage_off + stage_bytes;
  }
  return s;
}

// bytes of the extended observations (a copy of the observations the program reads,
// then the regions' blocks of shared per-point values), rounded up to 256; 0 without
size_t derived_bytes(const Plan& p, size_t elem) {
  if (p.derive.empty()) return 0;
  return ((size_t)(p.n_obs_min + p.derived_elems) * elem + 255) / 256 * 256;
}

// Fill the extended observations at `ext`: copy obs[0 .. n_obs_min), then run the derive
// plans, one lane per point of each region, each lane's parameters being its point's
// observation record (params = obs + base, P = stride).
ndvm_status run_derive(const Plan& p, const DevPlan& dp, ndvm_dtype dtype, const void* obs, void* ext, int* err,
                       void* stream) {
  const size_t elem = dtype == NDVM_F32 ? sizeof(float) : sizeof(double);
  cudaError_t e = cudaMemcpyAsync(ext, obs, (size_t)p.n_obs_min * elem, cudaMemcpyDeviceToDevice, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "copy observations");
  for (size_t k = 0; k < p.derive.size(); k++) {
    const Plan& q = p.derive[k];
    const DeriveInfo& di = p.derive_info[k];
    const DevPlan& dq = dp.derive[k];
    if (di.n_points <= 0) continue;
    const Shape sh = launch_shape(q, elem, di.n_points);
    ReplayArgs a;
    a.code = dq.code;
    a.n_code = (int)q.code.size();
    a.args = dq.args;
    a.consts = dtype == NDVM_F32 ? (const void*)dq.consts_f : (const void*)dq.consts_d;
    a.obs = obs;
    a.params = static_cast<const char*>(obs) + (size_t)di.base * elem;
    a.loss = nullptr;
    a.grad = nullptr;
    a.save = static_cast<char*>(ext) + (size_t)(p.n_obs_min + di.offset) * elem;
    a.save_ld = di.n_points;
    a.P = (int)di.stride;
    a.log2g = sh.log2g;
    a.shared_lane = sh.shared;
    a.sstride = sh.sstride;
    a.staged = sh.staged;
    a.stage_off = sh.stage_off;
    a.err = err;
    a.lane0 = 0;
    a.lane_end = di.n_points;
    const int64_t lanes_per_block = sh.tpb >> sh.log2g;
    const int64_t blocks = (di.n_points + lanes_per_block - 1) / lanes_per_block;
    {
      std::lock_guard<std::mutex> lk(g_launch_mu);
      e = launch_replay(a, dtype == NDVM_F32, (int)blocks, sh.tpb, sh.smem, (cudaStream_t)stream);
      g_launches++;
    }
    if (e != cudaSuccess) return cuda_fail(e, "derive launch");
  }
  return NDVM_OK;
}

ndvm_status run(ndvm_tape* t, bool grad, ndvm_dtype dtype, int64_t B, const void* params, const void* obs,
                int64_t n_obs, void* loss, void* gradp, void* ws, size_t ws_bytes, void* stream) {
  if (!t) return fail(NDVM_E_INVALID_ARG, "null tape");
  if (dtype != NDVM_F64 && dtype != NDVM_F32) return fail(NDVM_E_INVALID_ARG, "bad dtype");
  if (B < 0) return fail(NDVM_E_INVALID_ARG, "B must be >= 0");
  if (B == 0) return NDVM_OK;
  const Plan& p = grad ? t->grad_plan : t->value_plan;
  if (B > (int64_t)1 << 40) return fail(NDVM_E_INVALID_ARG, "B too large");
  if (p.n_params > 0 && !params) return fail(NDVM_E_INVALID_ARG, "null params");
  if (!loss) return fail(NDVM_E_INVALID_ARG, "null loss");
  if (grad && p.n_params > 0 && !gradp) return fail(NDVM_E_INVALID_ARG, "null grad");
  if (n_obs < p.n_obs_min) return fail(NDVM_E_INVALID_ARG, "obs holds " + std::to_string(n_obs) + " values but the program reads " + std::to_string(p.n_obs_min));
  if (p.n_obs_min > 0 && !obs) return fail(NDVM_E_INVALID_ARG, "null obs");
  const size_t elem = dtype == NDVM_F32 ? sizeof(float) : sizeof(double);
  const Shape sh = launch_shape(p, elem, B);
  const int tpb = sh.tpb, log2g = sh.log2g;
  const size_t smem = sh.smem;
  if (smem > kSmemLimit) return fail(NDVM_E_UNSUPPORTED, "tape needs " + std::to_string(p.n_slots) + " slots per lane, more than shared memory holds");
  const int lanes_per_block = tpb >> log2g;
  // the workspace holds the shared per-point values first, then the per-lane saves
  const size_t der_bytes = grad ? derived_bytes(p, elem) : 0;
  if (der_bytes > 0 && (!ws || ws_bytes < der_bytes))
    return fail(NDVM_E_INVALID_ARG, "this tape needs a workspace of at least " + std::to_string(der_bytes) + " bytes");
  void* lane_ws = der_bytes > 0 ? static_cast<char*>(ws) + der_bytes : ws;
  if (der_bytes > 0) ws_bytes -= der_bytes;
  int64_t chunk = B;
  if (grad && p.n_save > 0) {
    const size_t per_lane = (size_t)p.n_save * elem;
    if (!ws) return fail(NDVM_E_INVALID_ARG, "this tape needs a workspace of " + std::to_string(per_lane) + " bytes per lane");
    int64_t fit = (int64_t)(ws_bytes / per_lane);
    if (fit > kMaxChunk) fit = kMaxChunk;
    if (fit < B) {
      fit -= fit % lanes_per_block;
      if (fit < lanes_per_block)
        return fail(NDVM_E_INVALID_ARG, "workspace too small: need at least " + std::to_string(per_lane * lanes_per_block) + " bytes");
      chunk = fit;
    }
  }
  DevCache* dc = nullptr;
  ndvm_status s = device_cache(t, &dc);
  if (s != NDVM_OK) return s;
  const DevPlan& dp = grad ? dc->grad : dc->value;
  if (der_bytes > 0 && (s = run_derive(p, dp, dtype, obs, ws, dc->err, stream)) != NDVM_OK) return s;
  ReplayArgs a;
  // the staged and element-split variants run the paired stream; the plain one does not
  // carry the paired instruction (it would cost its register budget)
  const bool paired = (sh.staged || sh.shared) && dp.code_paired != nullptr;
  a.code = paired ? dp.code_paired : dp.code;
  a.n_code = (int)(paired ? p.code_paired.size() : p.code.size());
  a.args = dp.args;
  a.consts = dtype == NDVM_F32 ? (const void*)dp.consts_f : (const void*)dp.consts_d;
  a.obs = der_bytes > 0 ? ws : obs;  // the extended observations when the tape has shared values
  a.params = params;
  a.loss = loss;
  a.grad = gradp;
  a.save = lane_ws;
  a.save_ld = chunk;
  a.P = p.n_params;
  a.log2g = log2g;
  a.shared_lane = sh.shared;
  a.sstride = sh.sstride;
  a.staged = sh.staged;
  a.stage_off = sh.stage_off;
  a.err = dc->err;
  for (int64_t l0 = 0; l0 < B; l0 += chunk) {
    a.lane0 = l0;
    a.lane_end = l0 + chunk < B ? l0 + chunk : B;
    const int64_t lanes = a.lane_end - l0;
    const int64_t blocks = (lanes + lanes_per_block - 1) / lanes_per_block;
    if (blocks > 0x7fffffff) return fail(NDVM_E_INVALID_ARG, "too many lanes for one launch");
    cudaError_t e;
    {
      std::lock_guard<std::mutex> lk(g_launch_mu);
      e = launch_replay(a, dtype == NDVM_F32, (int)blocks, tpb, smem, (cudaStream_t)stream);
      g_launches++;
    }
    if (e != cudaSuccess) return cuda_fail(e, "replay launch");
  }
  return NDVM_OK;
}

// resident blocks per SM of a launch shape (shared memory and registers)
int resident_blocks(const Shape& s) {
  const int by_smem = (int)(kSmemPerSm / (s.smem + kSmemPerBlockReserved));
  const int regs = (s.shared || s.staged) ? kMaxRegsStagedOrShared : kMaxRegsPlain;
  const int by_regs = kRegsPerSm / (regs * s.tpb);
  return std::max(1, std::min(by_smem, by_regs));
}

// One replay of a batched launch: its arguments, its blocks and its launch shape.
struct Member {
  ReplayArgs a;
  int64_t blocks;
  Shape sh;
};

// Launches the members in as few kernels as possible: one per run of members with the
// same kernel variant, block size, threads per lane and resident blocks per SM (so that
// the launch's shared memory, its largest member's, costs no member its occupancy), at
// most kMultiMax members and 2^31 - 1 blocks per launch.
ndvm_status launch_members(std::vector<Member>& ms, bool f32, void* stream) {
  auto key = [](const Member& m) {
    return std::vector<int>{m.sh.shared, m.sh.staged, m.sh.log2g, m.sh.tpb, resident_blocks(m.sh)};
  };
  std::stable_sort(ms.begin(), ms.end(), [&](const Member& x, const Member& y) { return key(x) < key(y); });
  std::unique_ptr<MultiArgs> table(new MultiArgs);  // about 31 KB: on the heap
  for (size_t i = 0; i < ms.size();) {
    MultiArgs& m = *table;
    m.n = 0;
    int64_t blocks = 0;
    size_t smem = 0;
    const std::vector<int> k = key(ms[i]);
    while (i < ms.size() && m.n < kMultiMax && key(ms[i]) == k && blocks + ms[i].blocks <= 0x7fffffff) {
      m.start[m.n] = (int)blocks;
      m.a[m.n] = ms[i].a;
      blocks += ms[i].blocks;
      smem = std::max(smem, ms[i].sh.smem);
      m.n++;
      i++;
    }
    if (m.n == 0) return fail(NDVM_E_INVALID_ARG, "too many lanes for one launch");
    m.start[m.n] = (int)blocks;
    cudaError_t e;
    {
      std::lock_guard<std::mutex> lk(g_launch_mu);
      e = launch_replay_multi(m, f32, (int)blocks, k[3], smem, (cudaStream_t)stream);
      g_launches++;
    }
    if (e != cudaSuccess) return cuda_fail(e, "batched replay launch");
  }
  return NDVM_OK;
}

// Workspace of a batch: per tape with lanes, a 256-byte aligned region holding its
// extended observations (shared per-point values) and then its lanes' saved values.
// Returns the bytes needed; offsets[k] receives tape k's region (relative to the base).
size_t multi_layout(ndvm_tape* const* tapes, int32_t n, const int64_t* B, size_t elem, std::vector<size_t>* offsets) {
  size_t cur = 0;
  for (int32_t k = 0; k < n; k++) {
    size_t off = 0;
    if (tapes[k] && B[k] > 0) {
      const Plan& p = tapes[k]->grad_plan;
      const size_t need = derived_bytes(p, elem) + (size_t)p.n_save * elem * (size_t)B[k];
      if (need > 0) {
        cur = (cur + 255) / 256 * 256;
        off = cur;
        cur += need;
      }
    }
    if (offsets) offsets->push_back(off);
  }
  return cur;
}

ndvm_status run_multi(ndvm_tape* const* tapes, int32_t n, ndvm_dtype dtype, const int64_t* B,
                      const void* const* params, const void* const* obs, const int64_t* n_obs, void* const* loss,
                      void* const* grad, void* ws, size_t ws_bytes, void* stream) {
  if (n < 0) return fail(NDVM_E_INVALID_ARG, "negative tape count");
  if (n == 0) return NDVM_OK;
  if (!tapes || !B || !params || !obs || !n_obs || !loss || !grad) return fail(NDVM_E_INVALID_ARG, "null argument array");
  if (dtype != NDVM_F64 && dtype != NDVM_F32) return fail(NDVM_E_INVALID_ARG, "bad dtype");
  if (ws && (reinterpret_cast<uintptr_t>(ws) & 255)) return fail(NDVM_E_INVALID_ARG, "workspace must be 256-byte aligned");
  const size_t elem = dtype == NDVM_F32 ? sizeof(float) : sizeof(double);
  for (int32_t k = 0; k < n; k++) {
    const std::string at = " (tape " + std::to_string(k) + ")";
    if (!tapes[k]) return fail(NDVM_E_INVALID_ARG, "null tape" + at);
    if (B[k] < 0) return fail(NDVM_E_INVALID_ARG, "B must be >= 0" + at);
    if (B[k] > (int64_t)1 << 40) return fail(NDVM_E_INVALID_ARG, "B too large" + at);
    if (B[k] == 0) continue;
    const Plan& p = tapes[k]->grad_plan;
    if (p.n_params > 0 && (!params[k] || !grad[k])) return fail(NDVM_E_INVALID_ARG, "null params or grad" + at);
    if (!loss[k]) return fail(NDVM_E_INVALID_ARG, "null loss" + at);
    if (n_obs[k] < p.n_obs_min) return fail(NDVM_E_INVALID_ARG, "obs holds too few values" + at);
    if (p.n_obs_min > 0 && !obs[k]) return fail(NDVM_E_INVALID_ARG, "null obs" + at);
    if (launch_shape(p, elem, B[k]).smem > kSmemLimit)
      return fail(NDVM_E_UNSUPPORTED, "tape needs more slots per lane than shared memory holds" + at);
  }
  std::vector<size_t> off;
  const size_t need = multi_layout(tapes, n, B, elem, &off);
  if (need > 0 && (!ws || ws_bytes < need))
    return fail(NDVM_E_INVALID_ARG, "this batch needs a workspace of " + std::to_string(need) + " bytes");
  std::vector<Member> main, der;
  std::unique_ptr<CopyRuns> runs(new CopyRuns);
  runs->n = 0;
  std::vector<CopyRuns> run_batches;
  for (int32_t k = 0; k < n; k++) {
    if (B[k] == 0) continue;
    ndvm_tape* t = tapes[k];
    const Plan& p = t->grad_plan;
    DevCache* dc = nullptr;
    ndvm_status st = device_cache(t, &dc);
    if (st != NDVM_OK) return st;
    const DevPlan& dp = dc->grad;
    char* base = static_cast<char*>(ws) + off[(size_t)k];
    const size_t der_bytes = derived_bytes(p, elem);
    if (der_bytes > 0) {
      // the observations the program reads, then the derive plans (one lane per point)
      if (p.n_obs_min > 0) {
        if (runs->n == kCopyRunsMax) { run_batches.push_back(*runs); runs->n = 0; }
        runs->src[runs->n] = obs[k];
        runs->dst[runs->n] = base;
        runs->words[runs->n] = (int64_t)((size_t)p.n_obs_min * elem / 4);
        runs->n++;
      }
      for (size_t q = 0; q < p.derive.size(); q++) {
        const Plan& dq = p.derive[q];
        const DeriveInfo& di = p.derive_info[q];
        const DevPlan& dd = dp.derive[q];
        if (di.n_points <= 0) continue;
        Member m;
        m.sh = launch_shape(dq, elem, di.n_points);
        ReplayArgs& a = m.a;
        a.code = dd.code;
        a.n_code = (int)dq.code.size();
        a.args = dd.args;
        a.consts = dtype == NDVM_F32 ? (const void*)dd.consts_f : (const void*)dd.consts_d;
        a.obs = obs[k];
        a.params = static_cast<const char*>(obs[k]) + (size_t)di.base * elem;
        a.loss = nullptr;
        a.grad = nullptr;
        a.save = base + (size_t)(p.n_obs_min + di.offset) * elem;
        a.save_ld = di.n_points;
        a.P = (int)di.stride;
        a.log2g = m.sh.log2g;
        a.shared_lane = m.sh.shared;
        a.sstride = m.sh.sstride;
        a.staged = m.sh.staged;
        a.stage_off = m.sh.stage_off;
        a.err = dc->err;
        a.lane0 = 0;
        a.lane_end = di.n_points;
        const int64_t lpb = m.sh.tpb >> m.sh.log2g;
        m.blocks = (di.n_points + lpb - 1) / lpb;
        der.push_back(m);
      }
    }
    Member m;
    m.sh = launch_shape(p, elem, B[k]);
    ReplayArgs& a = m.a;
    const bool paired = (m.sh.staged || m.sh.shared) && dp.code_paired != nullptr;
    a.code = paired ? dp.code_paired : dp.code;
    a.n_code = (int)(paired ? p.code_paired.size() : p.code.size());
    a.args = dp.args;
    a.consts = dtype == NDVM_F32 ? (const void*)dp.consts_f : (const void*)dp.consts_d;
    a.obs = der_bytes > 0 ? (const void*)base : obs[k];
    a.params = params[k];
    a.loss = loss[k];
    a.grad = grad[k];
    a.save = base + der_bytes;
    a.save_ld = B[k];
    a.P = p.n_params;
    a.log2g = m.sh.log2g;
    a.shared_lane = m.sh.shared;
    a.sstride = m.sh.sstride;
    a.staged = m.sh.staged;
    a.stage_off = m.sh.stage_off;
    a.err = dc->err;
    a.lane0 = 0;
    a.lane_end = B[k];
    const int64_t lpb = m.sh.tpb >> m.sh.log2g;
    m.blocks = (B[k] + lpb - 1) / lpb;
    if (m.blocks > 0x7fffffff) return fail(NDVM_E_INVALID_ARG, "too many lanes for one launch");
    main.push_back(m);
  }
  if (runs->n > 0) run_batches.push_back(*runs);
  for (const CopyRuns& c : run_batches) {
    cudaError_t e;
    {
      std::lock_guard<std::mutex> lk(g_launch_mu);
      e = launch_copy_runs(c, (cudaStream_t)stream);
      g_launches++;
    }
    if (e != cudaSuccess) return cuda_fail(e, "observation copies");
  }
  ndvm_status st = launch_members(der, dtype == NDVM_F32, stream);
  if (st != NDVM_OK) return st;
  return launch_members(main, dtype == NDVM_F32, stream);
}

ndvm_status ensure(void** buf, size_t* have, size_t need) {
  if (*have >= need && *buf) return NDVM_OK;
  cudaFree(*buf);
  *buf = nullptr;
  *have = 0;
  cudaError_t e = cudaMalloc(buf, need ? need : 16);
  if (e != cudaSuccess) return e == cudaErrorMemoryAllocation ? fail(NDVM_E_OOM, "device allocation failed") : cuda_fail(e, "cudaMalloc");
  *have = need;
  return NDVM_OK;
}

}  // namespace

extern "C" {

ndvm_status ndvm_trace_build(const char* program, size_t len, ndvm_frontend fe, ndvm_tape** out) {
  if (!program || !out) return fail(NDVM_E_INVALID_ARG, "null argument");
  if (fe != NDVM_FE_SCHEME && fe != NDVM_FE_BYTECODE) return fail(NDVM_E_INVALID_ARG, "unknown front end");
  *out = nullptr;
  try {
    Builder b;
    std::string err;
    if (fe == NDVM_FE_SCHEME) trace_scheme(program, len, b, err);
    else trace_bytecode(program, len, b, err);
    if (b.t.loss < 0) return fail(NDVM_E_PARSE, "program produced no result");
    ndvm_tape* t = new ndvm_tape();
    t->tape = std::move(b.t);
    t->grad_plan = make_plan(t->tape, true);
    t->value_plan = make_plan(t->tape, false);
    std::string why;
    if (!validate_plan(t->grad_plan, t->tape.consts.size(), why) || !validate_plan(t->value_plan, t->tape.consts.size(), why)) {
      delete t;
      return fail(NDVM_E_UNSUPPORTED, "internal plan check failed: " + why);
    }
    *out = t;
    return NDVM_OK;
  } catch (const BuildError& e) {
    return fail((ndvm_status)e.code, e.msg);
  } catch (const std::bad_alloc&) {
    return fail(NDVM_E_OOM, "host allocation failed");
  } catch (const std::exception& e) {
    return fail(NDVM_E_UNSUPPORTED, e.what());
  }
}

ndvm_status ndvm_tape_info(const ndvm_tape* t, int64_t* n_nodes, int32_t* n_params, int64_t* n_obs, int64_t* n_slots,
                           uint64_t* hash) {
  if (!t) return fail(NDVM_E_INVALID_ARG, "null tape");
  if (n_nodes) *n_nodes = (int64_t)t->tape.nodes.size();
  if (n_params) *n_params = t->tape.n_params;
  if (n_obs) *n_obs = t->tape.n_obs_min;
  if (n_slots) *n_slots = t->grad_plan.n_slots;
  if (hash) *hash = t->tape.hash();
  return NDVM_OK;
}

ndvm_status ndvm_tape_cost(const ndvm_tape* t, double* work_fwd, double* work_rev, int64_t* save_elems,
                           int32_t* flags) {
  if (!t) return fail(NDVM_E_INVALID_ARG, "null tape");
  const Plan& p = t->grad_plan;
  if (work_fwd) *work_fwd = p.work_fwd;
  if (work_rev) *work_rev = p.work_rev;
  if (save_elems) *save_elems = p.n_save;
  if (flags) *flags = (p.has_regions ? 1 : 0) | (p.spill ? 2 : 0);
  return NDVM_OK;
}

ndvm_status ndvm_tape_shared_work(const ndvm_tape* t, double* work_per_call) {
  if (!t || !work_per_call) return fail(NDVM_E_INVALID_ARG, "null argument");
  double w = 0;
  for (const DeriveInfo& di : t->grad_plan.derive_info) w += di.work * (double)di.n_points;
  *work_per_call = w;
  return NDVM_OK;
}

ndvm_status ndvm_tape_serialize(const ndvm_tape* t, void* buf, size_t cap, size_t* len) {
  if (!t || !len) return fail(NDVM_E_INVALID_ARG, "null argument");
  std::vector<uint8_t> s = t->tape.serialize();
  *len = s.size();
  if (!buf && cap == 0) return NDVM_OK;
  if (!buf || cap < s.size()) return fail(NDVM_E_INVALID_ARG, "buffer too small");
  std::memcpy(buf, s.data(), s.size());
  return NDVM_OK;
}

void ndvm_tape_free(ndvm_tape* t) {
  if (!t) return;
  int cur = 0;
  cudaGetDevice(&cur);
  for (auto& kv : t->dev) {
    cudaSetDevice(kv.first);
    DevCache& c = kv.second;
    free_plan(c.grad); free_plan(c.value);
    cudaFree(c.err);
    cudaFree(c.h_params); cudaFree(c.h_obs); cudaFree(c.h_loss); cudaFree(c.h_grad); cudaFree(c.h_ws);
  }
  if (!t->dev.empty()) cudaSetDevice(cur);
  delete t;
}

size_t ndvm_workspace_bytes(const ndvm_tape* t, int64_t B, ndvm_dtype dtype) {
  if (!t || B <= 0) return 0;
  size_t elem = dtype == NDVM_F32 ? sizeof(float) : sizeof(double);
  return derived_bytes(t->grad_plan, elem) + (size_t)t->grad_plan.n_save * elem * (size_t)B;
}

ndvm_status ndvm_forward(const ndvm_tape* tape, ndvm_dtype dtype, int64_t B, const void* params, const void* obs,
                         int64_t n_obs, void* loss, void* stream) {
  return run(const_cast<ndvm_tape*>(tape), false, dtype, B, params, obs, n_obs, loss, nullptr, nullptr, 0, stream);
}

ndvm_status ndvm_value_and_grad(const ndvm_tape* tape, ndvm_dtype dtype, int64_t B, const void* params,
                                const void* obs, int64_t n_obs, void* loss, void* grad, void* ws, size_t ws_bytes,
                                void* stream) {
  return run(const_cast<ndvm_tape*>(tape), true, dtype, B, params, obs, n_obs, loss, grad, ws, ws_bytes, stream);
}

size_t ndvm_workspace_bytes_multi(const ndvm_tape* const* tapes, int32_t n_tapes, const int64_t* B, ndvm_dtype dtype) {
  if (!tapes || !B || n_tapes <= 0) return 0;
  for (int32_t k = 0; k < n_tapes; k++)
    if (B[k] < 0) return 0;
  return multi_layout(const_cast<ndvm_tape* const*>(tapes), n_tapes, B, dtype == NDVM_F32 ? sizeof(float) : sizeof(double),
                      nullptr);
}

ndvm_status ndvm_value_and_grad_multi(const ndvm_tape* const* tapes, int32_t n_tapes, ndvm_dtype dtype, const int64_t* B,
                                      const void* const* params, const void* const* obs, const int64_t* n_obs,
                                      void* const* loss, void* const* grad, void* workspace, size_t ws_bytes,
                                      void* stream) {
  return run_multi(const_cast<ndvm_tape* const*>(tapes), n_tapes, dtype, B, params, obs, n_obs, loss, grad, workspace,
                   ws_bytes, stream);
}

}  // extern "C"

namespace {

// host-buffer replay: copies in, replay, copies out, on one stream; `sync` waits for them
ndvm_status host_replay(const ndvm_tape* tape, ndvm_dtype dtype, int64_t B, const void* params, const void* obs,
                        int64_t n_obs, void* loss, void* grad, void* stream, bool sync) {
  ndvm_tape* t = const_cast<ndvm_tape*>(tape);
  if (!t) return fail(NDVM_E_INVALID_ARG, "null tape");
  if (B < 0 || n_obs < 0) return fail(NDVM_E_INVALID_ARG, "negative size");
  if (B == 0) return NDVM_OK;
  if (!loss || (t->tape.n_params > 0 && !params) || (n_obs > 0 && !obs)) return fail(NDVM_E_INVALID_ARG, "null argument");
  DevCache* dc = nullptr;
  ndvm_status s = device_cache(t, &dc);
  if (s != NDVM_OK) return s;
  const size_t elem = dtype == NDVM_F32 ? sizeof(float) : sizeof(double);
  const size_t pb = (size_t)B * t->tape.n_params * elem, ob = (size_t)n_obs * elem, lb = (size_t)B * elem;
  const bool want_grad = grad != nullptr;
  size_t wsb = want_grad ? ndvm_workspace_bytes(t, B, dtype) : 0;
  std::lock_guard<std::mutex> lk(t->host_mu);
  if ((s = ensure(&dc->h_params, &dc->h_params_bytes, pb)) != NDVM_OK) return s;
  if ((s = ensure(&dc->h_obs, &dc->h_obs_bytes, ob)) != NDVM_OK) return s;
  if ((s = ensure(&dc->h_loss, &dc->h_loss_bytes, lb)) != NDVM_OK) return s;
  if (want_grad && (s = ensure(&dc->h_grad, &dc->h_grad_bytes, pb)) != NDVM_OK) return s;
  if (wsb && (s = ensure(&dc->h_ws, &dc->h_ws_bytes, wsb)) != NDVM_OK) return s;
  cudaStream_t st = (cudaStream_t)stream;
  cudaError_t e;
  if (pb && (e = cudaMemcpyAsync(dc->h_params, params, pb, cudaMemcpyHostToDevice, st)) != cudaSuccess) return cuda_fail(e, "copy params");
  if (ob && (e = cudaMemcpyAsync(dc->h_obs, obs, ob, cudaMemcpyHostToDevice, st)) != cudaSuccess) return cuda_fail(e, "copy obs");
  if (want_grad)
    s = run(t, true, dtype, B, dc->h_params, n_obs ? dc->h_obs : nullptr, n_obs, dc->h_loss, dc->h_grad, dc->h_ws, wsb, stream);
  else
    s = run(t, false, dtype, B, dc->h_params, n_obs ? dc->h_obs : nullptr, n_obs, dc->h_loss, nullptr, nullptr, 0, stream);
  if (s != NDVM_OK) return s;
  if ((e = cudaMemcpyAsync(loss, dc->h_loss, lb, cudaMemcpyDeviceToHost, st)) != cudaSuccess) return cuda_fail(e, "copy loss");
  if (want_grad && pb && (e = cudaMemcpyAsync(grad, dc->h_grad, pb, cudaMemcpyDeviceToHost, st)) != cudaSuccess) return cuda_fail(e, "copy grad");
  if (sync && (e = cudaStreamSynchronize(st)) != cudaSuccess) return cuda_fail(e, "synchronize");
  return NDVM_OK;
}

}  // namespace

extern "C" {

ndvm_status ndvm_value_and_grad_host(const ndvm_tape* tape, ndvm_dtype dtype, int64_t B, const void* params,
                                     const void* obs, int64_t n_obs, void* loss, void* grad, void* stream) {
  return host_replay(tape, dtype, B, params, obs, n_obs, loss, grad, stream, true);
}

ndvm_status ndvm_value_and_grad_host_async(const ndvm_tape* tape, ndvm_dtype dtype, int64_t B, const void* params,
                                           const void* obs, int64_t n_obs, void* loss, void* grad, void* stream) {
  return host_replay(tape, dtype, B, params, obs, n_obs, loss, grad, stream, false);
}

ndvm_status ndvm_check_device(const ndvm_tape* tape) {
  ndvm_tape* t = const_cast<ndvm_tape*>(tape);
  if (!t) return fail(NDVM_E_INVALID_ARG, "null tape");
  DevCache* dc = nullptr;
  ndvm_status s = device_cache(t, &dc);
  if (s != NDVM_OK) return s;
  int flag = 0;
  cudaError_t e = cudaDeviceSynchronize();
  if (e != cudaSuccess) return cuda_fail(e, "synchronize");
  if ((e = cudaMemcpy(&flag, dc->err, sizeof(int), cudaMemcpyDeviceToHost)) != cudaSuccess) return cuda_fail(e, "read flag");
  if (flag) {
    cudaMemset(dc->err, 0, sizeof(int));
    return fail(NDVM_E_DEVICE_CHECK, "a replay kernel met an invalid instruction");
  }
  return NDVM_OK;
}

ndvm_status ndvm_measure_fp64_peak(double* flops_per_s, void* stream) {
  if (!flops_per_s) return fail(NDVM_E_INVALID_ARG, "null output");
  cudaError_t e = measure_fp64_peak(flops_per_s, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "fp64 peak probe");
  return NDVM_OK;
}

ndvm_status ndvm_measure_op_cost(int fn, int iters, double* ns_per_call, void* stream) {
  if (!ns_per_call) return fail(NDVM_E_INVALID_ARG, "null output");
  if (fn < 0 || fn >= NDVM_PROBE_COUNT || iters < 1) return fail(NDVM_E_INVALID_ARG, "unknown probe or iters < 1");
  cudaError_t e = measure_op_cost(fn, iters, ns_per_call, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "function cost probe");
  return NDVM_OK;
}

unsigned long long ndvm_launch_count(void) {
  std::lock_guard<std::mutex> lk(g_launch_mu);
  return g_launches;
}

const char* ndvm_last_error(void) { return g_last_error.c_str(); }

const char* ndvm_version(void) { return "ndvm-gb300 0.1"; }

// Value and gradient without allocating: the workspace is the library's fixed
// scratch array (replay.cu) instead of caller memory, and the tape must already be
// resident on the current device.  No cudaMalloc, cudaFree or other allocating
// call is made here.
ndvm_status ndvm_value_and_grad_noalloc(const ndvm_tape* tape, ndvm_dtype dtype, int64_t B, const void* params,
                                        const void* obs, int64_t n_obs, void* loss, void* grad, void* stream) {
  ndvm_tape* t = const_cast<ndvm_tape*>(tape);
  if (!t) return fail(NDVM_E_INVALID_ARG, "null tape");
  if (dtype != NDVM_F64 && dtype != NDVM_F32) return fail(NDVM_E_INVALID_ARG, "bad dtype");
  if (B < 0) return fail(NDVM_E_INVALID_ARG, "B must be >= 0");
  if (B == 0) return NDVM_OK;
  if (B > (int64_t)1 << 40) return fail(NDVM_E_INVALID_ARG, "B too large");
  const Plan& p = t->grad_plan;
  if (p.n_params > 0 && (!params || !grad)) return fail(NDVM_E_INVALID_ARG, "null params or grad");
  if (!loss) return fail(NDVM_E_INVALID_ARG, "null loss");
  if (n_obs < p.n_obs_min) return fail(NDVM_E_INVALID_ARG, "obs holds fewer values than the program reads");
  if (p.n_obs_min > 0 && !obs) return fail(NDVM_E_INVALID_ARG, "null obs");
  const size_t elem = dtype == NDVM_F32 ? sizeof(float) : sizeof(double);
  const Shape sh = launch_shape(p, elem, B);
  const int tpb = sh.tpb, log2g = sh.log2g;
  const size_t smem = sh.smem;
  if (smem > kSmemLimit) return fail(NDVM_E_UNSUPPORTED, "tape needs more slots per lane than shared memory holds");
  const int lanes_per_block = tpb >> log2g;
  // the scratch holds the shared per-point values first, then the per-lane saves
  const size_t der_bytes = derived_bytes(p, elem);
  const size_t lane_scratch = der_bytes <= kNoAllocScratchBytes ? kNoAllocScratchBytes - der_bytes : 0;
  int64_t chunk = B;
  if (der_bytes > kNoAllocScratchBytes)
    return fail(NDVM_E_INVALID_ARG, "this tape's extended observations need " + std::to_string(der_bytes) +
                                        " bytes; the fixed scratch holds " + std::to_string(kNoAllocScratchBytes) + " bytes");
  if (p.n_save > 0) {
    const size_t per_lane = (size_t)p.n_save * elem;
    const size_t per_block = per_lane * lanes_per_block;
    if (per_block > lane_scratch)
      return fail(NDVM_E_INVALID_ARG, "this tape needs " + std::to_string(per_block) + " bytes of workspace per block of " +
                                          std::to_string(lanes_per_block) + " lanes; the fixed scratch holds " +
                                          std::to_string(kNoAllocScratchBytes) + " bytes");
    int64_t fit = (int64_t)(lane_scratch / per_lane);
    if (fit < B) chunk = fit - fit % lanes_per_block;
  }
  // one launch covers at most kMaxChunk lanes, so its grid stays far below 2^31 blocks
  if (chunk > kMaxChunk) chunk = kMaxChunk - kMaxChunk % lanes_per_block;
  if ((chunk + lanes_per_block - 1) / lanes_per_block > 0x7fffffff)
    return fail(NDVM_E_INVALID_ARG, "too many lanes for one launch");
  DevCache* dc = nullptr;
  {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    std::lock_guard<std::mutex> lk(t->mu);
    auto it = t->dev.find(dev);
    if (it == t->dev.end())
      return fail(NDVM_E_INVALID_ARG, "tape is not resident on this device; one ndvm_forward or ndvm_value_and_grad "
                                      "call uploads it (that call allocates)");
    dc = &it->second;
  }
  void* scratch = nullptr;
  cudaError_t e = noalloc_scratch(&scratch);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetSymbolAddress");
  if (der_bytes > 0) {
    ndvm_status s = run_derive(p, dc->grad, dtype, obs, scratch, dc->err, stream);
    if (s != NDVM_OK) return s;
  }
  ReplayArgs a;
  const bool paired = (sh.staged || sh.shared) && dc->grad.code_paired != nullptr;
  a.code = paired ? dc->grad.code_paired : dc->grad.code;
  a.n_code = (int)(paired ? p.code_paired.size() : p.code.size());
  a.args = dc->grad.args;
  a.consts = dtype == NDVM_F32 ? (const void*)dc->grad.consts_f : (const void*)dc->grad.consts_d;
  a.obs = der_bytes > 0 ? scratch : obs;
  a.params = params;
  a.loss = loss;
  a.grad = grad;
  a.save = static_cast<char*>(scratch) + der_bytes;
  a.save_ld = chunk;
  a.P = p.n_params;
  a.log2g = log2g;
  a.shared_lane = sh.shared;
  a.sstride = sh.sstride;
  a.staged = sh.staged;
  a.stage_off = sh.stage_off;
  a.err = dc->err;
  for (int64_t l0 = 0; l0 < B; l0 += chunk) {
    a.lane0 = l0;
    a.lane_end = l0 + chunk < B ? l0 + chunk : B;
    const int64_t blocks = (a.lane_end - l0 + lanes_per_block - 1) / lanes_per_block;
    {
      std::lock_guard<std::mutex> lk(g_launch_mu);
      e = launch_replay(a, dtype == NDVM_F32, (int)blocks, tpb, smem, (cudaStream_t)stream);
      g_launches++;
    }
    if (e != cudaSuccess) return cuda_fail(e, "replay launch");
  }
  return NDVM_OK;
}

}  // extern "C"
