// Test infrastructure: FNV-1a 64 over the replay plans of the given programs (gradient
// and value plans: instruction streams, paired streams, argument lists, slot and
// workspace sizes, shared-value plans, extra constants), so that a test can tell
// whether the planner still emits the plans a recorded measurement was taken on.
// Usage: planhash FRONTEND FILE... (0 Scheme-style, 1 stack bytecode); prints the hash.
#include <cstdint>
#include <cstdio>
#include <cstdlib>
#include <fstream>
#include <sstream>
#include <string>

#include "plan.h"
#include "tape.h"

using namespace ndvm;

static uint64_t fnv(const void* p, size_t n, uint64_t h) {
  const unsigned char* b = static_cast<const unsigned char*>(p);
  for (size_t i = 0; i < n; i++) {
    h ^= b[i];
    h *= 1099511628211ULL;
  }
  return h;
}

int main(int argc, char** argv) {
  if (argc < 3) return 2;
  const int fe = std::atoi(argv[1]);
  uint64_t h = 1469598103934665603ULL;
  for (int i = 2; i < argc; i++) {
    std::ifstream f(argv[i]);
    std::stringstream ss;
    ss << f.rdbuf();
    const std::string s = ss.str();
    Builder b;
    std::string err;
    if (fe == 0) trace_scheme(s.data(), s.size(), b, err);
    else trace_bytecode(s.data(), s.size(), b, err);
    for (int g = 0; g < 2; g++) {
      const Plan p = make_plan(b.t, g == 1);
      h = fnv(p.code.data(), p.code.size() * sizeof(DInst), h);
      h = fnv(p.code_paired.data(), p.code_paired.size() * sizeof(DInst), h);
      h = fnv(p.args.data(), p.args.size() * sizeof(int32_t), h);
      h = fnv(&p.n_slots, sizeof p.n_slots, h);
      h = fnv(&p.n_save, sizeof p.n_save, h);
      for (const Plan& q : p.derive) {
        h = fnv(q.code.data(), q.code.size() * sizeof(DInst), h);
        h = fnv(&q.n_slots, sizeof q.n_slots, h);
      }
      h = fnv(p.extra_consts.data(), p.extra_consts.size() * sizeof(double), h);
    }
  }
  std::printf("%016llx\n", static_cast<unsigned long long>(h));
  return 0;
}
