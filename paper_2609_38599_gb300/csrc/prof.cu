// Kernel launch counting and optional CUDA-event timing per kernel name.
#include <string.h>

#include <vector>

#include "jarq_internal.cuh"

namespace jarq {
namespace {

const char *const kNames[] = {"validate", "residual", "init_rows", "hr_full", "grad", "gram",
                              "scale_solve", "phase_hr", "babai", "symmetrize", "group_factor",
                              "slices", "slice_rows", "proj", "whw", "rhs", "htilde", "ptilde",
                              "target", "syrk", "mu_combine", "own_rhs",
                              "scale_fit", "probe"};
constexpr int kNumNames = sizeof(kNames) / sizeof(kNames[0]);

struct Pending {
    int id;
    cudaEvent_t a, b;
};

bool g_enabled = false;
long long g_launches = 0;
long long g_count[kNumNames] = {};
double g_ms[kNumNames] = {};
std::vector<Pending> g_pending;
std::vector<cudaEvent_t> g_pool;

cudaEvent_t take_event() {
    if (!g_pool.empty()) {
        cudaEvent_t e = g_pool.back();
        g_pool.pop_back();
        return e;
    }
    cudaEvent_t e = nullptr;
    if (cudaEventCreate(&e) != cudaSuccess) {
        (void)cudaGetLastError();
        return nullptr;
    }
    return e;
}

int name_id(const char *name) {
    for (int i = 0; i < kNumNames; ++i)
        if (!strcmp(kNames[i], name)) return i;
    return -1;
}

}  // namespace

void count_launches(int n) { g_launches += n; }

ProfScope::ProfScope(const char *name, cudaStream_t s) : id_(-1), s_(s), a_(nullptr) {
    if (!g_enabled) return;
    id_ = name_id(name);
    if (id_ < 0) return;
    a_ = take_event();
    if (a_) cudaEventRecord(a_, s_);
}

void ProfScope::done() {
    if (id_ < 0 || !a_) return;
    cudaEvent_t b = take_event();
    if (!b) return;
    cudaEventRecord(b, s_);
    g_pending.push_back(Pending{id_, a_, b});
    a_ = nullptr;
}

void prof_collect() {
    for (auto &p : g_pending) {
        float ms = 0.f;
        if (cudaEventSynchronize(p.b) == cudaSuccess &&
            cudaEventElapsedTime(&ms, p.a, p.b) == cudaSuccess) {
            g_count[p.id] += 1;
            g_ms[p.id] += ms;
        }
        (void)cudaGetLastError();
        g_pool.push_back(p.a);
        g_pool.push_back(p.b);
    }
    g_pending.clear();
}

}  // namespace jarq

extern "C" {

void jarq_profile_enable(int on) { jarq::g_enabled = on != 0; }

void jarq_profile_reset(void) {
    jarq::prof_collect();
    for (int i = 0; i < jarq::kNumNames; ++i) {
        jarq::g_count[i] = 0;
        jarq::g_ms[i] = 0.0;
    }
}

int jarq_profile_read(const char *kernel, long long *launches, double *total_ms) {
    jarq::prof_collect();
    int id = kernel ? jarq::name_id(kernel) : -1;
    if (id < 0) return -1;
    if (launches) *launches = jarq::g_count[id];
    if (total_ms) *total_ms = jarq::g_ms[id];
    return 0;
}

long long jarq_launch_count(void) { return jarq::g_launches; }

}  // extern "C"
