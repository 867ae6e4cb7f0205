// C ABI: plans, the JIT tuner, the process plan cache and the run entry points.
//
// Sec. 3 of the paper: compose the lite space for the operator, evaluate the candidates
// on the device one after another, keep the fastest, and store it in a kernel database
// keyed by (kernel type t, shape s, primitive vector rho, device id) (Sec. 5.3).  Here
// the database is an in-process map keyed by type, shape, layout, strides, dtype and
// the device's name, compute capability and SM count.
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <chrono>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <map>
#include <memory>
#include <mutex>
#include <string>
#include <vector>

#include "../../include/nnjit.h"
#include "launch.h"
#include "space.h"

using namespace nnjit;

// ------------------------------------------------------------------------ errors
namespace {

thread_local std::string t_last_error;

nnjit_status fail(nnjit_status s, const std::string& msg) {
    t_last_error = msg;
    return s;
}

nnjit_status cuda_fail(cudaError_t e, const char* what) {
    std::string m = std::string(what) + ": " + cudaGetErrorName(e) + " (" + cudaGetErrorString(e) + ")";
    t_last_error = m;
    if (e == cudaErrorMemoryAllocation) return NNJIT_ERR_OOM;
    return NNJIT_ERR_CUDA;
}

bool env_flag(const char* name) {
    const char* v = std::getenv(name);
    return v && *v && std::strcmp(v, "0") != 0;
}

// Host-side fault injection for testing the tuner's failure handling without faulting
// the GPU: NNJIT_FAULT="launch:<i>" makes candidate i's launch report an error,
// "timeout:<i>" makes it report an expired kernel watchdog.
struct FaultSpec {
    int kind = 0;  // 0 none, 1 launch, 2 timeout
    int index = -1;
};

FaultSpec read_fault() {
    FaultSpec f;
    const char* v = std::getenv("NNJIT_FAULT");
    if (!v) return f;
    int idx = -1;
    if (std::sscanf(v, "launch:%d", &idx) == 1) { f.kind = 1; f.index = idx; }
    else if (std::sscanf(v, "timeout:%d", &idx) == 1) { f.kind = 2; f.index = idx; }
    return f;
}

}  // namespace

namespace nnjit {
// Record a failure detail for nnjit_last_error() from other translation units.
void set_last_error(const char* msg) { t_last_error = msg; }

namespace {
std::mutex g_attr_mu;
std::map<std::pair<int, const void*>, int> g_dyn_smem;  // (device, function) -> bytes set
std::map<int, int> g_sm_count;                          // device -> SMs
}  // namespace

cudaError_t ensure_dynamic_smem(const void* func, int smem_bytes) {
    if (smem_bytes <= 48 * 1024) return cudaSuccess;  // within the default limit
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    std::lock_guard<std::mutex> lk(g_attr_mu);
    int& have = g_dyn_smem[{dev, func}];
    if (have >= smem_bytes) return cudaSuccess;
    e = cudaFuncSetAttribute(func, cudaFuncAttributeMaxDynamicSharedMemorySize, smem_bytes);
    if (e == cudaSuccess) have = smem_bytes;
    return e;
}

int current_sm_count() {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 1;
    std::lock_guard<std::mutex> lk(g_attr_mu);
    auto it = g_sm_count.find(dev);
    if (it != g_sm_count.end()) return it->second;
    int sms = 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms <= 0) sms = 1;
    g_sm_count[dev] = sms;
    return sms;
}
}  // namespace nnjit

// ------------------------------------------------------------------------ plan
struct nnjit_plan_s {
    Problem p;
    int family = 0;
    int device = 0;
    nnjit_candidate cand{};
    int chosen_index = 0;
    int space_size = 0;
    int64_t naive = 0;
    std::vector<std::pair<int, double>> timings;  // (space index, median microseconds)
    std::vector<int> failed;                      // space indices skipped as failing
    double tune_ms = 0.0;
    bool from_cache = false;
    bool timed = false;
    nnjit_settings settings = nnjit::free_settings();  // the fixed settings its space was built with
    float* ws = nullptr;
    size_t ws_bytes = 0;
    int* err = nullptr;
    std::mutex mu;  // guards the tensor-map cache and the host staging buffers
    const void* tm_A = nullptr;
    const void* tm_B = nullptr;
    const void* tm_C = nullptr;
    bool tm_valid = false;
    nnjit_candidate tm_cand{};  // the candidate the cached tensor maps were encoded for
    bool tm_c_ok = false;
    CUtensorMap ta, tb, tc;
    void* hA = nullptr;  // device staging for run_host
    void* hB = nullptr;
    float* hbias = nullptr;
    float* hC = nullptr;
    // Online tuning (Sec. 3): serve each call with the incumbent candidate or with the
    // next one of the queue, timed by CUDA events read back on later calls.
    struct Online {
        bool active = false;
        bool done = false;
        std::vector<nnjit_candidate> space;
        std::string key;
        bool store = true;
        int best = 0;            // incumbent (space index)
        double best_us = -1.0;   // its median, once measured
        int eval = 0;            // candidate being evaluated
        int issued = 0;          // timed launches issued for `eval`
        std::vector<std::vector<double>> samples;
        struct Pending { int idx; cudaEvent_t e0, e1; };
        std::vector<Pending> pending;
        std::vector<cudaEvent_t> free_events;
    } online;
    std::mutex online_mu;
};

namespace {

struct CacheEntry {
    nnjit_candidate cand;
    int chosen_index;
    int space_size;
    int64_t naive;
    std::vector<std::pair<int, double>> timings;
    double tune_ms;
    bool timed;
};

std::mutex g_cache_mu;
std::map<std::string, CacheEntry>& cache() {
    static std::map<std::string, CacheEntry> m;
    return m;
}

// Process-wide fixed settings (nnjit_settings_set).
std::mutex g_set_mu;
nnjit_settings g_settings = free_settings();

nnjit_settings current_settings() {
    std::lock_guard<std::mutex> lk(g_set_mu);
    return g_settings;
}

bool any_fixed(const nnjit_settings& s) {
    for (int a = 0; a < kSettingAxes; ++a)
        if (setting_of(s, a) != NNJIT_SETTING_FREE) return true;
    return false;
}

std::mutex g_lim_mu;
std::map<int, nnjit_device_limits> g_limits;
std::map<int, std::string> g_dev_name;

nnjit_status query_limits(int dev, nnjit_device_limits* out) {
    {
        std::lock_guard<std::mutex> lk(g_lim_mu);
        auto it = g_limits.find(dev);
        if (it != g_limits.end()) { *out = it->second; return NNJIT_OK; }
    }
    cudaDeviceProp prop;
    cudaError_t e = cudaGetDeviceProperties(&prop, dev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetDeviceProperties");
    nnjit_device_limits L{};
    L.sm_count = prop.multiProcessorCount;
    L.smem_per_sm = (int32_t)prop.sharedMemPerMultiprocessor;
    L.smem_per_block_optin = (int32_t)prop.sharedMemPerBlockOptin;
    L.regs_per_sm = prop.regsPerMultiprocessor;
    L.max_threads_per_sm = prop.maxThreadsPerMultiProcessor;
    L.max_blocks_per_sm = prop.maxBlocksPerMultiProcessor;
    L.tmem_cols_per_sm = prop.major == 10 ? 512 : 0;
    L.l2_bytes = prop.l2CacheSize;
    L.cc_major = prop.major;
    L.cc_minor = prop.minor;
    std::lock_guard<std::mutex> lk(g_lim_mu);
    g_limits[dev] = L;
    g_dev_name[dev] = prop.name;
    *out = L;
    return NNJIT_OK;
}

std::string cache_key(const Problem& p, int dev, const nnjit_device_limits& L, const nnjit_settings& set) {
    char buf[512];
    std::string name;
    {
        std::lock_guard<std::mutex> lk(g_lim_mu);
        name = g_dev_name[dev];
    }
    std::snprintf(buf, sizeof buf,
                  "t=matmul|s=%lld,%lld,%lld,%lld|dt=%d|bl=%d|ld=%lld,%lld,%lld|st=%lld,%lld,%lld|"
                  "bias=%d|dev=%s,cc%d%d,sm%d",
                  (long long)p.M, (long long)p.N, (long long)p.K, (long long)p.batch, p.dtype,
                  p.b_layout, (long long)p.lda, (long long)p.ldb, (long long)p.ldc,
                  (long long)p.stride_a, (long long)p.stride_b, (long long)p.stride_c, p.has_bias,
                  name.c_str(), L.cc_major, L.cc_minor, L.sm_count);
    std::string key = buf;
    if (p.epilogue != NNJIT_EPI_NONE) key += "|ep=" + std::to_string(p.epilogue);
    if (any_fixed(set)) {
        std::snprintf(buf, sizeof buf, "|set=%d,%d,%d", set.raster, set.kgroup, set.reduce);
        key += buf;
    }
    return key;
}

// Split-K partials go to a workspace unless they are reduced inside a cluster.
bool uses_workspace(const nnjit_candidate& c) { return c.split_k > 1 && c.reduce == 0; }

// A CTA-pair candidate with stream-K over its last waves (reduce 2).
bool pair_stream_k(const nnjit_candidate& c) { return c.cluster_m == 2 && c.reduce == 2; }

size_t ws_bytes_for(const Problem& p, const nnjit_candidate& c) {
    (void)p;
    if (pair_stream_k(c)) return (size_t)tc2_sk_ws_bytes(std::max(1, c.grid / 2));
    if (!uses_workspace(c)) return 0;
    return (size_t)c.split_k * (size_t)p.batch * (size_t)p.M * (size_t)p.N * sizeof(float);
}

// Launch the plan's kernels for one product (the body of nnjit_matmul_run).
nnjit_status run_impl(nnjit_plan pl, const void* A, const void* B, const float* bias, float* C,
                      cudaStream_t s, const nnjit_candidate* override_cand = nullptr,
                      float* override_ws = nullptr) {
    const Problem& p = pl->p;
    const nnjit_candidate& c = override_cand ? *override_cand : pl->cand;
    float* ws = override_ws ? override_ws : pl->ws;
    if (p.M == 0 || p.N == 0) return NNJIT_OK;
    if (!C) return fail(NNJIT_ERR_INVALID_ARG, "C is NULL");
    if (p.K == 0) {
        cudaError_t e = launch_fill_bias(p, bias, C, s);
        return e == cudaSuccess ? NNJIT_OK : cuda_fail(e, "fill (K = 0)");
    }
    if (!A || !B) return fail(NNJIT_ERR_INVALID_ARG, "A or B is NULL");
    const uintptr_t ua = reinterpret_cast<uintptr_t>(A), ub = reinterpret_cast<uintptr_t>(B);
    if ((reinterpret_cast<uintptr_t>(C) & 3) || (bias && (reinterpret_cast<uintptr_t>(bias) & 3)))
        return fail(NNJIT_ERR_INVALID_ARG, "C and bias must be 4-byte aligned");
    if (c.family == NNJIT_FAMILY_FFMA) {
        if ((ua & 3) || (ub & 3)) return fail(NNJIT_ERR_INVALID_ARG, "A and B must be 4-byte aligned");
    } else if ((ua & 15) || (ub & 15)) {
        return fail(NNJIT_ERR_UNSUPPORTED, "tensor-core and GEMV paths need 16-byte aligned A and B");
    }
    const bool two_pass = uses_workspace(c);
    if (two_pass && !ws) return fail(NNJIT_ERR_INVALID_ARG, "split-K workspace missing");
    LaunchArgs la;
    la.p = &p;
    la.c = &c;
    la.A = A;
    la.B = B;
    la.bias = two_pass ? nullptr : bias;
    la.C = C;
    la.ws = ws;
    la.err = pl->err;
    la.stream = s;
    cudaError_t e = cudaSuccess;
    const bool tc = c.family == NNJIT_FAMILY_TC;
    const bool w4 = gemv_uses_w4(c);
    if (w4 != (p.dtype == NNJIT_W4_BF16)) return fail(NNJIT_ERR_INVALID_ARG, "candidate does not match the dtype");
    if (tc || gemv_uses_tma(c) || w4) {
        CUtensorMap ta, tb, tcm;
        bool c_ok = false;
        const char* why = "";
        float* out = two_pass ? ws : C;
        {
            std::lock_guard<std::mutex> lk(pl->mu);
            if (override_cand || !pl->tm_valid || pl->tm_A != A || pl->tm_B != B || pl->tm_C != out ||
                std::memcmp(&pl->tm_cand, &c, sizeof(c)) != 0) {
                e = tc ? encode_tc_tensor_maps(p, c, A, B, &ta, &tb, &why)
                    : w4 ? encode_gemv_w4_maps(p, c, A, B, &ta, &tb, &tcm, &why)
                         : encode_gemv_tensor_maps(p, c, A, B, &ta, &tb, &why);
                if (e != cudaSuccess) return fail(NNJIT_ERR_UNSUPPORTED, why);
                if (tc) encode_tc_output_map(p, c, out, two_pass, &tcm, &c_ok);
                if (w4) c_ok = true;  // third map: the group scales
                if (!override_cand) {
                    pl->ta = ta; pl->tb = tb; pl->tc = tcm; pl->tm_c_ok = c_ok;
                    pl->tm_A = A; pl->tm_B = B; pl->tm_C = out; pl->tm_cand = c; pl->tm_valid = true;
                }
            } else {
                ta = pl->ta; tb = pl->tb; tcm = pl->tc; c_ok = pl->tm_c_ok;
            }
        }
        la.tmap_a = &ta;
        la.tmap_b = &tb;
        la.tmap_c = c_ok ? &tcm : nullptr;
        e = tc ? launch_tc(la) : launch_gemv(la);
    } else if (c.family == NNJIT_FAMILY_FFMA) {
        e = launch_ffma(la);
    } else {
        e = launch_gemv(la);
    }
    if (e != cudaSuccess) return cuda_fail(e, "kernel launch");
    if (two_pass) {
        e = launch_splitk_reduce(ws, c.split_k, p, bias, C, s);
        if (e != cudaSuccess) return cuda_fail(e, "split-K reduce launch");
    }
    return NNJIT_OK;
}

double now_ms() {
    using namespace std::chrono;
    return duration<double, std::milli>(steady_clock::now().time_since_epoch()).count();
}

struct DevBuf {
    void* p = nullptr;
    ~DevBuf() { if (p) cudaFree(p); }
};

// Tuning scratch: `sets` independent operand sets so that back-to-back repetitions do
// not find their operands in L2 (rotation), plus one workspace big enough for any
// candidate's split-K partials.
struct Scratch {
    DevBuf A, B, bias, C, ws;
    int sets = 1;
    size_t a_elems = 0, b_elems = 0, c_elems = 0;
};

nnjit_status make_scratch(const Problem& p, const std::vector<nnjit_candidate>& space,
                          const nnjit_device_limits& L, Scratch* s) {
    const int e = p.elem_bytes();
    // element extents covering every batch item with the plan's strides (B in units of
    // e bytes, so 4-bit weight blobs are covered too)
    s->a_elems = (size_t)((p.batch - 1) * p.stride_a + (p.M - 1) * p.lda + p.K);
    s->b_elems = (size_t)((p.b_bytes() + e - 1) / e);
    s->c_elems = (size_t)((p.batch - 1) * p.stride_c + (p.M - 1) * p.ldc + p.N);
    // round each set up to 256 bytes so every set keeps 16-byte alignment
    auto r256 = [](size_t b) { return (b + 255) / 256 * 256; };
    const size_t set_bytes = r256(s->a_elems * e) + r256(s->b_elems * e) + r256(s->c_elems * 4);
    const size_t want = 3ull * (size_t)std::max(L.l2_bytes, 1);
    size_t sets = (want + set_bytes - 1) / set_bytes;
    sets = std::max<size_t>(1, std::min<size_t>(sets, 16));
    while (sets > 1 && sets * set_bytes > (size_t)4 << 30) --sets;
    s->sets = (int)sets;
    size_t ws_max = 0;
    for (const auto& c : space) ws_max = std::max(ws_max, ws_bytes_for(p, c));
    cudaError_t err;
    if ((err = cudaMalloc(&s->A.p, sets * r256(s->a_elems * e))) != cudaSuccess) return cuda_fail(err, "scratch A");
    if ((err = cudaMalloc(&s->B.p, sets * r256(s->b_elems * e))) != cudaSuccess) return cuda_fail(err, "scratch B");
    if ((err = cudaMalloc(&s->C.p, sets * r256(s->c_elems * 4))) != cudaSuccess) return cuda_fail(err, "scratch C");
    if ((err = cudaMalloc(&s->bias.p, r256((size_t)p.N * 4))) != cudaSuccess) return cuda_fail(err, "scratch bias");
    if (ws_max && (err = cudaMalloc(&s->ws.p, ws_max)) != cudaSuccess) return cuda_fail(err, "scratch workspace");
    // stream-K candidates keep hand-off flags in the workspace: zero before first use
    if (ws_max && (err = cudaMemset(s->ws.p, 0, ws_max)) != cudaSuccess) return cuda_fail(err, "scratch workspace");
    if ((err = launch_fill_scratch(s->A.p, (int64_t)(sets * r256(s->a_elems * e) / e), e, 1u, 0)) != cudaSuccess ||
        (err = launch_fill_scratch(s->B.p, (int64_t)(sets * r256(s->b_elems * e) / e), e, 2u, 0)) != cudaSuccess ||
        (err = launch_fill_scratch(s->bias.p, p.N, 4, 3u, 0)) != cudaSuccess)
        return cuda_fail(err, "scratch fill");
    err = cudaDeviceSynchronize();
    if (err != cudaSuccess) return cuda_fail(err, "scratch fill sync");
    return NNJIT_OK;
}

const void* set_ptr(const DevBuf& b, size_t elems, int e, int i) {
    const size_t stride = (elems * e + 255) / 256 * 256;
    return static_cast<const char*>(b.p) + (size_t)i * stride;
}

// Time one candidate: median over 3 trials of (R back-to-back launches rotating operand
// sets, captured in a CUDA graph so host launch overhead is not measured) / R, in
// microseconds.  Returns false if the candidate failed (it is then skipped); *fatal is
// set for a sticky CUDA error.
bool time_candidate(nnjit_plan pl, const nnjit_candidate& c, const Scratch& sc, int idx,
                    const FaultSpec& fault, double* us, nnjit_status* fatal) {
    const Problem& p = pl->p;
    const int e = p.elem_bytes();
    const float* bias = p.has_bias ? static_cast<const float*>(sc.bias.p) : nullptr;
    float* ws = static_cast<float*>(sc.ws.p);
    if (fault.kind == 1 && fault.index == idx) return false;
    cudaStream_t s = nullptr;
    if (cudaStreamCreateWithFlags(&s, cudaStreamNonBlocking) != cudaSuccess) {
        *fatal = fail(NNJIT_ERR_CUDA, "stream create");
        return false;
    }
    struct StreamGuard {
        cudaStream_t s;
        ~StreamGuard() { cudaStreamDestroy(s); }
    } sg{s};
    auto launch = [&](int set) -> nnjit_status {
        return run_impl(pl, set_ptr(sc.A, sc.a_elems, e, set), set_ptr(sc.B, sc.b_elems, e, set), bias,
                        const_cast<float*>(static_cast<const float*>(set_ptr(sc.C, sc.c_elems, 4, set))),
                        s, &c, ws);
    };
    auto sticky = [&](cudaError_t err, const char* what) {
        cudaGetLastError();
        if (cudaDeviceSynchronize() != cudaSuccess) *fatal = cuda_fail(err, what);
    };
    auto watchdog_fired = [&]() {
        int word = 0;
        cudaMemcpy(&word, pl->err, sizeof(int), cudaMemcpyDeviceToHost);
        if (fault.kind == 2 && fault.index == idx) word = 0x1FF;
        if (word != 0) {
            cudaMemset(pl->err, 0, sizeof(int));
            // a stopped stream-K launch may have left hand-off flags raised
            if (ws && pair_stream_k(c)) cudaMemset(ws, 0, ws_bytes_for(p, c));
        }
        return word != 0;
    };
    nnjit_status st = launch(0);
    cudaError_t err = cudaStreamSynchronize(s);
    if (err != cudaSuccess) { sticky(err, "tuning launch"); return false; }
    if (st != NNJIT_OK) return false;
    if (watchdog_fired()) return false;
    cudaEvent_t e0, e1;
    cudaEventCreate(&e0);
    cudaEventCreate(&e1);
    struct EventGuard {
        cudaEvent_t a, b;
        ~EventGuard() { cudaEventDestroy(a); cudaEventDestroy(b); }
    } eg{e0, e1};
    // estimate one launch, then size the repetitions to ~1 ms of device time (3..50)
    cudaEventRecord(e0, s);
    launch(1 % sc.sets);
    cudaEventRecord(e1, s);
    cudaEventSynchronize(e1);
    float ms1 = 0.f;
    cudaEventElapsedTime(&ms1, e0, e1);
    const int reps = (int)std::min(50.0, std::max(3.0, 1.0 / std::max(1e-4, (double)ms1)));
    cudaGraph_t graph = nullptr;
    cudaGraphExec_t exec = nullptr;
    int set = 0;
    bool captured = cudaStreamBeginCapture(s, cudaStreamCaptureModeThreadLocal) == cudaSuccess;
    if (captured) {
        for (int r = 0; r < reps; ++r) {
            launch(set);
            set = (set + 1) % sc.sets;
        }
        captured = cudaStreamEndCapture(s, &graph) == cudaSuccess && graph &&
                   cudaGraphInstantiate(&exec, graph, 0) == cudaSuccess;
    }
    if (!captured) cudaGetLastError();
    std::vector<double> trials;
    for (int t = 0; t < 3; ++t) {
        cudaEventRecord(e0, s);
        if (captured) {
            cudaGraphLaunch(exec, s);
        } else {
            for (int r = 0; r < reps; ++r) {
                launch(set);
                set = (set + 1) % sc.sets;
            }
        }
        cudaEventRecord(e1, s);
        cudaEventSynchronize(e1);
        float ms = 0.f;
        cudaEventElapsedTime(&ms, e0, e1);
        trials.push_back(1000.0 * ms / reps);
    }
    if (exec) cudaGraphExecDestroy(exec);
    if (graph) cudaGraphDestroy(graph);
    err = cudaStreamSynchronize(s);
    if (err == cudaSuccess) err = cudaGetLastError();
    if (err != cudaSuccess) { sticky(err, "tuning repetitions"); return false; }
    if (watchdog_fired()) return false;
    std::sort(trials.begin(), trials.end());
    *us = trials[trials.size() / 2];
    return true;
}

nnjit_status alloc_plan_buffers(nnjit_plan pl) {
    cudaError_t e = cudaMalloc(&pl->err, sizeof(int));
    if (e != cudaSuccess) return cuda_fail(e, "watchdog word");
    e = cudaMemset(pl->err, 0, sizeof(int));
    if (e != cudaSuccess) return cuda_fail(e, "watchdog word");
    pl->ws_bytes = ws_bytes_for(pl->p, pl->cand);
    if (pl->ws_bytes) {
        e = cudaMalloc(&pl->ws, pl->ws_bytes);
        if (e != cudaSuccess) return cuda_fail(e, "split-K workspace");
        e = cudaMemset(pl->ws, 0, pl->ws_bytes);  // stream-K hand-off flags start at zero
        if (e != cudaSuccess) return cuda_fail(e, "split-K workspace");
    }
    return NNJIT_OK;
}

void free_plan(nnjit_plan pl) {
    if (!pl) return;
    for (auto e : pl->online.free_events) cudaEventDestroy(e);
    for (auto& pd : pl->online.pending) {
        cudaEventDestroy(pd.e0);
        cudaEventDestroy(pd.e1);
    }
    if (pl->err) cudaFree(pl->err);
    if (pl->ws) cudaFree(pl->ws);
    if (pl->hA) cudaFree(pl->hA);
    if (pl->hB) cudaFree(pl->hB);
    if (pl->hbias) cudaFree(pl->hbias);
    if (pl->hC) cudaFree(pl->hC);
    delete pl;
}

nnjit_status plan_common(const nnjit_matmul_desc* d, nnjit_plan* out, Problem* prob,
                         nnjit_device_limits* L, int* dev, std::vector<nnjit_candidate>* space,
                         int64_t* naive, const nnjit_settings& set) {
    if (!out) return fail(NNJIT_ERR_INVALID_ARG, "out is NULL");
    *out = nullptr;
    std::string err;
    nnjit_status st = resolve_problem(d, prob, &err);
    if (st != NNJIT_OK) return fail(st, err);
    cudaError_t e = cudaGetDevice(dev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    e = cudaFree(nullptr);  // make sure a context exists
    if (e != cudaSuccess) return cuda_fail(e, "context");
    st = query_limits(*dev, L);
    if (st != NNJIT_OK) return st;
    st = build_space(*prob, *L, set, space, naive, &err);
    if (st != NNJIT_OK) return fail(st, err);
    return NNJIT_OK;
}

// Online tuning parameters: timed launches per candidate and the margin by which a
// newcomer must beat the incumbent ("significantly faster", Sec. 3).
constexpr int kOnlineSamples = 3;
constexpr double kOnlineMargin = 0.02;
constexpr int kOnlineEventPairs = 8;

double median_of(std::vector<double> v) {
    std::sort(v.begin(), v.end());
    return v[v.size() / 2];
}

// Read back finished timings and advance the evaluation queue.  Caller holds online_mu.
void online_poll(nnjit_plan pl) {
    auto& o = pl->online;
    for (size_t i = 0; i < o.pending.size();) {
        auto& pd = o.pending[i];
        if (cudaEventQuery(pd.e1) != cudaSuccess) { ++i; continue; }
        float ms = 0.f;
        if (cudaEventElapsedTime(&ms, pd.e0, pd.e1) == cudaSuccess) o.samples[pd.idx].push_back(1000.0 * ms);
        o.free_events.push_back(pd.e0);
        o.free_events.push_back(pd.e1);
        o.pending.erase(o.pending.begin() + (long)i);
    }
    while (!o.done && (int)o.samples[o.eval].size() >= kOnlineSamples) {
        const double med = median_of(o.samples[o.eval]);
        pl->timings.emplace_back(o.eval, med);
        if (o.best_us < 0 || (o.eval != o.best && med < o.best_us * (1.0 - kOnlineMargin))) {
            o.best = o.eval;
            o.best_us = med;
        }
        o.issued = 0;
        if (++o.eval >= (int)o.space.size()) o.done = true;
    }
    pl->cand = o.space[o.best];
    pl->chosen_index = o.best;
    if (o.done && o.store && !o.key.empty()) {
        CacheEntry ce{pl->cand, pl->chosen_index, pl->space_size, pl->naive, pl->timings,
                      pl->tune_ms, true};
        std::lock_guard<std::mutex> lk(g_cache_mu);
        cache()[o.key] = ce;
        o.store = false;
    }
}

// One call of an online plan.
nnjit_status online_run(nnjit_plan pl, const void* A, const void* B, const float* bias, float* C,
                        cudaStream_t s) {
    std::lock_guard<std::mutex> lk(pl->online_mu);
    auto& o = pl->online;
    online_poll(pl);
    const bool explore = !o.done && o.issued < kOnlineSamples && o.free_events.size() >= 2;
    const int idx = explore ? o.eval : o.best;
    cudaEvent_t e0 = nullptr, e1 = nullptr;
    if (explore) {
        e0 = o.free_events.back(); o.free_events.pop_back();
        e1 = o.free_events.back(); o.free_events.pop_back();
        cudaEventRecord(e0, s);
    }
    nnjit_status st = run_impl(pl, A, B, bias, C, s, &o.space[idx], pl->ws);
    if (explore) {
        if (st != NNJIT_OK) {
            // a failing newcomer is skipped; the call is served by the incumbent
            o.free_events.push_back(e0);
            o.free_events.push_back(e1);
            pl->failed.push_back(idx);
            o.samples[idx].assign(kOnlineSamples, 1e300);
            online_poll(pl);
            return run_impl(pl, A, B, bias, C, s, &o.space[o.best], pl->ws);
        }
        cudaEventRecord(e1, s);
        o.pending.push_back({idx, e0, e1});
        ++o.issued;
    }
    return st;
}

}  // namespace

// ------------------------------------------------------------------------ C ABI
extern "C" {

const char* nnjit_status_string(nnjit_status s) {
    switch (s) {
        case NNJIT_OK: return "NNJIT_OK";
        case NNJIT_ERR_INVALID_ARG: return "NNJIT_ERR_INVALID_ARG";
        case NNJIT_ERR_UNSUPPORTED: return "NNJIT_ERR_UNSUPPORTED";
        case NNJIT_ERR_CUDA: return "NNJIT_ERR_CUDA";
        case NNJIT_ERR_OOM: return "NNJIT_ERR_OOM";
        case NNJIT_ERR_TIMEOUT: return "NNJIT_ERR_TIMEOUT";
        case NNJIT_ERR_BUDGET: return "NNJIT_ERR_BUDGET";
    }
    return "NNJIT_ERR_UNKNOWN";
}

const char* nnjit_last_error(void) { return t_last_error.c_str(); }

int32_t nnjit_version(void) { return 100; }

}  // extern "C"

namespace {

// Kernel choices recorded by nnjit_attention_tune, keyed by shape, mask and device.
std::mutex g_attn_mu;
std::map<std::string, int> g_attn_choice;

std::string attention_key(const nnjit_attention_desc& d, int dev) {
    char buf[160];
    std::snprintf(buf, sizeof buf, "attn|%lld,%lld,%lld,%lld|c%d|dev%d", (long long)d.batch, (long long)d.Lq,
                  (long long)d.Lk, (long long)d.d, d.causal, dev);
    return buf;
}

nnjit_status attention_validate(const nnjit_attention_desc* d, const void* Q, const void* K, const void* V,
                                const float* O) {
    if (!d) return fail(NNJIT_ERR_INVALID_ARG, "descriptor is NULL");
    const int64_t lim = (int64_t)1 << 31;
    if (d->batch < 1 || d->Lq < 0 || d->Lk < 0 || d->batch >= lim || d->Lq >= lim || d->Lk >= lim)
        return fail(NNJIT_ERR_INVALID_ARG, "need batch >= 1 and 0 <= Lq, Lk < 2^31");
    if (d->causal != 0 && d->causal != 1) return fail(NNJIT_ERR_INVALID_ARG, "causal must be 0 or 1");
    if (!std::isfinite(d->scale)) return fail(NNJIT_ERR_INVALID_ARG, "scale must be finite");
    if (d->d != 64 && d->d != 128) return fail(NNJIT_ERR_UNSUPPORTED, "head dimension must be 64 or 128");
    if (d->kernel < NNJIT_ATTN_AUTO || d->kernel > NNJIT_ATTN_TCGEN05_2T)
        return fail(NNJIT_ERR_INVALID_ARG, "unknown kernel");
    if (d->Lq == 0) return NNJIT_OK;
    if (!Q || !O || (d->Lk > 0 && (!K || !V))) return fail(NNJIT_ERR_INVALID_ARG, "NULL pointer");
    auto a16 = [](const void* p) { return !p || (reinterpret_cast<uintptr_t>(p) & 15) == 0; };
    if (!a16(Q) || !a16(K) || !a16(V) || !a16(O)) return fail(NNJIT_ERR_UNSUPPORTED, "pointers must be 16-byte aligned");
    return NNJIT_OK;
}

cudaError_t attention_launch(const nnjit_attention_desc& d, int kernel, const void* Q, const void* K,
                             const void* V, float* O, cudaStream_t s) {
    if (kernel == NNJIT_ATTN_MMA) return launch_attention(d, Q, K, V, O, s);
    return launch_attention_tc(d, Q, K, V, O, s, kernel == NNJIT_ATTN_TCGEN05_2T);
}

}  // namespace

extern "C" {

nnjit_status nnjit_attention(const nnjit_attention_desc* d, const void* Q, const void* K, const void* V,
                             float* O, void* stream) {
    nnjit_status st = attention_validate(d, Q, K, V, O);
    if (st != NNJIT_OK || d->Lq == 0) return st;
    int kernel = d->kernel;
    if (kernel == NNJIT_ATTN_AUTO) {
        // without a record: the two-tile kernel once its 256-query items fill at least half
        // of the SMs (it was the faster on both benchmark shapes), else the one-tile kernel,
        // whose 128-query items give small problems twice the CTAs
        const long long items2 = d->batch * ((d->Lq + 255) / 256);
        kernel = 2 * items2 >= current_sm_count() ? NNJIT_ATTN_TCGEN05_2T : NNJIT_ATTN_TCGEN05;
        int dev = 0;
        cudaGetDevice(&dev);
        std::lock_guard<std::mutex> lk(g_attn_mu);
        auto it = g_attn_choice.find(attention_key(*d, dev));
        if (it != g_attn_choice.end()) kernel = it->second;
    }
    cudaError_t e = attention_launch(*d, kernel, Q, K, V, O, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "attention launch");
    return NNJIT_OK;
}

nnjit_status nnjit_attention_tune(const nnjit_attention_desc* d, const void* Q, const void* K, const void* V,
                                  float* O, int32_t reps, double* times_us, int32_t* chosen) {
    nnjit_status st = attention_validate(d, Q, K, V, O);
    if (st != NNJIT_OK) return st;
    if (reps < 1 || reps > 100) return fail(NNJIT_ERR_INVALID_ARG, "reps must be 1..100");
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    const int kernels[3] = {NNJIT_ATTN_TCGEN05, NNJIT_ATTN_MMA, NNJIT_ATTN_TCGEN05_2T};
    double med[3] = {0.0, 0.0, 0.0};
    if (d->Lq > 0) {
        cudaStream_t s = nullptr;
        if ((e = cudaStreamCreateWithFlags(&s, cudaStreamNonBlocking)) != cudaSuccess) return cuda_fail(e, "stream");
        cudaEvent_t e0 = nullptr, e1 = nullptr;
        cudaEventCreate(&e0);
        cudaEventCreate(&e1);
        for (int k = 0; k < 3 && e == cudaSuccess; ++k) {
            e = attention_launch(*d, kernels[k], Q, K, V, O, s);  // warm-up
            std::vector<double> trials;
            for (int t = 0; t < 3 && e == cudaSuccess; ++t) {
                cudaEventRecord(e0, s);
                for (int r = 0; r < reps && e == cudaSuccess; ++r) e = attention_launch(*d, kernels[k], Q, K, V, O, s);
                cudaEventRecord(e1, s);
                if (e == cudaSuccess) e = cudaEventSynchronize(e1);
                float ms = 0.f;
                cudaEventElapsedTime(&ms, e0, e1);
                trials.push_back(1000.0 * ms / reps);
            }
            if (e == cudaSuccess) {
                std::sort(trials.begin(), trials.end());
                med[k] = trials[1];
            }
        }
        cudaEventDestroy(e0);
        cudaEventDestroy(e1);
        cudaStreamDestroy(s);
        if (e != cudaSuccess) return cuda_fail(e, "attention tuning");
        int word = 0;
        if ((e = attention_watchdog_take(&word)) != cudaSuccess) return cuda_fail(e, "attention watchdog read");
        if (word != 0) return fail(NNJIT_ERR_TIMEOUT, "attention wait expired while tuning");
    }
    int bk = 0;  // the lowest median (the first on a tie)
    for (int k = 1; k < 3; ++k)
        if (med[k] < med[bk]) bk = k;
    const int best = kernels[bk];
    {
        std::lock_guard<std::mutex> lk(g_attn_mu);
        g_attn_choice[attention_key(*d, dev)] = best;
    }
    if (times_us)
        for (int k = 0; k < 3; ++k) times_us[k] = med[k];
    if (chosen) *chosen = best;
    return NNJIT_OK;
}

nnjit_status nnjit_attention_check(void) {
    cudaError_t e = cudaDeviceSynchronize();
    if (e != cudaSuccess) return cuda_fail(e, "attention check");
    int word = 0;
    e = attention_watchdog_take(&word);
    if (e != cudaSuccess) return cuda_fail(e, "attention watchdog read");
    if (word != 0) {
        char msg[64];
        std::snprintf(msg, sizeof msg, "attention wait expired (code 0x%x)", word);
        return fail(NNJIT_ERR_TIMEOUT, msg);
    }
    return NNJIT_OK;
}

nnjit_status nnjit_w4_layout(int64_t N, int64_t K, int64_t ldb, int64_t* scale_offset_bytes,
                             int64_t* total_bytes) {
    if (N < 0 || K < 0 || ldb < K || ldb % 32 != 0 || N % 8 != 0)
        return fail(NNJIT_ERR_INVALID_ARG, "4-bit layout needs N >= 0 a multiple of 8, ldb >= K a multiple of 32");
    Problem p;
    p.dtype = NNJIT_W4_BF16;
    p.N = N; p.K = K; p.ldb = ldb;
    if (scale_offset_bytes) *scale_offset_bytes = p.w4_scale_offset();
    if (total_bytes) *total_bytes = p.w4_blob_bytes();
    return NNJIT_OK;
}

nnjit_status nnjit_device_limits_query(int32_t device, nnjit_device_limits* out) {
    if (!out) return fail(NNJIT_ERR_INVALID_ARG, "out is NULL");
    return query_limits(device, out);
}

nnjit_status nnjit_space_enumerate(const nnjit_matmul_desc* d, const nnjit_device_limits* lim,
                                   nnjit_candidate* out, int32_t capacity, int32_t* count,
                                   int64_t* naive_count) {
    if (!lim || !count || capacity < 0 || (capacity > 0 && !out))
        return fail(NNJIT_ERR_INVALID_ARG, "bad output arguments");
    Problem p;
    std::string err;
    nnjit_status st = resolve_problem(d, &p, &err);
    if (st != NNJIT_OK) return fail(st, err);
    std::vector<nnjit_candidate> v;
    int64_t naive = 0;
    st = build_space(p, *lim, current_settings(), &v, &naive, &err);
    if (st != NNJIT_OK) return fail(st, err);
    *count = (int32_t)v.size();
    for (int32_t i = 0; i < capacity && i < (int32_t)v.size(); ++i) out[i] = v[i];
    if (naive_count) *naive_count = naive;
    return NNJIT_OK;
}

}  // extern "C"

namespace {

// The body of nnjit_matmul_plan_ex with explicit fixed settings (the settings study
// builds its spaces with every setting searched).
nnjit_status plan_ex_impl(const nnjit_matmul_desc* d, double budget_ms, const nnjit_settings& set,
                          nnjit_plan* out) {
    const double t0 = now_ms();
    if (!(budget_ms >= 0.0)) return fail(NNJIT_ERR_INVALID_ARG, "tune_budget_ms must be >= 0");
    Problem p;
    nnjit_device_limits L;
    int dev = 0;
    std::vector<nnjit_candidate> space;
    int64_t naive = 0;
    nnjit_status st = plan_common(d, out, &p, &L, &dev, &space, &naive, set);
    if (st != NNJIT_OK) return st;
    std::unique_ptr<nnjit_plan_s> pl(new nnjit_plan_s);
    pl->p = p;
    pl->device = dev;
    pl->family = space[0].family;
    pl->space_size = (int)space.size();
    pl->naive = naive;
    pl->settings = set;
    const bool use_cache = !(p.flags & NNJIT_PLAN_NO_CACHE) && !(p.flags & NNJIT_PLAN_EXHAUSTIVE);
    const std::string key = cache_key(p, dev, L, set);
    if (use_cache) {
        std::lock_guard<std::mutex> lk(g_cache_mu);
        auto it = cache().find(key);
        // an entry (possibly loaded from a file) is honoured only if its candidate is
        // still a member of the space built now
        int member = -1;
        if (it != cache().end())
            for (size_t i = 0; i < space.size() && member < 0; ++i)
                if (std::memcmp(&space[i], &it->second.cand, sizeof(nnjit_candidate)) == 0) member = (int)i;
        if (it != cache().end() && member >= 0) {
            const CacheEntry& ce = it->second;
            pl->cand = ce.cand;
            pl->chosen_index = member;
            pl->timings = ce.timings;
            pl->tune_ms = ce.tune_ms;
            pl->timed = ce.timed;
            pl->from_cache = true;
        }
    }
    if (!pl->from_cache) {
        const bool require = (p.flags & NNJIT_PLAN_REQUIRE_TIMED) != 0;
        const bool exhaustive = (p.flags & NNJIT_PLAN_EXHAUSTIVE) != 0;
        if (p.degenerate() || (budget_ms == 0.0 && !exhaustive)) {
            if (!p.degenerate() && require)
                return fail(NNJIT_ERR_BUDGET, "budget 0 with NNJIT_PLAN_REQUIRE_TIMED");
            pl->cand = space[0];
            pl->chosen_index = 0;
        } else {
            // the plan's watchdog word is needed while timing candidates
            cudaError_t e = cudaMalloc(&pl->err, sizeof(int));
            if (e != cudaSuccess) return cuda_fail(e, "watchdog word");
            cudaMemset(pl->err, 0, sizeof(int));
            Scratch sc;
            st = make_scratch(p, space, L, &sc);
            if (st != NNJIT_OK) { cudaFree(pl->err); pl->err = nullptr; return st; }
            const FaultSpec fault = read_fault();
            const bool log = env_flag("NNJIT_LOG");
            std::vector<std::pair<int, double>> timed;
            nnjit_status fatal = NNJIT_OK;
            for (int i = 0; i < (int)space.size(); ++i) {
                if (!exhaustive && !timed.empty() && now_ms() - t0 >= budget_ms) break;
                double us = 0.0;
                if (time_candidate(pl.get(), space[i], sc, i, fault, &us, &fatal)) {
                    timed.emplace_back(i, us);
                    if (log) std::fprintf(stderr, "[nnjit] cand %d family %d bn %d split %d: %.3f us\n",
                                          i, space[i].family, space[i].bn, space[i].split_k, us);
                } else {
                    pl->failed.push_back(i);
                    if (log) std::fprintf(stderr, "[nnjit] cand %d failed (skipped)\n", i);
                }
                if (fatal != NNJIT_OK) { cudaFree(pl->err); pl->err = nullptr; return fatal; }
            }
            if (timed.empty()) {
                cudaFree(pl->err);
                pl->err = nullptr;
                return fail(NNJIT_ERR_CUDA, "every timed candidate failed");
            }
            // Re-time the three fastest interleaved (noise between the first pass and now
            // hits all of them alike); keep the fastest re-timed one, ties to lower index.
            std::vector<std::pair<int, double>> order = timed;
            std::stable_sort(order.begin(), order.end(),
                             [](const std::pair<int, double>& a, const std::pair<int, double>& b) {
                                 return a.second < b.second;
                             });
            const int top = std::min<int>(3, (int)order.size());
            std::vector<std::vector<double>> again(top);
            if (top > 1) {
                for (int round = 0; round < 3; ++round)
                    for (int j = 0; j < top; ++j) {
                        double us = 0.0;
                        if (time_candidate(pl.get(), space[order[j].first], sc, order[j].first,
                                           FaultSpec{}, &us, &fatal))
                            again[j].push_back(us);
                        if (fatal != NNJIT_OK) { cudaFree(pl->err); pl->err = nullptr; return fatal; }
                    }
            }
            int best = order[0].first;
            double best_us = 1e300;
            for (int j = 0; j < top; ++j) {
                double med = order[j].second;
                if (!again[j].empty()) {
                    std::sort(again[j].begin(), again[j].end());
                    med = again[j][again[j].size() / 2];
                }
                if (med < best_us || (med == best_us && order[j].first < best)) {
                    best_us = med;
                    best = order[j].first;
                }
                for (auto& t : timed)
                    if (t.first == order[j].first) t.second = med;
            }
            pl->cand = space[best];
            pl->chosen_index = best;
            pl->timings = timed;
            pl->timed = true;
            cudaFree(pl->err);
            pl->err = nullptr;
        }
        pl->tune_ms = now_ms() - t0;
        if (use_cache) {
            CacheEntry ce{pl->cand, pl->chosen_index, pl->space_size, pl->naive, pl->timings,
                          pl->tune_ms, pl->timed};
            std::lock_guard<std::mutex> lk(g_cache_mu);
            cache()[key] = ce;
        }
    }
    st = alloc_plan_buffers(pl.get());
    if (st != NNJIT_OK) { free_plan(pl.release()); return st; }
    *out = pl.release();
    return NNJIT_OK;
}

}  // namespace

extern "C" {

nnjit_status nnjit_matmul_plan_ex(const nnjit_matmul_desc* d, double budget_ms, nnjit_plan* out) {
    return plan_ex_impl(d, budget_ms, current_settings(), out);
}

nnjit_status nnjit_settings_set(const nnjit_settings* s) {
    const nnjit_settings v = s ? *s : free_settings();
    std::string err;
    if (!settings_valid(v, &err)) return fail(NNJIT_ERR_INVALID_ARG, err);
    std::lock_guard<std::mutex> lk(g_set_mu);
    g_settings = v;
    return NNJIT_OK;
}

nnjit_status nnjit_settings_get(nnjit_settings* out) {
    if (!out) return fail(NNJIT_ERR_INVALID_ARG, "out is NULL");
    *out = current_settings();
    return NNJIT_OK;
}

nnjit_status nnjit_settings_study(const nnjit_matmul_desc* descs, int32_t count, nnjit_settings* out,
                                  char* report, size_t report_len, size_t* report_needed) {
    if (!descs || count < 1 || !out) return fail(NNJIT_ERR_INVALID_ARG, "need descs, count >= 1 and out");
    static const char* names[kSettingAxes] = {"raster", "kgroup", "reduce"};
    const nnjit_settings free_set = free_settings();
    int vote[kSettingAxes];      // value every decisive vote agreed on; -1 none yet; -2 conflict
    for (int a = 0; a < kSettingAxes; ++a) vote[a] = -1;
    std::string js = "{\"products\":[";
    char tmp[512];
    for (int32_t i = 0; i < count; ++i) {
        nnjit_matmul_desc d = descs[i];
        d.flags |= NNJIT_PLAN_EXHAUSTIVE | NNJIT_PLAN_NO_CACHE;
        nnjit_plan raw = nullptr;
        nnjit_status st = plan_ex_impl(&d, 0.0, free_set, &raw);
        if (st != NNJIT_OK) return st;
        std::unique_ptr<nnjit_plan_s, void (*)(nnjit_plan)> pl(raw, free_plan);
        const Problem& p = pl->p;
        nnjit_device_limits L;
        st = query_limits(pl->device, &L);
        if (st != NNJIT_OK) return st;
        std::vector<nnjit_candidate> space;
        int64_t naive = 0;
        std::string err;
        st = build_space(p, L, free_set, &space, &naive, &err);
        if (st != NNJIT_OK) return fail(st, err);
        std::vector<double> us(space.size(), -1.0);
        for (const auto& t : pl->timings)
            if (t.first >= 0 && t.first < (int)space.size()) us[t.first] = t.second;
        const int best = pl->chosen_index;
        std::snprintf(tmp, sizeof tmp,
                      "%s{\"M\":%lld,\"N\":%lld,\"K\":%lld,\"batch\":%lld,\"dtype\":%d,\"b_layout\":%d,"
                      "\"space_size\":%d,\"best_index\":%d,\"best_us\":%.4f,\"best\":{\"bm\":%d,\"bn\":%d,"
                      "\"split_k\":%d,\"raster\":%d,\"kgroup\":%d,\"reduce\":%d},\"settings\":{",
                      i ? "," : "", (long long)p.M, (long long)p.N, (long long)p.K, (long long)p.batch, p.dtype,
                      p.b_layout, (int)space.size(), best, us[best], space[best].bm, space[best].bn,
                      space[best].split_k, candidate_setting(p, space[best], 0), candidate_setting(p, space[best], 1),
                      candidate_setting(p, space[best], 2));
        js += tmp;
        for (int a = 0; a < kSettingAxes; ++a) {
            int twin = -1;
            for (int j = 0; j < (int)space.size() && twin < 0; ++j)
                if (setting_twins(p, space[best], space[j], a)) twin = j;
            const int mine = candidate_setting(p, space[best], a);
            const char* verdict = "no twin";
            if (twin >= 0 && us[twin] > 0.0 && us[best] > 0.0) {
                if (us[twin] > 1.02 * us[best]) {
                    verdict = "decisive";
                    vote[a] = (vote[a] == -1 || vote[a] == mine) ? mine : -2;
                } else {
                    verdict = "tie";
                }
            }
            std::snprintf(tmp, sizeof tmp, "%s\"%s\":{\"value\":%d,\"twin_value\":%d,\"twin_us\":%.4f,\"verdict\":\"%s\"}",
                          a ? "," : "", names[a], mine, twin >= 0 ? candidate_setting(p, space[twin], a) : -1,
                          twin >= 0 ? us[twin] : -1.0, verdict);
            js += tmp;
        }
        js += "}}";
    }
    nnjit_settings res = free_set;
    int* fields[kSettingAxes] = {&res.raster, &res.kgroup, &res.reduce};
    for (int a = 0; a < kSettingAxes; ++a) *fields[a] = vote[a] >= 0 ? vote[a] : NNJIT_SETTING_FREE;
    std::snprintf(tmp, sizeof tmp, "],\"fixed\":{\"raster\":%d,\"kgroup\":%d,\"reduce\":%d}}",
                  res.raster, res.kgroup, res.reduce);
    js += tmp;
    *out = res;
    if (report_needed) *report_needed = js.size() + 1;
    if (report && report_len > 0) {
        const size_t n = std::min(report_len - 1, js.size());
        std::memcpy(report, js.data(), n);
        report[n] = '\0';
    }
    return NNJIT_OK;
}

nnjit_status nnjit_matmul_plan(int64_t M, int64_t N, int64_t K, nnjit_dtype dt, double budget_ms,
                               nnjit_plan* out) {
    nnjit_matmul_desc d{};
    d.M = M; d.N = N; d.K = K; d.batch = 1;
    d.dtype = dt;
    d.b_layout = NNJIT_B_KN;
    d.has_bias = 1;
    return nnjit_matmul_plan_ex(&d, budget_ms, out);
}

nnjit_status nnjit_matmul_plan_candidate(const nnjit_matmul_desc* d, int32_t index, nnjit_plan* out) {
    Problem p;
    nnjit_device_limits L;
    int dev = 0;
    std::vector<nnjit_candidate> space;
    int64_t naive = 0;
    const nnjit_settings set = current_settings();
    nnjit_status st = plan_common(d, out, &p, &L, &dev, &space, &naive, set);
    if (st != NNJIT_OK) return st;
    if (index < 0 || index >= (int32_t)space.size())
        return fail(NNJIT_ERR_INVALID_ARG, "candidate index out of range");
    std::unique_ptr<nnjit_plan_s> pl(new nnjit_plan_s);
    pl->p = p;
    pl->device = dev;
    pl->family = space[index].family;
    pl->cand = space[index];
    pl->chosen_index = index;
    pl->space_size = (int)space.size();
    pl->naive = naive;
    pl->settings = set;
    st = alloc_plan_buffers(pl.get());
    if (st != NNJIT_OK) { free_plan(pl.release()); return st; }
    *out = pl.release();
    return NNJIT_OK;
}

nnjit_status nnjit_matmul_run(nnjit_plan p, const void* A, const void* B, const float* bias,
                              float* C, void* stream) {
    if (!p) return fail(NNJIT_ERR_INVALID_ARG, "plan is NULL");
    if (p->online.active) return online_run(p, A, B, bias, C, static_cast<cudaStream_t>(stream));
    return run_impl(p, A, B, bias, C, static_cast<cudaStream_t>(stream));
}

nnjit_status nnjit_matmul_plan_online(const nnjit_matmul_desc* d, nnjit_plan* out) {
    const double t0 = now_ms();
    Problem p;
    nnjit_device_limits L;
    int dev = 0;
    std::vector<nnjit_candidate> space;
    int64_t naive = 0;
    const nnjit_settings set = current_settings();
    nnjit_status st = plan_common(d, out, &p, &L, &dev, &space, &naive, set);
    if (st != NNJIT_OK) return st;
    std::unique_ptr<nnjit_plan_s> pl(new nnjit_plan_s);
    pl->p = p;
    pl->device = dev;
    pl->settings = set;
    pl->family = space[0].family;
    pl->cand = space[0];
    pl->chosen_index = 0;
    pl->space_size = (int)space.size();
    pl->naive = naive;
    pl->timed = true;
    auto& o = pl->online;
    o.active = !p.degenerate();
    o.space = space;
    o.samples.assign(space.size(), {});
    o.key = (p.flags & NNJIT_PLAN_NO_CACHE) ? std::string() : cache_key(p, dev, L, set);
    // the workspace serves every candidate of the queue
    nnjit_candidate widest = space[0];
    for (const auto& c : space)
        if (ws_bytes_for(p, c) > ws_bytes_for(p, widest)) widest = c;
    pl->cand = widest;
    st = alloc_plan_buffers(pl.get());
    pl->cand = space[0];
    if (st != NNJIT_OK) { free_plan(pl.release()); return st; }
    for (int i = 0; i < 2 * kOnlineEventPairs; ++i) {
        cudaEvent_t e;
        if (cudaEventCreate(&e) != cudaSuccess) { free_plan(pl.release()); return fail(NNJIT_ERR_CUDA, "event create"); }
        o.free_events.push_back(e);
    }
    pl->tune_ms = now_ms() - t0;
    *out = pl.release();
    return NNJIT_OK;
}

nnjit_status nnjit_plan_online_progress(nnjit_plan p, int32_t* evaluated, int32_t* space_size,
                                        int32_t* current_index, int32_t* done) {
    if (!p) return fail(NNJIT_ERR_INVALID_ARG, "plan is NULL");
    std::lock_guard<std::mutex> lk(p->online_mu);
    if (p->online.active) online_poll(p);
    if (evaluated) *evaluated = p->online.active ? p->online.eval : p->space_size;
    if (space_size) *space_size = p->space_size;
    if (current_index) *current_index = p->chosen_index;
    if (done) *done = (!p->online.active || p->online.done) ? 1 : 0;
    return NNJIT_OK;
}

nnjit_status nnjit_matmul_run_batched(nnjit_plan p, const void* A, const void* B, float* C,
                                      void* stream) {
    return nnjit_matmul_run(p, A, B, nullptr, C, stream);
}

namespace {

// Byte sizes of a packed plan's host operands and its device staging buffers (allocated on
// first use and kept by the plan).  UNSUPPORTED for plans with padded strides.
nnjit_status host_staging(nnjit_plan pl, size_t* a_bytes, size_t* b_bytes, size_t* c_bytes) {
    const Problem& p = pl->p;
    const int64_t b_rows = p.b_layout == NNJIT_B_KN ? p.K : p.N;
    const int64_t b_cols = p.b_layout == NNJIT_B_KN ? p.N : p.K;
    const bool packed = p.lda == std::max<int64_t>(p.K, 1) && p.ldb == std::max<int64_t>(b_cols, 1) &&
                        p.ldc == std::max<int64_t>(p.N, 1) && p.stride_a == p.M * p.lda &&
                        p.stride_b == b_rows * p.ldb && p.stride_c == p.M * p.ldc;
    if (!packed) return fail(NNJIT_ERR_UNSUPPORTED, "run_host needs a packed plan");
    const size_t e = (size_t)p.elem_bytes();
    *a_bytes = (size_t)(p.batch * p.M * p.K) * e;
    *b_bytes = (size_t)p.b_bytes();
    *c_bytes = (size_t)(p.batch * p.M * p.N) * 4;
    if (p.M == 0 || p.N == 0) return NNJIT_OK;
    std::lock_guard<std::mutex> lk(pl->mu);
    cudaError_t err = cudaSuccess;
    if (!pl->hA && *a_bytes && (err = cudaMalloc(&pl->hA, *a_bytes)) != cudaSuccess) return cuda_fail(err, "staging A");
    if (!pl->hB && *b_bytes && (err = cudaMalloc(&pl->hB, *b_bytes)) != cudaSuccess) return cuda_fail(err, "staging B");
    if (!pl->hbias && (err = cudaMalloc(&pl->hbias, (size_t)p.N * 4)) != cudaSuccess) return cuda_fail(err, "staging bias");
    if (!pl->hC && (err = cudaMalloc(&pl->hC, *c_bytes)) != cudaSuccess) return cuda_fail(err, "staging C");
    return NNJIT_OK;
}

// Copy streams (host to device, device to host) and a pool of events of one device, used
// by nnjit_matmul_run_host_seq; `mu` serialises the calls that enqueue on them.
struct CopyLanes {
    std::mutex mu;
    cudaStream_t in = nullptr, out = nullptr;
    std::vector<cudaEvent_t> events;
};
std::mutex g_lanes_mu;
std::map<int, std::unique_ptr<CopyLanes>> g_lanes;

CopyLanes* copy_lanes(int dev) {
    std::lock_guard<std::mutex> lk(g_lanes_mu);
    auto& l = g_lanes[dev];
    if (!l) l.reset(new CopyLanes);
    return l.get();
}

}  // namespace

nnjit_status nnjit_matmul_run_host(nnjit_plan pl, const void* hA, const void* hB,
                                   const float* hbias, float* hC, void* stream) {
    if (!pl) return fail(NNJIT_ERR_INVALID_ARG, "plan is NULL");
    const Problem& p = pl->p;
    size_t a_bytes = 0, b_bytes = 0, c_bytes = 0;
    if (!hC && p.M > 0 && p.N > 0) return fail(NNJIT_ERR_INVALID_ARG, "NULL host buffer");
    if (p.M > 0 && p.N > 0 && p.K > 0 && (!hA || !hB)) return fail(NNJIT_ERR_INVALID_ARG, "NULL host buffer");
    nnjit_status st = host_staging(pl, &a_bytes, &b_bytes, &c_bytes);
    if (st != NNJIT_OK || p.M == 0 || p.N == 0) return st;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    cudaError_t err;
    if (a_bytes && (err = cudaMemcpyAsync(pl->hA, hA, a_bytes, cudaMemcpyHostToDevice, s)) != cudaSuccess)
        return cuda_fail(err, "copy A");
    if (b_bytes && (err = cudaMemcpyAsync(pl->hB, hB, b_bytes, cudaMemcpyHostToDevice, s)) != cudaSuccess)
        return cuda_fail(err, "copy B");
    if (hbias && (err = cudaMemcpyAsync(pl->hbias, hbias, (size_t)p.N * 4, cudaMemcpyHostToDevice, s)) != cudaSuccess)
        return cuda_fail(err, "copy bias");
    st = run_impl(pl, pl->hA, pl->hB, hbias ? pl->hbias : nullptr, pl->hC, s);
    if (st != NNJIT_OK) return st;
    if ((err = cudaMemcpyAsync(hC, pl->hC, c_bytes, cudaMemcpyDeviceToHost, s)) != cudaSuccess)
        return cuda_fail(err, "copy C");
    return NNJIT_OK;
}

nnjit_status nnjit_matmul_run_host_seq(int32_t count, const nnjit_plan* plans, const void* const* hA,
                                       const void* const* hB, const float* const* hbias,
                                       float* const* hC, void* stream) {
    if (count < 0 || (count > 0 && (!plans || !hA || !hB || !hC)))
        return fail(NNJIT_ERR_INVALID_ARG, "count < 0 or NULL array");
    if (count == 0) return NNJIT_OK;
    int dev = 0;
    cudaError_t err = cudaGetDevice(&dev);
    if (err != cudaSuccess) return cuda_fail(err, "current device");
    std::vector<size_t> ab(count), bb(count), cb(count);
    for (int32_t i = 0; i < count; ++i) {
        nnjit_plan pl = plans[i];
        if (!pl) return fail(NNJIT_ERR_INVALID_ARG, "plan is NULL");
        if (pl->device != dev) return fail(NNJIT_ERR_INVALID_ARG, "every plan must belong to the current device");
        const Problem& p = pl->p;
        if (p.M > 0 && p.N > 0 && (!hC[i] || (p.K > 0 && (!hA[i] || !hB[i]))))
            return fail(NNJIT_ERR_INVALID_ARG, "NULL host buffer");
        nnjit_status st = host_staging(pl, &ab[i], &bb[i], &cb[i]);
        if (st != NNJIT_OK) return st;
    }
    CopyLanes* L = copy_lanes(dev);
    std::lock_guard<std::mutex> lk(L->mu);
    if (!L->in && (err = cudaStreamCreateWithFlags(&L->in, cudaStreamNonBlocking)) != cudaSuccess)
        return cuda_fail(err, "copy stream");
    if (!L->out && (err = cudaStreamCreateWithFlags(&L->out, cudaStreamNonBlocking)) != cudaSuccess)
        return cuda_fail(err, "copy stream");
    // events: [0] the start, then per product: inputs landed, kernels done, result copied
    const size_t need = 1 + 3 * (size_t)count;
    while (L->events.size() < need) {
        cudaEvent_t e;
        if ((err = cudaEventCreateWithFlags(&e, cudaEventDisableTiming)) != cudaSuccess)
            return cuda_fail(err, "event");
        L->events.push_back(e);
    }
    cudaEvent_t* ev = L->events.data();
    auto ev_in = [&](int i) { return ev[1 + 3 * i]; };
    auto ev_k = [&](int i) { return ev[2 + 3 * i]; };
    auto ev_out = [&](int i) { return ev[3 + 3 * i]; };
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    // both copy streams start after the work already queued on `stream`
    if ((err = cudaEventRecord(ev[0], s)) != cudaSuccess ||
        (err = cudaStreamWaitEvent(L->in, ev[0], 0)) != cudaSuccess ||
        (err = cudaStreamWaitEvent(L->out, ev[0], 0)) != cudaSuccess)
        return cuda_fail(err, "stream join");
    for (int32_t i = 0; i < count; ++i) {
        nnjit_plan pl = plans[i];
        const Problem& p = pl->p;
        // an earlier product of the same plan: its staging buffers are reused, so this
        // product's inputs wait for its kernels and this product's kernels for its result
        int prev = -1;
        for (int32_t j = i - 1; j >= 0 && prev < 0; --j)
            if (plans[j] == pl) prev = j;
        if (prev >= 0 && (err = cudaStreamWaitEvent(L->in, ev_k(prev), 0)) != cudaSuccess)
            return cuda_fail(err, "stream join");
        const bool work = p.M > 0 && p.N > 0;
        if (work && ab[i] && (err = cudaMemcpyAsync(pl->hA, hA[i], ab[i], cudaMemcpyHostToDevice, L->in)) != cudaSuccess)
            return cuda_fail(err, "copy A");
        if (work && bb[i] && (err = cudaMemcpyAsync(pl->hB, hB[i], bb[i], cudaMemcpyHostToDevice, L->in)) != cudaSuccess)
            return cuda_fail(err, "copy B");
        const float* bias_i = hbias ? hbias[i] : nullptr;
        if (work && bias_i &&
            (err = cudaMemcpyAsync(pl->hbias, bias_i, (size_t)p.N * 4, cudaMemcpyHostToDevice, L->in)) != cudaSuccess)
            return cuda_fail(err, "copy bias");
        if ((err = cudaEventRecord(ev_in(i), L->in)) != cudaSuccess ||
            (err = cudaStreamWaitEvent(s, ev_in(i), 0)) != cudaSuccess)
            return cuda_fail(err, "stream join");
        if (prev >= 0 && (err = cudaStreamWaitEvent(s, ev_out(prev), 0)) != cudaSuccess)
            return cuda_fail(err, "stream join");
        if (work) {
            nnjit_status st = run_impl(pl, pl->hA, pl->hB, bias_i ? pl->hbias : nullptr, pl->hC, s);
            if (st != NNJIT_OK) return st;
        }
        if ((err = cudaEventRecord(ev_k(i), s)) != cudaSuccess ||
            (err = cudaStreamWaitEvent(L->out, ev_k(i), 0)) != cudaSuccess)
            return cuda_fail(err, "stream join");
        if (work && (err = cudaMemcpyAsync(hC[i], pl->hC, cb[i], cudaMemcpyDeviceToHost, L->out)) != cudaSuccess)
            return cuda_fail(err, "copy C");
        if ((err = cudaEventRecord(ev_out(i), L->out)) != cudaSuccess) return cuda_fail(err, "event");
    }
    // later work on `stream` starts after the last result has reached the host (the copy-out
    // stream runs in order, so its last event covers every earlier copy)
    if ((err = cudaStreamWaitEvent(s, ev_out(count - 1), 0)) != cudaSuccess) return cuda_fail(err, "stream join");
    return NNJIT_OK;
}

nnjit_status nnjit_plan_check(nnjit_plan p) {
    if (!p) return fail(NNJIT_ERR_INVALID_ARG, "plan is NULL");
    int cur = 0;
    cudaGetDevice(&cur);
    if (cur != p->device) cudaSetDevice(p->device);
    cudaError_t e = cudaDeviceSynchronize();
    int word = 0;
    if (e == cudaSuccess) e = cudaMemcpy(&word, p->err, sizeof(int), cudaMemcpyDeviceToHost);
    if (e == cudaSuccess && word != 0) {
        cudaMemset(p->err, 0, sizeof(int));
        // a stopped stream-K launch may have left hand-off flags raised
        if (p->ws && p->ws_bytes) cudaMemset(p->ws, 0, p->ws_bytes);
    }
    if (cur != p->device) cudaSetDevice(cur);
    if (e != cudaSuccess) return cuda_fail(e, "plan check");
    if (word != 0) {
        char buf[96];
        std::snprintf(buf, sizeof buf, "kernel watchdog expired (code 0x%x)", word);
        return fail(NNJIT_ERR_TIMEOUT, buf);
    }
    return NNJIT_OK;
}

nnjit_status nnjit_plan_candidate(nnjit_plan p, nnjit_candidate* out) {
    if (!p || !out) return fail(NNJIT_ERR_INVALID_ARG, "NULL argument");
    *out = p->cand;
    return NNJIT_OK;
}

nnjit_status nnjit_plan_describe(nnjit_plan pl, char* buf, size_t len, size_t* needed) {
    if (!pl) return fail(NNJIT_ERR_INVALID_ARG, "plan is NULL");
    const Problem& p = pl->p;
    const nnjit_candidate& c = pl->cand;
    std::string s;
    char tmp[1024];
    std::snprintf(tmp, sizeof tmp,
                  "{\"M\":%lld,\"N\":%lld,\"K\":%lld,\"batch\":%lld,\"dtype\":%d,\"b_layout\":%d,"
                  "\"family\":%d,\"chosen_index\":%d,\"space_size\":%d,\"naive_space\":%lld,"
                  "\"tune_ms\":%.3f,\"from_cache\":%s,\"timed\":%s,"
                  "\"candidate\":{\"bm\":%d,\"bn\":%d,\"bk\":%d,\"tm\":%d,\"tn\":%d,\"stages\":%d,"
                  "\"split_k\":%d,\"raster\":%d,\"threads\":%d,\"smem_bytes\":%d,\"tmem_cols\":%d,"
                  "\"regs_per_thread\":%d,\"blocks_per_sm\":%d,\"grid\":%d,\"wave_eff_ppm\":%d,"
                  "\"instance\":%d,\"predicted_cost\":%lld},\"settings\":[%d,%d,%d],\"timings_us\":[",
                  (long long)p.M, (long long)p.N, (long long)p.K, (long long)p.batch, p.dtype,
                  p.b_layout, pl->family, pl->chosen_index, pl->space_size, (long long)pl->naive,
                  pl->tune_ms, pl->from_cache ? "true" : "false", pl->timed ? "true" : "false",
                  c.bm, c.bn, c.bk, c.tm, c.tn, c.stages, c.split_k, c.raster, c.threads,
                  c.smem_bytes, c.tmem_cols, c.regs_per_thread, c.blocks_per_sm, c.grid,
                  c.wave_eff_ppm, c.instance, (long long)c.predicted_cost, pl->settings.raster,
                  pl->settings.kgroup, pl->settings.reduce);
    s += tmp;
    for (size_t i = 0; i < pl->timings.size(); ++i) {
        std::snprintf(tmp, sizeof tmp, "%s[%d,%.4f]", i ? "," : "", pl->timings[i].first,
                      pl->timings[i].second);
        s += tmp;
    }
    s += "],\"failed\":[";
    for (size_t i = 0; i < pl->failed.size(); ++i) {
        std::snprintf(tmp, sizeof tmp, "%s%d", i ? "," : "", pl->failed[i]);
        s += tmp;
    }
    s += "]}";
    if (needed) *needed = s.size() + 1;
    if (buf && len > 0) {
        const size_t n = std::min(len - 1, s.size());
        std::memcpy(buf, s.data(), n);
        buf[n] = '\0';
    }
    return NNJIT_OK;
}

nnjit_status nnjit_plan_destroy(nnjit_plan p) {
    free_plan(p);
    return NNJIT_OK;
}

nnjit_status nnjit_cache_clear(void) {
    std::lock_guard<std::mutex> lk(g_cache_mu);
    cache().clear();
    return NNJIT_OK;
}

int32_t nnjit_cache_size(void) {
    std::lock_guard<std::mutex> lk(g_cache_mu);
    return (int32_t)cache().size();
}

// File format: a header line, then one line per entry:
//   key \t 20 candidate integers \t chosen_index space_size naive tune_ms timed \t
//   n (index us)*n
static const char* kCacheHeader = "nnjit-plan-cache v3";

nnjit_status nnjit_cache_save(const char* path) {
    if (!path) return fail(NNJIT_ERR_INVALID_ARG, "path is NULL");
    std::string tmp = std::string(path) + ".tmp";
    FILE* f = std::fopen(tmp.c_str(), "w");
    if (!f) return fail(NNJIT_ERR_INVALID_ARG, std::string("cannot write ") + path);
    std::fprintf(f, "%s\n", kCacheHeader);
    {
        std::lock_guard<std::mutex> lk(g_cache_mu);
        for (const auto& kv : cache()) {
            const CacheEntry& e = kv.second;
            const nnjit_candidate& c = e.cand;
            std::fprintf(f, "%s\t%d %d %d %d %d %d %d %d %d %d %d %d %d %d %d %d %d %lld %d %d\t%d %d %lld %.6f %d\t%zu",
                         kv.first.c_str(), c.family, c.bm, c.bn, c.bk, c.tm, c.tn, c.stages,
                         c.split_k, c.raster, c.threads, c.smem_bytes, c.tmem_cols,
                         c.regs_per_thread, c.blocks_per_sm, c.grid, c.wave_eff_ppm, c.instance,
                         (long long)c.predicted_cost, c.reduce, c.cluster_m, e.chosen_index, e.space_size,
                         (long long)e.naive, e.tune_ms, e.timed ? 1 : 0, e.timings.size());
            for (const auto& t : e.timings) std::fprintf(f, " %d %.6f", t.first, t.second);
            std::fprintf(f, "\n");
        }
    }
    const bool ok = std::fclose(f) == 0 && std::rename(tmp.c_str(), path) == 0;
    if (!ok) return fail(NNJIT_ERR_INVALID_ARG, std::string("cannot write ") + path);
    return NNJIT_OK;
}

nnjit_status nnjit_cache_load(const char* path, int32_t* loaded) {
    if (!path) return fail(NNJIT_ERR_INVALID_ARG, "path is NULL");
    FILE* f = std::fopen(path, "r");
    if (!f) return fail(NNJIT_ERR_INVALID_ARG, std::string("cannot read ") + path);
    std::string content;
    char buf[4096];
    size_t n;
    while ((n = std::fread(buf, 1, sizeof buf, f)) > 0) content.append(buf, n);
    std::fclose(f);
    size_t pos = content.find('\n');
    if (pos == std::string::npos || content.substr(0, pos) != kCacheHeader)
        return fail(NNJIT_ERR_INVALID_ARG, "not an nnjit plan cache file");
    std::map<std::string, CacheEntry> got;
    while (pos != std::string::npos && pos + 1 < content.size()) {
        const size_t end = content.find('\n', pos + 1);
        const std::string line = content.substr(pos + 1, end == std::string::npos ? std::string::npos : end - pos - 1);
        pos = end;
        if (line.empty()) continue;
        const size_t t1 = line.find('\t');
        if (t1 == std::string::npos) return fail(NNJIT_ERR_INVALID_ARG, "malformed cache line");
        CacheEntry e{};
        nnjit_candidate& c = e.cand;
        long long cost = 0, naive = 0;
        int timed = 0;
        size_t ntim = 0;
        int used = 0;
        const char* rest = line.c_str() + t1 + 1;
        if (std::sscanf(rest, "%d %d %d %d %d %d %d %d %d %d %d %d %d %d %d %d %d %lld %d %d %d %d %lld %lf %d %zu%n",
                        &c.family, &c.bm, &c.bn, &c.bk, &c.tm, &c.tn, &c.stages, &c.split_k,
                        &c.raster, &c.threads, &c.smem_bytes, &c.tmem_cols, &c.regs_per_thread,
                        &c.blocks_per_sm, &c.grid, &c.wave_eff_ppm, &c.instance, &cost, &c.reduce,
                        &c.cluster_m, &e.chosen_index, &e.space_size, &naive, &e.tune_ms, &timed,
                        &ntim, &used) != 26 ||
            ntim > 4096)
            return fail(NNJIT_ERR_INVALID_ARG, "malformed cache line");
        c.predicted_cost = cost;
        e.naive = naive;
        e.timed = timed != 0;
        rest += used;
        for (size_t i = 0; i < ntim; ++i) {
            int idx = 0;
            double us = 0;
            int u2 = 0;
            if (std::sscanf(rest, " %d %lf%n", &idx, &us, &u2) != 2)
                return fail(NNJIT_ERR_INVALID_ARG, "malformed cache timings");
            rest += u2;
            e.timings.emplace_back(idx, us);
        }
        got[line.substr(0, t1)] = e;
    }
    {
        std::lock_guard<std::mutex> lk(g_cache_mu);
        for (auto& kv : got) cache()[kv.first] = kv.second;
    }
    if (loaded) *loaded = (int32_t)got.size();
    return NNJIT_OK;
}

}  // extern "C"
