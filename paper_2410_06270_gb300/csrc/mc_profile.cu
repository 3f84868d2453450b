// mc_profile.cu -- per-kernel CUDA-event timing of the library's launches.
#include <mutex>
#include <vector>

#include "mc_host.h"
#include "mc_profile.h"

namespace mc {

namespace {
struct Rec {
    int id;
    cudaEvent_t a, b;
    bool graph;  // recorded by event nodes of a captured graph: re-recorded by every replay
};
std::mutex g_mu;
bool g_on = false;
unsigned g_mask = ~0u;  // kernel ids recorded while on
std::vector<Rec> g_recs;
std::vector<cudaEvent_t> g_pool;
cudaEvent_t g_pending[kKCount];
const char *g_names[kKCount] = {"route", "permute", "gemv_w13", "gemv_w2", "combine",
                                "frag_x", "gemm_w13", "gemm_w2", "rmsnorm", "importance", "x_img"};

// An event record on st; inside stream capture it becomes an event node of the
// graph, so every replay of the graph records it again.
bool record(cudaEvent_t e, cudaStream_t st)
{
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    if (cudaStreamIsCapturing(st, &cs) == cudaSuccess && cs == cudaStreamCaptureStatusActive) {
        cudaEventRecordWithFlags(e, st, cudaEventRecordExternal);
        return true;
    }
    cudaEventRecord(e, st);
    return false;
}

cudaEvent_t take_event()
{
    if (!g_pool.empty()) {
        cudaEvent_t e = g_pool.back();
        g_pool.pop_back();
        return e;
    }
    cudaEvent_t e = nullptr;
    cudaEventCreate(&e);
    return e;
}
}  // namespace

bool profile_on() { return g_on; }

void profile_begin(int id, cudaStream_t st)
{
    if (!g_on || !((g_mask >> id) & 1u)) return;
    std::lock_guard<std::mutex> lk(g_mu);
    g_pending[id] = take_event();
    record(g_pending[id], st);
}

void profile_end(int id, cudaStream_t st)
{
    if (!g_on || !((g_mask >> id) & 1u)) return;
    std::lock_guard<std::mutex> lk(g_mu);
    cudaEvent_t b = take_event();
    const bool graph = record(b, st);
    g_recs.push_back({id, g_pending[id], b, graph});
}

}  // namespace mc

using namespace mc;

extern "C" {

int mc_profile_enable(int on)
{
    std::lock_guard<std::mutex> lk(g_mu);
    int old = g_on;
    g_on = on != 0;
    return old;
}

unsigned mc_profile_select(unsigned mask)
{
    std::lock_guard<std::mutex> lk(g_mu);
    const unsigned old = g_mask;
    g_mask = mask;
    return old;
}

int mc_profile_read(double *ms_out, int *count_out, int n)
{
    clear_error();
    std::vector<Rec> recs, kept;
    {
        std::lock_guard<std::mutex> lk(g_mu);
        recs.swap(g_recs);
    }
    for (auto &r : recs)
        if (r.graph) kept.push_back(r);
    for (int i = 0; i < n; ++i) {
        if (ms_out) ms_out[i] = 0;
        if (count_out) count_out[i] = 0;
    }
    int rc = MC_OK;
    for (auto &r : recs) {
        if (cudaEventSynchronize(r.b) != cudaSuccess) rc = set_error(MC_ERR_CUDA, "event sync failed");
        float ms = 0.f;
        if (cudaEventElapsedTime(&ms, r.a, r.b) != cudaSuccess) rc = set_error(MC_ERR_CUDA, "elapsed failed");
        if (r.id < n) {
            if (ms_out) ms_out[r.id] += ms;
            if (count_out) count_out[r.id] += 1;
        }
    }
    std::lock_guard<std::mutex> lk(g_mu);
    for (auto &r : recs) {
        if (r.graph) continue;
        g_pool.push_back(r.a);
        g_pool.push_back(r.b);
    }
    g_recs.insert(g_recs.begin(), kept.begin(), kept.end());
    return rc;
}

int mc_profile_clear(void)
{
    std::lock_guard<std::mutex> lk(g_mu);
    for (auto &r : g_recs) {
        g_pool.push_back(r.a);
        g_pool.push_back(r.b);
    }
    g_recs.clear();
    return MC_OK;
}

const char *mc_profile_name(int id) { return (id >= 0 && id < kKCount) ? g_names[id] : ""; }

}  // extern "C"
