// noalloc.cu -- switchsd_step_static_workspace: switchsd_step for callers that cannot allocate.
//
// switchsd_step with the two-layer probe needs device scratch between its two kernels (the first
// layer's split-K partial sums), which the caller normally passes in params->workspace.  Some callers cannot hand
// the library device memory at call time: an inference server that gives all of the GPU's memory to
// its own pool when it starts, or a host program with no CUDA allocator of its own.  This entry point
// serves them from a fixed array compiled into the library instead, and allocates nothing.
//
// The array is a file-scope __device__ variable: every GPU that loads the library holds it (16 MiB)
// until the process exits.  Host code cannot use the variable's name as a device address, so the
// first call on each device asks the runtime for the array's address (cudaGetSymbolAddress) with that
// device current, and every later call on the device reuses it.  A device reset (cudaDeviceReset) ends
// the context the address belongs to, so the cached address is not valid after one: a process that
// resets a device must not call this entry point on it again.
#include <mutex>

#include "common.cuh"

namespace {

// Two-layer probe scratch: S x B x H1p floats (switchsd_workspace_bytes).
constexpr size_t kStaticWorkspaceFloats = size_t(4) << 20;  // 16 MiB
static __device__ __align__(256) float g_static_workspace[kStaticWorkspaceFloats];

constexpr int kMaxDevices = 64;
std::mutex g_lock;
void *g_address[kMaxDevices] = {};

// The array's device address on the current device, looked up once per device; NULL on failure.
void *static_workspace_address() {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
    std::lock_guard<std::mutex> guard(g_lock);
    if (g_address[dev] == nullptr) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_static_workspace) != cudaSuccess) {
            (void)cudaGetLastError();  // leave no error behind for the caller's next runtime check
            return nullptr;
        }
        g_address[dev] = p;
    }
    return g_address[dev];
}

}  // namespace

extern "C" int switchsd_step_static_workspace(const int32_t *ctx_tokens, const int32_t *ctx_lens,
                                              const uint16_t *hidden, const uint16_t *probe_w,
                                              const switchsd_params *params, int32_t *out_draft,
                                              int32_t *out_len, int32_t *out_mode, float *out_score) {
    if (params == nullptr) return SWITCHSD_ERR_ARG;
    const size_t need = switchsd_workspace_bytes(params);
    if (need > sizeof(g_static_workspace)) return SWITCHSD_ERR_SHAPE;  // S(d) * B * H1p > 4 Mi floats
    switchsd_params p = *params;
    if (need > 0) {
        void *ws = static_workspace_address();
        if (ws == nullptr) return SWITCHSD_ERR_CUDA;
        p.workspace = ws;
        p.workspace_bytes = sizeof(g_static_workspace);
    }
    return switchsd_step(ctx_tokens, ctx_lens, hidden, probe_w, &p, out_draft, out_len, out_mode, out_score);
}
