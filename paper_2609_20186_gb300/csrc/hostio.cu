// hostio.cu -- switchsd_step_host / switchsd_verify_step_host: one call with host-side inputs and results.
//
// A caller whose per-step inputs arrive in host memory and who reads the decisions back on the host
// (mode, draft, accepted length) would otherwise make three calls per step -- a host-to-device copy,
// the step, a device-to-host copy -- and a stream synchronisation.  These entry points make them in
// one foreign call, ordered on the step's stream.
//
// The copies.  On this machine a copy-engine transfer costs ~10 us of latency on the GPU's timeline,
// more than the step itself, while the GPU reads and writes page-locked host memory directly at
// little cost (the host is attached over a coherent link).  So when a host buffer is page-locked and
// mapped into the device's address space (every pinned allocation is, with unified addressing) the
// copy is a small kernel of 16-byte loads and stores through its device address; a pageable buffer
// goes through cudaMemcpyAsync.  The input-copy kernel is launched in stream order without
// programmatic serialization and the step after it keeps its prefetch bits only for inputs that the
// copy does not write; the output-copy kernel, launched the same way, starts after the step is
// complete and its writes are visible to the host once the stream is synchronised.
#include "common.cuh"

namespace {

constexpr int kCopyThreads = 256;

struct CopyArgs {
    void *dst;
    const void *src;
    size_t bytes;
};

__global__ void __launch_bounds__(kCopyThreads) host_copy_kernel(const CopyArgs a) {
    const size_t stride = size_t(gridDim.x) * kCopyThreads;
    const size_t t0 = size_t(blockIdx.x) * kCopyThreads + threadIdx.x;
    if (((reinterpret_cast<uintptr_t>(a.dst) | reinterpret_cast<uintptr_t>(a.src) | a.bytes) & 15) == 0) {
        const uint4 *src = static_cast<const uint4 *>(a.src);
        uint4 *dst = static_cast<uint4 *>(a.dst);
        const size_t n = a.bytes / 16;
        size_t i = t0;
        for (; i + 3 * stride < n; i += 4 * stride) {  // four loads in flight per thread
            const uint4 v0 = src[i], v1 = src[i + stride], v2 = src[i + 2 * stride], v3 = src[i + 3 * stride];
            dst[i] = v0;
            dst[i + stride] = v1;
            dst[i + 2 * stride] = v2;
            dst[i + 3 * stride] = v3;
        }
        for (; i < n; i += stride) dst[i] = src[i];
    } else {
        const uint8_t *src = static_cast<const uint8_t *>(a.src);
        uint8_t *dst = static_cast<uint8_t *>(a.dst);
        for (size_t i = t0; i < a.bytes; i += stride) dst[i] = src[i];
    }
}

// The device address of page-locked, mapped host memory at `host`; NULL for any other pointer
// (pageable memory, device memory, an unknown address).
void *mapped_address(const void *host) {
    cudaPointerAttributes at;
    if (cudaPointerGetAttributes(&at, host) != cudaSuccess) {
        cudaGetLastError();
        return nullptr;
    }
    return at.type == cudaMemoryTypeHost ? at.devicePointer : nullptr;
}

unsigned copy_blocks(size_t bytes) {
    const size_t words = (bytes + 15) / 16;
    const size_t blocks = (words + 4 * kCopyThreads - 1) / (4 * kCopyThreads);
    return unsigned(blocks < 1 ? 1 : (blocks > 1024 ? 1024 : blocks));
}

int copy_by_kernel(void *dst, const void *src, size_t bytes, cudaStream_t s) {
    CopyArgs a{dst, src, bytes};
    host_copy_kernel<<<copy_blocks(bytes), kCopyThreads, 0, s>>>(a);
    return cudaGetLastError() == cudaSuccess ? SWITCHSD_OK : SWITCHSD_ERR_CUDA;
}

// *by_kernel: whether the copy ran as a kernel (which then immediately precedes the step).
int stage_in(const switchsd_host_io *io, cudaStream_t s, bool *by_kernel) {
    *by_kernel = false;
    if (io->in_bytes == 0) return SWITCHSD_OK;
    if (const void *src = mapped_address(io->in_host)) {
        *by_kernel = true;
        return copy_by_kernel(io->in_dev, src, io->in_bytes, s);
    }
    return cudaMemcpyAsync(io->in_dev, io->in_host, io->in_bytes, cudaMemcpyHostToDevice, s) == cudaSuccess
               ? SWITCHSD_OK
               : SWITCHSD_ERR_CUDA;
}

int stage_out(const switchsd_host_io *io, cudaStream_t s) {
    if (io->out_bytes > 0) {
        if (void *dst = mapped_address(io->out_host)) {
            const int code = copy_by_kernel(dst, io->out_dev, io->out_bytes, s);
            if (code != SWITCHSD_OK) return code;
        } else if (cudaMemcpyAsync(io->out_host, io->out_dev, io->out_bytes, cudaMemcpyDeviceToHost, s) !=
                   cudaSuccess) {
            return SWITCHSD_ERR_CUDA;
        }
    }
    if (io->synchronize && cudaStreamSynchronize(s) != cudaSuccess) return SWITCHSD_ERR_CUDA;
    return SWITCHSD_OK;
}

bool io_ok(const switchsd_host_io *io) {
    return io != nullptr && (io->in_bytes == 0 || (io->in_host != nullptr && io->in_dev != nullptr)) &&
           (io->out_bytes == 0 || (io->out_host != nullptr && io->out_dev != nullptr));
}

bool overlaps(const void *a, size_t an, const void *b, size_t bn) {
    const uintptr_t x = reinterpret_cast<uintptr_t>(a), y = reinterpret_cast<uintptr_t>(b);
    return b != nullptr && an > 0 && bn > 0 && x < y + bn && y < x + an;
}

// The step's parameters after an input copy by kernel: a prefetch bit stays only if the copied range
// misses every input that bit lets the step read before the copy kernel is done.
switchsd_params after_copy_kernel(const switchsd_params &p, const switchsd_host_io *io, const void *ctx,
                                  const void *lens, const void *hidden, const void *probe_w) {
    switchsd_params q = p;
    const size_t B = p.B > 0 ? size_t(p.B) : 0, d = p.d > 0 ? size_t(p.d) : 0;
    const size_t rows = p.hidden_rows > 1 ? size_t(p.hidden_rows) : 1;
    const size_t w_bytes = p.probe_kind == SWITCHSD_PROBE_MLP && p.probe_hidden > 0
                               ? (size_t(p.probe_hidden) * d + size_t(p.probe_hidden)) * 2
                               : d * 2;
    if (overlaps(io->in_dev, io->in_bytes, hidden, B * rows * d * 2) ||
        overlaps(io->in_dev, io->in_bytes, probe_w, w_bytes))
        q.prefetch &= ~SWITCHSD_PREFETCH_PROBE;
    if (overlaps(io->in_dev, io->in_bytes, ctx, B * (p.cap > 0 ? size_t(p.cap) : 0) * 4) ||
        overlaps(io->in_dev, io->in_bytes, lens, B * 4))
        q.prefetch &= ~SWITCHSD_PREFETCH_CONTEXT;
    return q;
}

}  // namespace

extern "C" int switchsd_step_host(const switchsd_host_io *io, const int32_t *ctx_tokens, const int32_t *ctx_lens,
                                  const uint16_t *hidden, const uint16_t *probe_w, const switchsd_params *params,
                                  int32_t *out_draft, int32_t *out_len, int32_t *out_mode, float *out_score) {
    if (!io_ok(io) || params == nullptr) return SWITCHSD_ERR_ARG;
    cudaStream_t s = static_cast<cudaStream_t>(params->stream);
    bool by_kernel = false;
    int code = stage_in(io, s, &by_kernel);
    if (code != SWITCHSD_OK) return code;
    const switchsd_params q = by_kernel ? after_copy_kernel(*params, io, ctx_tokens, ctx_lens, hidden, probe_w)
                                        : *params;
    code = switchsd_step(ctx_tokens, ctx_lens, hidden, probe_w, &q, out_draft, out_len, out_mode, out_score);
    if (code != SWITCHSD_OK) return code;
    return stage_out(io, s);
}

extern "C" int switchsd_verify_step_host(const switchsd_host_io *io, const int32_t *draft,
                                         const int32_t *target_argmax, const int32_t *draft_len,
                                         int32_t *out_accept, int32_t *ctx_tokens, int32_t *ctx_lens,
                                         const uint16_t *hidden, const uint16_t *probe_w,
                                         const switchsd_params *params, int32_t *out_draft, int32_t *out_len,
                                         int32_t *out_mode, float *out_score) {
    if (!io_ok(io) || params == nullptr) return SWITCHSD_ERR_ARG;
    cudaStream_t s = static_cast<cudaStream_t>(params->stream);
    bool by_kernel = false;
    int code = stage_in(io, s, &by_kernel);
    if (code != SWITCHSD_OK) return code;
    const switchsd_params q = by_kernel ? after_copy_kernel(*params, io, ctx_tokens, ctx_lens, hidden, probe_w)
                                        : *params;
    code = switchsd_verify_step(draft, target_argmax, draft_len, out_accept, ctx_tokens, ctx_lens, hidden, probe_w,
                                &q, out_draft, out_len, out_mode, out_score);
    if (code != SWITCHSD_OK) return code;
    return stage_out(io, s);
}

extern "C" int switchsd_verify_sampled_step_host(const switchsd_host_io *io, const int32_t *draft,
                                                 const float *p_draft, const float *q_draft, const float *u,
                                                 const int32_t *resample, const int32_t *draft_len,
                                                 int32_t *out_accept, int32_t *ctx_tokens, int32_t *ctx_lens,
                                                 const uint16_t *hidden, const uint16_t *probe_w,
                                                 const switchsd_params *params, int32_t *out_draft,
                                                 int32_t *out_len, int32_t *out_mode, float *out_score) {
    if (!io_ok(io) || params == nullptr) return SWITCHSD_ERR_ARG;
    cudaStream_t s = static_cast<cudaStream_t>(params->stream);
    bool by_kernel = false;
    int code = stage_in(io, s, &by_kernel);
    if (code != SWITCHSD_OK) return code;
    const switchsd_params q = by_kernel ? after_copy_kernel(*params, io, ctx_tokens, ctx_lens, hidden, probe_w)
                                        : *params;
    code = switchsd_verify_sampled_step(draft, p_draft, q_draft, u, resample, draft_len, out_accept, ctx_tokens,
                                        ctx_lens, hidden, probe_w, &q, out_draft, out_len, out_mode, out_score);
    if (code != SWITCHSD_OK) return code;
    return stage_out(io, s);
}

// ------------------------------------------------------------------------------------------------
// switchsd_plan: the host-staged step recorded once as a CUDA graph and replayed per call.
//
// A graph holding input copy -> step launch(es) -> output copy is handed to the GPU in one submission.
// It is recorded by stream capture of exactly the calls switchsd_*_host makes, on a private stream; a
// replay with other host buffers only retargets the two copy nodes (kernel or copy-engine nodes, as
// recorded).
// ------------------------------------------------------------------------------------------------
struct switchsd_plan {
    cudaGraph_t graph = nullptr;
    cudaGraphExec_t exec = nullptr;
    cudaGraphNode_t in_node = nullptr, out_node = nullptr;
    bool in_kernel = false, out_kernel = false;  // copy by kernel (mapped host memory) or copy engine
    switchsd_host_io io = {};
    cudaStream_t stream = nullptr;  // where replays are launched (the step's params->stream)
};

namespace {

void plan_free(switchsd_plan *p) {
    if (p == nullptr) return;
    if (p->exec) cudaGraphExecDestroy(p->exec);
    if (p->graph) cudaGraphDestroy(p->graph);
    delete p;
}

// The recorded copy whose source (src_end) or destination is `end`: a host_copy_kernel node when
// `kernel` (end is then a device address), else a memcpy node (end is the host pointer).
cudaGraphNode_t find_copy(cudaGraph_t g, bool kernel, const void *end, bool src_end) {
    cudaGraphNode_t nodes[64];
    size_t n = 0;
    if (cudaGraphGetNodes(g, nullptr, &n) != cudaSuccess || n == 0 || n > 64) return nullptr;
    if (cudaGraphGetNodes(g, nodes, &n) != cudaSuccess) return nullptr;
    for (size_t i = 0; i < n; ++i) {
        cudaGraphNodeType t;
        if (cudaGraphNodeGetType(nodes[i], &t) != cudaSuccess) continue;
        if (kernel && t == cudaGraphNodeTypeKernel) {
            cudaKernelNodeParams kp = {};
            if (cudaGraphKernelNodeGetParams(nodes[i], &kp) != cudaSuccess) continue;
            if (kp.func != reinterpret_cast<void *>(host_copy_kernel) || kp.kernelParams == nullptr) continue;
            const CopyArgs *a = static_cast<const CopyArgs *>(kp.kernelParams[0]);
            if ((src_end ? a->src : static_cast<const void *>(a->dst)) == end) return nodes[i];
        } else if (!kernel && t == cudaGraphNodeTypeMemcpy) {
            cudaMemcpy3DParms m = {};
            if (cudaGraphMemcpyNodeGetParams(nodes[i], &m) != cudaSuccess) continue;
            if ((src_end ? m.srcPtr.ptr : m.dstPtr.ptr) == end) return nodes[i];
        }
    }
    return nullptr;
}

int retarget_kernel(cudaGraphExec_t exec, cudaGraphNode_t node, CopyArgs a) {
    void *args[1] = {&a};
    cudaKernelNodeParams kp = {};
    kp.func = reinterpret_cast<void *>(host_copy_kernel);
    kp.gridDim = dim3(copy_blocks(a.bytes));
    kp.blockDim = dim3(kCopyThreads);
    kp.sharedMemBytes = 0;
    kp.kernelParams = args;
    kp.extra = nullptr;
    return cudaGraphExecKernelNodeSetParams(exec, node, &kp) == cudaSuccess ? SWITCHSD_OK : SWITCHSD_ERR_CUDA;
}

}  // namespace

extern "C" int switchsd_plan_create(const switchsd_step_args *a, const switchsd_host_io *io, switchsd_plan **out) {
    if (out == nullptr) return SWITCHSD_ERR_ARG;
    *out = nullptr;
    if (a == nullptr || a->params == nullptr || !io_ok(io)) return SWITCHSD_ERR_ARG;
    const bool verify = a->draft != nullptr || a->target_argmax != nullptr || a->draft_len != nullptr;
    if (verify && (a->draft == nullptr || a->target_argmax == nullptr || a->draft_len == nullptr))
        return SWITCHSD_ERR_ARG;
    const bool sampled = a->p_draft != nullptr || a->u != nullptr || a->q_draft != nullptr;
    if (sampled && (!verify || a->p_draft == nullptr || a->u == nullptr)) return SWITCHSD_ERR_ARG;
    switchsd_plan *p = new switchsd_plan;
    p->io = *io;
    p->io.synchronize = 0;
    p->stream = static_cast<cudaStream_t>(a->params->stream);
    cudaStream_t cap = nullptr;
    if (cudaStreamCreateWithFlags(&cap, cudaStreamNonBlocking) != cudaSuccess) {
        cudaGetLastError();
        plan_free(p);
        return SWITCHSD_ERR_CUDA;
    }
    int code = SWITCHSD_OK;
    if (cudaStreamBeginCapture(cap, cudaStreamCaptureModeRelaxed) != cudaSuccess) {
        code = SWITCHSD_ERR_CUDA;
    } else {
        code = stage_in(&p->io, cap, &p->in_kernel);
        switchsd_params q = p->in_kernel ? after_copy_kernel(*a->params, &p->io, a->ctx_tokens, a->ctx_lens,
                                                             a->hidden, a->probe_w)
                                         : *a->params;
        q.stream = cap;
        if (code == SWITCHSD_OK)
            code = sampled ? switchsd_verify_sampled_step(a->draft, a->p_draft, a->q_draft, a->u, a->target_argmax,
                                                          a->draft_len, a->out_accept, a->ctx_tokens, a->ctx_lens,
                                                          a->hidden, a->probe_w, &q, a->out_draft, a->out_len,
                                                          a->out_mode, a->out_score)
                   : verify ? switchsd_verify_step(a->draft, a->target_argmax, a->draft_len, a->out_accept,
                                                   a->ctx_tokens, a->ctx_lens, a->hidden, a->probe_w, &q, a->out_draft,
                                                   a->out_len, a->out_mode, a->out_score)
                            : switchsd_step(a->ctx_tokens, a->ctx_lens, a->hidden, a->probe_w, &q, a->out_draft,
                                            a->out_len, a->out_mode, a->out_score);
        p->out_kernel = p->io.out_bytes > 0 && mapped_address(p->io.out_host) != nullptr;
        if (code == SWITCHSD_OK) code = stage_out(&p->io, cap);  // synchronize is 0: queues the copy only
        cudaGraph_t g = nullptr;
        const cudaError_t e = cudaStreamEndCapture(cap, &g);     // always ends the capture
        if (code == SWITCHSD_OK && e != cudaSuccess) code = SWITCHSD_ERR_CUDA;
        p->graph = g;
    }
    if (code == SWITCHSD_OK && p->graph == nullptr) code = SWITCHSD_ERR_CUDA;
    if (code == SWITCHSD_OK && cudaGraphInstantiate(&p->exec, p->graph, 0) != cudaSuccess) code = SWITCHSD_ERR_CUDA;
    if (code == SWITCHSD_OK && io->in_bytes > 0) {
        const void *end = p->in_kernel ? mapped_address(io->in_host) : io->in_host;
        if ((p->in_node = find_copy(p->graph, p->in_kernel, end, true)) == nullptr) code = SWITCHSD_ERR_CUDA;
    }
    if (code == SWITCHSD_OK && io->out_bytes > 0) {
        const void *end = p->out_kernel ? mapped_address(io->out_host) : io->out_host;
        if ((p->out_node = find_copy(p->graph, p->out_kernel, end, false)) == nullptr) code = SWITCHSD_ERR_CUDA;
    }
    cudaStreamDestroy(cap);
    if (code != SWITCHSD_OK) {
        cudaGetLastError();  // clear the (non-sticky) error a failed capture or instantiation leaves
        plan_free(p);
        return code;
    }
    *out = p;
    return SWITCHSD_OK;
}

extern "C" int switchsd_plan_run(switchsd_plan *p, const void *in_host, void *out_host, int32_t synchronize) {
    if (p == nullptr || p->exec == nullptr) return SWITCHSD_ERR_ARG;
    if (in_host == nullptr) in_host = p->io.in_host;
    if (out_host == nullptr) out_host = p->io.out_host;
    if (p->in_node != nullptr && in_host != p->io.in_host) {
        int code;
        if (p->in_kernel) {
            const void *src = mapped_address(in_host);
            if (src == nullptr) return SWITCHSD_ERR_ARG;  // recorded as a kernel copy: needs pinned memory
            code = retarget_kernel(p->exec, p->in_node, CopyArgs{p->io.in_dev, src, p->io.in_bytes});
        } else {
            code = cudaGraphExecMemcpyNodeSetParams1D(p->exec, p->in_node, p->io.in_dev, in_host, p->io.in_bytes,
                                                      cudaMemcpyHostToDevice) == cudaSuccess
                       ? SWITCHSD_OK
                       : SWITCHSD_ERR_CUDA;
        }
        if (code != SWITCHSD_OK) return code;
        p->io.in_host = in_host;
    }
    if (p->out_node != nullptr && out_host != p->io.out_host) {
        int code;
        if (p->out_kernel) {
            void *dst = mapped_address(out_host);
            if (dst == nullptr) return SWITCHSD_ERR_ARG;
            code = retarget_kernel(p->exec, p->out_node, CopyArgs{dst, p->io.out_dev, p->io.out_bytes});
        } else {
            code = cudaGraphExecMemcpyNodeSetParams1D(p->exec, p->out_node, out_host, p->io.out_dev, p->io.out_bytes,
                                                      cudaMemcpyDeviceToHost) == cudaSuccess
                       ? SWITCHSD_OK
                       : SWITCHSD_ERR_CUDA;
        }
        if (code != SWITCHSD_OK) return code;
        p->io.out_host = out_host;
    }
    if (cudaGraphLaunch(p->exec, p->stream) != cudaSuccess) return SWITCHSD_ERR_CUDA;
    if (synchronize && cudaStreamSynchronize(p->stream) != cudaSuccess) return SWITCHSD_ERR_CUDA;
    return SWITCHSD_OK;
}

extern "C" void switchsd_plan_destroy(switchsd_plan *p) { plan_free(p); }
