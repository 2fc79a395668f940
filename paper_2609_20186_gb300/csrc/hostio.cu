// hostio.cu -- switchsd_step_host / switchsd_verify_step_host: one call with host-side inputs and results.
//
// A caller whose per-step inputs arrive in host memory and who reads the decisions back on the host
// (mode, draft, accepted length) would otherwise make three calls per step -- a host-to-device copy,
// the step, a device-to-host copy -- and a stream synchronisation.  These entry points make them in
// one foreign call: both copies are cudaMemcpyAsync on the step's stream around the unchanged step
// launch, so the GPU runs copy, step, copy back to back while the host returns (or waits, when asked).
#include "common.cuh"

namespace {

int stage_in(const switchsd_host_io *io, cudaStream_t s) {
    if (io->in_bytes == 0) return SWITCHSD_OK;
    return cudaMemcpyAsync(io->in_dev, io->in_host, io->in_bytes, cudaMemcpyHostToDevice, s) == cudaSuccess
               ? SWITCHSD_OK
               : SWITCHSD_ERR_CUDA;
}

int stage_out(const switchsd_host_io *io, cudaStream_t s) {
    if (io->out_bytes > 0 &&
        cudaMemcpyAsync(io->out_host, io->out_dev, io->out_bytes, cudaMemcpyDeviceToHost, s) != cudaSuccess)
        return SWITCHSD_ERR_CUDA;
    if (io->synchronize && cudaStreamSynchronize(s) != cudaSuccess) return SWITCHSD_ERR_CUDA;
    return SWITCHSD_OK;
}

bool io_ok(const switchsd_host_io *io) {
    return io != nullptr && (io->in_bytes == 0 || (io->in_host != nullptr && io->in_dev != nullptr)) &&
           (io->out_bytes == 0 || (io->out_host != nullptr && io->out_dev != nullptr));
}

}  // namespace

extern "C" int switchsd_step_host(const switchsd_host_io *io, const int32_t *ctx_tokens, const int32_t *ctx_lens,
                                  const uint16_t *hidden, const uint16_t *probe_w, const switchsd_params *params,
                                  int32_t *out_draft, int32_t *out_len, int32_t *out_mode, float *out_score) {
    if (!io_ok(io) || params == nullptr) return SWITCHSD_ERR_ARG;
    cudaStream_t s = static_cast<cudaStream_t>(params->stream);
    int code = stage_in(io, s);
    if (code != SWITCHSD_OK) return code;
    code = switchsd_step(ctx_tokens, ctx_lens, hidden, probe_w, params, out_draft, out_len, out_mode, out_score);
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
    int code = stage_in(io, s);
    if (code != SWITCHSD_OK) return code;
    code = switchsd_verify_step(draft, target_argmax, draft_len, out_accept, ctx_tokens, ctx_lens, hidden, probe_w,
                                params, out_draft, out_len, out_mode, out_score);
    if (code != SWITCHSD_OK) return code;
    return stage_out(io, s);
}
