// api.cu -- library-wide entry points of the C ABI (error text, ABI version).
#include "common.cuh"

extern "C" const char *switchsd_strerror(int code) {
    switch (code) {
        case SWITCHSD_OK: return "ok";
        case SWITCHSD_ERR_ARG: return "bad argument (NULL or misaligned pointer, or bad enum)";
        case SWITCHSD_ERR_SHAPE: return "unsupported shape";
        case SWITCHSD_ERR_CUDA: return "CUDA launch failed";
        case SWITCHSD_ROW_CAPACITY: return "row: append does not fit in cap";
        case SWITCHSD_ROW_BAD_LEN: return "row: length out of range";
        case SWITCHSD_ROW_TIMEOUT: return "row: on-chip copy did not complete in time";
        default: return "unknown code";
    }
}

extern "C" int switchsd_abi_version(void) { return SWITCHSD_ABI_VERSION; }
