// labels.cu -- switchsd_copy_labels: copy-mode labels of every position of B rows (§3.2).
//
// Position j of a row is labelled 1 when it lies in a window of n consecutive tokens that also occurs
// starting at an earlier position of the row (the paper trains its probe on these labels with
// n = n_train = 5).  Two kernels over a per-row open-addressing table in the caller's workspace:
//
//   insert  thread per window start s: hash the n tokens, probe linearly; an empty slot is claimed with
//           atomicCAS, a slot whose window holds the same tokens takes atomicMin(slot, s).  Every slot
//           then holds the smallest start among the windows with its tokens -- the same value whatever
//           order the inserts ran in.  The slot of s is recorded in where[s].
//   label   CTA per 256 positions: for the window starts s in [j0 - n + 1, j0 + 256) it reads the slot
//           of s and marks s when the slot's smallest start is below s (the window repeats); position
//           j is then the OR of the marks of the n windows that cover it.
//
// The table has a power of two >= 2 * cap slots per row (load factor <= 1/2), so every probe sequence
// ends within the table.  Windows are compared token by token, so hash collisions cost time only.
#include "common.cuh"

namespace switchsd {

constexpr int kLabelThreads = 256;

struct LabelArgs {
    const int32_t *ctx, *lens;
    int32_t *table;     // [B][T]
    int32_t *where;     // [B][cap]: the slot of each window start
    uint8_t *labels;    // [B][cap]
    int32_t B, cap, n;
    uint32_t tmask;     // T - 1
};

__device__ __forceinline__ uint32_t window_hash(const int32_t *w, int n, uint32_t tmask) {
    uint64_t h = 0x9E3779B97F4A7C15ull ^ uint64_t(n);
    for (int i = 0; i < n; ++i) {
        h = (h ^ uint64_t(uint32_t(w[i]))) * 0xBF58476D1CE4E5B9ull;
        h ^= h >> 31;
    }
    return uint32_t(h ^ (h >> 32)) & tmask;
}

__device__ __forceinline__ bool same_window(const int32_t *a, const int32_t *b, int n) {
    for (int i = 0; i < n; ++i)
        if (a[i] != b[i]) return false;
    return true;
}

__device__ __forceinline__ int32_t row_length(const LabelArgs &a, int b) {
    const int32_t L = a.lens[b];
    return (L >= 0 && L <= a.cap) ? L : 0;  // a length outside [0, cap] labels nothing
}

__global__ void __launch_bounds__(kLabelThreads) label_insert_kernel(const LabelArgs a) {
    const int b = blockIdx.y;
    const int32_t s = int32_t(blockIdx.x) * kLabelThreads + threadIdx.x;
    pdl_wait();
    pdl_trigger();
    const int32_t L = row_length(a, b);
    if (s + a.n > L) return;
    const int32_t *x = a.ctx + size_t(b) * size_t(a.cap);
    int32_t *tab = a.table + size_t(b) * (size_t(a.tmask) + 1);
    int32_t *where = a.where + size_t(b) * size_t(a.cap);
    uint32_t h = window_hash(x + s, a.n, a.tmask);
    for (uint32_t probe = 0; probe <= a.tmask; ++probe, h = (h + 1) & a.tmask) {
        // Claim the slot if empty; otherwise the CAS returns its start (one round trip either way).
        const int32_t v = atomicCAS(&tab[h], -1, s);
        if (v < 0) {
            where[s] = int32_t(h);
            return;
        }
        if (same_window(x + v, x + s, a.n)) {
            atomicMin(&tab[h], s);
            where[s] = int32_t(h);
            return;
        }
    }
}

__global__ void __launch_bounds__(kLabelThreads) label_mark_kernel(const LabelArgs a) {
    __shared__ uint8_t s_rep[kLabelThreads + SWITCHSD_NMAX];  // window repeats, for starts j0 - n + 1 ..
    const int b = blockIdx.y;
    const int32_t j0 = int32_t(blockIdx.x) * kLabelThreads;
    pdl_wait();
    pdl_trigger();
    const int32_t L = row_length(a, b);
    const int32_t *tab = a.table + size_t(b) * (size_t(a.tmask) + 1);
    const int32_t *where = a.where + size_t(b) * size_t(a.cap);
    const int32_t first = j0 - a.n + 1;
    for (int t = threadIdx.x; t < kLabelThreads + a.n - 1; t += kLabelThreads) {
        const int32_t s = first + t;
        uint8_t rep = 0;
        if (s >= 0 && s + a.n <= L) {
            const int32_t h = where[s];  // written by the insert of s
            rep = h >= 0 && uint32_t(h) <= a.tmask && tab[h] < s;
        }
        s_rep[t] = rep;
    }
    __syncthreads();
    const int32_t j = j0 + int32_t(threadIdx.x);
    if (j >= a.cap) return;
    uint8_t y = 0;
    if (j < L)
        for (int i = 0; i < a.n; ++i) y |= s_rep[threadIdx.x + i];  // windows starting at j - n + 1 .. j
    a.labels[size_t(b) * size_t(a.cap) + j] = y;
}

static uint32_t table_slots(int32_t cap) {
    uint32_t t = 16;
    while (t < 2u * uint32_t(cap)) t <<= 1;
    return t;
}

}  // namespace switchsd

using namespace switchsd;

extern "C" size_t switchsd_labels_workspace_bytes(int32_t B, int32_t cap) {
    if (B < 1 || cap < 1) return 0;
    return size_t(B) * (size_t(table_slots(cap)) + size_t(cap)) * sizeof(int32_t);
}

extern "C" int switchsd_copy_labels(const int32_t *ctx_tokens, const int32_t *ctx_lens, int32_t B, int32_t cap,
                                    int32_t n, uint8_t *out_labels, void *workspace, size_t workspace_bytes,
                                    void *stream) {
    if (!ctx_tokens || !ctx_lens || !out_labels || !workspace) return SWITCHSD_ERR_ARG;
    if ((reinterpret_cast<uintptr_t>(workspace) & 3) != 0) return SWITCHSD_ERR_ARG;
    if (B < 1 || B > 65535 || cap < 1 || cap > (1 << 30) || n < 1 || n > SWITCHSD_NMAX) return SWITCHSD_ERR_SHAPE;
    if (workspace_bytes < switchsd_labels_workspace_bytes(B, cap)) return SWITCHSD_ERR_ARG;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const uint32_t T = table_slots(cap);
    if (cudaMemsetAsync(workspace, 0xff, size_t(B) * T * sizeof(int32_t), s) != cudaSuccess) return SWITCHSD_ERR_CUDA;
    LabelArgs a;
    a.ctx = ctx_tokens;
    a.lens = ctx_lens;
    a.table = static_cast<int32_t *>(workspace);
    a.where = a.table + size_t(B) * T;
    a.labels = out_labels;
    a.B = B;
    a.cap = cap;
    a.n = n;
    a.tmask = T - 1;
    const dim3 grid(unsigned((cap + kLabelThreads - 1) / kLabelThreads), unsigned(B));
    if (launch_pdl(label_insert_kernel, grid, dim3(kLabelThreads), 0, s, 0u, a) != cudaSuccess)
        return SWITCHSD_ERR_CUDA;
    if (launch_pdl(label_mark_kernel, grid, dim3(kLabelThreads), 0, s, 0u, a) != cudaSuccess)
        return SWITCHSD_ERR_CUDA;
    return SWITCHSD_OK;
}
