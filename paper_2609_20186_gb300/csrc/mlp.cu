// mlp.cu -- first layer of the two-layer copy-intent probe z = w2 . ReLU(W1 h + b1) + b2, on the tensor cores.
//
// The paper's probe is linear (Eq. 3); this two-layer form is an extension used with probe_kind
// SWITCHSD_PROBE_MLP.  Its first layer is a real contraction, Z1[B, H1] = H[B, d] . W1[H1, d]^T, so it
// runs on tcgen05.  K = d is split S ways: CTA (s, n, m) stages its K chunks of H rows [128 m, +128) and
// W1 units [64 n, +64) in shared memory with TMA (128-byte swizzle, zero fill past the tensor edges), one
// thread issues tcgen05.mma (bf16 x bf16, fp32 accumulators in 64 TMEM columns), the four warps read
// their 32 rows back with tcgen05.ld and store them as the split-K partial sums
//     part[s][b][u]  (fp32, s < S, b < B, u < H1p = H1 rounded up to 64; units >= H1 hold zeros).
// The step kernel that follows adds the S partials of its row in order, then b1, ReLU, w2 and b2: every
// sum has a fixed order, so the result is deterministic.  No cluster and no cross-CTA exchange here.
#include <cudaTypedefs.h>

#include <algorithm>

#include "common.cuh"
#include "mlp.cuh"

namespace switchsd {

constexpr int kMlpM = 128;             // rows (sequences) per tile: the MMA's M
constexpr int kMlpN = 64;              // hidden units per tile: the MMA's N
constexpr int kMlpKc = 64;             // K elements per staged chunk: one 128-byte swizzle row
constexpr int kMlpThreads = 128;       // four warps: one per 32 TMEM lanes
constexpr uint32_t kAChunk = kMlpM * kMlpKc * 2;    // 16 KB
constexpr uint32_t kBChunk = kMlpN * kMlpKc * 2;    // 8 KB
constexpr uint32_t kTmemCols = 64;
static_assert(kMaxMlpChunks * (kAChunk + kBChunk) + 1024 + 64 <= 227 * 1024,
              "operands, alignment slack and static shared memory must fit one CTA");
static_assert(kMlpThreads == kMlpM && kMlpN == 64, "one thread per tile row; 16 chunks of 16 bytes per row");

// Instruction descriptor of tcgen05.mma kind::f16: D fp32, A and B bf16, both K-major, M = 128, N = 64.
constexpr uint32_t kIdesc = (1u << 4) | (1u << 7) | (1u << 10) | (uint32_t(kMlpN >> 3) << 17) |
                            (uint32_t(kMlpM >> 4) << 24);

struct MlpArgs {
    float *part;   // [S][B][H1p]
    int32_t B, H1p, nchunks, prefetch;
    int32_t stages;  // operand stages: chunk c goes to stage c % stages, refilled once its MMAs are done
};

// Shared-memory matrix descriptor: K-major, 128-byte swizzle, 8-row groups 1024 bytes apart.
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr) {
    return uint64_t((saddr & 0x3FFFFu) >> 4) | (uint64_t(1) << 16) | (uint64_t(1024 >> 4) << 32) |
           (uint64_t(1) << 46) | (uint64_t(2) << 61);
}

__device__ __forceinline__ void tma_load_2d(void *dst, const CUtensorMap *map, int32_t x, int32_t y, uint64_t *bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];\n" ::"r"(
            smem_addr(dst)),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(smem_addr(bar))
        : "memory");
}

__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float *v) {
    uint32_t r[32];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
        "%15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];\n"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
          "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
          "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr));
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

__global__ void __launch_bounds__(kMlpThreads) mlp_tc_kernel(const __grid_constant__ CUtensorMap tm_h,
                                                             const __grid_constant__ CUtensorMap tm_w,
                                                             const MlpArgs a) {
    extern __shared__ uint8_t smem_raw[];
    __shared__ __align__(8) uint64_t full[kMaxMlpChunks], empty[kMaxMlpChunks], mma_bar;
    __shared__ uint32_t s_tmem;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int S = int(gridDim.x), ks = blockIdx.x;
    const int n_tile = blockIdx.y, m0 = blockIdx.z * kMlpM, n0 = n_tile * kMlpN;
    const int per = (a.nchunks + S - 1) / S;
    const int c0 = ks * per;
    const int nck = max(0, min(a.nchunks, c0 + per) - c0);
    const int st = a.stages;  // 1 .. kMaxMlpChunks
    // 1024-byte aligned operand stages (the swizzle atom): A chunks, then B chunks.
    uint8_t *base = smem_raw + ((1024u - (smem_addr(smem_raw) & 1023u)) & 1023u);
    uint8_t *opA = base;
    uint8_t *opB = base + size_t(st) * kAChunk;
    auto issue = [&](int c) {  // chunk c of this CTA's K slice into stage c % st
        const int sg = c % st;
        mbar_arrive_expect_tx(&full[sg], kAChunk + kBChunk);
        tma_load_2d(opA + size_t(sg) * kAChunk, &tm_h, (c0 + c) * kMlpKc, m0, &full[sg]);
        tma_load_2d(opB + size_t(sg) * kBChunk, &tm_w, (c0 + c) * kMlpKc, n0, &full[sg]);
    };
    const int first = min(nck, st);  // chunks issued up front

    if (tid == 0) {
        for (int i = 0; i < st; ++i) {
            mbar_init(&full[i], 1);
            mbar_init(&empty[i], 1);
        }
        mbar_init(&mma_bar, 1);
        fence_mbar_init();
        // With the probe prefetch bit the caller guarantees that the preceding kernel writes neither
        // the hidden states nor W1, so their copies may start before the grid-dependency wait.
        if (a.prefetch)
            for (int c = 0; c < first; ++c) issue(c);
    }
    // With the prefetch bit this kernel reads nothing the preceding kernel writes, and the step kernel it
    // releases reads before its own wait only what the caller's prefetch bits cover: both start at once.
    // That kernel's wait covers this whole grid, whose stores follow this grid's own wait below.
    if (a.prefetch) pdl_trigger();
    if (warp == 0) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;\n" ::"r"(smem_addr(&s_tmem)),
                     "r"(kTmemCols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;\n" ::: "memory");
    }
    if (!a.prefetch) {
        pdl_wait();  // the operands may come from the preceding kernel
        pdl_trigger();
        if (tid == 0)
            for (int c = 0; c < first; ++c) issue(c);
    }
    asm volatile("tcgen05.fence::before_thread_sync;\n" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;\n" ::: "memory");
    const uint32_t tmem = s_tmem;

    // One thread: wait for chunk c, issue its MMAs, commit them to the stage's empty barrier; a stage is
    // refilled (chunk c + st) once those MMAs have read it.  ok = every copy and commit arrived in time.
    bool ok = true;
    if (tid == 0) {
        int landed = 0, issued = first;
        for (int c = 0; c < nck; ++c) {
            const int sg = c % st;
            const uint32_t ph = uint32_t(c / st) & 1u;
            if (!mbar_wait(&full[sg], ph)) {
                ok = false;
                break;
            }
            landed = c + 1;
            asm volatile("tcgen05.fence::after_thread_sync;\n" ::: "memory");
            const uint64_t da = sw128_desc(smem_addr(opA + size_t(sg) * kAChunk));
            const uint64_t db = sw128_desc(smem_addr(opB + size_t(sg) * kBChunk));
#pragma unroll
            for (int j = 0; j < kMlpKc / 16; ++j) {
                const uint32_t acc = (c | j) != 0;
                // advance both descriptors by j * 32 bytes inside the swizzle row
                asm volatile(
                    "{\n"
                    ".reg .pred p;\n"
                    "setp.ne.b32 p, %4, 0;\n"
                    "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n"
                    "}\n" ::"r"(tmem),
                    "l"(da + uint64_t(2 * j)), "l"(db + uint64_t(2 * j)), "r"(kIdesc), "r"(acc)
                    : "memory");
            }
            if (c + st < nck) {
                asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n" ::"r"(
                                 smem_addr(&empty[sg]))
                             : "memory");
                if (!mbar_wait(&empty[sg], ph)) {
                    ok = false;
                    break;
                }
                issue(c + st);
                issued = c + st + 1;
            }
        }
        if (landed > 0) {
            // arrives once every MMA issued has completed (on the failure path too: they read the stages)
            asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n" ::"r"(
                             smem_addr(&mma_bar))
                         : "memory");
        } else {
            // nothing to accumulate, or the first copy did not land: release the waiters
            asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];\n" ::"r"(smem_addr(&mma_bar)) : "memory");
        }
        // copies issued but not waited for (a wait gave up): a second bounded wait before the stages go
        for (int c = landed; c < issued; ++c) (void)mbar_wait(&full[c % st], uint32_t(c / st) & 1u);
    }
    const bool mma_done = mbar_wait(&mma_bar, 0);
    asm volatile("tcgen05.fence::after_thread_sync;\n" ::: "memory");
    ok = __syncthreads_and(ok && mma_done);

    // Row tid of the tile: its 64 accumulators (zero when this CTA had no K chunk; NaN when a copy or
    // the MMAs did not complete in time, so the row's logit shows the failure).
    float v[kMlpN];
    if (nck > 0 && ok) {
        const uint32_t taddr = tmem + (uint32_t(warp * 32) << 16);
        tmem_ld32(taddr, v);
        tmem_ld32(taddr + 32, v + 32);
        asm volatile("tcgen05.wait::ld.sync.aligned;\n" ::: "memory");
    } else {
        const float fill = ok ? 0.f : __int_as_float(0x7fc00000);
#pragma unroll
        for (int i = 0; i < kMlpN; ++i) v[i] = fill;
    }
    // The tile goes out through shared memory (the operand stages are free: every MMA has completed), so
    // that each warp store writes two whole 256-byte rows instead of one 16-byte piece of 32 rows.  Row r
    // keeps its 16-byte chunk q at position q ^ (r % 16): both the row-wise writes below and the reads
    // across rows hit distinct banks.
    // The partial sums overwrite what an earlier step kernel may still read: with the prefetch bit the
    // copies and the MMAs above ran before the wait, the stores come after it.
    if (a.prefetch) pdl_wait();
    float4 *tile = reinterpret_cast<float4 *>(base);  // [kMlpM rows][16 chunks]
#pragma unroll
    for (int q = 0; q < kMlpN / 4; ++q)
        tile[tid * 16 + (q ^ (tid & 15))] = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
    asm volatile("tcgen05.fence::before_thread_sync;\n" ::: "memory");
    __syncthreads();
#pragma unroll 4
    for (int i = 0; i < 16; ++i) {  // warp w writes rows 32 w .. 32 w + 31, two per store
        const int r = warp * 32 + 2 * i + (lane >> 4), c = lane & 15;
        if (m0 + r < a.B)
            reinterpret_cast<float4 *>(a.part + (size_t(ks) * a.B + size_t(m0 + r)) * a.H1p + n0)[c] =
                tile[r * 16 + (c ^ (r & 15))];
    }
    if (warp == 0)
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;\n" ::"r"(tmem), "r"(kTmemCols) : "memory");
}

// ------------------------------------------------------------------------------------------------
// Host side.
// ------------------------------------------------------------------------------------------------
static PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    if (fn == nullptr) {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    }
    return fn;
}

// 2-D bf16 tensor map: rows of `d` elements, box = kMlpKc x box_rows, 128-byte swizzle, zero fill.
static bool encode_rows(CUtensorMap *map, const uint16_t *ptr, int rows, int d, int box_rows) {
    PFN_cuTensorMapEncodeTiled_v12000 fn = encode_fn();
    if (fn == nullptr) return false;
    const cuuint64_t dims[2] = {cuuint64_t(d), cuuint64_t(rows)};
    const cuuint64_t strides[1] = {cuuint64_t(d) * 2};
    const cuuint32_t box[2] = {cuuint32_t(kMlpKc), cuuint32_t(box_rows)};
    const cuuint32_t estr[2] = {1, 1};
    return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<uint16_t *>(ptr), dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int mlp_split(int d) {
    const int nchunks = (d + kMlpKc - 1) / kMlpKc;
    int s = 1;
    while (s < kMaxMlpSplit && s * 2 <= nchunks) s *= 2;
    return s;
}

bool mlp_shape_ok(int d, int H1) {
    const int nchunks = (d + kMlpKc - 1) / kMlpKc;
    const int s = mlp_split(d);
    return (nchunks + s - 1) / s <= kMaxMlpChunks && H1 >= 1 && H1 <= kMaxMlpHidden && d >= 8 && d % 8 == 0;
}

int mlp_hidden_padded(int H1) { return (H1 + kMlpN - 1) / kMlpN * kMlpN; }

cudaError_t launch_mlp_tc(const uint16_t *hidden, const uint16_t *W1, float *part, int B, int d, int H1,
                          bool prefetch, cudaStream_t stream, int stages) {
    CUtensorMap tm_h, tm_w;
    if (!encode_rows(&tm_h, hidden, B, d, kMlpM) || !encode_rows(&tm_w, W1, H1, d, kMlpN))
        return cudaErrorInvalidValue;
    const int nchunks = (d + kMlpKc - 1) / kMlpKc;
    const int S = mlp_split(d);
    const int per = (nchunks + S - 1) / S;
    const int st = stages >= 1 && stages < per ? stages : per;
    // the operand stages, which also hold the output tile (kMlpM x kMlpN fp32) once the MMAs are done
    const size_t smem = 1024 + std::max(size_t(st) * (kAChunk + kBChunk), size_t(kMlpM) * kMlpN * 4);
    static bool attr_done[64] = {false};
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev >= 0 && dev < 64 && !attr_done[dev]) {
        const cudaError_t e = cudaFuncSetAttribute(mlp_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                   int(1024 + size_t(kMaxMlpChunks) * (kAChunk + kBChunk)));
        if (e != cudaSuccess) return e;
        attr_done[dev] = true;
    }
    MlpArgs a;
    a.part = part;
    a.B = B;
    a.H1p = mlp_hidden_padded(H1);
    a.nchunks = nchunks;
    a.prefetch = prefetch ? 1 : 0;
    a.stages = st;
    const dim3 grid(unsigned(S), unsigned(a.H1p / kMlpN), unsigned((B + kMlpM - 1) / kMlpM));
    // An explicit one-CTA cluster: the copies and the MMA commit address shared::cluster.
    return launch_pdl(mlp_tc_kernel, grid, dim3(kMlpThreads), smem, stream, 1u, tm_h, tm_w, a);
}

}  // namespace switchsd
