// mlp.cu -- the two-layer copy-intent probe z = w2 . ReLU(W1 h + b1) + b2 on the tensor cores.
//
// The paper's probe is linear (Eq. 3); this two-layer form is an extension used with probe_kind
// SWITCHSD_PROBE_MLP.  Its first layer is a real contraction, Z1[B, H1] = H[B, d] . W1[H1, d]^T, so it
// runs on tcgen05: each thread-block cluster of S CTAs owns one 128-row x 64-unit tile of Z1 and
// splits K = d between its CTAs.  A CTA stages its K chunks of H and W1 in shared memory with TMA
// (128-byte swizzle, zero fill past the tensor edges), one thread issues tcgen05.mma (bf16 x bf16,
// fp32 accumulators in 64 TMEM columns), and the four warps read their 32 rows back with tcgen05.ld.
// After a cluster barrier (every CTA's MMAs complete) the S partial tiles are reduce-scattered across
// the cluster with st.async into the freed operand areas (CTA r owns 64/S columns); the owner adds
// b1, applies ReLU, weights by w2 and sums its columns; the leader adds the S owners' sums in a fixed
// order and writes the tile's partial logit zpart[n_tile][b] to the caller's workspace.  The step kernel adds the n_tile partials (fixed order) and b2.  Deterministic: every sum
// has a fixed order.
#include <cudaTypedefs.h>

#include "common.cuh"
#include "mlp.cuh"

namespace switchsd {

constexpr int kMlpM = 128;             // rows (sequences) per tile: the MMA's M
constexpr int kMlpN = 64;              // hidden units per tile: the MMA's N
constexpr int kMlpKc = 64;             // K elements per staged chunk: one 128-byte swizzle row
constexpr int kMlpThreads = 128;       // four warps: one per 32 TMEM lanes
constexpr uint32_t kAChunk = kMlpM * kMlpKc * 2;    // 16 KB
constexpr uint32_t kBChunk = kMlpN * kMlpKc * 2;    // 8 KB
constexpr uint32_t kRecvBytes = kMlpM * kMlpN * 4;  // 32 KB: the columns a CTA owns, from every CTA
constexpr uint32_t kTmemCols = 64;
static_assert(kMaxMlpChunks * (kAChunk + kBChunk) + 1024 + 16 * 128 * 4 + 64 <= 227 * 1024,
              "operands, alignment slack and static shared memory must fit one CTA");

// Instruction descriptor of tcgen05.mma kind::f16: D fp32, A and B bf16, both K-major, M = 128, N = 64.
constexpr uint32_t kIdesc = (1u << 4) | (1u << 7) | (1u << 10) | (uint32_t(kMlpN >> 3) << 17) |
                            (uint32_t(kMlpM >> 4) << 24);

struct MlpArgs {
    const float *b1;
    const uint16_t *w2;
    float *zpart;  // [NT][B]
    int32_t B, d, H1, nchunks;
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

__device__ __forceinline__ void st_async_f32(uint32_t cluster_addr, float v, uint32_t cluster_mbar) {
    asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.b32 [%0], %1, [%2];\n" ::"r"(cluster_addr),
                 "r"(__float_as_uint(v)), "r"(cluster_mbar)
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
    __shared__ __align__(8) uint64_t tma_bar, mma_bar, red_bar, fin_bar;
    __shared__ uint32_t s_tmem;
    __shared__ float s_fin[kMaxMlpSplit][kMlpM];  // leader: every owner's per-row sum

    const int tid = threadIdx.x, warp = tid >> 5;
    const uint32_t rank = cluster_ctarank();
    const uint32_t S = cluster_nctarank();
    const int n_tile = blockIdx.y, m0 = blockIdx.z * kMlpM, n0 = n_tile * kMlpN;
    const int W = kMlpN / int(S);  // columns owned by each CTA
    const int per = (a.nchunks + int(S) - 1) / int(S);
    const int c0 = int(rank) * per;
    const int nck = max(0, min(a.nchunks, c0 + per) - c0);
    // 1024-byte aligned operand area (the swizzle atom): A chunks, then B chunks.
    uint8_t *base = smem_raw + ((1024u - (smem_addr(smem_raw) & 1023u)) & 1023u);
    uint8_t *opA = base;
    uint8_t *opB = base + size_t(per) * kAChunk;
    // The reduce-scatter lands on the operand area: it is written only after every CTA of the cluster
    // has finished its MMAs (cluster barrier below).
    float *recv = reinterpret_cast<float *>(base);  // [S][128][W]

    if (tid == 0) {
        mbar_init(&tma_bar, 1);
        mbar_init(&mma_bar, 1);
        mbar_init(&red_bar, 1);
        mbar_arrive_expect_tx(&red_bar, kRecvBytes);
        if (rank == 0) {
            mbar_init(&fin_bar, 1);
            mbar_arrive_expect_tx(&fin_bar, S * kMlpM * 4u);
        }
        fence_mbar_init();
    }
    if (warp == 0) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;\n" ::"r"(smem_addr(&s_tmem)),
                     "r"(kTmemCols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;\n" ::: "memory");
    }
    pdl_wait();
    pdl_trigger();

    if (tid == 0 && nck > 0) {
        mbar_arrive_expect_tx(&tma_bar, uint32_t(nck) * (kAChunk + kBChunk));
        for (int c = 0; c < nck; ++c) {
            tma_load_2d(opA + size_t(c) * kAChunk, &tm_h, (c0 + c) * kMlpKc, m0, &tma_bar);
            tma_load_2d(opB + size_t(c) * kBChunk, &tm_w, (c0 + c) * kMlpKc, n0, &tma_bar);
        }
    }
    asm volatile("tcgen05.fence::before_thread_sync;\n" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;\n" ::: "memory");
    const uint32_t tmem = s_tmem;

    bool ok = true;
    if (tid == 0) {
        if (nck > 0 && mbar_wait(&tma_bar, 0)) {
            for (int c = 0; c < nck; ++c) {
                const uint64_t da = sw128_desc(smem_addr(opA + size_t(c) * kAChunk));
                const uint64_t db = sw128_desc(smem_addr(opB + size_t(c) * kBChunk));
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
            }
            asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n" ::"r"(
                             smem_addr(&mma_bar))
                         : "memory");
        } else {
            // nothing to accumulate, or the copies did not land: release the waiters, flag the tile
            if (nck > 0) ok = false;
            asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];\n" ::"r"(smem_addr(&mma_bar)) : "memory");
        }
    }
    const bool mma_done = mbar_wait(&mma_bar, 0);
    asm volatile("tcgen05.fence::after_thread_sync;\n" ::: "memory");
    ok = __syncthreads_and(ok && mma_done);

    // Row tid of the tile: its 64 accumulators (zero when this CTA had no K chunk).
    float v[kMlpN];
    if (nck > 0 && ok) {
        const uint32_t taddr = tmem + (uint32_t(warp * 32) << 16);
        tmem_ld32(taddr, v);
        tmem_ld32(taddr + 32, v + 32);
        asm volatile("tcgen05.wait::ld.sync.aligned;\n" ::: "memory");
    } else {
#pragma unroll
        for (int i = 0; i < kMlpN; ++i) v[i] = 0.f;
    }

    // Once every CTA has arrived, all MMAs of the cluster are complete (operand areas free) and every
    // barrier is initialised: the reduce-scatter may start.
    cluster_arrive_release();
    cluster_wait_acquire();
    // Reduce-scatter: columns [o W, (o+1) W) go to CTA o, into its recv[rank][tid][0..W).
    for (int o = 0; o < int(S); ++o) {
        const uint32_t mb = map_to_rank(&red_bar, uint32_t(o));
        for (int q = 0; q < W; q += 4) {
            const int col = o * W + q;
            uint4 u;
            u.x = __float_as_uint(v[col]);
            u.y = __float_as_uint(v[col + 1]);
            u.z = __float_as_uint(v[col + 2]);
            u.w = __float_as_uint(v[col + 3]);
            st_async_v4(map_to_rank(&recv[(size_t(rank) * kMlpM + tid) * W + q], uint32_t(o)), u, mb);
        }
    }
    // Owner: add the S partials in order, then b1, ReLU and w2 over the owned columns.
    const bool got = mbar_wait(&red_bar, 0);
    float zt = 0.f;
    for (int c = 0; c < W; ++c) {
        float sum = 0.f;
        for (uint32_t src = 0; src < S; ++src) sum += recv[(size_t(src) * kMlpM + tid) * W + c];
        const int u = n0 + int(rank) * W + c;
        if (u < a.H1) {
            const float pre = sum + (a.b1 ? a.b1[u] : 0.f);
            zt = fmaf(bf16_lo(uint32_t(a.w2[u])), fmaxf(pre, 0.f), zt);
        }
    }
    if (!(got && ok)) zt = __int_as_float(0x7fc00000);  // NaN marks a tile that did not complete
    st_async_f32(map_to_rank(&s_fin[rank][tid], 0), zt, map_to_rank(&fin_bar, 0));
    if (rank == 0) {
        const bool all_in = mbar_wait(&fin_bar, 0);
        float z = 0.f;
        for (uint32_t src = 0; src < S; ++src) z += s_fin[src][tid];
        if (!all_in) z = __int_as_float(0x7fc00000);
        if (m0 + tid < a.B) a.zpart[size_t(n_tile) * a.B + m0 + tid] = z;
    }
    asm volatile("tcgen05.fence::before_thread_sync;\n" ::: "memory");
    __syncthreads();
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

int mlp_tiles_n(int H1) { return (H1 + kMlpN - 1) / kMlpN; }

cudaError_t launch_mlp_tc(const uint16_t *hidden, const uint16_t *W1, const uint16_t *w2, const float *b1, float *zpart,
                          int B, int d, int H1, cudaStream_t stream) {
    CUtensorMap tm_h, tm_w;
    if (!encode_rows(&tm_h, hidden, B, d, kMlpM) || !encode_rows(&tm_w, W1, H1, d, kMlpN))
        return cudaErrorInvalidValue;
    const int nchunks = (d + kMlpKc - 1) / kMlpKc;
    const int S = mlp_split(d);
    const int per = (nchunks + S - 1) / S;
    const size_t ops = size_t(per) * (kAChunk + kBChunk);
    const size_t smem = 1024 + (ops > kRecvBytes ? ops : size_t(kRecvBytes));
    static bool attr_done[64] = {false};
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev >= 0 && dev < 64 && !attr_done[dev]) {
        cudaError_t e = cudaFuncSetAttribute(mlp_tc_kernel, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
        if (e != cudaSuccess) return e;
        e = cudaFuncSetAttribute(mlp_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 int(1024 + size_t(kMaxMlpChunks) * (kAChunk + kBChunk)));
        if (e != cudaSuccess) return e;
        attr_done[dev] = true;
    }
    MlpArgs a;
    a.b1 = b1;
    a.w2 = w2;
    a.zpart = zpart;
    a.B = B;
    a.d = d;
    a.H1 = H1;
    a.nchunks = nchunks;
    const dim3 grid(unsigned(S), unsigned(mlp_tiles_n(H1)), unsigned((B + kMlpM - 1) / kMlpM));
    return launch_pdl(mlp_tc_kernel, grid, dim3(kMlpThreads), smem, stream, unsigned(S), tm_h, tm_w, a);
}

}  // namespace switchsd
