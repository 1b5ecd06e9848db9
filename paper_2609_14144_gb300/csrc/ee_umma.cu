// Fifth-generation tensor-core projections of the multi-position layer pass
// (the prompt and the full-depth re-pass, ee_rows.cu) on sm_103a: tcgen05.mma
// with operands staged in shared memory by TMA and the fp32 accumulator in
// tensor memory.
//
// One projection of a batch of M <= 128 positions: Y[row][n] = sum_k W[n][k]
// x[row][k] for the n_rows x K tile-packed bf16 weights W.  Each activation
// is carried as three bf16 parts (x = high + middle + low, ee_rows.cu), and
// the three part arrays of a block of 64 positions are stacked as 192
// operand rows, so one MMA of shape M = 128 (weight rows) x N = 192 (3 parts
// x 64 positions) multiplies every part of a block at once, into one of two
// accumulators (one per block); bf16 products are exact in the fp32
// accumulator and the epilogue adds the three columns of each position.
//
// CTA (x, s): weight rows [128 x, 128 x + 128) (four 32-row tiles) over the
// K range of split s, 64 columns per pipeline stage:
//   - warp 0, lane 0 loads a stage: the 128 x 64 weight block with one TMA
//     tensor copy (a four-dimensional view of the tile-packed layout whose
//     box lands in shared memory in the UMMA canonical K-major layout with
//     no swizzle: 8-row x 16-byte core matrices, 128 bytes apart along the
//     rows, 2048 along K) and the two 192 x 64 activation blocks with one
//     bulk copy (the activation buffer is stored chunk-major, so a stage is
//     one contiguous 48 KB range in the same canonical layout: a block's
//     192 rows 3072 bytes long, the two blocks of a chunk side by side, 6144
//     bytes apart along K);
//   - warp 1, lane 0 issues four K = 16 MMAs per stage and row block (the
//     second block only when the batch has rows there) into the tensor-memory
//     accumulators and commits each stage back to its producer barrier;
//   - after the last stage all four warps read the accumulators (warp w holds
//     tensor-memory lanes 32 w .. 32 w + 31, the weight rows of tile w) and
//     write the split's partial sums part[s][row][n], which the consumer adds
//     in split order as with the warp-level path.
// Every wait is bounded; after a wait runs out the kernel flags kErrStall in
// the device error word, waits (bounded, whatever the word says) for its
// copies in flight and for the MMAs it issued, frees its tensor memory and
// returns.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <algorithm>
#include <mutex>

#include "ee_internal.h"

namespace ee {
namespace {

constexpr int kUThreads = 128;
constexpr int kUStages = 3;
constexpr int kUMRows = 128;                       // weight rows per CTA (UMMA M)
constexpr int kUBlocks = kRowsMax / kRowsHalf;     // row blocks of a batch, one accumulator each
constexpr int kUN = 3 * kRowsHalf;                 // operand rows of one block's activations (UMMA N)
constexpr int kUKStage = 64;                       // K columns per stage
constexpr int kUABytes = kUMRows * kUKStage * 2;   // 16 KB
constexpr int kUBBlock = kUN * 16;                 // one block's three parts of one 16-byte chunk: 3 KB
constexpr int kUBBytes = kUBlocks * kUN * kUKStage * 2;  // 48 KB
constexpr int kUStageBytes = kUABytes + kUBBytes;  // 64 KB
constexpr int kUAccCols = 256;                     // tensor-memory columns per accumulator (>= kUN)
constexpr int kUTmemCols = kUBlocks * kUAccCols;   // 512
constexpr long long kUWaitCycles = 4000000000ll;   // about 2 s

__device__ __forceinline__ uint32_t u_saddr(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ void u_mb_init(uint64_t* b, int n) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(u_saddr(b)), "r"(n) : "memory");
}
__device__ __forceinline__ bool u_mb_test(uint64_t* b, int parity) {
    uint32_t ok;
    asm volatile(
        "{ .reg .pred p; mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2; selp.u32 %0, 1, 0, p; }"
        : "=r"(ok)
        : "r"(u_saddr(b)), "r"(parity)
        : "memory");
    return ok != 0;
}
// Wait for the phase of parity `parity`; false after the bound, or (when
// `err` is given) once the error word carries kErrStall.
__device__ __forceinline__ bool u_mb_wait(uint64_t* b, int parity, const volatile int* err) {
    if (u_mb_test(b, parity)) return true;
    const long long t0 = clock64();
    for (unsigned it = 1;; ++it) {
        if (u_mb_test(b, parity)) return true;
        if ((it & 255) == 0) {
            if (clock64() - t0 > kUWaitCycles) return false;
            if (err && (*err & kErrStall)) return false;
        }
    }
}

// ---------------------------------------------------------------- tcgen05
// Shared-memory operand descriptor: start address, leading (K-direction) and
// stride (row-direction) byte offsets of the core matrices, no swizzle.
__device__ __forceinline__ uint64_t u_desc(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
    uint64_t d = 0;
    d |= (uint64_t)((saddr >> 4) & 0x3fffu);
    d |= (uint64_t)((lbo >> 4) & 0x3fffu) << 16;
    d |= (uint64_t)((sbo >> 4) & 0x3fffu) << 32;
    d |= (uint64_t)1 << 46;  // descriptor version of sm_100 and later
    return d;                // base offset 0, layout type 0 (no swizzle)
}
// Instruction descriptor of kind::f16: fp32 accumulator, bf16 A and B, both
// K-major, N = kUN, M = kUMRows.
constexpr uint32_t kUIdesc = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(kUN >> 3) << 17) |
                             ((uint32_t)(kUMRows >> 4) << 24);

__device__ __forceinline__ void u_mma(uint32_t tmem_d, uint64_t a, uint64_t b, uint32_t accumulate) {
    asm volatile(
        "{ .reg .pred p; setp.ne.u32 p, %4, 0; tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p; }" ::"r"(
            tmem_d),
        "l"(a), "l"(b), "r"(kUIdesc), "r"(accumulate)
        : "memory");
}
__device__ __forceinline__ void u_commit(uint64_t* bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(u_saddr(bar))
                 : "memory");
}
__device__ __forceinline__ void u_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void u_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }

// 16 consecutive fp32 columns of this thread's tensor-memory lane.
__device__ __forceinline__ void u_ld16(uint32_t taddr, float (&v)[16]) {
    uint32_t r[16];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr)
        : "memory");
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

// ---------------------------------------------------------------- copies
__device__ __forceinline__ void u_expect_tx(uint64_t* bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(u_saddr(bar)), "r"(bytes) : "memory");
}
// The 128 x 64 weight block at (tile t0, 16-byte column chunk c0) of the
// four-dimensional view {8 elements, 32 rows, tiles, chunks}.
__device__ __forceinline__ void u_tma_w(void* dst, const CUtensorMap* map, int t0, int c0, uint64_t* bar) {
    asm volatile(
        "cp.async.bulk.tensor.4d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4, %5}], "
        "[%6];" ::"r"(u_saddr(dst)),
        "l"(map), "r"(0), "r"(0), "r"(t0), "r"(c0), "r"(u_saddr(bar))
        : "memory");
}
__device__ __forceinline__ void u_bulk(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
    asm volatile("cp.async.bulk.shared::cta.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                     u_saddr(dst)),
                 "l"(src), "r"(bytes), "r"(u_saddr(bar))
                 : "memory");
}

__global__ void __launch_bounds__(kUThreads, 1)
    k_rows_umma(const __grid_constant__ CUtensorMap wmap, const uint16_t* __restrict__ x3, int n_tiles, int K, int M,
                int S, float* __restrict__ part, int Np, int* err) {
    extern __shared__ __align__(1024) uint8_t u_smem_raw[];
    uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(u_smem_raw) + 1023) & ~(uintptr_t)1023);
    uint64_t* full = reinterpret_cast<uint64_t*>(sm + kUStages * kUStageBytes);
    uint64_t* empty = full + kUStages;
    uint64_t* done = empty + kUStages;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(done + 1);
    const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int tile0 = blockIdx.x * 4, s = blockIdx.y;
    const int nk = (K + kUKStage - 1) / kUKStage;
    const int k0 = (int)((int64_t)nk * s / S), k1 = (int)((int64_t)nk * (s + 1) / S), ks = k1 - k0;
    volatile int* everr = err;

    if (threadIdx.x == 0) {
        for (int i = 0; i < kUStages; ++i) {
            u_mb_init(&full[i], 1);
            u_mb_init(&empty[i], 1);
        }
        u_mb_init(done, 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (w == 0) {  // tensor memory for the accumulator
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(u_saddr(tmem_slot)),
                     "r"(kUTmemCols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    u_fence_before();
    __syncthreads();
    u_fence_after();
    const uint32_t tmem = *tmem_slot;
    // The weights do not depend on the previous kernel: the first stages'
    // weight blocks are requested before the programmatic wait, so that
    // their HBM latency overlaps the previous kernel's tail.
    const int pre = ks < kUStages ? ks : kUStages;
    if (w == 0 && lane == 0)
        for (int i = 0; i < pre; ++i) {
            u_expect_tx(&full[i], kUStageBytes);
            u_tma_w(sm + i * kUStageBytes, &wmap, tile0, (k0 + i) * (kUKStage / 8), &full[i]);
        }
    // the set-up above overlaps the previous kernel (programmatic launch)
    asm volatile("griddepcontrol.wait;" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

    if (w == 0 && lane == 0) {
        // producer: stage i of this split, the ring reused once its MMAs are done
        int issued = 0;
        bool ok = true;
        for (int i = 0; i < ks && ok; ++i) {
            const int st = i % kUStages;
            if (i >= kUStages && !u_mb_wait(&empty[st], ((i / kUStages) - 1) & 1, everr)) {
                atomicOr(err, kErrStall);
                ok = false;
                break;
            }
            uint8_t* a = sm + st * kUStageBytes;
            const int kc = (k0 + i) * (kUKStage / 8);  // first 16-byte chunk of the stage
            if (i >= pre) {  // (the first stages' weights are in flight already)
                u_expect_tx(&full[st], kUStageBytes);
                u_tma_w(a, &wmap, tile0, kc, &full[st]);
            }
            u_bulk(a + kUABytes, x3 + (int64_t)kc * kUBlocks * kUN * 8, kUBBytes, &full[st]);
            ++issued;
        }
        // every issued copy lands before the CTA may leave
        for (int i = issued > kUStages ? issued - kUStages : 0; i < issued; ++i)
            u_mb_wait(&full[i % kUStages], (i / kUStages) & 1, nullptr);
    } else if (w == 1 && lane == 0) {
        // MMA issuer
        for (int i = 0; i < ks; ++i) {
            const int st = i % kUStages;
            if (!u_mb_wait(&full[st], (i / kUStages) & 1, everr)) {
                atomicOr(err, kErrStall);
                break;
            }
            u_fence_after();
            const uint32_t a = u_saddr(sm + st * kUStageBytes), b = a + kUABytes;
#pragma unroll
            for (int kk = 0; kk < kUKStage / 16; ++kk)
#pragma unroll
                for (int rb = 0; rb < kUBlocks; ++rb)
                    if (rb * kRowsHalf < M)
                        u_mma(tmem + rb * kUAccCols, u_desc(a + kk * 2 * 2048, 2048, 128),
                              u_desc(b + rb * kUBBlock + kk * 2 * kUBlocks * kUBBlock, kUBlocks * kUBBlock, 128),
                              (i > 0 || kk > 0) ? 1u : 0u);
            u_commit(&empty[st]);
        }
        u_commit(done);  // after every MMA this thread issued
    }
    __syncwarp();
    // epilogue: every thread is one weight row (tensor-memory lane)
    bool have = u_mb_wait(done, 0, nullptr);  // the MMA thread commits done after every wait of its own
    if (!have) have = u_mb_wait(done, 0, nullptr);
    u_fence_after();
    // the tensor-memory loads are warp-wide: the whole warp reads or none of it
    if (__all_sync(0xffffffffu, have && ks > 0 && !(*everr & kErrStall))) {
        const int n = (tile0 + w) * 32 + lane;  // output row of the projection
        const uint32_t lane_addr = tmem + ((uint32_t)(32 * w) << 16);
        float* ps = part + (int64_t)s * M * Np;
        for (int c0 = 0; c0 < M; c0 += 16) {
            const uint32_t acc = lane_addr + (c0 / kRowsHalf) * kUAccCols + c0 % kRowsHalf;  // row block's accumulator
            float hi[16], md[16], lo[16];
            u_ld16(acc, hi);
            u_ld16(acc + kRowsHalf, md);
            u_ld16(acc + 2 * kRowsHalf, lo);
            if (tile0 + w < n_tiles)
#pragma unroll
                for (int i = 0; i < 16; ++i)
                    if (c0 + i < M) ps[(int64_t)(c0 + i) * Np + n] = (hi[i] + md[i]) + lo[i];
        }
    }
    u_fence_before();
    __syncthreads();
    if (w == 0) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kUTmemCols) : "memory");
}

// ---------------------------------------------------------------- host side
PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
std::once_flag g_encode_once;

bool encode_fn() {
    std::call_once(g_encode_once, [] {
        void* fn = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
        cudaGetLastError();
    });
    return g_encode != nullptr;
}

// The tile-packed weights as {8 elements, 32 rows, tiles, 16-byte chunks}
// with byte strides {-, 16, 64 K, 512}; a box of {8, 32, 4, kUKStage / 8} lands as
// row * 16 + chunk * 2048 bytes (row = 32 tile + row within the tile).
bool weight_map(CUtensorMap* map, const uint16_t* W, int64_t n_tiles, int K) {
    if (!encode_fn() || K % 8 || ((uintptr_t)W & 15)) return false;
    const cuuint64_t dim[4] = {8, 32, (cuuint64_t)n_tiles, (cuuint64_t)(K / 8)};
    const cuuint64_t stride[3] = {16, (cuuint64_t)K * 64, 512};
    const cuuint32_t box[4] = {8, 32, 4, kUKStage / 8};
    const cuuint32_t estr[4] = {1, 1, 1, 1};
    return g_encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<uint16_t*>(W), dim, stride, box, estr,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

size_t umma_smem() { return (size_t)kUStages * kUStageBytes + 256 + 1024; }

}  // namespace

bool umma_available() {
    static int ok = -1;
    if (ok < 0) {
        int dev = 0, major = 0, minor = 0;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
        cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
        CUtensorMap probe;
        static uint16_t dummy[64 * 8] __attribute__((aligned(16)));
        ok = major == 10 && encode_fn() && weight_map(&probe, dummy, 4, 64) &&
             cudaFuncSetAttribute(k_rows_umma, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)umma_smem()) ==
                 cudaSuccess;
        cudaGetLastError();
    }
    return ok == 1;
}

// K splits: as many as keep the grid within one wave (one CTA per SM: the
// stages take most of the shared memory), at most one per stage.
int umma_splits(int64_t n_tiles, int K, int n_sm) {
    const int64_t mt = (n_tiles + 3) / 4;
    const int nk = (K + kUKStage - 1) / kUKStage;
    const int64_t want = n_sm / mt;
    return (int)std::max<int64_t>(1, std::min<int64_t>(want, nk));
}

cudaError_t launch_mm_umma(const uint16_t* W, int64_t n_rows, int K, const uint16_t* x3, int M, int S, float* part,
                           int Np, int* err, cudaStream_t s) {
    const int64_t nt = tile_count(n_rows);
    CUtensorMap map;
    if (!weight_map(&map, W, nt, K)) return cudaErrorNotSupported;
    const dim3 grid((unsigned)((nt + 3) / 4), (unsigned)S);
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = grid;
    cfg.blockDim = dim3(kUThreads);
    cfg.dynamicSmemBytes = umma_smem();
    cfg.stream = s;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, k_rows_umma, map, x3, (int)nt, K, M, S, part, Np, err);
}

}  // namespace ee
