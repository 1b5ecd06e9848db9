// Fifth-generation tensor-core projections of the multi-position layer pass
// (the prompt and the full-depth re-pass, ee_rows.cu) on sm_103a: tcgen05.mma
// with operands staged in shared memory by TMA and the fp32 accumulator in
// tensor memory.
//
// One projection of a batch of M <= 256 positions: Y[row][n] = sum_k W[n][k]
// x[row][k] for the n_rows x K tile-packed bf16 weights W.  Each activation
// is carried as three bf16 parts (x = high + middle + low, ee_rows.cu), each
// part of the batch stored as N operand rows; every K = 16 step issues
// three MMAs of shape M = 128 (weight rows) x N (the batch's rows rounded up
// to 16), one per part, into two fp32 accumulators whose column is the batch
// row: the high parts' products into the first, the middle and low parts'
// (2^-8 of the size and less) into the second, so that their small terms are
// not added into the large sum step by step; the epilogue adds the two.  The
// bf16 products are exact.
//
// CTA (x, s): weight rows [128 x, 128 x + 128) (four 32-row tiles) over the
// K range of split s, 32 columns per pipeline stage, four stages in flight:
//   - warp 0, lane 0 loads a stage: the 128 x 32 weight block with one TMA
//     tensor copy (a three-dimensional view of the tile-packed layout whose
//     box lands in shared memory in the UMMA canonical K-major layout with
//     no swizzle: 8-row x 16-byte core matrices, 128 bytes apart along the
//     rows, 2048 along K) and the batch's activations with bulk copies (the
//     activation buffer is stored chunk-major with a row stride of N, so a
//     stage is one contiguous range in the same canonical layout: a part's N
//     rows N x 16 bytes long, the three parts of a chunk side by side, chunks
//     3 N x 16 bytes apart along K; 48 KB for a full batch);
//   - warp 1, lane 0 issues six MMAs per stage into the tensor-memory
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
constexpr int kUStages = 4;
constexpr int kUMRows = 128;                        // weight rows per CTA (UMMA M)
constexpr int kUKStage = 32;                        // K columns per stage
constexpr int kUABytes = kUMRows * kUKStage * 2;    // 8 KB
constexpr int kUBBytes = kUKStage / 8 * 3 * kRowsMax * 16;  // a full batch's activations: 48 KB
constexpr int kUStageBytes = kUABytes + kUBBytes;   // 56 KB
constexpr int kUTmemCols = 2 * kRowsMax;            // two accumulators of one fp32 column per position
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
// K-major, M = kUMRows, N = n (a multiple of 16, 16 <= n <= 256).
__device__ __forceinline__ uint32_t u_idesc(int n) {
    return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(n >> 3) << 17) | ((uint32_t)(kUMRows >> 4) << 24);
}

__device__ __forceinline__ void u_mma(uint32_t tmem_d, uint64_t a, uint64_t b, uint32_t idesc, uint32_t accumulate) {
    asm volatile(
        "{ .reg .pred p; setp.ne.u32 p, %4, 0; tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p; }" ::"r"(
            tmem_d),
        "l"(a), "l"(b), "r"(idesc), "r"(accumulate)
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
// three-dimensional view {256 elements (one chunk of a 32-row tile), tiles,
// chunks}.
__device__ __forceinline__ void u_tma_w(void* dst, const CUtensorMap* map, int t0, int c0, uint64_t* bar) {
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4}], "
        "[%5];" ::"r"(u_saddr(dst)),
        "l"(map), "r"(0), "r"(t0), "r"(c0), "r"(u_saddr(bar))
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
    // operand rows of the batch (UMMA N): M rounded up to 16; the rows past M
    // give accumulator columns that are never read
    // (the activation parts are stored with this row stride, x3_rows(M))
    const int N = x3_rows(M);
    const int part_bytes = N * 16;  // one part of one 16-byte chunk
    const uint32_t act_bytes = (uint32_t)(kUKStage / 8 * 3 * part_bytes);
    const uint32_t stage_tx = (uint32_t)kUABytes + act_bytes;
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
            u_expect_tx(&full[i], stage_tx);
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
                u_expect_tx(&full[st], stage_tx);
                u_tma_w(a, &wmap, tile0, kc, &full[st]);
            }
            // the stage's activations: one contiguous range
            u_bulk(a + kUABytes, x3 + (int64_t)kc * 3 * N * 8, act_bytes, &full[st]);
            ++issued;
        }
        // every issued copy lands before the CTA may leave
        for (int i = issued > kUStages ? issued - kUStages : 0; i < issued; ++i)
            u_mb_wait(&full[i % kUStages], (i / kUStages) & 1, nullptr);
    } else if (w == 1 && lane == 0) {
        // MMA issuer
        const uint32_t idesc = u_idesc(N);
        for (int i = 0; i < ks; ++i) {
            const int st = i % kUStages;
            if (!u_mb_wait(&full[st], (i / kUStages) & 1, everr)) {
                atomicOr(err, kErrStall);
                break;
            }
            u_fence_after();
            const uint32_t a = u_saddr(sm + st * kUStageBytes), b = a + kUABytes;
            // each K = 16 step: the weights times the high parts of the batch
            // into the first accumulator, times the middle and the low parts
            // into the second
#pragma unroll
            for (int kk = 0; kk < kUKStage / 16; ++kk)
#pragma unroll
                for (int pp = 0; pp < 3; ++pp)
                    u_mma(tmem + (pp ? kRowsMax : 0), u_desc(a + kk * 2 * 2048, 2048, 128),
                          u_desc(b + (kk * 2 * 3 + pp) * part_bytes, 3 * part_bytes, 128), idesc,
                          (i > 0 || kk > 0 || pp == 2) ? 1u : 0u);
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
        for (int c0 = 0; c0 < M; c0 += 16) {  // accumulator column = batch row
            float hi[16], ml[16];
            u_ld16(lane_addr + c0, hi);
            u_ld16(lane_addr + kRowsMax + c0, ml);
            if (tile0 + w < n_tiles)
#pragma unroll
                for (int i = 0; i < 16; ++i)
                    if (c0 + i < M) ps[(int64_t)(c0 + i) * Np + n] = hi[i] + ml[i];
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

// The tile-packed weights as {256 elements, tiles, 16-byte chunks} with byte
// strides {-, 64 K, 512}: the 32 rows of one tile's chunk are 512 contiguous
// bytes.  A box of {256, 4, kUKStage / 8} lands as row * 16 + chunk * 2048
// bytes (row = 32 tile + row within the tile), the canonical layout, in 512-byte
// rows of the copy.
bool weight_map(CUtensorMap* map, const uint16_t* W, int64_t n_tiles, int K) {
    if (!encode_fn() || K % 8 || ((uintptr_t)W & 15)) return false;
    const cuuint64_t dim[3] = {256, (cuuint64_t)n_tiles, (cuuint64_t)(K / 8)};
    const cuuint64_t stride[2] = {(cuuint64_t)K * 64, 512};
    const cuuint32_t box[3] = {256, 4, kUKStage / 8};
    const cuuint32_t estr[3] = {1, 1, 1};
    return g_encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<uint16_t*>(W), dim, stride, box, estr,
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
