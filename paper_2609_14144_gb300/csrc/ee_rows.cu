// Multi-position layer pass for sm_103a: the prompt (Section 2's prefill,
// full depth with no gate) and Section 11's full-depth re-pass of exited
// positions run each layer over a batch of up to kRowsMax positions, so a
// weight byte is read once per batch instead of once per position.
//
// A layer is ten launches, each reading what the previous one wrote:
//   k_rows_add_norm  residual add of the previous projection's split
//                    partials (in a fixed order), then RMSNorm with the next
//                    gain, written as three bf16 parts
//   k_rows_umma / k_rows_mm   a projection: Y[row][n] = sum_k W[n][k] x[row][k]
//   k_rows_qkv       split sum, bias, RoPE at each row's position; q kept in
//                    fp32, k and v stored bf16 into the paged cache
//   k_rows_fattn     causal attention of every row over the cache up to its
//                    position on the tensor cores, keys split over CTAs
//                    (rows of the batch at earlier positions were written by
//                    k_rows_qkv of this layer); k_rows_amerge combines the
//                    splits
//   the O projection, k_rows_add_norm (mid residual, MLP norm), the gate/up
//   projection, k_rows_swiglu, the down projection
//
// Projections run on the tcgen05 tensor cores by default (k_rows_umma,
// ee_umma.cu).  The warp-level build here (EE_OPT_ROWS = 2) uses the legacy
// mma (m16n8k16, bf16 operands, fp32 accumulation).  A warp owns one (32-row weight tile, K
// range) unit: the tiled weight layout gives each lane the 16-byte chunk of
// one row, and the order of k inside one mma is free as long as both
// operands agree, so a lane's chunk feeds its A fragment as loaded (slots
// 2q, 2q+1, 2q+8, 2q+9 of the lane's k group q take the chunk's first four
// elements, the second mma the last four) and the activations are read in the
// same order.  Activations keep fp32 precision: each is split into three
// bf16 parts, x = high + middle + low (each the rounding of what the parts
// before it leave, 24 significant bits in all), and the weights are
// multiplied with each; bf16 products are exact in the fp32 accumulator.  Weights are the
// A operand (16 output rows per mma), positions the B operand (8 per mma).
//
// Partial sums of the K splits go to a scratch buffer and the consumer adds
// them in split order, so results do not depend on scheduling.

#include <cuda_bf16.h>
#include <math.h>
#include <stdint.h>

#include <algorithm>

#include "ee_internal.h"

namespace ee {
namespace {

constexpr int kRowsThreads = 256;
constexpr int kRowsWarps = kRowsThreads / 32;

__device__ __forceinline__ float r_bf2f(uint16_t b) { return __uint_as_float((uint32_t)b << 16); }
__device__ __forceinline__ uint16_t r_f2bf(float f) { return __bfloat16_as_ushort(__float2bfloat16_rn(f)); }

// A product's input as three bf16 parts, stored chunk-major: for each
// 16-byte column chunk (8 columns), the high parts of the batch's rows, then
// the middle parts, then the low parts, 16 bytes per row and `rows` rows a
// part (the batch's row count rounded up to 16).  One part of a chunk is then
// the tensor cores' operand of N = rows rows in their canonical layout
// (ee_umma.cu), a few chunks one contiguous stage whatever the batch size,
// and a warp-level product reads a row's chunk of one part as 16 contiguous
// bytes.
struct Parts {
    uint16_t* p;
    int rows;
};
__device__ __forceinline__ int64_t x3_index(int part, int row, int col, int rows) {
    return (((int64_t)(col >> 3) * 3 + part) * rows + row) * 8 + (col & 7);
}

// The three bf16 parts of x at (row, col): high = bf16(x), middle = bf16(x -
// high), low = bf16(x - high - middle) (each difference exact in fp32).
__device__ __forceinline__ void split_store(float x, const Parts& p, int row, int col) {
    const uint16_t h = r_f2bf(x);
    const float r1 = x - r_bf2f(h);
    const uint16_t md = r_f2bf(r1);
    p.p[x3_index(0, row, col, p.rows)] = h;
    p.p[x3_index(1, row, col, p.rows)] = md;
    p.p[x3_index(2, row, col, p.rows)] = r_f2bf(r1 - r_bf2f(md));
}
// Columns from n up to the next multiple of 64 (a tensor-core stage) read as 0.
__host__ __device__ __forceinline__ int pad64(int n) { return (n + 63) & ~63; }

// Weights are read once per batch: streamed past L1, first out of L2.
__device__ __forceinline__ uint4 ld_weights(const uint4* p) {
    uint64_t pol;
    asm("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
    uint4 r;
    asm volatile("ld.global.nc.L1::no_allocate.L2::cache_hint.v4.u32 {%0,%1,%2,%3}, [%4], %5;"
                 : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
                 : "l"(p), "l"(pol));
    return r;
}
__device__ __forceinline__ uint4 ld_act(const uint16_t* p) { return __ldg(reinterpret_cast<const uint4*>(p)); }

__device__ __forceinline__ void mma_16816(float (&c)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                          uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
        "{%0,%1,%2,%3};"
        : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

__device__ __forceinline__ float r_warp_sum(float v) {
#pragma unroll
    for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// Programmatic dependent launch: every kernel of the pass waits for its
// predecessor's results first, then lets its successor launch, so that a
// launch's setup overlaps the kernel before it.
__device__ __forceinline__ void r_pdl() {
    asm volatile("griddepcontrol.wait;" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

__device__ __forceinline__ int64_t slot_offset(const DevModel& m, int j, int pos) {
    const int page = m.page_table[pos / m.page_size];
    const int slot = pos - (pos / m.page_size) * m.page_size;
    return (int64_t)j * m.kv_layer_stride + ((int64_t)page * m.KH * m.page_size + slot) * m.D;
}

// ------------------------------------------------------------------ projection
//
// part[s][row][n] = sum over the k of split s of W[n][k] x[row][k], for the
// M rows of x (three bf16 parts, chunk-major) and every output n of
// the tiled weights.  A unit is (tile, split, row group): NB blocks of 8 rows
// starting at row group * 8 NB (rows past M read as zero and are not
// stored); the row groups of one (tile, split) are neighbouring warps, so a
// weight chunk read for one is an L2 hit for the others.  K splits cover
// whole 32-column steps, U steps loaded before any is multiplied; a chunk
// past K reads as zero on both sides.
template <int NB, int U>
__global__ void __launch_bounds__(kRowsThreads) k_rows_mm(const uint4* __restrict__ W, int n_tiles, int K,
                                                          const Parts x3, int ldx, int M, int S,
                                                          int RG, float* __restrict__ part, int Np) {
    r_pdl();
    const int lane = threadIdx.x & 31, g = lane >> 2, q = lane & 3;
    const int Rc = K >> 3;             // 16-byte chunks per weight row
    const int nsteps = (Rc + 3) >> 2;  // 32-column steps
    const int units = n_tiles * S * RG;
    const int nw = gridDim.x * kRowsWarps;
    for (int u = blockIdx.x * kRowsWarps + (threadIdx.x >> 5); u < units; u += nw) {
        const int ts = u / RG, rg = u - ts * RG;
        const int tile = ts / S, s = ts - tile * S;
        const int r0 = rg * 8 * NB;
        const int st0 = (int)((int64_t)nsteps * s / S), st1 = (int)((int64_t)nsteps * (s + 1) / S);
        const uint4* wt = W + (int64_t)tile * Rc * 32;
        // the high parts' products and the middle and low parts' products in
        // separate accumulators (small terms added into a large running sum
        // lose their low bits), added at the end
        float acc[2][NB][4], acm[2][NB][4];
#pragma unroll
        for (int a = 0; a < 2; ++a)
#pragma unroll
            for (int n = 0; n < NB; ++n)
#pragma unroll
                for (int e = 0; e < 4; ++e) acc[a][n][e] = acm[a][n][e] = 0.f;
        for (int st = st0; st < st1; st += U) {
            uint4 w[U][4], bh[U][NB], bm[U][NB], bl[U][NB];
#pragma unroll
            for (int v = 0; v < U; ++v) {
                const int ch = (st + v) * 4 + q;  // this lane's chunk of the step
                const bool ok = st + v < st1 && ch < Rc;
#pragma unroll
                for (int r = 0; r < 4; ++r)  // rows g, g+8, g+16, g+24 of the tile
                    w[v][r] = ok ? ld_weights(wt + (int64_t)ch * 32 + g + 8 * r) : make_uint4(0u, 0u, 0u, 0u);
#pragma unroll
                for (int n = 0; n < NB; ++n) {
                    const int row = r0 + n * 8 + g;
                    const bool okx = ok && row < M;
                    const uint16_t* at = x3.p + x3_index(0, okx ? row : 0, ch * 8, x3.rows);
                    bh[v][n] = okx ? ld_act(at) : make_uint4(0u, 0u, 0u, 0u);
                    bm[v][n] = okx ? ld_act(at + x3.rows * 8) : make_uint4(0u, 0u, 0u, 0u);
                    bl[v][n] = okx ? ld_act(at + 2 * x3.rows * 8) : make_uint4(0u, 0u, 0u, 0u);
                }
            }
#pragma unroll
            for (int v = 0; v < U; ++v) {
                const uint4* x = w[v];
#pragma unroll
                for (int n = 0; n < NB; ++n) {
                    const uint4 parts[3] = {bh[v][n], bm[v][n], bl[v][n]};
#pragma unroll
                    for (int pp = 0; pp < 3; ++pp) {
                        const uint4 b = parts[pp];
                        float(&c0)[4] = pp ? acm[0][n] : acc[0][n];
                        float(&c1)[4] = pp ? acm[1][n] : acc[1][n];
                        // first mma of the step: chunk elements 0..3; second: 4..7
                        mma_16816(c0, x[0].x, x[1].x, x[0].y, x[1].y, b.x, b.y);
                        mma_16816(c0, x[0].z, x[1].z, x[0].w, x[1].w, b.z, b.w);
                        mma_16816(c1, x[2].x, x[3].x, x[2].y, x[3].y, b.x, b.y);
                        mma_16816(c1, x[2].z, x[3].z, x[2].w, x[3].w, b.z, b.w);
                    }
                }
            }
        }
        // accumulator e of block (a, n): output row tile*32 + a*16 + g (+8 for
        // e >= 2), batch row r0 + n*8 + 2q (+1 for odd e)
        float* ps = part + (int64_t)s * M * Np;
#pragma unroll
        for (int a = 0; a < 2; ++a)
#pragma unroll
            for (int n = 0; n < NB; ++n)
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const int row = r0 + n * 8 + 2 * q + (e & 1);
                    const int out = tile * 32 + a * 16 + g + (e >> 1) * 8;
                    if (row < M) ps[(int64_t)row * Np + out] = acc[a][n][e] + acm[a][n][e];
                }
    }
}

// ------------------------------------------------------------------ per-row epilogues

constexpr int kNormThreads = 768;  // residual add + RMSNorm: one CTA per row

// Sum over the block of NT threads; every thread gets the same value (fixed order).
template <int NT>
__device__ __forceinline__ float r_block_sum(float v, float* red) {
    v = r_warp_sum(v);
    const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
    __syncthreads();
    if (l == 0) red[w] = v;
    __syncthreads();
    float t = l < NT / 32 ? red[l] : 0.f;
    return r_warp_sum(t);
}

// Sum of the S split partials p[0], p[stride], ..., in a fixed order: four
// running sums over splits s = 4k + r, added pairwise at the end, so that
// several loads are in flight.
__device__ __forceinline__ float split_sum(const float* __restrict__ p, int64_t stride, int S) {
    float a0 = 0.f, a1 = 0.f, a2 = 0.f, a3 = 0.f;
    int s = 0;
#pragma unroll 2
    for (; s + 4 <= S; s += 4) {
        a0 += p[(int64_t)s * stride];
        a1 += p[(int64_t)(s + 1) * stride];
        a2 += p[(int64_t)(s + 2) * stride];
        a3 += p[(int64_t)(s + 3) * stride];
    }
    for (; s < S; ++s) a0 += p[(int64_t)s * stride];
    return (a0 + a1) + (a2 + a3);
}

// One CTA per row i < M_norm.  Rows below M_add first add the split partials
// of a d-output projection (split stride M_add rows) to their residual.  With
// a gain, the row's RMSNorm h / sqrt(mean(h^2) + eps) * g goes to x as three
// bf16 parts.
__global__ void __launch_bounds__(kNormThreads) k_rows_add_norm(float* __restrict__ H, int d,
                                                                const float* __restrict__ part, int S, int M_add,
                                                                int Np, const uint16_t* __restrict__ gain, float eps,
                                                                const Parts x3, int ldx) {
    r_pdl();
    __shared__ float red[kNormThreads / 32];
    const int i = blockIdx.x;
    float* h = H + (int64_t)i * d;
    float ss = 0.f;
    for (int n = threadIdx.x; n < d; n += kNormThreads) {
        float v = h[n];
        if (i < M_add) {
            v += split_sum(part + (int64_t)i * Np + n, (int64_t)M_add * Np, S);
            h[n] = v;
        }
        ss = fmaf(v, v, ss);
    }
    if (!gain) return;  // uniform over the block
    ss = r_block_sum<kNormThreads>(ss, red);
    const float inv = 1.0f / sqrtf(ss / (float)d + eps);
    for (int n = threadIdx.x; n < pad64(d); n += kNormThreads)
        split_store(n < d ? h[n] * inv * r_bf2f(gain[n]) : 0.f, x3, i, n);
}

// Q/K/V of layer j for row blockIdx.y: thread = one unit (the packed row pair
// i, i + D/2 of one head; Q heads, then K, then V).  Split sum, bias, RoPE at
// the row's position; q stays fp32, k and v go to the cache as bf16.
__global__ void __launch_bounds__(kRowsThreads) k_rows_qkv(DevModel m, int j, const float* __restrict__ part,
                                                           int S, int M, int Np, const int32_t* __restrict__ pos,
                                                           float* __restrict__ Q) {
    r_pdl();
    const int i = blockIdx.y;
    const int u = blockIdx.x * kRowsThreads + threadIdx.x;
    const int half = m.D >> 1;
    const int nq = m.A * half, nk = m.KH * half;
    if (u >= nq + 2 * nk) return;
    const float* p = part + (int64_t)i * Np + 2 * u;
    float r0 = split_sum(p, (int64_t)M * Np, S), r1 = split_sum(p + 1, (int64_t)M * Np, S);
    if (m.qkv_bias) {
        const uint16_t* b = m.layers + (int64_t)j * m.layer_stride + m.off_bqkv;
        r0 += r_bf2f(b[2 * u]);
        r1 += r_bf2f(b[2 * u + 1]);
    }
    const int t = pos[i];
    if (u < nq) {
        const int h = u / half, e = u - h * half;
        const float2 c = m.rope[(int64_t)t * half + e];
        float* qh = Q + (int64_t)i * m.A * m.D + h * m.D;
        qh[e] = r0 * c.x - r1 * c.y;
        qh[e + half] = r0 * c.y + r1 * c.x;
    } else if (u < nq + nk) {
        const int uu = u - nq, g = uu / half, e = uu - g * half;
        const float2 c = m.rope[(int64_t)t * half + e];
        uint16_t* k = m.kpool + slot_offset(m, j, t) + (int64_t)g * m.page_size * m.D;
        k[e] = r_f2bf(r0 * c.x - r1 * c.y);
        k[e + half] = r_f2bf(r0 * c.y + r1 * c.x);
    } else {
        const int uu = u - nq - nk, g = uu / half, e = uu - g * half;
        uint16_t* v = m.vpool + slot_offset(m, j, t) + (int64_t)g * m.page_size * m.D;
        v[e] = r_f2bf(r0);
        v[e + half] = r_f2bf(r1);
    }
    if (u == 0) m.kv_src[(int64_t)j * m.max_ctx + t] = 1;
}

// SwiGLU of row blockIdx.y: a = silu(gate) * up from the split sums of the
// packed (gate, up) row pair, as three bf16 parts.
__global__ void __launch_bounds__(kRowsThreads) k_rows_swiglu(const float* __restrict__ part, int S, int M, int Np,
                                                              int F, const Parts x3, int ldx) {
    r_pdl();
    const int i = blockIdx.y;
    const int f = blockIdx.x * kRowsThreads + threadIdx.x;
    if (f >= pad64(F)) return;
    if (f >= F) {
        split_store(0.f, x3, i, f);
        return;
    }
    const float* p = part + (int64_t)i * Np + 2 * f;
    const float gs = split_sum(p, (int64_t)M * Np, S), us = split_sum(p + 1, (int64_t)M * Np, S);
    const float a = gs / (1.0f + expf(-gs)) * us;
    split_store(a, x3, i, f);
}

// Starting residual of row blockIdx.x: the embedding of ids[i] (a prompt;
// the row's position pos_base + i is recorded in pos) or the residual its
// position exited with.
__global__ void __launch_bounds__(kRowsThreads) k_rows_init(DevModel m, float* __restrict__ H, int32_t* pos,
                                                            const int32_t* __restrict__ ids, int pos_base) {
    r_pdl();
    const int i = blockIdx.x;
    float* h = H + (int64_t)i * m.d;
    if (ids) {
        int tok = ids[i];
        if (tok < 0 || tok >= m.V) {
            if (threadIdx.x == 0) atomicOr(&m.ctl->err, kErrTokenRange);
            tok = 0;
        }
        const uint16_t* e = m.embed + (int64_t)tok * m.d;
        for (int n = threadIdx.x; n < m.d; n += kRowsThreads) h[n] = r_bf2f(e[n]);
        if (threadIdx.x == 0) pos[i] = pos_base + i;
    } else {
        const float* src = m.h_exit + (int64_t)pos[i] * m.d;
        for (int n = threadIdx.x; n < m.d; n += kRowsThreads) h[n] = src[n];
    }
}

__global__ void k_rows_prefill_done(DevModel m, int n) {
    r_pdl();
    if (threadIdx.x != 0) return;
    Ctl* c = m.ctl;
    c->pos = n;
    c->pend_lo = n;  // prompt positions ran every layer
    c->prefill_i = n;
    c->exit_readout = -1;
    c->n_evaluated = 0;
    c->full_token = -1;
    c->nucleus_member = -1;
}

// ------------------------------------------------------------ flash attention
//
// Causal attention of the batch on the tensor cores, its keys split over
// CTAs (flash-decoding over a prompt batch).  CTA (kv head g, key split s,
// z = (row block b, head z' of the group)) takes query head h = g G + z' for
// the 64 rows of block b of the batch (4 warps x 16 rows) against keys [s KC, (s + 1) KC) of the
// layer's cache, in blocks of kFaKeys keys staged in shared memory:
//   S = Q K^T as mma m16n8k16 with the query (scaled by 1/sqrt(D)) split into
//     three bf16 parts (high + middle + low = q exactly), each multiplied
//     with the bf16 keys into the same fp32 accumulators (exact products);
//   keys past a row's position are masked (Section 2's causal softmax), and
//     a running maximum and sum per row rescale the output as blocks pass;
//   O += P V with the probabilities split into three bf16 parts the same
//     way, the values read transposed from shared memory (ldmatrix.trans).
// Each split writes its unnormalised output, maximum and sum per (row,
// head); k_rows_amerge combines the splits of each row in split order and
// writes the attention output as the O projection's three bf16 parts.
constexpr int kFaWarps = 4;
constexpr int kFaThreads = 32 * kFaWarps;
constexpr int kFaKeys = 64;        // keys per shared-memory block
constexpr int kFaMaxSplits = 32;   // key splits per batch (at most)

__host__ __device__ constexpr int fa_ld(int D) { return D + 8; }  // padded row (bf16): conflict-free ldmatrix
__host__ __device__ constexpr size_t fa_smem(int D) {  // queries, then two blocks of keys and values
    return (size_t)(kFaWarps * 3 * 16 + 4 * kFaKeys) * fa_ld(D) * 2;
}

__device__ __forceinline__ uint32_t fa_saddr(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }
// 16 bytes global -> shared, asynchronously; the bytes past src_bytes (0 or 16) are zero.
__device__ __forceinline__ void fa_cp16(uint32_t dst, const void* src, int src_bytes) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(src_bytes) : "memory");
}
__device__ __forceinline__ void ldsm_x4(uint32_t a, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(a));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t a, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(a));
}
// Two floats as three packed bf16 parts (high, middle, low; the first float
// in the low halves).
__device__ __forceinline__ void fa_split2(float x0, float x1, uint32_t& hi, uint32_t& md, uint32_t& lo) {
    const uint16_t h0 = r_f2bf(x0), h1 = r_f2bf(x1);
    const float a0 = x0 - r_bf2f(h0), a1 = x1 - r_bf2f(h1);
    const uint16_t m0 = r_f2bf(a0), m1 = r_f2bf(a1);
    hi = (uint32_t)h0 | ((uint32_t)h1 << 16);
    md = (uint32_t)m0 | ((uint32_t)m1 << 16);
    lo = (uint32_t)r_f2bf(a0 - r_bf2f(m0)) | ((uint32_t)r_f2bf(a1 - r_bf2f(m1)) << 16);
}

template <int D>
__global__ void __launch_bounds__(kFaThreads) k_rows_fattn(DevModel m, int j, const float* __restrict__ Q,
                                                           const int32_t* __restrict__ pos, int Mj, int KC,
                                                           int t_max, float* __restrict__ part) {
    r_pdl();
    constexpr int LD = fa_ld(D);
    constexpr int NT = D / 8;   // n8 tiles of the output
    constexpr int KS = D / 16;  // k16 steps of a score
    extern __shared__ __align__(16) uint16_t fsm[];
    uint16_t* qs = fsm;                                // [warp][part][16][LD]
    uint16_t* ks = qs + kFaWarps * 3 * 16 * LD;        // [2][kFaKeys][LD]
    uint16_t* vs = ks + 2 * kFaKeys * LD;              // [2][kFaKeys][LD]
    const int g = blockIdx.x, s = blockIdx.y, G = m.A / m.KH, h = g * G + (int)blockIdx.z % G;
    const int row0 = ((int)blockIdx.z / G) * kFaWarps * 16;  // the CTA's first row of the batch
    if (row0 >= Mj) return;                                  // a block with no row at this layer
    const int tid = threadIdx.x, w = tid >> 5, lane = tid & 31, g8 = lane >> 2, t4 = lane & 3;
    const int k0 = s * KC;
    // the CTA's keys end at the split's end or past the batch's last position
    const int kend = min(k0 + KC, t_max);
    const int64_t head_off = (int64_t)g * m.page_size * D;
    // A block of keys and values into buffer `buf`: cp.async, all of a
    // thread's copies issued together; keys past kend read as zero.
    auto load_block = [&](int kb, int buf) {
        const uint32_t kd = fa_saddr(ks + buf * kFaKeys * LD), vd = fa_saddr(vs + buf * kFaKeys * LD);
#pragma unroll
        for (int u = 0; u < kFaKeys * (D / 8) / kFaThreads; ++u) {
            const int e = tid + u * kFaThreads, r = e / (D / 8), c = e - r * (D / 8), t = kb + r;
            const bool ok = t < kend;
            const int64_t off = ok ? slot_offset(m, j, t) + head_off + c * 8 : 0;
            fa_cp16(kd + (r * LD + c * 8) * 2, m.kpool + off, ok ? 16 : 0);
            fa_cp16(vd + (r * LD + c * 8) * 2, m.vpool + off, ok ? 16 : 0);
        }
        asm volatile("cp.async.commit_group;" ::: "memory");
    };
    if (k0 < kend) load_block(k0, 0);
    // rows of this warp, their positions (-1: not in the batch)
    const int r0 = row0 + 16 * w + g8, r1 = r0 + 8;
    const int p0 = r0 < Mj ? pos[r0] : -1, p1 = r1 < Mj ? pos[r1] : -1;
    int pw = max(p0, p1);
#pragma unroll
    for (int o = 4; o < 32; o <<= 1) pw = max(pw, __shfl_xor_sync(0xffffffffu, pw, o));
    const bool act = pw >= k0;  // this warp has a row with a key in the split
    // the warp's queries, scaled, as three bf16 parts (all loads issued first)
    const float scale = 1.0f / sqrtf((float)D);
    uint16_t* qw = qs + w * 3 * 16 * LD;
    {
        constexpr int QV = 16 * D / 4 / 32;  // float4 per lane
        float4 qv[QV];
#pragma unroll
        for (int u = 0; u < QV; ++u) {
            const int e = lane + 32 * u, r = e / (D / 4), c = 4 * (e - r * (D / 4)), i = row0 + 16 * w + r;
            qv[u] = i < Mj ? *reinterpret_cast<const float4*>(Q + (int64_t)i * m.A * D + (int64_t)h * D + c)
                           : make_float4(0.f, 0.f, 0.f, 0.f);
        }
#pragma unroll
        for (int u = 0; u < QV; ++u) {
            const int e = lane + 32 * u, r = e / (D / 4), c = 4 * (e - r * (D / 4));
            uint32_t h0, m0, l0_, h1, m1, l1_;
            fa_split2(qv[u].x * scale, qv[u].y * scale, h0, m0, l0_);
            fa_split2(qv[u].z * scale, qv[u].w * scale, h1, m1, l1_);
            *reinterpret_cast<uint2*>(qw + (0 * 16 + r) * LD + c) = make_uint2(h0, h1);
            *reinterpret_cast<uint2*>(qw + (1 * 16 + r) * LD + c) = make_uint2(m0, m1);
            *reinterpret_cast<uint2*>(qw + (2 * 16 + r) * LD + c) = make_uint2(l0_, l1_);
        }
    }
    float o[NT][4];
#pragma unroll
    for (int n = 0; n < NT; ++n) o[n][0] = o[n][1] = o[n][2] = o[n][3] = 0.f;
    float mr0 = -INFINITY, mr1 = -INFINITY, l0 = 0.f, l1 = 0.f;
    // ldmatrix row addresses: matrix q = lane / 8, row lane % 8
    const int lq = lane >> 3, lr = lane & 7;
    const uint32_t qa = fa_saddr(qw) + ((lq & 1) * 8 + lr) * LD * 2 + (lq >> 1) * 16;       // A: rows +8, cols +8
    const uint32_t kb_a0 = fa_saddr(ks) + ((lq >> 1) * 8 + lr) * LD * 2 + (lq & 1) * 16;    // B of K: keys +8, dims +8
    const uint32_t vb_a0 = fa_saddr(vs) + ((lq & 1) * 8 + lr) * LD * 2 + (lq >> 1) * 16;    // B of V^T: keys +8, dims +8
    int buf = 0;
    for (int kb = k0; kb < kend; kb += kFaKeys, buf ^= 1) {
        // the next block into the other buffer (free: every warp passed the
        // barrier at the end of the previous block), then wait for this one
        const bool next = kb + kFaKeys < kend;
        if (next) load_block(kb + kFaKeys, buf ^ 1);
        if (next)
            asm volatile("cp.async.wait_group 1;" ::: "memory");
        else
            asm volatile("cp.async.wait_group 0;" ::: "memory");
        __syncthreads();  // the block (and the queries) visible to every warp
        const uint32_t kb_a = kb_a0 + buf * kFaKeys * LD * 2, vb_a = vb_a0 + buf * kFaKeys * LD * 2;
        if (act && kb <= pw) {
            // scores of the warp's 16 rows against the block's 64 keys
            float sc[8][4];
#pragma unroll
            for (int n = 0; n < 8; ++n) sc[n][0] = sc[n][1] = sc[n][2] = sc[n][3] = 0.f;
#pragma unroll
            for (int kk = 0; kk < KS; ++kk) {
                uint32_t a[3][4];
#pragma unroll
                for (int pt = 0; pt < 3; ++pt)
                    ldsm_x4(qa + pt * 16 * LD * 2 + kk * 32, a[pt][0], a[pt][1], a[pt][2], a[pt][3]);
#pragma unroll
                for (int np = 0; np < 4; ++np) {
                    uint32_t b0, b1, b2, b3;
                    ldsm_x4(kb_a + np * 16 * LD * 2 + kk * 32, b0, b1, b2, b3);
#pragma unroll
                    for (int pt = 0; pt < 3; ++pt) {
                        mma_16816(sc[2 * np], a[pt][0], a[pt][1], a[pt][2], a[pt][3], b0, b1);
                        mma_16816(sc[2 * np + 1], a[pt][0], a[pt][1], a[pt][2], a[pt][3], b2, b3);
                    }
                }
            }
            // causal mask, block maxima, rescale
            float bm0 = -INFINITY, bm1 = -INFINITY;
#pragma unroll
            for (int n = 0; n < 8; ++n) {
                const int t = kb + n * 8 + 2 * t4;
                sc[n][0] = t <= p0 ? sc[n][0] : -INFINITY;
                sc[n][1] = t + 1 <= p0 ? sc[n][1] : -INFINITY;
                sc[n][2] = t <= p1 ? sc[n][2] : -INFINITY;
                sc[n][3] = t + 1 <= p1 ? sc[n][3] : -INFINITY;
                bm0 = fmaxf(bm0, fmaxf(sc[n][0], sc[n][1]));
                bm1 = fmaxf(bm1, fmaxf(sc[n][2], sc[n][3]));
            }
            bm0 = fmaxf(bm0, __shfl_xor_sync(0xffffffffu, bm0, 1));
            bm0 = fmaxf(bm0, __shfl_xor_sync(0xffffffffu, bm0, 2));
            bm1 = fmaxf(bm1, __shfl_xor_sync(0xffffffffu, bm1, 1));
            bm1 = fmaxf(bm1, __shfl_xor_sync(0xffffffffu, bm1, 2));
            const float mn0 = fmaxf(mr0, bm0), mn1 = fmaxf(mr1, bm1);
            // a row with no key yet keeps maximum -inf, probabilities 0
            const float c0 = mn0 == -INFINITY ? 1.f : expf(mr0 - mn0);
            const float c1 = mn1 == -INFINITY ? 1.f : expf(mr1 - mn1);
            float s0 = 0.f, s1 = 0.f;
#pragma unroll
            for (int n = 0; n < 8; ++n) {
                sc[n][0] = mn0 == -INFINITY ? 0.f : expf(sc[n][0] - mn0);
                sc[n][1] = mn0 == -INFINITY ? 0.f : expf(sc[n][1] - mn0);
                sc[n][2] = mn1 == -INFINITY ? 0.f : expf(sc[n][2] - mn1);
                sc[n][3] = mn1 == -INFINITY ? 0.f : expf(sc[n][3] - mn1);
                s0 += sc[n][0] + sc[n][1];
                s1 += sc[n][2] + sc[n][3];
            }
            s0 += __shfl_xor_sync(0xffffffffu, s0, 1);
            s0 += __shfl_xor_sync(0xffffffffu, s0, 2);
            s1 += __shfl_xor_sync(0xffffffffu, s1, 1);
            s1 += __shfl_xor_sync(0xffffffffu, s1, 2);
            l0 = l0 * c0 + s0;
            l1 = l1 * c1 + s1;
            mr0 = mn0;
            mr1 = mn1;
#pragma unroll
            for (int n = 0; n < NT; ++n) {
                o[n][0] *= c0;
                o[n][1] *= c0;
                o[n][2] *= c1;
                o[n][3] *= c1;
            }
            // O += P V over the block's keys, 16 at a time
#pragma unroll
            for (int kk = 0; kk < kFaKeys / 16; ++kk) {
                uint32_t a[3][4];
                fa_split2(sc[2 * kk][0], sc[2 * kk][1], a[0][0], a[1][0], a[2][0]);
                fa_split2(sc[2 * kk][2], sc[2 * kk][3], a[0][1], a[1][1], a[2][1]);
                fa_split2(sc[2 * kk + 1][0], sc[2 * kk + 1][1], a[0][2], a[1][2], a[2][2]);
                fa_split2(sc[2 * kk + 1][2], sc[2 * kk + 1][3], a[0][3], a[1][3], a[2][3]);
#pragma unroll
                for (int np = 0; np < NT / 2; ++np) {
                    uint32_t b0, b1, b2, b3;
                    ldsm_x4_t(vb_a + kk * 16 * LD * 2 + np * 32, b0, b1, b2, b3);
#pragma unroll
                    for (int pt = 0; pt < 3; ++pt) {
                        mma_16816(o[2 * np], a[pt][0], a[pt][1], a[pt][2], a[pt][3], b0, b1);
                        mma_16816(o[2 * np + 1], a[pt][0], a[pt][1], a[pt][2], a[pt][3], b2, b3);
                    }
                }
            }
        }
        __syncthreads();  // every warp is done with this buffer before the next load into it
    }
    if (!act) return;
    // the split's unnormalised output, maximum and sum of each row:
    // part[((s kRowsMax + row) A + h)][D + 2]
    const int ld = D + 2;
    float* q0 = part + ((int64_t)(s * kRowsMax + r0) * m.A + h) * ld;
    float* q1 = part + ((int64_t)(s * kRowsMax + r1) * m.A + h) * ld;
#pragma unroll
    for (int n = 0; n < NT; ++n) {
        const int c = n * 8 + 2 * t4;
        if (p0 >= 0) {
            q0[c] = o[n][0];
            q0[c + 1] = o[n][1];
        }
        if (p1 >= 0) {
            q1[c] = o[n][2];
            q1[c + 1] = o[n][3];
        }
    }
    if (t4 == 0) {
        if (p0 >= 0) {
            q0[D] = mr0;
            q0[D + 1] = l0;
        }
        if (p1 >= 0) {
            q1[D] = mr1;
            q1[D + 1] = l1;
        }
    }
}

// The splits of row i, head h (blockIdx.x = h, blockIdx.y = i; D threads):
// o = sum_s exp(m_s - M) o_s / sum_s exp(m_s - M) l_s over the splits that
// hold a key at or before the row's position, in split order; written as the
// O projection's three bf16 parts at column h D + e.
template <int D>
__global__ void __launch_bounds__(D) k_rows_amerge(DevModel m, const float* __restrict__ part,
                                                   const int32_t* __restrict__ pos, int KC, const Parts x3) {
    r_pdl();
    const int h = blockIdx.x, i = blockIdx.y, e = threadIdx.x;
    const int ns = pos[i] / KC + 1, ld = D + 2;
    const float* q = part + ((int64_t)i * m.A + h) * ld;
    const int64_t step = (int64_t)kRowsMax * m.A * ld;  // one split
    float M = -INFINITY;
    for (int s = 0; s < ns; ++s) M = fmaxf(M, q[s * step + D]);
    float num = 0.f, den = 0.f;
    for (int s = 0; s < ns; ++s) {
        const float* qs = q + s * step;
        const float wgt = expf(qs[D] - M);
        num = fmaf(wgt, qs[e], num);
        den = fmaf(wgt, qs[D + 1], den);
    }
    split_store(num / den, x3, i, h * D + e);
    if (h == 0)  // the columns past A D up to the tensor cores' stage
        for (int col = m.A * D + e; col < pad64(m.A * D); col += D) split_store(0.f, x3, i, col);
}

// ------------------------------------------------------------------ host side

template <class... KArgs, class... Args>
cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s, Args... args) {
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, static_cast<KArgs>(args)...);
}

// The activation parts of a batch of M rows (row stride M rounded up to 16,
// the operand rows of the tensor-core products).
Parts parts(const RowsBuf& b, int M) { return Parts{b.x3, x3_rows(M)}; }

#define RCKA(x)                                   \
    do {                                          \
        cudaError_t e_ = (x);                     \
        if (e_ != cudaSuccess) return e_;         \
    } while (0)

// Row blocks of 8 a warp takes (1, 2 or 4) and the row groups of a batch.
void row_groups(int M, int& NB, int& RG) {
    const int blocks = (M + 7) / 8;
    NB = blocks <= 1 ? 1 : blocks <= 2 ? 2 : 4;
    RG = (blocks + NB - 1) / NB;
}

// Keys per split of the flash attention: a multiple of kFaKeys, large enough
// that the splits of a batch whose last position is t_max - 1, times the
// (query head, block of 64 rows) pairs, make about one wave of CTAs (one
// resident per SM: its stages take over half the shared memory), and at most
// kFaMaxSplits.  (Two or four waves of shorter splits were slower: every
// split is a partial result written, merged and read again.)
int fa_keys_per_split(int t_max, int units, int n_sm) {
    const int target = std::max(1, std::min(kFaMaxSplits, n_sm / std::max(1, units)));
    int kc = (t_max + target - 1) / target;
    kc = std::max(kFaKeys, (kc + kFaKeys - 1) / kFaKeys * kFaKeys);
    while ((t_max + kc - 1) / kc > kFaMaxSplits) kc += kFaKeys;
    return kc;
}

// The batch's attention at layer j: the split kernel, then the merge into
// the O projection's input parts.
cudaError_t launch_attn(const DevModel& m, const RowsBuf& b, int j, int Mj, const int32_t* d_pos, int t_max,
                        cudaStream_t s) {
    const int row_blocks = (Mj + kFaWarps * 16 - 1) / (kFaWarps * 16);
    const int KC = fa_keys_per_split(t_max, m.A * row_blocks, b.n_sm);
    const int S = (t_max + KC - 1) / KC;
    const dim3 grid(m.KH, S, (m.A / m.KH) * row_blocks);
    if (m.D == 128) {
        RCKA(launch_pdl(k_rows_fattn<128>, grid, dim3(kFaThreads), fa_smem(128), s, m, j, (const float*)b.Q, d_pos, Mj,
                        KC, t_max, b.part));
        return launch_pdl(k_rows_amerge<128>, dim3(m.A, Mj), dim3(128), 0, s, m, (const float*)b.part, d_pos, KC,
                          parts(b, Mj));
    }
    RCKA(launch_pdl(k_rows_fattn<64>, grid, dim3(kFaThreads), fa_smem(64), s, m, j, (const float*)b.Q, d_pos, Mj, KC,
                    t_max, b.part));
    return launch_pdl(k_rows_amerge<64>, dim3(m.A, Mj), dim3(64), 0, s, m, (const float*)b.part, d_pos, KC, parts(b, Mj));
}

// One projection of the batch: W (n_rows x K, tiled) times the M rows of
// b.xhi / b.xmid / b.xlo into b.part; returns the split count and padded row count
// its consumer needs.
cudaError_t launch_mm(const uint16_t* W, int64_t n_rows, int K, const RowsBuf& b, int M, int& S, int& Np,
                      cudaStream_t s) {
    const int64_t nt = tile_count(n_rows);
    if (b.umma) {
        Np = (int)(nt * kTileRows);
        S = umma_splits(nt, K, b.n_sm);
        S = (int)std::max<int64_t>(1, std::min<int64_t>(S, b.part_floats / ((int64_t)M * Np)));
        return launch_mm_umma(W, n_rows, K, b.x3, M, S, b.part, Np, b.err, s);
    }
    int NB, RG;
    row_groups(M, NB, RG);
    S = rows_splits(nt, K, M);
    Np = (int)(nt * kTileRows);
    const int64_t units = nt * S * RG;
    const int grid = (int)std::min<int64_t>((units + kRowsWarps - 1) / kRowsWarps, 65535);
    const uint4* w = reinterpret_cast<const uint4*>(W);
    if (NB == 1)
        return launch_pdl(k_rows_mm<1, 2>, dim3(grid), dim3(kRowsThreads), 0, s, w, (int)nt, K, parts(b, M), b.ldx, M, S, RG,
                          b.part, Np);
    else if (NB == 2)
        return launch_pdl(k_rows_mm<2, 2>, dim3(grid), dim3(kRowsThreads), 0, s, w, (int)nt, K, parts(b, M), b.ldx, M, S, RG,
                          b.part, Np);
    else
        return launch_pdl(k_rows_mm<4, 1>, dim3(grid), dim3(kRowsThreads), 0, s, w, (int)nt, K, parts(b, M), b.ldx, M, S, RG,
                          b.part, Np);
}

}  // namespace

// Enough (tile, split, row group) units to give every resident warp of the
// GPU one (16 warps per SM; 24 with four row blocks a warp, whose registers
// leave room for three CTAs), each at least one 32-column step, and split
// partials (written and read once, in L2) at most the weight bytes,
// S * M * 4 B * 2 <= K * 2 B, or twice that with four row blocks a warp
// (whose units are otherwise too few to cover the SMs).
int rows_splits(int64_t n_tiles, int K, int M) {
    const int nsteps = ((K >> 3) + 3) >> 2;
    const int Mp = std::max(8, (M + 7) & ~7);
    int NB, RG;
    row_groups(M, NB, RG);
    const int64_t target = NB == 4 ? kRowsTargetUnits * 3 / 2 : kRowsTargetUnits;
    int S = (int)((target + n_tiles * RG - 1) / (n_tiles * RG));
    S = std::min(S, std::max(1, K / ((NB == 4 ? 2 : 4) * Mp)));
    S = std::min(S, nsteps);
    return std::max(S, 1);
}

cudaError_t configure_rows() {
    cudaError_t e = cudaFuncSetAttribute(k_rows_fattn<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)fa_smem(128));
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(k_rows_fattn<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)fa_smem(64));
    return e;
}

int64_t rows_part_floats(int d, int A, int KH, int D, int F) {
    const int64_t rows[4] = {(int64_t)(A + 2 * KH) * D, d, 2LL * F, d};
    const int K[4] = {d, A * D, d, F};
    int64_t most = 0;
    for (int M = 8; M <= kRowsMax; M += 8)
        for (int p = 0; p < 4; ++p) {
            const int64_t nt = tile_count(rows[p]);
            most = std::max(most, (int64_t)rows_splits(nt, K[p], M) * M * nt * kTileRows);
        }
    // the flash attention's split outputs: [kFaMaxSplits][kRowsMax][A][D + 2]
    return std::max(most, (int64_t)kFaMaxSplits * kRowsMax * A * (D + 2));
}

#define RCK(x)                                    \
    do {                                          \
        cudaError_t e_ = (x);                     \
        if (e_ != cudaSuccess) return e_;         \
    } while (0)

cudaError_t rows_pass(const DevModel& m, const RowsBuf& b, const int* start, int M, int32_t* d_pos,
                      const int32_t* ids, int pos_base, int t_max, bool kv_only, cudaStream_t s) {
    if (M <= 0) return cudaSuccess;
    if (t_max <= 0 || t_max > m.max_ctx) return cudaErrorInvalidValue;
    if (M > kRowsMax || start[0] < 0 || start[M - 1] >= m.L) return cudaErrorInvalidValue;
    for (int i = 1; i < M; ++i)
        if (start[i] < start[i - 1]) return cudaErrorInvalidValue;
    const int L = m.L, d = m.d, AD = m.A * m.D;
    const int64_t nqkv = (int64_t)(m.A + 2 * m.KH) * m.D;
    RCK(launch_pdl(k_rows_init, dim3(M), dim3(kRowsThreads), 0, s, m, b.H, d_pos, ids, pos_base));
    int M_prev = 0, S_prev = 1, Np_prev = 0;
    for (int j = start[0]; j < L; ++j) {
        int Mj = M_prev;
        while (Mj < M && start[Mj] <= j) ++Mj;
        const uint16_t* lw = m.layers + (int64_t)j * m.layer_stride;
        int S = 1, Np = 0;
        // the previous layer's down projection into the residual, this layer's input norm
        RCK(launch_pdl(k_rows_add_norm, dim3(Mj), dim3(kNormThreads), 0, s, b.H, d, (const float*)b.part, S_prev, M_prev,
                       Np_prev, lw + m.off_gattn, m.eps, parts(b, Mj), b.ldx));
        RCK(launch_mm(lw + m.off_wqkv, nqkv, d, b, Mj, S, Np, s));
        const int nu = (int)(nqkv / 2);
        RCK(launch_pdl(k_rows_qkv, dim3((nu + kRowsThreads - 1) / kRowsThreads, Mj), dim3(kRowsThreads), 0, s, m, j,
                       (const float*)b.part, S, Mj, Np, (const int32_t*)d_pos, b.Q));
        if (kv_only && j == L - 1) return cudaSuccess;
        RCK(launch_attn(m, b, j, Mj, d_pos, t_max, s));
        RCK(launch_mm(lw + m.off_wo, d, AD, b, Mj, S, Np, s));
        RCK(launch_pdl(k_rows_add_norm, dim3(Mj), dim3(kNormThreads), 0, s, b.H, d, (const float*)b.part, S, Mj, Np,
                       lw + m.off_gmlp, m.eps, parts(b, Mj), b.ldx));
        RCK(launch_mm(lw + m.off_wgu, 2LL * m.F, d, b, Mj, S, Np, s));
        RCK(launch_pdl(k_rows_swiglu, dim3((pad64(m.F) + kRowsThreads - 1) / kRowsThreads, Mj), dim3(kRowsThreads), 0, s,
                       (const float*)b.part, S, Mj, Np, m.F, parts(b, Mj), b.ldx));
        RCK(launch_mm(lw + m.off_wd, d, m.F, b, Mj, S, Np, s));
        M_prev = Mj;
        S_prev = S;
        Np_prev = Np;
    }
    // the last down projection into the residual (no norm)
    return launch_pdl(k_rows_add_norm, dim3(M_prev), dim3(kNormThreads), 0, s, b.H, d, (const float*)b.part, S_prev,
                      M_prev, Np_prev, (const uint16_t*)nullptr, m.eps, parts(b, M_prev), b.ldx);
}

cudaError_t launch_rows_prefill_done(const DevModel& m, int n, cudaStream_t s) {
    return launch_pdl(k_rows_prefill_done, dim3(1), dim3(32), 0, s, m, n);
}

}  // namespace ee
