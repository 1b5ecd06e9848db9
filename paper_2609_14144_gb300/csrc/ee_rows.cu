// Multi-position layer pass for sm_103a: the prompt (Section 2's prefill,
// full depth with no gate) and Section 11's full-depth re-pass of exited
// positions run each layer over a batch of up to kRowsMax positions, so a
// weight byte is read once per batch instead of once per position.
//
// A layer is nine launches, each reading what the previous one wrote:
//   k_rows_add_norm  residual add of the previous projection's split
//                    partials (in a fixed order), then RMSNorm with the next
//                    gain, written as three bf16 parts
//   k_rows_mm        a projection: Y[row][n] = sum_k W[n][k] x[row][k]
//   k_rows_qkv       split sum, bias, RoPE at each row's position; q kept in
//                    fp32, k and v stored bf16 into the paged cache
//   k_rows_attn      causal attention of every row over the cache up to its
//                    position (rows of the batch at earlier positions were
//                    written by k_rows_qkv of this layer)
//   k_rows_mm (O), k_rows_add_norm (mid residual, MLP norm),
//   k_rows_mm (gate/up), k_rows_swiglu, k_rows_mm (down)
//
// Projections use the legacy warp-level tensor-core mma (m16n8k16, bf16
// operands, fp32 accumulation).  A warp owns one (32-row weight tile, K
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
constexpr int kKeysPerChunk = kRowsThreads;  // attention: one key per thread per chunk

__device__ __forceinline__ float r_bf2f(uint16_t b) { return __uint_as_float((uint32_t)b << 16); }
__device__ __forceinline__ uint16_t r_f2bf(float f) { return __bfloat16_as_ushort(__float2bfloat16_rn(f)); }
__device__ __forceinline__ float r_lo(uint32_t u) { return __uint_as_float(u << 16); }
__device__ __forceinline__ float r_hi(uint32_t u) { return __uint_as_float(u & 0xffff0000u); }

// A product's input as three bf16 parts, stored chunk-major: for each
// 16-byte column chunk (8 columns), the high parts of the kRowsMax rows, then
// the middle parts, then the low parts, 16 bytes per row.  Eight chunks are
// then one contiguous block in the tensor cores' canonical operand layout
// (ee_umma.cu), and a warp-level product reads a row's chunk of one part as
// 16 contiguous bytes.
struct Parts {
    uint16_t* p;
};
__device__ __forceinline__ int64_t x3_index(int part, int row, int col) {
    return ((int64_t)((col >> 3) * 3 + part) * kRowsMax + row) * 8 + (col & 7);
}

// The three bf16 parts of x at (row, col): high = bf16(x), middle = bf16(x -
// high), low = bf16(x - high - middle) (each difference exact in fp32).
__device__ __forceinline__ void split_store(float x, const Parts& p, int row, int col) {
    const uint16_t h = r_f2bf(x);
    const float r1 = x - r_bf2f(h);
    const uint16_t md = r_f2bf(r1);
    p.p[x3_index(0, row, col)] = h;
    p.p[x3_index(1, row, col)] = md;
    p.p[x3_index(2, row, col)] = r_f2bf(r1 - r_bf2f(md));
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
__device__ __forceinline__ float r_warp_max(float v) {
#pragma unroll
    for (int o = 16; o; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
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
        float acc[2][NB][4];
#pragma unroll
        for (int a = 0; a < 2; ++a)
#pragma unroll
            for (int n = 0; n < NB; ++n)
#pragma unroll
                for (int e = 0; e < 4; ++e) acc[a][n][e] = 0.f;
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
                    const uint16_t* at = x3.p + x3_index(0, okx ? row : 0, ch * 8);
                    bh[v][n] = okx ? ld_act(at) : make_uint4(0u, 0u, 0u, 0u);
                    bm[v][n] = okx ? ld_act(at + kRowsMax * 8) : make_uint4(0u, 0u, 0u, 0u);
                    bl[v][n] = okx ? ld_act(at + 2 * kRowsMax * 8) : make_uint4(0u, 0u, 0u, 0u);
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
                        // first mma of the step: chunk elements 0..3; second: 4..7
                        mma_16816(acc[0][n], x[0].x, x[1].x, x[0].y, x[1].y, b.x, b.y);
                        mma_16816(acc[0][n], x[0].z, x[1].z, x[0].w, x[1].w, b.z, b.w);
                        mma_16816(acc[1][n], x[2].x, x[3].x, x[2].y, x[3].y, b.x, b.y);
                        mma_16816(acc[1][n], x[2].z, x[3].z, x[2].w, x[3].w, b.z, b.w);
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
                    if (row < M) ps[(int64_t)row * Np + out] = acc[a][n][e];
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

// Causal attention of row blockIdx.y and kv head blockIdx.x over cache
// positions 0..pos[i] of layer j, for the head group's G query heads, in
// chunks of one key per thread: scores q.k / sqrt(D) per thread, a running
// maximum and sum per head, and the weighted values summed with each warp
// taking its own 32 keys of the chunk (lane l owning dimensions
// l*D/32 .. l*D/32 + D/32 - 1 of every head), rescaled whenever the maximum
// grows; the warps' sums are added in warp order at the end (Section 2's
// softmax attention).  Output o at column h*D + e as three bf16 parts.
template <int D>
__global__ void __launch_bounds__(kRowsThreads) k_rows_attn(DevModel m, int j, const float* __restrict__ Q,
                                                            const int32_t* __restrict__ pos, const Parts x3,
                                                            int ldx) {
    r_pdl();
    constexpr int kG = kSegMaxGroup;  // query heads per kv head (at most)
    constexpr int DL = D / 32;        // dimensions per lane in the value sums
    constexpr int CPR = D / 8;        // 16-byte chunks of a key row
    extern __shared__ uint4 ksm[];    // [kKeysPerChunk][CPR + 1] keys, then [kKeysPerChunk][CPR] values
    uint4* vsm = ksm + kKeysPerChunk * (CPR + 1);
    __shared__ float qs[kG * D];
    __shared__ float ps[kG * kKeysPerChunk];
    __shared__ int64_t offs[kKeysPerChunk];
    __shared__ float redm[kRowsWarps][kG], reds[kRowsWarps][kG];
    __shared__ float mrun[kG], lrun[kG], resc[kG];
    const int g = blockIdx.x, i = blockIdx.y, G = m.A / m.KH;
    const int tid = threadIdx.x, lane = tid & 31, w = tid >> 5;
    const int T = pos[i] + 1;
    const float scale = 1.0f / sqrtf((float)D);
    const float* qrow = Q + (int64_t)i * m.A * D + (int64_t)g * G * D;
    for (int x = tid; x < G * D; x += kRowsThreads) qs[x] = qrow[x] * scale;
    if (tid < kG) {
        mrun[tid] = -INFINITY;
        lrun[tid] = 0.f;
    }
    float o[kG][DL];
#pragma unroll
    for (int h = 0; h < kG; ++h)
#pragma unroll
        for (int x = 0; x < DL; ++x) o[h][x] = 0.f;
    const int64_t head_off = (int64_t)g * m.page_size * D;
    __syncthreads();
    for (int c0 = 0; c0 < T; c0 += kKeysPerChunk) {
        const int t = c0 + tid;
        const bool valid = t < T;
        const int64_t off = valid ? slot_offset(m, j, t) + head_off : 0;
        offs[tid] = off;
        __syncthreads();
        // the chunk's key and value rows into shared memory, consecutive
        // threads along a row (coalesced); key rows padded by 16 bytes
        // (conflict-free row reads), value rows past T zero
        for (int e = tid; e < kKeysPerChunk * CPR; e += kRowsThreads) {
            const int r = e / CPR, c = e - r * CPR;
            if (c0 + r < T) {
                ksm[r * (CPR + 1) + c] = *reinterpret_cast<const uint4*>(m.kpool + offs[r] + c * 8);
                vsm[r * CPR + c] = *reinterpret_cast<const uint4*>(m.vpool + offs[r] + c * 8);
            } else {
                vsm[r * CPR + c] = make_uint4(0u, 0u, 0u, 0u);
            }
        }
        __syncthreads();
        float sc[kG];
#pragma unroll
        for (int h = 0; h < kG; ++h) sc[h] = 0.f;
        if (valid) {
            uint4 kv[D / 8];
#pragma unroll
            for (int c = 0; c < D / 8; ++c) kv[c] = ksm[tid * (CPR + 1) + c];
#pragma unroll
            for (int c = 0; c < D / 8; ++c) {
                const float kf[8] = {r_lo(kv[c].x), r_hi(kv[c].x), r_lo(kv[c].y), r_hi(kv[c].y),
                                     r_lo(kv[c].z), r_hi(kv[c].z), r_lo(kv[c].w), r_hi(kv[c].w)};
#pragma unroll
                for (int h = 0; h < kG; ++h) {
                    if (h < G) {
                        const float* qh = qs + h * D + c * 8;
                        float a = sc[h];
#pragma unroll
                        for (int e = 0; e < 8; ++e) a = fmaf(qh[e], kf[e], a);
                        sc[h] = a;
                    }
                }
            }
        }
#pragma unroll
        for (int h = 0; h < kG; ++h) {
            if (h < G) {
                sc[h] = valid ? sc[h] : -INFINITY;
                const float mx = r_warp_max(sc[h]);
                if (lane == 0) redm[w][h] = mx;
            }
        }
        __syncthreads();
        if (tid < G) {
            float cm = redm[0][tid];
            for (int ww = 1; ww < kRowsWarps; ++ww) cm = fmaxf(cm, redm[ww][tid]);
            const float mo = mrun[tid], mn = fmaxf(mo, cm);
            resc[tid] = mo == -INFINITY ? 0.f : expf(mo - mn);
            mrun[tid] = mn;
        }
        __syncthreads();
#pragma unroll
        for (int h = 0; h < kG; ++h) {
            if (h < G) {
                const float p = valid ? expf(sc[h] - mrun[h]) : 0.f;
                ps[h * kKeysPerChunk + tid] = p;
                const float sum = r_warp_sum(p);
                if (lane == 0) reds[w][h] = sum;
            }
        }
        __syncthreads();
        if (tid < G) {
            float sum = 0.f;
            for (int ww = 0; ww < kRowsWarps; ++ww) sum += reds[ww][tid];
            lrun[tid] = lrun[tid] * resc[tid] + sum;
        }
#pragma unroll
        for (int h = 0; h < kG; ++h) {
            const float r = h < G ? resc[h] : 0.f;
#pragma unroll
            for (int x = 0; x < DL; ++x) o[h][x] *= r;
        }
        // this warp's keys of the chunk (invalid keys have p = 0 and offset 0)
        const int k0 = w * 32;
#pragma unroll 8
        for (int kk = 0; kk < 32; ++kk) {
            const int tt = k0 + kk;
            const uint16_t* vr = reinterpret_cast<const uint16_t*>(vsm + tt * CPR) + lane * DL;
            float v[DL];
            if constexpr (DL == 4) {
                const uint2 u = *reinterpret_cast<const uint2*>(vr);
                v[0] = r_lo(u.x);
                v[1] = r_hi(u.x);
                v[2] = r_lo(u.y);
                v[3] = r_hi(u.y);
            } else {
                const uint32_t u = *reinterpret_cast<const uint32_t*>(vr);
                v[0] = r_lo(u);
                v[1] = r_hi(u);
            }
#pragma unroll
            for (int h = 0; h < kG; ++h) {
                if (h < G) {
                    const float p = ps[h * kKeysPerChunk + tt];
#pragma unroll
                    for (int x = 0; x < DL; ++x) o[h][x] = fmaf(p, v[x], o[h][x]);
                }
            }
        }
        __syncthreads();
    }
    // add the warps' sums in warp order through shared memory (ps is free)
    float* acc = ps;  // kG * D <= kG * kKeysPerChunk floats
    for (int ww = 0; ww < kRowsWarps; ++ww) {
        if (w == ww) {
#pragma unroll
            for (int h = 0; h < kG; ++h) {
                if (h < G) {
#pragma unroll
                    for (int x = 0; x < DL; ++x) {
                        float* a = acc + h * D + lane * DL + x;
                        *a = ww == 0 ? o[h][x] : *a + o[h][x];
                    }
                }
            }
        }
        __syncthreads();
    }
    for (int idx = tid; idx < G * D; idx += kRowsThreads) {
        const int h = idx / D, e = idx - h * D;
        const int col = (g * G + h) * D + e;
        split_store(acc[idx] / lrun[h], x3, i, col);
    }
    if (g == 0)  // the columns past A D up to the tensor cores' stage
        for (int col = m.A * D + tid; col < pad64(m.A * D); col += kRowsThreads) split_store(0.f, x3, i, col);
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

Parts parts(const RowsBuf& b) { return Parts{b.x3}; }

size_t attn_smem(int D) { return (size_t)kKeysPerChunk * (2 * (D / 8) + 1) * 16; }

// Row blocks of 8 a warp takes (1, 2 or 4) and the row groups of a batch.
void row_groups(int M, int& NB, int& RG) {
    const int blocks = (M + 7) / 8;
    NB = blocks <= 1 ? 1 : blocks <= 2 ? 2 : 4;
    RG = (blocks + NB - 1) / NB;
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
        return launch_pdl(k_rows_mm<1, 2>, dim3(grid), dim3(kRowsThreads), 0, s, w, (int)nt, K, parts(b), b.ldx, M, S, RG,
                          b.part, Np);
    else if (NB == 2)
        return launch_pdl(k_rows_mm<2, 2>, dim3(grid), dim3(kRowsThreads), 0, s, w, (int)nt, K, parts(b), b.ldx, M, S, RG,
                          b.part, Np);
    else
        return launch_pdl(k_rows_mm<4, 1>, dim3(grid), dim3(kRowsThreads), 0, s, w, (int)nt, K, parts(b), b.ldx, M, S, RG,
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
    cudaError_t e = cudaFuncSetAttribute(k_rows_attn<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)attn_smem(128));
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(k_rows_attn<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)attn_smem(64));
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
    return most;
}

#define RCK(x)                                    \
    do {                                          \
        cudaError_t e_ = (x);                     \
        if (e_ != cudaSuccess) return e_;         \
    } while (0)

cudaError_t rows_pass(const DevModel& m, const RowsBuf& b, const int* start, int M, int32_t* d_pos,
                      const int32_t* ids, int pos_base, bool kv_only, cudaStream_t s) {
    if (M <= 0) return cudaSuccess;
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
                       Np_prev, lw + m.off_gattn, m.eps, parts(b), b.ldx));
        RCK(launch_mm(lw + m.off_wqkv, nqkv, d, b, Mj, S, Np, s));
        const int nu = (int)(nqkv / 2);
        RCK(launch_pdl(k_rows_qkv, dim3((nu + kRowsThreads - 1) / kRowsThreads, Mj), dim3(kRowsThreads), 0, s, m, j,
                       (const float*)b.part, S, Mj, Np, (const int32_t*)d_pos, b.Q));
        if (kv_only && j == L - 1) return cudaSuccess;
        if (m.D == 128)
            RCK(launch_pdl(k_rows_attn<128>, dim3(m.KH, Mj), dim3(kRowsThreads), attn_smem(128), s, m, j,
                           (const float*)b.Q, (const int32_t*)d_pos, parts(b), b.ldx));
        else
            RCK(launch_pdl(k_rows_attn<64>, dim3(m.KH, Mj), dim3(kRowsThreads), attn_smem(64), s, m, j,
                           (const float*)b.Q, (const int32_t*)d_pos, parts(b), b.ldx));
        RCK(launch_mm(lw + m.off_wo, d, AD, b, Mj, S, Np, s));
        RCK(launch_pdl(k_rows_add_norm, dim3(Mj), dim3(kNormThreads), 0, s, b.H, d, (const float*)b.part, S, Mj, Np,
                       lw + m.off_gmlp, m.eps, parts(b), b.ldx));
        RCK(launch_mm(lw + m.off_wgu, 2LL * m.F, d, b, Mj, S, Np, s));
        RCK(launch_pdl(k_rows_swiglu, dim3((pad64(m.F) + kRowsThreads - 1) / kRowsThreads, Mj), dim3(kRowsThreads), 0, s,
                       (const float*)b.part, S, Mj, Np, m.F, parts(b), b.ldx));
        RCK(launch_mm(lw + m.off_wd, d, m.F, b, Mj, S, Np, s));
        M_prev = Mj;
        S_prev = S;
        Np_prev = Np;
    }
    // the last down projection into the residual (no norm)
    return launch_pdl(k_rows_add_norm, dim3(M_prev), dim3(kNormThreads), 0, s, b.H, d, (const float*)b.part, S_prev,
                      M_prev, Np_prev, (const uint16_t*)nullptr, m.eps, parts(b), b.ldx);
}

cudaError_t launch_rows_prefill_done(const DevModel& m, int n, cudaStream_t s) {
    return launch_pdl(k_rows_prefill_done, dim3(1), dim3(32), 0, s, m, n);
}

}  // namespace ee
