// Multi-position layer pass for sm_103a: the prompt (Section 2's prefill,
// full depth with no gate) and Section 11's full-depth re-pass of exited
// positions run each layer over a batch of up to kRowsMax positions, so a
// weight byte is read once per batch instead of once per position.
//
// A layer is nine launches, each reading what the previous one wrote:
//   k_rows_add_norm  residual add of the previous projection's split
//                    partials (in split order), then RMSNorm with the next
//                    gain, written as bf16 high and low parts
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
// same order.  Activations stay fp32 in meaning: each is split into a bf16
// high part and the bf16 rounding of the remainder, and both are multiplied
// (16 significant bits, within ~1e-5 relative of fp32).  Weights are the
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

// x as bf16 high part and the bf16 rounding of x - high.
__device__ __forceinline__ void split_store(float x, uint16_t* hi, uint16_t* lo) {
    const uint16_t h = r_f2bf(x);
    *hi = h;
    *lo = r_f2bf(x - r_bf2f(h));
}

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

__device__ __forceinline__ int64_t slot_offset(const DevModel& m, int j, int pos) {
    const int page = m.page_table[pos / m.page_size];
    const int slot = pos - (pos / m.page_size) * m.page_size;
    return (int64_t)j * m.kv_layer_stride + ((int64_t)page * m.KH * m.page_size + slot) * m.D;
}

// ------------------------------------------------------------------ projection
//
// part[s][row][n] = sum over the k of split s of W[n][k] x[row][k], for the
// M rows of x (bf16 high and low parts, row stride ldx) and every output n of
// the tiled weights.  NB blocks of 8 rows (rows past M read as zero and are
// not stored).  K splits cover whole 32-column steps; a chunk past K reads as
// zero on both sides.
template <int NB>
__global__ void __launch_bounds__(kRowsThreads) k_rows_mm(const uint4* __restrict__ W, int n_tiles, int K,
                                                          const uint16_t* __restrict__ xhi,
                                                          const uint16_t* __restrict__ xlo, int ldx, int M, int S,
                                                          float* __restrict__ part, int Np) {
    const int lane = threadIdx.x & 31, g = lane >> 2, q = lane & 3;
    const int Rc = K >> 3;             // 16-byte chunks per weight row
    const int nsteps = (Rc + 3) >> 2;  // 32-column steps
    const int units = n_tiles * S;
    const int nw = gridDim.x * kRowsWarps;
    for (int u = blockIdx.x * kRowsWarps + (threadIdx.x >> 5); u < units; u += nw) {
        const int tile = u / S, s = u - tile * S;
        const int st0 = (int)((int64_t)nsteps * s / S), st1 = (int)((int64_t)nsteps * (s + 1) / S);
        const uint4* wt = W + (int64_t)tile * Rc * 32;
        float acc[2][NB][4];
#pragma unroll
        for (int a = 0; a < 2; ++a)
#pragma unroll
            for (int n = 0; n < NB; ++n)
#pragma unroll
                for (int e = 0; e < 4; ++e) acc[a][n][e] = 0.f;
        for (int st = st0; st < st1; ++st) {
            const int ch = st * 4 + q;  // this lane's chunk of the step
            const bool ok = ch < Rc;
            uint4 w[4];
#pragma unroll
            for (int r = 0; r < 4; ++r)  // rows g, g+8, g+16, g+24 of the tile
                w[r] = ok ? ld_weights(wt + (int64_t)ch * 32 + g + 8 * r) : make_uint4(0u, 0u, 0u, 0u);
            uint4 bh[NB], bl[NB];
#pragma unroll
            for (int n = 0; n < NB; ++n) {
                const int row = n * 8 + g;
                const bool okx = ok && row < M;
                const int64_t at = (int64_t)row * ldx + ch * 8;
                bh[n] = okx ? ld_act(xhi + at) : make_uint4(0u, 0u, 0u, 0u);
                bl[n] = okx ? ld_act(xlo + at) : make_uint4(0u, 0u, 0u, 0u);
            }
#pragma unroll
            for (int n = 0; n < NB; ++n) {
                // first mma of the step: chunk elements 0..3; second: 4..7
                mma_16816(acc[0][n], w[0].x, w[1].x, w[0].y, w[1].y, bh[n].x, bh[n].y);
                mma_16816(acc[0][n], w[0].x, w[1].x, w[0].y, w[1].y, bl[n].x, bl[n].y);
                mma_16816(acc[0][n], w[0].z, w[1].z, w[0].w, w[1].w, bh[n].z, bh[n].w);
                mma_16816(acc[0][n], w[0].z, w[1].z, w[0].w, w[1].w, bl[n].z, bl[n].w);
                mma_16816(acc[1][n], w[2].x, w[3].x, w[2].y, w[3].y, bh[n].x, bh[n].y);
                mma_16816(acc[1][n], w[2].x, w[3].x, w[2].y, w[3].y, bl[n].x, bl[n].y);
                mma_16816(acc[1][n], w[2].z, w[3].z, w[2].w, w[3].w, bh[n].z, bh[n].w);
                mma_16816(acc[1][n], w[2].z, w[3].z, w[2].w, w[3].w, bl[n].z, bl[n].w);
            }
        }
        // accumulator e of block (a, n): output row tile*32 + a*16 + g (+8 for
        // e >= 2), batch row n*8 + 2q (+1 for odd e)
        float* ps = part + (int64_t)s * M * Np;
#pragma unroll
        for (int a = 0; a < 2; ++a)
#pragma unroll
            for (int n = 0; n < NB; ++n)
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const int row = n * 8 + 2 * q + (e & 1);
                    const int out = tile * 32 + a * 16 + g + (e >> 1) * 8;
                    if (row < M) ps[(int64_t)row * Np + out] = acc[a][n][e];
                }
    }
}

// ------------------------------------------------------------------ per-row epilogues

// Sum over the block; every thread gets the same value (fixed order).
__device__ __forceinline__ float r_block_sum(float v, float* red) {
    v = r_warp_sum(v);
    const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
    __syncthreads();
    if (l == 0) red[w] = v;
    __syncthreads();
    float t = l < kRowsWarps ? red[l] : 0.f;
    return r_warp_sum(t);
}

// One CTA per row i < M_norm.  Rows below M_add first add the split partials
// of a d-output projection (split stride M_add rows) to their residual.  With
// a gain, the row's RMSNorm h / sqrt(mean(h^2) + eps) * g goes to x as bf16
// high and low parts.
__global__ void __launch_bounds__(kRowsThreads) k_rows_add_norm(float* __restrict__ H, int d,
                                                                const float* __restrict__ part, int S, int M_add,
                                                                int Np, const uint16_t* __restrict__ gain, float eps,
                                                                uint16_t* __restrict__ xhi, uint16_t* __restrict__ xlo,
                                                                int ldx) {
    __shared__ float red[kRowsWarps];
    const int i = blockIdx.x;
    float* h = H + (int64_t)i * d;
    float ss = 0.f;
    for (int n = threadIdx.x; n < d; n += kRowsThreads) {
        float v = h[n];
        if (i < M_add) {
            float a = 0.f;
            for (int s = 0; s < S; ++s) a += part[((int64_t)s * M_add + i) * Np + n];
            v += a;
            h[n] = v;
        }
        ss = fmaf(v, v, ss);
    }
    if (!gain) return;  // uniform over the block
    ss = r_block_sum(ss, red);
    const float inv = 1.0f / sqrtf(ss / (float)d + eps);
    for (int n = threadIdx.x; n < d; n += kRowsThreads) {
        const float x = h[n] * inv * r_bf2f(gain[n]);
        split_store(x, xhi + (int64_t)i * ldx + n, xlo + (int64_t)i * ldx + n);
    }
}

// Q/K/V of layer j for row blockIdx.y: thread = one unit (the packed row pair
// i, i + D/2 of one head; Q heads, then K, then V).  Split sum, bias, RoPE at
// the row's position; q stays fp32, k and v go to the cache as bf16.
__global__ void __launch_bounds__(kRowsThreads) k_rows_qkv(DevModel m, int j, const float* __restrict__ part,
                                                           int S, int M, int Np, const int32_t* __restrict__ pos,
                                                           float* __restrict__ Q) {
    const int i = blockIdx.y;
    const int u = blockIdx.x * kRowsThreads + threadIdx.x;
    const int half = m.D >> 1;
    const int nq = m.A * half, nk = m.KH * half;
    if (u >= nq + 2 * nk) return;
    float r0 = 0.f, r1 = 0.f;
    for (int s = 0; s < S; ++s) {
        const float* p = part + ((int64_t)s * M + i) * Np + 2 * u;
        r0 += p[0];
        r1 += p[1];
    }
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
// packed (gate, up) row pair, as bf16 high and low parts.
__global__ void __launch_bounds__(kRowsThreads) k_rows_swiglu(const float* __restrict__ part, int S, int M, int Np,
                                                              int F, uint16_t* __restrict__ xhi,
                                                              uint16_t* __restrict__ xlo, int ldx) {
    const int i = blockIdx.y;
    const int f = blockIdx.x * kRowsThreads + threadIdx.x;
    if (f >= F) return;
    float gs = 0.f, us = 0.f;
    for (int s = 0; s < S; ++s) {
        const float* p = part + ((int64_t)s * M + i) * Np + 2 * f;
        gs += p[0];
        us += p[1];
    }
    const float a = gs / (1.0f + expf(-gs)) * us;
    split_store(a, xhi + (int64_t)i * ldx + f, xlo + (int64_t)i * ldx + f);
}

// Starting residual of row blockIdx.x: the embedding of ids[i] (a prompt;
// the row's position pos_base + i is recorded in pos) or the residual its
// position exited with.
__global__ void __launch_bounds__(kRowsThreads) k_rows_init(DevModel m, float* __restrict__ H, int32_t* pos,
                                                            const int32_t* __restrict__ ids, int pos_base) {
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
    if (threadIdx.x != 0) return;
    Ctl* c = m.ctl;
    c->pos = n;
    c->prefill_i = n;
    c->exit_readout = -1;
    c->n_evaluated = 0;
    c->full_token = -1;
    c->nucleus_member = -1;
}

// Causal attention of row blockIdx.y and kv head blockIdx.x over cache
// positions 0..pos[i] of layer j, for the head group's G query heads: keys
// in chunks of one per thread, a running maximum and sum per head, the
// output rescaled with each new maximum (the result is Section 2's softmax
// attention).  Output o at column h*D + e as bf16 high and low parts.
__global__ void __launch_bounds__(kRowsThreads) k_rows_attn(DevModel m, int j, const float* __restrict__ Q,
                                                            const int32_t* __restrict__ pos,
                                                            uint16_t* __restrict__ xhi, uint16_t* __restrict__ xlo,
                                                            int ldx) {
    constexpr int kG = kSegMaxGroup;             // query heads per kv head (at most)
    constexpr int kOut = kG * 128 / kRowsThreads;  // outputs per thread (at most)
    __shared__ float qs[kG * 128];
    __shared__ float ps[kG * kKeysPerChunk];
    __shared__ int64_t offs[kKeysPerChunk];
    __shared__ float redm[kRowsWarps][kG], reds[kRowsWarps][kG];
    __shared__ float mrun[kG], lrun[kG], resc[kG];
    const int g = blockIdx.x, i = blockIdx.y, D = m.D, G = m.A / m.KH;
    const int tid = threadIdx.x, lane = tid & 31, w = tid >> 5;
    const int T = pos[i] + 1;
    const float scale = 1.0f / sqrtf((float)D);
    const float* qrow = Q + (int64_t)i * m.A * D + (int64_t)g * G * D;
    for (int x = tid; x < G * D; x += kRowsThreads) qs[x] = qrow[x] * scale;
    if (tid < kG) {
        mrun[tid] = -INFINITY;
        lrun[tid] = 0.f;
    }
    float o[kOut];
#pragma unroll
    for (int k = 0; k < kOut; ++k) o[k] = 0.f;
    const int64_t head_off = (int64_t)g * m.page_size * D;
    __syncthreads();
    for (int c0 = 0; c0 < T; c0 += kKeysPerChunk) {
        const int t = c0 + tid;
        const bool valid = t < T;
        const int64_t off = valid ? slot_offset(m, j, t) + head_off : 0;
        offs[tid] = off;
        float sc[kG];
#pragma unroll
        for (int h = 0; h < kG; ++h) sc[h] = 0.f;
        if (valid) {
            const uint16_t* kr = m.kpool + off;
            for (int c = 0; c < D; c += 8) {
                const uint4 kv = *reinterpret_cast<const uint4*>(kr + c);
                const float kf[8] = {r_lo(kv.x), r_hi(kv.x), r_lo(kv.y), r_hi(kv.y),
                                     r_lo(kv.z), r_hi(kv.z), r_lo(kv.w), r_hi(kv.w)};
#pragma unroll
                for (int h = 0; h < kG; ++h) {
                    if (h < G) {
                        const float* qh = qs + h * D + c;
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
        const int nk = min(kKeysPerChunk, T - c0);
#pragma unroll
        for (int k = 0; k < kOut; ++k) {
            const int idx = tid + kRowsThreads * k;
            if (idx < G * D) {
                const int h = idx / D, e = idx - h * D;
                const float* ph = ps + h * kKeysPerChunk;
                float a = o[k] * resc[h];
                for (int tt = 0; tt < nk; ++tt) a = fmaf(ph[tt], r_bf2f(m.vpool[offs[tt] + e]), a);
                o[k] = a;
            }
        }
        __syncthreads();
    }
#pragma unroll
    for (int k = 0; k < kOut; ++k) {
        const int idx = tid + kRowsThreads * k;
        if (idx < G * D) {
            const int h = idx / D, e = idx - h * D;
            const int64_t col = (int64_t)(g * G + h) * D + e;
            split_store(o[k] / lrun[h], xhi + (int64_t)i * ldx + col, xlo + (int64_t)i * ldx + col);
        }
    }
}

// ------------------------------------------------------------------ host side

// One projection of the batch: W (n_rows x K, tiled) times the M rows of
// b.xhi / b.xlo into b.part; returns the split count and padded row count
// its consumer needs.
cudaError_t launch_mm(const uint16_t* W, int64_t n_rows, int K, const RowsBuf& b, int M, int& S, int& Np,
                      cudaStream_t s) {
    const int64_t nt = tile_count(n_rows);
    S = rows_splits(nt, K, M);
    Np = (int)(nt * kTileRows);
    const int64_t units = nt * S;
    const int grid = (int)std::min<int64_t>((units + kRowsWarps - 1) / kRowsWarps, 65535);
    const uint4* w = reinterpret_cast<const uint4*>(W);
    const int nb = (M + 7) / 8;
    if (nb <= 1)
        k_rows_mm<1><<<grid, kRowsThreads, 0, s>>>(w, (int)nt, K, b.xhi, b.xlo, b.ldx, M, S, b.part, Np);
    else if (nb <= 2)
        k_rows_mm<2><<<grid, kRowsThreads, 0, s>>>(w, (int)nt, K, b.xhi, b.xlo, b.ldx, M, S, b.part, Np);
    else if (nb <= 4)
        k_rows_mm<4><<<grid, kRowsThreads, 0, s>>>(w, (int)nt, K, b.xhi, b.xlo, b.ldx, M, S, b.part, Np);
    else
        k_rows_mm<8><<<grid, kRowsThreads, 0, s>>>(w, (int)nt, K, b.xhi, b.xlo, b.ldx, M, S, b.part, Np);
    return cudaGetLastError();
}

}  // namespace

// Enough (tile, split) units to give every warp slot of the GPU one, each at
// least one 32-column step, and split partials (written and read once) at
// most half the weight bytes: S * M * 4 B * 2 <= K * 2 B / 2.
int rows_splits(int64_t n_tiles, int K, int M) {
    const int nsteps = ((K >> 3) + 3) >> 2;
    const int Mp = std::max(8, (M + 7) & ~7);
    int S = (int)((kRowsTargetUnits + n_tiles - 1) / n_tiles);
    S = std::min(S, std::max(1, K / (8 * Mp)));
    S = std::min(S, nsteps);
    return std::max(S, 1);
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
    k_rows_init<<<M, kRowsThreads, 0, s>>>(m, b.H, d_pos, ids, pos_base);
    RCK(cudaGetLastError());
    int M_prev = 0, S_prev = 1, Np_prev = 0;
    for (int j = start[0]; j < L; ++j) {
        int Mj = M_prev;
        while (Mj < M && start[Mj] <= j) ++Mj;
        const uint16_t* lw = m.layers + (int64_t)j * m.layer_stride;
        int S = 1, Np = 0;
        // the previous layer's down projection into the residual, this layer's input norm
        k_rows_add_norm<<<Mj, kRowsThreads, 0, s>>>(b.H, d, b.part, S_prev, M_prev, Np_prev, lw + m.off_gattn, m.eps,
                                                     b.xhi, b.xlo, b.ldx);
        RCK(cudaGetLastError());
        RCK(launch_mm(lw + m.off_wqkv, nqkv, d, b, Mj, S, Np, s));
        const int nu = (int)(nqkv / 2);
        k_rows_qkv<<<dim3((nu + kRowsThreads - 1) / kRowsThreads, Mj), kRowsThreads, 0, s>>>(m, j, b.part, S, Mj, Np,
                                                                                             d_pos, b.Q);
        RCK(cudaGetLastError());
        if (kv_only && j == L - 1) return cudaSuccess;
        k_rows_attn<<<dim3(m.KH, Mj), kRowsThreads, 0, s>>>(m, j, b.Q, d_pos, b.xhi, b.xlo, b.ldx);
        RCK(cudaGetLastError());
        RCK(launch_mm(lw + m.off_wo, d, AD, b, Mj, S, Np, s));
        k_rows_add_norm<<<Mj, kRowsThreads, 0, s>>>(b.H, d, b.part, S, Mj, Np, lw + m.off_gmlp, m.eps, b.xhi, b.xlo,
                                                     b.ldx);
        RCK(cudaGetLastError());
        RCK(launch_mm(lw + m.off_wgu, 2LL * m.F, d, b, Mj, S, Np, s));
        k_rows_swiglu<<<dim3((m.F + kRowsThreads - 1) / kRowsThreads, Mj), kRowsThreads, 0, s>>>(b.part, S, Mj, Np, m.F,
                                                                                                 b.xhi, b.xlo, b.ldx);
        RCK(cudaGetLastError());
        RCK(launch_mm(lw + m.off_wd, d, m.F, b, Mj, S, Np, s));
        M_prev = Mj;
        S_prev = S;
        Np_prev = Np;
    }
    // the last down projection into the residual (no norm)
    k_rows_add_norm<<<M_prev, kRowsThreads, 0, s>>>(b.H, d, b.part, S_prev, M_prev, Np_prev, nullptr, m.eps, b.xhi,
                                                    b.xlo, b.ldx);
    return cudaGetLastError();
}

cudaError_t launch_rows_prefill_done(const DevModel& m, int n, cudaStream_t s) {
    k_rows_prefill_done<<<1, 32, 0, s>>>(m, n);
    return cudaGetLastError();
}

}  // namespace ee
