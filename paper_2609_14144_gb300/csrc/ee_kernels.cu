// sm_103a kernels of the confidence-gated early-exit decode step.
//
// Batch-1 decode is a chain of M = 1 matrix-vector products: about one flop
// per weight byte, so every kernel here is bound by HBM bandwidth, not by the
// tensor cores.  The design goals are therefore (1) every weight byte read
// once, with 16-byte coalesced loads and enough of them in flight,
// (2) perfect balance across the 152 SMs, and (3) no launch-gap bubbles
// (programmatic dependent launch: each kernel prefetches its weights into L2
// before it waits for its predecessor's activations).
//
// The streaming GEMV core ("flat GEMV"): a weight matrix of n_units units,
// each NR rows of K bf16 values stored contiguously, is viewed as one array
// of 16-byte chunks.  Every warp owns an equal contiguous slice of that array
// (or, in the row-aligned variant, an equal run of whole units).  Lanes read
// consecutive chunks (512 bytes per warp instruction), multiply by the
// activation vector held in shared memory as fp32, and keep one running sum
// per lane; a warp reduction closes each row.  Units cut by a slice boundary
// are finished by whichever contributing warp arrives last, summing the
// contributions in warp order, so results do not depend on timing.
#include <algorithm>
#include <cooperative_groups.h>
#include <cuda_bf16.h>
#include <math.h>
#include <math_constants.h>

#include "ee_internal.h"
#include "ee_vocab.cuh"

namespace ee {

// ------------------------------------------------------------------ helpers

__device__ __forceinline__ float bf_lo(uint32_t u) { return __uint_as_float(u << 16); }
__device__ __forceinline__ float bf_hi(uint32_t u) { return __uint_as_float(u & 0xffff0000u); }
__device__ __forceinline__ float bf2f(uint16_t b) { return __uint_as_float((uint32_t)b << 16); }
__device__ __forceinline__ uint16_t f2bf(float f) { return __bfloat16_as_ushort(__float2bfloat16_rn(f)); }

// L2 policy for data read once per step (weights): its lines are the first
// evicted, so the streamed matrices do not push out the KV cache and the
// activations.  (Not volatile: a pure value the compiler may hoist.)
__device__ __forceinline__ uint64_t l2_evict_first_policy() {
    uint64_t pol;
    asm("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
    return pol;
}
// Streaming 16-byte load of read-only weights: no L1 allocation, 256-byte
// L2 sector promotion, evict-first in L2.
__device__ __forceinline__ uint4 ldg_stream(const uint4* p) {
    uint4 r;
    asm volatile("ld.global.nc.L1::no_allocate.L2::cache_hint.L2::256B.v4.u32 {%0,%1,%2,%3}, [%4], %5;"
        : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
        : "l"(p), "l"(l2_evict_first_policy()));
    return r;
}

__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_launch_dependents() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

__device__ __forceinline__ void prefetch_l2(const void* p, uint32_t bytes) {
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p), "r"(bytes) : "memory");
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// Sum over the block; every thread gets the same value (fixed order).
__device__ __forceinline__ float block_sum(float v, float* red) {
    v = warp_sum(v);
    const int w = threadIdx.x >> 5, l = threadIdx.x & 31, nw = blockDim.x >> 5;
    __syncthreads();
    if (l == 0) red[w] = v;
    __syncthreads();
    float t = (l < nw) ? red[l] : 0.f;
    return warp_sum(t);
}

// x = src / sqrt(mean(src^2) + eps) * g, fp32 statistics, into smem.
__device__ __forceinline__ void rmsnorm_to_smem(const float* src, const uint16_t* g, int d, float eps, float* x,
                                                float* red) {
    float ss = 0.f;
    for (int i = threadIdx.x; i < d; i += blockDim.x) {
        const float v = src[i];
        ss = fmaf(v, v, ss);
    }
    ss = block_sum(ss, red);
    const float inv = 1.0f / sqrtf(ss / (float)d + eps);
    for (int i = threadIdx.x; i < d; i += blockDim.x) x[i] = src[i] * inv * bf2f(g[i]);
    __syncthreads();
}

// Dot product of 8 packed bf16 weights with 8 fp32 activations.
__device__ __forceinline__ float dot8(const uint4 w, const float* x) {
    const float4 a = *reinterpret_cast<const float4*>(x);
    const float4 b = *reinterpret_cast<const float4*>(x + 4);
    float s = bf_lo(w.x) * a.x;
    s = fmaf(bf_hi(w.x), a.y, s);
    s = fmaf(bf_lo(w.y), a.z, s);
    s = fmaf(bf_hi(w.y), a.w, s);
    s = fmaf(bf_lo(w.z), b.x, s);
    s = fmaf(bf_hi(w.z), b.y, s);
    s = fmaf(bf_lo(w.w), b.z, s);
    s = fmaf(bf_hi(w.w), b.w, s);
    return s;
}

// Chunk range [c0, c1) of `warp` out of `nwarps` over n_units units of Cu chunks.
template <bool ALIGNED>
__device__ __forceinline__ void warp_range(int64_t n_units, int64_t Cu, int warp, int nwarps, int64_t& c0,
                                           int64_t& c1) {
    if (ALIGNED) {
        c0 = (n_units * warp / nwarps) * Cu;
        c1 = (n_units * (warp + 1) / nwarps) * Cu;
    } else {
        const int64_t Ct = n_units * Cu;
        c0 = Ct * warp / nwarps;
        c1 = Ct * (warp + 1) / nwarps;
    }
}

// The flat GEMV core (see the file comment).  Epi is called by lane 0 with
// the unit index and its NR row sums.  Requires K % 8 == 0 and K >= 256.
template <int NR, bool ALIGNED, int U, class Epi>
__device__ __forceinline__ void flat_gemv(const uint16_t* __restrict__ W, int K, int64_t n_units,
                                          const float* __restrict__ xs, int warp, int nwarps,
                                          float* __restrict__ part, int* __restrict__ ticket, Epi& epi) {
    const int lane = threadIdx.x & 31;
    const int Rc = K >> 3;
    const int64_t Cu = (int64_t)NR * Rc;
    const int64_t Ct = n_units * Cu;
    int64_t c0, c1;
    warp_range<ALIGNED>(n_units, Cu, warp, nwarps, c0, c1);
    if (c0 >= c1) return;
    const uint4* Wc = reinterpret_cast<const uint4*>(W);

    int64_t row = c0 / Rc;
    int o0 = (int)(c0 - row * Rc);  // offset of lane 0's chunk inside `row`, in [0, Rc)
    int col = o0 + lane;            // offset of this lane's chunk inside its row
    if (col >= Rc) col -= Rc;
    float acc = 0.f;
    float rs[NR];
#pragma unroll
    for (int r = 0; r < NR; ++r) rs[r] = 0.f;

    auto owner = [&](int64_t c) -> int64_t { return ((c + 1) * (int64_t)nwarps - 1) / Ct; };

    auto finish_row = [&](int64_t rw, float s) {
        const int64_t unit = rw / NR;
        const int ri = (int)(rw - unit * NR);
#pragma unroll
        for (int r = 0; r < NR; ++r)
            if (r == ri) rs[r] = s;
        if (ri == NR - 1 || (rw + 1) * Rc >= c1) {
            const bool whole = ALIGNED || (unit * Cu >= c0 && (unit + 1) * Cu <= c1);
            if (lane == 0) {
                if (whole) {
                    epi(unit, rs);
                } else {
                    const bool first = unit * Cu < c0;
                    const int64_t slot = (int64_t)warp * 2 + (first ? 0 : 1);
#pragma unroll
                    for (int r = 0; r < NR; ++r) part[slot * NR + r] = rs[r];
                    __threadfence();
                    const int64_t wa = owner(unit * Cu), wb = owner((unit + 1) * Cu - 1);
                    const int n = (int)(wb - wa + 1);
                    const int old = atomicAdd(&ticket[unit], 1);
                    if (old == n - 1) {
                        __threadfence();
                        float sum[NR];
#pragma unroll
                        for (int r = 0; r < NR; ++r) sum[r] = __ldcg(&part[(wa * 2 + 1) * NR + r]);
                        for (int64_t w = wa + 1; w <= wb; ++w)
#pragma unroll
                            for (int r = 0; r < NR; ++r) sum[r] += __ldcg(&part[(w * 2) * NR + r]);
                        epi(unit, sum);
                        ticket[unit] = 0;
                    }
                }
            }
#pragma unroll
            for (int r = 0; r < NR; ++r) rs[r] = 0.f;
        }
    };

    for (int64_t g = c0; g < c1; g += 32 * U) {
        uint4 w[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int64_t c = g + 32 * u + lane;
            w[u] = (c < c1) ? ldg_stream(Wc + c) : make_uint4(0u, 0u, 0u, 0u);
        }
#pragma unroll
        for (int u = 0; u < U; ++u) {
            if (g + 32 * u >= c1) break;
            const float v = dot8(w[u], xs + col * 8);
            const int b = Rc - o0;  // first lane that belongs to the next row
            if (b < 32) {
                acc += (lane < b) ? v : 0.f;
                finish_row(row, warp_sum(acc));
                acc = (lane >= b) ? v : 0.f;
                ++row;
                o0 += 32 - Rc;
            } else {
                acc += v;
                o0 += 32;
                if (o0 == Rc) {
                    finish_row(row, warp_sum(acc));
                    acc = 0.f;
                    ++row;
                    o0 = 0;
                }
            }
            col += 32;
            if (col >= Rc) col -= Rc;
        }
    }
    if (row * Rc < c1) finish_row(row, warp_sum(acc));
}

__device__ __forceinline__ void cp_async16(void* smem, const void* gmem) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"((uint32_t)__cvta_generic_to_shared(smem)),
                 "l"(gmem)
                 : "memory");
}
// Weight copy that marks its L2 line first to be evicted (read once per step).
__device__ __forceinline__ void cp_async16_stream(void* smem, const void* gmem, uint64_t pol) {
    asm volatile("cp.async.cg.shared.global.L2::cache_hint [%0], [%1], 16, %2;"
                 ::"r"((uint32_t)__cvta_generic_to_shared(smem)), "l"(gmem), "l"(pol)
                 : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_all;" ::: "memory"); }

// Distributed shared memory: the address of a shared-memory location in the
// CTA of cluster rank `rank`, and a load from it.
__device__ __forceinline__ uint32_t dsmem_rank(uint32_t smem_addr, uint32_t rank) {
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(smem_addr), "r"(rank));
    return r;
}
__device__ __forceinline__ uint32_t dsmem_addr(const void* p, uint32_t rank) {
    return dsmem_rank((uint32_t)__cvta_generic_to_shared(p), rank);
}
__device__ __forceinline__ float ld_dsmem(uint32_t addr) {
    float v;
    asm volatile("ld.shared::cluster.f32 %0, [%1];" : "=f"(v) : "r"(addr) : "memory");
    return v;
}

// ------------------------------------------------------------------ tiled GEMV
//
// Engine weights are repacked into tiles of 32 rows: for each 16-byte column
// chunk c, the 32 rows' chunks are stored back to back (512 bytes), so one
// warp instruction streams 512 contiguous bytes and lane r owns row r of the
// tile: it accumulates that row's dot product on its own, and the activation
// chunk it multiplies is the same for every lane (a shared-memory broadcast).
// Element (row, k) of an n_rows x K matrix lives at
//     ((tile * Rc + c) * 32 + r) * 8 + e,   tile = row / 32, r = row % 32,
//     c = k / 8, e = k % 8, Rc = K / 8;   rows past n_rows are zero padding.
// An "item" is one (tile, c) pair; a matrix is n_tiles * Rc items.

constexpr int kWarps = kGemvThreads / 32;  // warps per GEMV CTA
constexpr int kSlotTiles = kGemvSlotTiles;  // tiles one CTA may touch
constexpr int kWindow = 8;                 // loads each lane issues per batch

// The items of one CTA: [C0, C1) of Ct, an equal share of the matrix
// (item counts fit in 32 bits: the engine checks).
struct CoopRange {
    int C0, C1, Ct;
    int Rc, cta, n_cta;
};

__device__ __forceinline__ CoopRange coop_range(int64_t n_tiles, int K, int cta, int n_cta) {
    CoopRange r;
    r.Rc = K >> 3;
    r.Ct = (int)(n_tiles * r.Rc);
    r.C0 = (int)((int64_t)r.Ct * cta / n_cta);
    r.C1 = (int)((int64_t)r.Ct * (cta + 1) / n_cta);
    r.cta = cta;
    r.n_cta = n_cta;
    return r;
}

// Warp w of the CTA consumes items C0 + w, C0 + w + 16, ...; the first
// kWindow of them are loaded here (before the kernel waits on its
// predecessor: weights never depend on it).
__device__ __forceinline__ void coop_prefetch(const uint4* W, const CoopRange& r, uint4 (&buf)[kWindow]) {
    const int lane = threadIdx.x & 31, wl = threadIdx.x >> 5;
#pragma unroll
    for (int u = 0; u < kWindow; ++u) {
        const int it = r.C0 + wl + kWarps * u;
        buf[u] = it < r.C1 ? ldg_stream(W + (int64_t)it * 32 + lane) : make_uint4(0u, 0u, 0u, 0u);
    }
}

// Stream the CTA's items against x (fp32 in shared memory), leaving each
// warp's share of every tile it touched in sm_part[tile][warp][lane], then
// synchronise the CTA.  Loads go in batches of kWindow issued back to back
// before any is used (the first batch was issued by coop_prefetch).  Returns
// false (before touching anything) if the CTA would touch more than
// kSlotTiles tiles.
__device__ __forceinline__ bool coop_stream(const uint4* __restrict__ W, const CoopRange& r,
                                            uint4 (&buf)[kWindow], const float* __restrict__ xs,
                                            float* __restrict__ sm_part) {
    const int lane = threadIdx.x & 31, wl = threadIdx.x >> 5;
    const int t_first = r.C0 / r.Rc, t_last = (r.C1 - 1) / r.Rc;
    if (t_last - t_first + 1 > kSlotTiles) return false;
    const int it = r.C0 + wl;
    int slot = it / r.Rc - t_first;
    int c = it - (slot + t_first) * r.Rc;
    float acc = 0.f;
    bool pending = false;
    for (int base = it; base < r.C1; base += kWarps * kWindow) {
        if (base != it) {
#pragma unroll
            for (int u = 0; u < kWindow; ++u) {
                const int cur = base + kWarps * u;
                buf[u] = cur < r.C1 ? ldg_stream(W + (int64_t)cur * 32 + lane) : make_uint4(0u, 0u, 0u, 0u);
            }
        }
#pragma unroll
        for (int u = 0; u < kWindow; ++u) {
            if (base + kWarps * u >= r.C1) break;
            acc += dot8(buf[u], xs + c * 8);
            pending = true;
            c += kWarps;
            if (c >= r.Rc) {
                sm_part[(slot * kWarps + wl) * 32 + lane] = acc;
                acc = 0.f;
                pending = false;
                c -= r.Rc;
                ++slot;
            }
        }
    }
    if (pending) sm_part[(slot * kWarps + wl) * 32 + lane] = acc;
    __syncthreads();
    return true;
}

// Combine a tile shared by several CTAs: each contributor leaves its
// 32 row sums in its slot; the last to arrive sums them in CTA order and
// runs the epilogue.  kind 0: the tile began before this CTA's range;
// kind 1: it began inside and runs past the end.
template <class Epi>
__device__ __forceinline__ void cross_cta_combine(const CoopRange& r, int tile, float s, int kind, float* g_part,
                                                  int slot_base, unsigned* ticket, const Epi& epi) {
    const int lane = threadIdx.x & 31;
    g_part[((int64_t)(slot_base + r.cta) * 2 + kind) * 32 + lane] = s;
    __threadfence();
    __syncwarp();
    unsigned old = 0;
    if (lane == 0) old = atomicAdd(&ticket[tile], 1u);
    old = __shfl_sync(0xffffffffu, old, 0);
    auto owner = [&](int64_t it) -> int { return (int)(((it + 1) * (int64_t)r.n_cta - 1) / r.Ct); };
    const int ca = owner((int64_t)tile * r.Rc), cb = owner((int64_t)(tile + 1) * r.Rc - 1);
    if ((int)old != cb - ca) return;
    __threadfence();
    float v = __ldcg(&g_part[((int64_t)(slot_base + ca) * 2 + 1) * 32 + lane]);
    for (int c = ca + 1; c <= cb; ++c) v += __ldcg(&g_part[((int64_t)(slot_base + c) * 2 + 0) * 32 + lane]);
    epi(tile, v);
    if (lane == 0) ticket[tile] = 0;
}

// Finish every tile the CTA touched (after coop_stream): sum the warps'
// shares in warp order; whole tiles run the epilogue here, tiles shared with
// a neighbouring CTA go through cross_cta_combine.
template <class Epi>
__device__ __forceinline__ void coop_finish(const CoopRange& r, const float* __restrict__ sm_part, float* g_part,
                                            int slot_base, unsigned* ticket, const Epi& epi) {
    const int lane = threadIdx.x & 31, wl = threadIdx.x >> 5;
    const int t_first = r.C0 / r.Rc, t_last = (r.C1 - 1) / r.Rc;
    for (int tt = t_first + wl; tt <= t_last; tt += kWarps) {
        float s = 0.f;
#pragma unroll
        for (int w = 0; w < kWarps; ++w) s += sm_part[((tt - t_first) * kWarps + w) * 32 + lane];
        const bool head = tt * r.Rc < r.C0, tail = (tt + 1) * r.Rc > r.C1;
        if (!head && !tail)
            epi(tt, s);
        else
            cross_cta_combine(r, tt, s, head ? 0 : 1, g_part, slot_base, ticket, epi);
    }
}

// Zero the per-warp tile partials (they must start at zero: a warp may not
// touch every tile of its CTA).
__device__ __forceinline__ void zero_sm_part(float* sm_part) {
    for (int i = threadIdx.x; i < kSlotTiles * kWarps * 32; i += blockDim.x) sm_part[i] = 0.f;
}

// Whole-tile mode (one CTA per tile, small matrices): the CTA's tile is
// copied into shared memory with cp.async before the kernel waits on its
// predecessor, so after the wait only the activation vector is fetched.
// The streaming mode (coop_prefetch / coop_stream) serves the rest.
template <bool WHOLE>
struct GemvFront {
    CoopRange r;
    uint4 buf[kWindow];
    __device__ __forceinline__ void begin(const uint4* W, int64_t n_tiles, int K, uint4* tile_sm) {
        if (WHOLE) {
            r.Rc = K >> 3;
            r.Ct = (int)(n_tiles * r.Rc);
            r.C0 = blockIdx.x * r.Rc;
            r.C1 = r.C0 + r.Rc;
            r.cta = blockIdx.x;
            r.n_cta = gridDim.x;
            const uint4* src = W + (int64_t)r.C0 * 32;
            const uint64_t pol = l2_evict_first_policy();
            for (int i = threadIdx.x; i < r.Rc * 32; i += blockDim.x) cp_async16_stream(tile_sm + i, src + i, pol);
            cp_async_commit();
        } else {
            r = coop_range(n_tiles, K, blockIdx.x, gridDim.x);
            coop_prefetch(W, r, buf);
        }
    }
    // Leaves each warp's share of the CTA's tiles in sm_part and synchronises.
    __device__ __forceinline__ bool stream(const uint4* W, const float* xs, float* sm_part, const uint4* tile_sm) {
        if (!WHOLE) return coop_stream(W, r, buf, xs, sm_part);
        const int lane = threadIdx.x & 31, wl = threadIdx.x >> 5;
        cp_async_wait_all();
        __syncthreads();
        float acc = 0.f;
        for (int it = wl; it < r.Rc; it += kWarps) acc += dot8(tile_sm[it * 32 + lane], xs + it * 8);
        sm_part[wl * 32 + lane] = acc;
        __syncthreads();
        return true;
    }
    // Columns [lo, hi) of x this CTA multiplies (all of them when the range
    // wraps or covers a whole row).
    __device__ __forceinline__ void x_range(int K, int& lo, int& hi) const {
        if (WHOLE || r.C1 - r.C0 >= r.Rc) {
            lo = 0;
            hi = K;
            return;
        }
        const int a = r.C0 % r.Rc, b = (r.C1 - 1) % r.Rc;
        if (a <= b) {
            lo = a * 8;
            hi = b * 8 + 8;
        } else {
            lo = 0;
            hi = K;
        }
    }
};

// Shared-memory pointer of the staged tile: after x, the tile partials and
// `extra` floats.
__device__ __forceinline__ uint4* sm_tile(float* xs, int K, int extra) {
    return reinterpret_cast<uint4*>(xs + ((K + 3) & ~3) + kSlotTiles * kWarps * 32 + extra);
}

// ------------------------------------------------------------------ epilogues
// Called by all 32 lanes of a warp with the tile index and lane's row sum.

// Q/K/V tile: 16 units of a row pair (i, i + D/2) of one head, first row on
// the even lane.  Q is rotated and kept in fp32; K is rotated and V copied
// into the paged cache as bf16.
struct EpiQKV {
    float* q;
    uint16_t* kdst;       // this layer's page slot, kv head 0
    uint16_t* vdst;
    int64_t head_stride;  // elements between kv heads inside a page
    const uint16_t* bias; // packed [unit][2] or null
    const float2* cs;     // rope row of this position
    int64_t unit_offset;  // unit index of the tile-0 unit
    int D, nq_units, nk_units;
    __device__ __forceinline__ void operator()(int64_t tile, float s) const {
        const int lane = threadIdx.x & 31, odd = lane & 1;
        const int64_t u = tile * 16 + (lane >> 1) + unit_offset;
        if (bias) s += bf2f(bias[2 * u + odd]);
        const float other = __shfl_xor_sync(0xffffffffu, s, 1);
        const float r0 = odd ? other : s, r1 = odd ? s : other;
        const int half = D >> 1;
        if (u < nq_units) {
            const int h = (int)(u / half), i = (int)(u - (int64_t)h * half);
            const float2 c = cs[i];
            if (!odd)
                q[h * D + i] = r0 * c.x - r1 * c.y;
            else
                q[h * D + i + half] = r0 * c.y + r1 * c.x;
        } else if (u < nq_units + nk_units) {
            const int64_t uu = u - nq_units;
            const int g = (int)(uu / half), i = (int)(uu - (int64_t)g * half);
            const float2 c = cs[i];
            uint16_t* k = kdst + g * head_stride;
            if (!odd)
                k[i] = f2bf(r0 * c.x - r1 * c.y);
            else
                k[i + half] = f2bf(r0 * c.y + r1 * c.x);
        } else {
            const int64_t uu = u - nq_units - nk_units;
            const int g = (int)(uu / half), i = (int)(uu - (int64_t)g * half);
            uint16_t* v = vdst + g * head_stride;
            if (!odd)
                v[i] = f2bf(r0);
            else
                v[i + half] = f2bf(r1);
        }
    }
};

// Residual add: h[row] += s.
struct EpiAddH {
    float* h;
    int n_rows;
    __device__ __forceinline__ void operator()(int64_t tile, float s) const {
        const int64_t row = tile * 32 + (threadIdx.x & 31);
        if (row < n_rows) h[row] += s;
    }
};

// Readout affine map: y[row] = s + b[row].
struct EpiBias {
    float* y;
    const uint16_t* b;
    int n_rows;
    __device__ __forceinline__ void operator()(int64_t tile, float s) const {
        const int64_t row = tile * 32 + (threadIdx.x & 31);
        if (row < n_rows) y[row] = s + bf2f(b[row]);
    }
};

// Gated FFN tile: 16 units (gate row on the even lane, up row on the odd).
struct EpiSwiGLU {
    float* a;
    int F;
    __device__ __forceinline__ void operator()(int64_t tile, float s) const {
        const int lane = threadIdx.x & 31;
        const float up = __shfl_xor_sync(0xffffffffu, s, 1);
        const int64_t u = tile * 16 + (lane >> 1);
        if (!(lane & 1) && u < F) a[u] = s / (1.0f + expf(-s)) * up;
    }
};


__device__ __forceinline__ const uint16_t* layer_base(const DevModel& m, int j) {
    return m.layers + (int64_t)j * m.layer_stride;
}

__device__ __forceinline__ int64_t kv_slot_offset(const DevModel& m, int j, int pos) {
    const int page = m.page_table[pos / m.page_size];
    const int slot = pos - (pos / m.page_size) * m.page_size;
    return (int64_t)j * m.kv_layer_stride + ((int64_t)page * m.KH * m.page_size + slot) * m.D;
}

__device__ __forceinline__ void global_warp(int& warp, int& nwarps) {
    const int wpb = blockDim.x >> 5;
    warp = blockIdx.x * wpb + (threadIdx.x >> 5);
    nwarps = gridDim.x * wpb;
}

__device__ __forceinline__ int64_t tiles_of(int64_t rows) { return (rows + 31) / 32; }

__device__ __forceinline__ void flag_error(Ctl* c, int bit) {
    if (c && threadIdx.x == 0) atomicOr(&c->err, bit);
}

// Shared-memory layout of every GEMV kernel: x (K floats), then the tile
// partials (kSlotTiles * kWarps * 32 floats), then a second K-float area
// for the first layer's embedding row.
__device__ __forceinline__ float* sm_partials(float* xs, int K) { return xs + ((K + 3) & ~3); }

// ------------------------------------------------------------------ kernels

// Attention input of layer j: [embedding gather,] RMSNorm, Q/K/V GEMV, RoPE,
// KV append at the step's position.
template <bool WHOLE>
__global__ void __launch_bounds__(kGemvThreads, 2) k_qkv(DevModel m, int layer, int first) {
    extern __shared__ float4 smem_f4[];
    float* xs = reinterpret_cast<float*>(smem_f4);
    float* sm_part = sm_partials(xs, m.d);
    uint4* tile_sm = sm_tile(xs, m.d, m.d);
    __shared__ float red[32];
    const uint16_t* lw = layer_base(m, layer);
    const uint4* W = reinterpret_cast<const uint4*>(lw + m.off_wqkv);
    const int64_t nq = (int64_t)m.A * m.D / 2, nk = (int64_t)m.KH * m.D / 2;
    GemvFront<WHOLE> fr;
    fr.begin(W, (nq + 2 * nk) / 16, m.d, tile_sm);
    const CoopRange& r = fr.r;
    if (!WHOLE) zero_sm_part(sm_part);
    pdl_wait();
    pdl_launch_dependents();
    Ctl* c = m.ctl;
    int pos = c->pos;
    const bool pos_ok = pos >= 0 && pos < m.max_ctx;
    if (!pos_ok) pos = 0;
    const float* src = m.h;
    if (first) {
        int tok = c->in_tok;
        const bool tok_ok = tok >= 0 && tok < m.V;
        if (!tok_ok) tok = 0;
        float* hl = sm_part + kSlotTiles * kWarps * 32;
        const uint16_t* e = m.embed + (int64_t)tok * m.d;
        for (int i = threadIdx.x; i < m.d; i += blockDim.x) {
            const float v = bf2f(e[i]);
            hl[i] = v;
            if (blockIdx.x == 0) m.h[i] = v;
        }
        if (blockIdx.x == 0 && threadIdx.x == 0) {
            c->exit_readout = -1;
            c->n_evaluated = 0;
            c->full_token = -1;
            c->nucleus_member = -1;
            if (!tok_ok) atomicOr(&c->err, kErrTokenRange);
        }
        __syncthreads();
        src = hl;
    }
    if (!pos_ok) {
        if (blockIdx.x == 0) flag_error(c, kErrPosition);
        cp_async_wait_all();
        return;
    }
    rmsnorm_to_smem(src, lw + m.off_gattn, m.d, m.eps, xs, red);
    if (!fr.stream(W, xs, sm_part, tile_sm)) {
        flag_error(c, kErrShape);
        return;
    }
    const int64_t kvo = kv_slot_offset(m, layer, pos);
    const EpiQKV epi{m.q, m.kpool + kvo, m.vpool + kvo, (int64_t)m.page_size * m.D,
                     m.qkv_bias ? lw + m.off_bqkv : nullptr, m.rope + (int64_t)pos * (m.D / 2), 0, m.D, (int)nq, (int)nk};
    coop_finish(r, sm_part, m.gemv_part, 0, m.gemv_ticket, epi);
    if (blockIdx.x == 0 && threadIdx.x == 0) m.kv_src[(int64_t)layer * m.max_ctx + pos] = 1;
}

// KV repair for the skipped layers exit_layer .. L-1 (0-based) at the step's
// position: K = RoPE(W_K RMSNorm_j(h_k)), V = W_V RMSNorm_j(h_k), stored bf16.
// blockIdx.y selects the layer; each layer's K/V tiles are split over
// gridDim.x CTAs.
template <bool WHOLE>
__global__ void __launch_bounds__(kGemvThreads, 2) k_kvfill(DevModel m, int exit_layer) {
    extern __shared__ float4 smem_f4[];
    float* xs = reinterpret_cast<float*>(smem_f4);
    float* sm_part = sm_partials(xs, m.d);
    uint4* tile_sm = sm_tile(xs, m.d, 0);
    __shared__ float red[32];
    const int j = exit_layer + blockIdx.y;
    const uint16_t* lw = layer_base(m, j);
    const int64_t nq = (int64_t)m.A * m.D / 2, nk = (int64_t)m.KH * m.D / 2;
    const uint4* W = reinterpret_cast<const uint4*>(lw + m.off_wqkv + nq * 2 * m.d);
    GemvFront<WHOLE> fr;
    fr.begin(W, 2 * nk / 16, m.d, tile_sm);
    const CoopRange& r = fr.r;
    if (!WHOLE) zero_sm_part(sm_part);
    pdl_wait();
    pdl_launch_dependents();
    const int pos = m.ctl->pos;
    if (pos < 0 || pos >= m.max_ctx) {
        cp_async_wait_all();
        return;
    }
    rmsnorm_to_smem(m.h, lw + m.off_gattn, m.d, m.eps, xs, red);
    if (!fr.stream(W, xs, sm_part, tile_sm)) {
        flag_error(m.ctl, kErrShape);
        return;
    }
    const int64_t kvo = kv_slot_offset(m, j, pos);
    const EpiQKV epi{m.q, m.kpool + kvo, m.vpool + kvo, (int64_t)m.page_size * m.D,
                     m.qkv_bias ? lw + m.off_bqkv : nullptr, m.rope + (int64_t)pos * (m.D / 2), nq, m.D, (int)nq, (int)nk};
    coop_finish(r, sm_part, m.gemv_part, blockIdx.y * gridDim.x, m.gemv_ticket + blockIdx.y * m.gemv_ticket_stride,
                epi);
    if (blockIdx.x == 0 && threadIdx.x == 0) m.kv_src[(int64_t)j * m.max_ctx + pos] = 2;
    if (blockIdx.x == 0 && blockIdx.y == 0) {  // what a later full-depth re-pass starts from
        for (int i = threadIdx.x; i < m.d; i += blockDim.x) m.h_exit[(int64_t)pos * m.d + i] = m.h[i];
        if (threadIdx.x == 0) m.exit_at[pos] = (int16_t)exit_layer;
    }
}

// An exit step under the deferred fill: record the residual the position
// exited with and its exit layer (what a later fill or re-pass starts from);
// its skipped layers' entries stay empty.
__global__ void k_record_exit(DevModel m, int exit_layer) {
    pdl_wait();
    pdl_launch_dependents();
    const int pos = m.ctl->pos;
    if (pos < 0 || pos >= m.max_ctx) return;
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < m.d; i += gridDim.x * blockDim.x)
        m.h_exit[(int64_t)pos * m.d + i] = m.h[i];
    if (blockIdx.x == 0 && threadIdx.x == 0) m.exit_at[pos] = (int16_t)exit_layer;
}

// The deferred KV fill (Section 4, step five): a skipped entry of layer j at
// position p is the residual p exited with, through layer j's input RMSNorm
// and its key and value matrices (the key rotated at p); deferred to the
// first later step that runs layer j, it changes no token, since only such
// a step reads it.  CTA (x, y) takes key/value tile x of layer j0 + y, staged
// once in shared memory, and fills every pending entry of that layer: each
// position p in [ctl->pend_lo, ctl->pos) that exited at a layer <= j
// (exit_at) and whose entry at layer j is still empty (kv_src 0).  The
// weights are read once for all pending positions.
constexpr int kFillThreads = 256;
__global__ void __launch_bounds__(kFillThreads) k_fill_pending(DevModel m, int j0) {
    extern __shared__ float4 smem_f4[];
    const int d = m.d, j = j0 + blockIdx.y, tile = blockIdx.x;
    float* xs = reinterpret_cast<float*>(smem_f4);                       // [d]
    float* part = xs + ((d + 3) & ~3);                                    // [8][32]
    int* list = reinterpret_cast<int*>(part + 8 * 32);                    // [kFillThreads] + count
    uint4* tile_sm = reinterpret_cast<uint4*>(list + kFillThreads + 4);   // 32 rows x d bf16, tile-packed
    __shared__ float red[32];
    const uint16_t* lw = m.layers + (int64_t)j * m.layer_stride;
    const int64_t nq = (int64_t)m.A * m.D / 2, nk = (int64_t)m.KH * m.D / 2;
    const int Rc = d >> 3;  // 16-byte column chunks
    const uint4* W = reinterpret_cast<const uint4*>(lw + m.off_wqkv + nq * 2 * d) + (int64_t)tile * Rc * 32;
    for (int i = threadIdx.x; i < Rc * 32; i += kFillThreads) cp_async16(tile_sm + i, W + i);
    cp_async_commit();
    pdl_wait();
    pdl_launch_dependents();
    const Ctl* c = m.ctl;
    const int pos = c->pos, lo = max(0, c->pend_lo);
    const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
    bool staged = false;
    for (int base = lo; base < pos; base += kFillThreads) {
        // this round's pending positions, in position order
        if (threadIdx.x == 0) list[kFillThreads] = 0;
        __syncthreads();
        const int p = base + threadIdx.x;
        const bool need = p < pos && m.exit_at[p] > 0 && m.exit_at[p] <= j &&
                          m.kv_src[(int64_t)j * m.max_ctx + p] == 0;
        const unsigned bal = __ballot_sync(0xffffffffu, need);
        if (lane == 0) red[w] = __int_as_float(__popc(bal));
        __syncthreads();
        int before = 0;
        for (int k = 0; k < w; ++k) before += __float_as_int(red[k]);
        if (need) list[before + __popc(bal & ((1u << lane) - 1))] = p;
        if (threadIdx.x == 0) {
            int n = 0;
            for (int k = 0; k < kFillThreads / 32; ++k) n += __float_as_int(red[k]);
            list[kFillThreads] = n;
        }
        __syncthreads();
        const int n = list[kFillThreads];
        if (n > 0 && !staged) {
            cp_async_wait_all();
            __syncthreads();
            staged = true;
        }
        for (int k = 0; k < n; ++k) {
            const int q = list[k];
            rmsnorm_to_smem(m.h_exit + (int64_t)q * d, lw + m.off_gattn, d, m.eps, xs, red);
            // lane = row of the tile, warp w the 16-byte column chunks w, w + 8, ...
            float acc = 0.f;
            for (int cc = w; cc < Rc; cc += kFillThreads / 32) acc += dot8(tile_sm[cc * 32 + lane], xs + cc * 8);
            part[w * 32 + lane] = acc;
            __syncthreads();
            if (w == 0) {
                float sum = 0.f;
#pragma unroll
                for (int k2 = 0; k2 < kFillThreads / 32; ++k2) sum += part[k2 * 32 + lane];
                const int64_t kvo = kv_slot_offset(m, j, q);
                const EpiQKV epi{nullptr, m.kpool + kvo, m.vpool + kvo, (int64_t)m.page_size * m.D,
                                 m.qkv_bias ? lw + m.off_bqkv : nullptr, m.rope + (int64_t)q * (m.D / 2), nq, m.D,
                                 (int)nq, (int)nk};
                epi(tile, sum);
            }
            if (tile == 0 && threadIdx.x == 0) m.kv_src[(int64_t)j * m.max_ctx + q] = 2;
            __syncthreads();
        }
    }
    if (!staged) cp_async_wait_all();
}

// Output projection with the residual add: h += W_o o.
template <bool WHOLE>
__global__ void __launch_bounds__(kGemvThreads, 2) k_oproj(DevModel m, int layer) {
    extern __shared__ float4 smem_f4[];
    float* xs = reinterpret_cast<float*>(smem_f4);
    const int K = m.A * m.D;
    float* sm_part = sm_partials(xs, K);
    uint4* tile_sm = sm_tile(xs, K, 0);
    const uint4* W = reinterpret_cast<const uint4*>(layer_base(m, layer) + m.off_wo);
    GemvFront<WHOLE> fr;
    fr.begin(W, tiles_of(m.d), K, tile_sm);
    const CoopRange& r = fr.r;
    if (!WHOLE) zero_sm_part(sm_part);
    pdl_wait();
    pdl_launch_dependents();
    int lo, hi;
    fr.x_range(K, lo, hi);
    for (int i = lo + threadIdx.x; i < hi; i += blockDim.x) xs[i] = m.o[i];
    __syncthreads();
    if (!fr.stream(W, xs, sm_part, tile_sm)) {
        flag_error(m.ctl, kErrShape);
        return;
    }
    const EpiAddH epi{m.h, m.d};
    coop_finish(r, sm_part, m.gemv_part, 0, m.gemv_ticket, epi);
}

// Gated feed-forward up: a = SiLU(W_g x) * (W_u x), x = RMSNorm(h) * g_mlp.
template <bool WHOLE>
__global__ void __launch_bounds__(kGemvThreads, 2) k_gateup(DevModel m, int layer) {
    extern __shared__ float4 smem_f4[];
    float* xs = reinterpret_cast<float*>(smem_f4);
    float* sm_part = sm_partials(xs, m.d);
    uint4* tile_sm = sm_tile(xs, m.d, 0);
    __shared__ float red[32];
    const uint16_t* lw = layer_base(m, layer);
    const uint4* W = reinterpret_cast<const uint4*>(lw + m.off_wgu);
    GemvFront<WHOLE> fr;
    fr.begin(W, tiles_of(2 * (int64_t)m.F), m.d, tile_sm);
    const CoopRange& r = fr.r;
    if (!WHOLE) zero_sm_part(sm_part);
    pdl_wait();
    pdl_launch_dependents();
    rmsnorm_to_smem(m.h, lw + m.off_gmlp, m.d, m.eps, xs, red);
    if (!fr.stream(W, xs, sm_part, tile_sm)) {
        flag_error(m.ctl, kErrShape);
        return;
    }
    const EpiSwiGLU epi{m.a, m.F};
    coop_finish(r, sm_part, m.gemv_part, 0, m.gemv_ticket, epi);
}

// Gated feed-forward down with the residual add: h += W_d a.
template <bool WHOLE>
__global__ void __launch_bounds__(kGemvThreads, 2) k_down(DevModel m, int layer) {
    extern __shared__ float4 smem_f4[];
    float* xs = reinterpret_cast<float*>(smem_f4);
    float* sm_part = sm_partials(xs, m.F);
    uint4* tile_sm = sm_tile(xs, m.F, 0);
    const uint4* W = reinterpret_cast<const uint4*>(layer_base(m, layer) + m.off_wd);
    GemvFront<WHOLE> fr;
    fr.begin(W, tiles_of(m.d), m.F, tile_sm);
    const CoopRange& r = fr.r;
    if (!WHOLE) zero_sm_part(sm_part);
    pdl_wait();
    pdl_launch_dependents();
    int lo, hi;
    fr.x_range(m.F, lo, hi);
    for (int i = lo + threadIdx.x; i < hi; i += blockDim.x) xs[i] = m.a[i];
    __syncthreads();
    if (!fr.stream(W, xs, sm_part, tile_sm)) {
        flag_error(m.ctl, kErrShape);
        return;
    }
    const EpiAddH epi{m.h, m.d};
    coop_finish(r, sm_part, m.gemv_part, 0, m.gemv_ticket, epi);
}

// Readout affine map r: y_r = W_r h + b_r; also keeps h_k for debug.
template <bool WHOLE>
__global__ void __launch_bounds__(kGemvThreads, 2) k_readout(DevModel m, int r) {
    extern __shared__ float4 smem_f4[];
    float* xs = reinterpret_cast<float*>(smem_f4);
    float* sm_part = sm_partials(xs, m.d);
    uint4* tile_sm = sm_tile(xs, m.d, 0);
    const uint4* W = reinterpret_cast<const uint4*>(m.ro_w[r]);
    GemvFront<WHOLE> fr;
    fr.begin(W, tiles_of(m.d), m.d, tile_sm);
    const CoopRange& rg = fr.r;
    if (!WHOLE) zero_sm_part(sm_part);
    pdl_wait();
    pdl_launch_dependents();
    for (int i = threadIdx.x; i < m.d; i += blockDim.x) {
        const float v = m.h[i];
        xs[i] = v;
        if (blockIdx.x == 0) m.hk[(int64_t)r * m.d + i] = v;
    }
    __syncthreads();
    if (!fr.stream(W, xs, sm_part, tile_sm)) {
        flag_error(m.ctl, kErrShape);
        return;
    }
    const EpiBias epi{m.y + (int64_t)r * m.d, m.ro_b[r], m.d};
    coop_finish(rg, sm_part, m.gemv_part, 0, m.gemv_ticket, epi);
}

// The logit of row x of the tiled unembedding, summed in the order the
// vocabulary pass sums it (chunk by chunk from 0), so the two agree bit for
// bit.  part: Rc floats of shared memory.  Every thread of the CTA calls it.
__device__ __forceinline__ float tiled_row_logit(const uint4* W, int64_t x, int Rc, const float* xs, float* part) {
    __shared__ float lx;
    const int64_t t = x >> 5, ln = x & 31;
    for (int c = threadIdx.x; c < Rc; c += blockDim.x) part[c] = dot8(__ldg(W + (t * Rc + c) * 32 + ln), xs + c * 8);
    __syncthreads();
    if (threadIdx.x == 0) {
        float acc = 0.f;
        for (int c = 0; c < Rc; ++c) acc += part[c];
        lx = acc;
    }
    __syncthreads();
    return lx;
}

// One pass over the (tiled) unembedding: z = RMSNorm(x) * gain, l = U z,
// with max, sum of exp and lowest argmax.  Each warp owns a run of whole
// tiles (no cross-warp combine), lane r the rows r, r + 32, ...
__global__ void __launch_bounds__(kGemvThreads, 2) k_vocab(VocabArgs v) {
    extern __shared__ float4 smem_f4[];
    float* xs = reinterpret_cast<float*>(smem_f4);
    __shared__ float red[32];
    const int lane = threadIdx.x & 31;
    int warp, nwarps;
    global_warp(warp, nwarps);
    const int Rc = v.d >> 3;
    const int64_t n_tiles = (v.V + 31) / 32;
    const int64_t t0 = n_tiles * warp / nwarps, t1 = n_tiles * (warp + 1) / nwarps;
    const int64_t i0 = t0 * Rc, i1 = t1 * Rc;
    const uint4* W = reinterpret_cast<const uint4*>(v.U);
    uint4 buf[kWindow];
#pragma unroll
    for (int u = 0; u < kWindow; ++u)
        buf[u] = i0 + u < i1 ? ldg_stream(W + (i0 + u) * 32 + lane) : make_uint4(0u, 0u, 0u, 0u);
    pdl_wait();
    pdl_launch_dependents();
    rmsnorm_to_smem(v.x, v.gain, v.d, v.eps, xs, red);
    const bool keep = v.logits && (!v.logits_if_dbg || (v.ctl && v.ctl->dbg));
    // nucleus tracking: on full steps, the tokens above readout 0's token
    const bool nucleus = v.mode == 2 && v.ctl->nucleus_on && v.ctl->n_evaluated > 0;
    int nx = -1;
    float lx = INFINITY;
    if (nucleus) {
        nx = v.ctl->readout_token[0];
        if (nx < 0 || nx >= v.V) nx = 0;  // the readout pass flags an out-of-range token
        lx = tiled_row_logit(W, nx, Rc, xs, xs + ((v.d + 3) & ~3));
    }
    LaneStats st;
    int64_t t = t0;
    int c = 0;
    float acc = 0.f;
    for (int64_t base = i0; base < i1; base += kWindow) {
        if (base != i0) {
#pragma unroll
            for (int u = 0; u < kWindow; ++u)
                buf[u] = base + u < i1 ? ldg_stream(W + (base + u) * 32 + lane) : make_uint4(0u, 0u, 0u, 0u);
        }
#pragma unroll
        for (int u = 0; u < kWindow; ++u) {
            if (base + u >= i1) break;
            acc += dot8(buf[u], xs + c * 8);
            if (++c == Rc) {
                const int64_t row = t * 32 + lane;
                if (row < v.V) {
                    if (keep) v.logits[row] = acc;
                    st.add(acc, (int)row, lx, nx);
                }
                acc = 0.f;
                c = 0;
                ++t;
            }
        }
    }
    vocab_finish(v, st, nucleus, (int)(blockDim.x >> 5), [] { __syncthreads(); });
}

// The same pass over a row-major [V, d] matrix (standalone op): the flat
// streaming core, one warp per run of whole rows.
struct EpiVocabRowMajor {
    float* logits;
    LaneStats st;
    __device__ __forceinline__ void operator()(int64_t u, const float* r) {
        if (logits) logits[u] = r[0];
        st.add(r[0], (int)u);
    }
};

__global__ void __launch_bounds__(kGemvThreads, 2) k_vocab_rowmajor(VocabArgs v) {
    extern __shared__ float4 smem_f4[];
    float* xs = reinterpret_cast<float*>(smem_f4);
    __shared__ float red[32];
    int warp, nwarps;
    global_warp(warp, nwarps);
    pdl_wait();
    pdl_launch_dependents();
    rmsnorm_to_smem(v.x, v.gain, v.d, v.eps, xs, red);
    EpiVocabRowMajor epi{v.logits, LaneStats()};
    flat_gemv<1, true, 8>(v.U, v.d, v.V, xs, warp, nwarps, nullptr, nullptr, epi);
    // lane 0 holds this warp's statistics; the others hold none
    LaneStats st = (threadIdx.x & 31) == 0 ? epi.st : LaneStats();
    vocab_finish(v, st, false, (int)(blockDim.x >> 5), [] { __syncthreads(); });
}

// Split-K decode attention over the paged cache.  Grid (splits, KH): CTA
// (s, g) covers a contiguous run of positions for the A/K query heads of
// key-value head g with a per-lane online softmax; the last CTA of head g
// merges the splits and writes o = softmax(q K^T / sqrt(D)) V (fp32).
template <int D>
__global__ void __launch_bounds__(kAttnThreads) k_attention(AttnArgs a) {
    constexpr int LPR = D / 8;  // lanes per position (8 dims each)
    constexpr int RPW = 32 / LPR;
    constexpr int NW = kAttnThreads / 32;
    constexpr int GMAX = 8;
    __shared__ __align__(16) float qs[GMAX * D];
    __shared__ float wm[NW][GMAX], wl[NW][GMAX];
    __shared__ __align__(16) float wacc[NW][GMAX][D];
    __shared__ int is_last;
    pdl_wait();
    pdl_launch_dependents();
    const int T = a.ctl ? a.ctl->pos + 1 : a.T;
    const int G = a.A / a.KH;
    int S = (T + kAttnMinRows - 1) / kAttnMinRows;
    if (S > (int)gridDim.x) S = gridDim.x;
    const int chunk = (T + S - 1) / S;
    const int s = blockIdx.x, g = blockIdx.y;
    if (s >= S) return;
    const int t0 = s * chunk, t1 = min(T, t0 + chunk);
    const float scale = 1.0f / sqrtf((float)D);
    for (int i = threadIdx.x; i < G * D; i += blockDim.x) qs[i] = a.q[(int64_t)g * G * D + i] * scale;
    __syncthreads();

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int grp = lane / LPR, e0 = (lane % LPR) * 8;
    float mx[GMAX], ls[GMAX], acc[GMAX][8];
#pragma unroll
    for (int h = 0; h < GMAX; ++h) {
        mx[h] = -CUDART_INF_F;
        ls[h] = 0.f;
#pragma unroll
        for (int e = 0; e < 8; ++e) acc[h][e] = 0.f;
    }
    const int P = a.page_size;
    for (int tt = t0 + warp * RPW; tt < t1; tt += NW * RPW) {
        const int t = tt + grp;
        const bool valid = t < t1;
        float kf[8], vf[8];
        if (valid) {
            const int page = a.page_table[t / P];
            const int64_t off = (((int64_t)page * a.KH + g) * P + (t % P)) * D + e0;
            const uint4 kw = *reinterpret_cast<const uint4*>(a.kp + off);
            const uint4 vw = *reinterpret_cast<const uint4*>(a.vp + off);
            kf[0] = bf_lo(kw.x); kf[1] = bf_hi(kw.x); kf[2] = bf_lo(kw.y); kf[3] = bf_hi(kw.y);
            kf[4] = bf_lo(kw.z); kf[5] = bf_hi(kw.z); kf[6] = bf_lo(kw.w); kf[7] = bf_hi(kw.w);
            vf[0] = bf_lo(vw.x); vf[1] = bf_hi(vw.x); vf[2] = bf_lo(vw.y); vf[3] = bf_hi(vw.y);
            vf[4] = bf_lo(vw.z); vf[5] = bf_hi(vw.z); vf[6] = bf_lo(vw.w); vf[7] = bf_hi(vw.w);
        } else {
#pragma unroll
            for (int e = 0; e < 8; ++e) kf[e] = vf[e] = 0.f;
        }
#pragma unroll
        for (int h = 0; h < GMAX; ++h) {
            if (h >= G) break;
            float d = 0.f;
#pragma unroll
            for (int e = 0; e < 8; ++e) d = fmaf(kf[e], qs[h * D + e0 + e], d);
#pragma unroll
            for (int o = LPR / 2; o; o >>= 1) d += __shfl_xor_sync(0xffffffffu, d, o);
            if (valid) {
                const float mn = fmaxf(mx[h], d);
                const float corr = expf(mx[h] - mn);
                const float p = expf(d - mn);
                ls[h] = ls[h] * corr + p;
#pragma unroll
                for (int e = 0; e < 8; ++e) acc[h][e] = fmaf(p, vf[e], acc[h][e] * corr);
                mx[h] = mn;
            }
        }
    }
    // merge the position groups of this warp (lanes with equal e0)
#pragma unroll
    for (int o = LPR; o < 32; o <<= 1) {
#pragma unroll
        for (int h = 0; h < GMAX; ++h) {
            if (h >= G) break;
            const float m2 = __shfl_xor_sync(0xffffffffu, mx[h], o);
            const float l2 = __shfl_xor_sync(0xffffffffu, ls[h], o);
            float a2[8];
#pragma unroll
            for (int e = 0; e < 8; ++e) a2[e] = __shfl_xor_sync(0xffffffffu, acc[h][e], o);
            const float M = fmaxf(mx[h], m2);
            if (M != -CUDART_INF_F) {
                const float c1 = expf(mx[h] - M), c2 = expf(m2 - M);
                ls[h] = ls[h] * c1 + l2 * c2;
#pragma unroll
                for (int e = 0; e < 8; ++e) acc[h][e] = acc[h][e] * c1 + a2[e] * c2;
                mx[h] = M;
            }
        }
    }
    if (grp == 0) {
#pragma unroll
        for (int h = 0; h < GMAX; ++h) {
            if (h >= G) break;
            if (lane == 0) {
                wm[warp][h] = mx[h];
                wl[warp][h] = ls[h];
            }
#pragma unroll
            for (int e = 0; e < 8; ++e) wacc[warp][h][e0 + e] = acc[h][e];
        }
    }
    __syncthreads();
    // merge warps; write this split's partial (acc[D], m, l) per query head
    const int S_stride = kAttnMaxSplits;
    for (int i = threadIdx.x; i < G * D; i += blockDim.x) {
        const int h = i / D, e = i - h * D;
        float M = -CUDART_INF_F, L = 0.f, O = 0.f;
        for (int w = 0; w < NW; ++w) {
            const float m2 = wm[w][h];
            const float Mn = fmaxf(M, m2);
            if (Mn == -CUDART_INF_F) continue;
            const float c1 = expf(M - Mn), c2 = expf(m2 - Mn);
            L = L * c1 + wl[w][h] * c2;
            O = O * c1 + wacc[w][h][e] * c2;
            M = Mn;
        }
        float* pp = a.part + ((int64_t)(g * G + h) * S_stride + s) * (D + 2);
        pp[e] = O;
        if (e == 0) {
            pp[D] = M;
            pp[D + 1] = L;
        }
    }
    __threadfence();
    __syncthreads();
    if (threadIdx.x == 0) is_last = atomicAdd(&a.ticket[g], 1) == S - 1;
    __syncthreads();
    if (!is_last) return;
    __threadfence();
    for (int i = threadIdx.x; i < G * D; i += blockDim.x) {
        const int h = i / D, e = i - h * D;
        const float* base = a.part + (int64_t)(g * G + h) * S_stride * (D + 2);
        float M = -CUDART_INF_F;
        for (int sp = 0; sp < S; ++sp) M = fmaxf(M, __ldcg(&base[sp * (D + 2) + D]));
        float L = 0.f, O = 0.f;
        for (int sp = 0; sp < S; ++sp) {
            const float ms = __ldcg(&base[sp * (D + 2) + D]);
            if (ms == -CUDART_INF_F) continue;
            const float c = expf(ms - M);
            L = fmaf(__ldcg(&base[sp * (D + 2) + D + 1]), c, L);
            O = fmaf(__ldcg(&base[sp * (D + 2) + e]), c, O);
        }
        a.out[(int64_t)(g * G + h) * D + e] = O / L;
    }
    if (threadIdx.x == 0) a.ticket[g] = 0;
}

// Decode attention of one layer on a thread-block cluster per key-value head
// (grid (CL, KH), cluster (CL, 1, 1)).  Rank r covers a contiguous run of
// positions for all A/K query heads of head g, in sub-chunks of NB positions
// staged in shared memory (K rows XOR-swizzled by 16-byte chunk so that four
// threads per position read without bank conflicts).  The first sub-chunk's
// past rows are copied (cp.async) before the kernel waits on the QKV kernel:
// only position T-1 is new.  Per sub-chunk: scores (4 threads per position),
// a running softmax per head, and P V with each thread owning output pairs;
// then the CL ranks merge through distributed shared memory, each finishing
// a share of o = softmax(q K^T / sqrt(D)) V (fp32).
namespace cg = cooperative_groups;


template <int D>
struct AttnSmem {
    static constexpr int NB = 16384 / D;  // positions per sub-chunk (K + V = 64 KB)
    static constexpr int CH = D / 8;      // 16-byte chunks per row
    static constexpr int GMAX = 8;
    static constexpr size_t bytes = (size_t)2 * NB * CH * 16 + (size_t)GMAX * D * 4 + (size_t)GMAX * NB * 4;
};

// Copy rows [r0, r1) of the CTA's sub-chunk (positions base + r) into smem.
template <int D>
__device__ __forceinline__ void attn_stage(const AttnArgs& a, int g, int base, int r0, int r1, uint4* Ks, uint4* Vs,
                                           bool async) {
    constexpr int CH = D / 8;
    const int P = a.page_size;
    for (int i = r0 * CH + threadIdx.x; i < r1 * CH; i += blockDim.x) {
        const int r = i / CH, c = i - r * CH;
        const int t = base + r;
        const int64_t off = (((int64_t)a.page_table[t / P] * a.KH + g) * P + (t % P)) * D + c * 8;
        uint4* kd = Ks + r * CH + (c ^ (r & (CH - 1)));
        uint4* vd = Vs + r * CH + c;
        if (async) {
            cp_async16(kd, a.kp + off);
            cp_async16(vd, a.vp + off);
        } else {
            *kd = *reinterpret_cast<const uint4*>(a.kp + off);
            *vd = *reinterpret_cast<const uint4*>(a.vp + off);
        }
    }
}

template <int D>
__global__ void __launch_bounds__(kAttnThreads) k_attn_cluster(AttnArgs a) {
    using S = AttnSmem<D>;
    constexpr int NB = S::NB, CH = S::CH, GMAX = S::GMAX;
    extern __shared__ __align__(16) unsigned char attn_sm[];
    uint4* Ks = reinterpret_cast<uint4*>(attn_sm);
    uint4* Vs = Ks + NB * CH;
    float* qs = reinterpret_cast<float*>(Vs + NB * CH);
    float* ps = qs + GMAX * D;
    __shared__ float hm[GMAX], hl[GMAX], hs[GMAX];
    cg::cluster_group cluster = cg::this_cluster();
    const int rank = (int)cluster.block_rank(), CL = (int)cluster.num_blocks();
    const int g = blockIdx.y, G = a.A / a.KH;
    const int T = a.ctl->pos + 1;
    const int chunk = (T + CL - 1) / CL;
    const int t0 = min(T, rank * chunk), t1 = min(T, t0 + chunk);
    // past rows of the first sub-chunk, before waiting on the QKV kernel
    const int first_end = min(t1, t0 + NB);
    attn_stage<D>(a, g, t0, 0, max(0, min(first_end, T - 1) - t0), Ks, Vs, true);
    cp_async_commit();
    if (threadIdx.x < GMAX) {
        hm[threadIdx.x] = -CUDART_INF_F;
        hl[threadIdx.x] = 0.f;
    }
    pdl_wait();
    pdl_launch_dependents();
    const float scale = 1.0f / sqrtf((float)D);
    for (int i = threadIdx.x; i < G * D; i += blockDim.x) qs[i] = a.q[(int64_t)g * G * D + i] * scale;
    if (T - 1 >= t0 && T - 1 < first_end) attn_stage<D>(a, g, t0, T - 1 - t0, T - t0, Ks, Vs, false);
    cp_async_wait_all();
    __syncthreads();

    // each thread owns output pairs (h, e, e+1) for items tid, tid + blockDim
    constexpr int ITEMS = (GMAX * D / 2 + kAttnThreads - 1) / kAttnThreads;
    float acc[ITEMS][2];
#pragma unroll
    for (int k = 0; k < ITEMS; ++k) acc[k][0] = acc[k][1] = 0.f;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    (void)lane;

    for (int base = t0; base < t1; base += NB) {
        const int nb = min(NB, t1 - base);
        if (base != t0) {
            __syncthreads();  // everyone is done with the previous sub-chunk
            attn_stage<D>(a, g, base, 0, nb, Ks, Vs, false);
            __syncthreads();
        }
        // scores: one thread per (head, position), the whole dot product
        for (int w = threadIdx.x; w < G * nb; w += blockDim.x) {
            const int h = w / nb, p = w - h * nb;
            const float* qh = qs + h * D;
            float d0 = 0.f, d1 = 0.f;
#pragma unroll
            for (int c = 0; c < CH; ++c) {
                const uint4 kw = Ks[p * CH + (c ^ (p & (CH - 1)))];
                const float4 q0 = *reinterpret_cast<const float4*>(qh + c * 8);
                const float4 q1 = *reinterpret_cast<const float4*>(qh + c * 8 + 4);
                d0 = fmaf(bf_lo(kw.x), q0.x, d0);
                d1 = fmaf(bf_hi(kw.x), q0.y, d1);
                d0 = fmaf(bf_lo(kw.y), q0.z, d0);
                d1 = fmaf(bf_hi(kw.y), q0.w, d1);
                d0 = fmaf(bf_lo(kw.z), q1.x, d0);
                d1 = fmaf(bf_hi(kw.z), q1.y, d1);
                d0 = fmaf(bf_lo(kw.w), q1.z, d0);
                d1 = fmaf(bf_hi(kw.w), q1.w, d1);
            }
            ps[h * NB + p] = d0 + d1;
        }
        __syncthreads();
        // softmax statistics of this sub-chunk, one warp per head
        if (warp < G) {
            const int h = warp;
            float m = -CUDART_INF_F;
            for (int p = lane; p < nb; p += 32) m = fmaxf(m, ps[h * NB + p]);
#pragma unroll
            for (int o = 16; o; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
            const float mo = hm[h];
            const float mn = fmaxf(mo, m);
            float l = 0.f;
            for (int p = lane; p < nb; p += 32) {
                const float e = expf(ps[h * NB + p] - mn);
                ps[h * NB + p] = e;
                l += e;
            }
            l = warp_sum(l);
            if (lane == 0) {
                const float sc = expf(mo - mn);  // 0 on the first sub-chunk
                hs[h] = sc;
                hl[h] = hl[h] * sc + l;
                hm[h] = mn;
            }
        }
        __syncthreads();
        // P V: acc(h, e..e+1) = acc * rescale + sum_p p(h, p) v(p, e..e+1)
#pragma unroll
        for (int k = 0; k < ITEMS; ++k) {
            const int it = threadIdx.x + k * kAttnThreads;
            if (it >= G * D / 2) break;
            const int h = it / (D / 2), e2 = it - h * (D / 2);
            const float sc = hs[h];
            float x0 = acc[k][0] * sc, x1 = acc[k][1] * sc;
            const uint32_t* vrow = reinterpret_cast<const uint32_t*>(Vs) + e2;
            const float* pr = ps + h * NB;
            for (int p = 0; p < nb; ++p) {
                const uint32_t v2 = vrow[p * (D / 2)];
                const float w = pr[p];
                x0 = fmaf(w, bf_lo(v2), x0);
                x1 = fmaf(w, bf_hi(v2), x1);
            }
            acc[k][0] = x0;
            acc[k][1] = x1;
        }
    }
    // this CTA's partial: (hm, hl) per head, accumulator pairs in qs (reused)
    __syncthreads();
#pragma unroll
    for (int k = 0; k < ITEMS; ++k) {
        const int it = threadIdx.x + k * kAttnThreads;
        if (it >= G * D / 2) break;
        qs[2 * it] = acc[k][0];
        qs[2 * it + 1] = acc[k][1];
    }
    cluster.sync();
    // merge the ranks' partials: thread (r, h) weighs rank r for head h
    // (shuffle reductions over the CL ranks of a head), then each output sums
    // the CL scaled partials, all remote loads issued before use; outputs are
    // spread over all ranks
    __shared__ float rw[16][GMAX];  // exp(m_r - M) / L per rank and head (CL <= 16)
    if (threadIdx.x < 16 * GMAX) {
        const int r = threadIdx.x & 15, h = threadIdx.x >> 4;  // 16 lanes per head
        const bool on = r < CL && h < G;
        const float mr = on ? ld_dsmem(dsmem_addr(&hm[h], r)) : -CUDART_INF_F;
        const float lr = on ? ld_dsmem(dsmem_addr(&hl[h], r)) : 0.f;
        float M = mr;
#pragma unroll
        for (int o = 8; o; o >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));
        const float c = mr == -CUDART_INF_F ? 0.f : expf(mr - M);
        float L = lr * c;
#pragma unroll
        for (int o = 8; o; o >>= 1) L += __shfl_xor_sync(0xffffffffu, L, o);
        if (on) rw[r][h] = c / L;
    }
    __syncthreads();
    for (int i = rank * blockDim.x + threadIdx.x; i < G * D; i += CL * blockDim.x) {
        const int h = i / D;
        const uint32_t base = (uint32_t)__cvta_generic_to_shared(qs + i);
        float part[16];
#pragma unroll
        for (int r = 0; r < 16; ++r)
            if (r < CL) part[r] = ld_dsmem(dsmem_rank(base, r));
        float O = 0.f;
#pragma unroll
        for (int r = 0; r < 16; ++r)
            if (r < CL) O = fmaf(rw[r][h], part[r], O);
        a.out[(int64_t)g * G * D + i] = O;
    }
    cluster.sync();  // keep every rank's shared memory alive until all have read it
}

// End of a decode step: emit, record, count, advance, feed the token back.
__global__ void k_step_end(DevModel m, int has_cond, cudaGraphConditionalHandle cond) {
    pdl_wait();
    pdl_launch_dependents();
    if (threadIdx.x != 0) return;
    Ctl* c = m.ctl;
    const int tok = c->token;
    const int r = c->exit_readout;
    const int st = c->step;
    float conf = 0.f;
    if (r >= 0)
        conf = c->conf[r];
    else if (c->n_evaluated > 0)
        conf = c->conf[c->n_evaluated - 1];
    if (c->out_tokens) c->out_tokens[st] = tok;
    if (c->out_exit) c->out_exit[st] = r;
    if (c->out_conf) c->out_conf[st] = conf;
    if (c->out_conf_all)
        for (int q = 0; q < m.n_readouts; ++q)
            c->out_conf_all[(int64_t)st * m.n_readouts + q] = q < c->n_evaluated ? c->conf[q] : NAN;
    if (c->out_member) c->out_member[st] = c->nucleus_member;
    if (c->out_mass) c->out_mass[st] = c->nucleus_member >= 0 ? c->nucleus_mass : NAN;
    c->steps += 1;
    if (r >= 0) {
        c->exits[r] += 1;
    } else {
        c->full_steps += 1;
        c->pend_lo = c->pos + 1;  // a full step ran every layer after filling what was pending
    }
    c->pos += 1;
    c->in_tok = (c->forced_in && st + 1 < c->n_steps) ? c->forced_in[st + 1] : tok;
    c->step = st + 1;
    if (has_cond) cudaGraphSetConditional(cond, (c->step < c->n_steps && c->err == 0) ? 1u : 0u);
}

// Prefill bookkeeping between prompt positions.
__global__ void k_prefill_advance(DevModel m, int has_cond, cudaGraphConditionalHandle cond) {
    pdl_wait();
    pdl_launch_dependents();
    if (threadIdx.x != 0) return;
    Ctl* c = m.ctl;
    c->pos += 1;
    c->prefill_i += 1;
    const int more = c->prefill_i < c->prefill_n;
    if (more) c->in_tok = c->prompt[c->prefill_i];
    if (has_cond) cudaGraphSetConditional(cond, (more && c->err == 0) ? 1u : 0u);
}

// After the prefill's LM head: the full model's token becomes the next input.
__global__ void k_prefill_end(DevModel m) {
    pdl_wait();
    pdl_launch_dependents();
    if (threadIdx.x != 0) return;
    Ctl* c = m.ctl;
    c->in_tok = c->token;
    c->exit_readout = -1;
    c->n_evaluated = 0;
    c->nucleus_member = -1;
    c->pend_lo = c->pos;  // prompt positions ran every layer
}

// Per-call inputs written into the control block ahead of a graph launch.
__global__ void k_set_inputs(Ctl* c, CtlInputs in) {
    if (threadIdx.x != 0) return;
    if (in.set_token) c->in_tok = in.in_tok;
    c->force = in.force;
    c->step = 0;
    c->n_steps = in.n_steps;
    c->dbg = in.dbg;
    c->conf_kind = in.conf_kind;
    c->nucleus_on = in.nucleus_on;
    c->nucleus_p = in.nucleus_p;
    c->out_conf_all = in.out_conf_all;
    c->out_member = in.out_member;
    c->out_mass = in.out_mass;
    c->forced_in = in.forced_in;
    for (int r = 0; r < kMaxReadouts; ++r) c->tau[r] = in.tau[r];
    c->sched = in.sched;
    c->out_tokens = in.out_tokens;
    c->out_exit = in.out_exit;
    c->out_conf = in.out_conf;
    if (in.prefill_n > 0) {
        c->prefill_n = in.prefill_n;
        c->prefill_i = 0;
        c->prompt = in.prompt;
    }
}

// Threshold selection (Section 4, step four).  Each thread takes one
// candidate threshold (-inf, then each observed confidence), counts the
// early positions (conf > candidate) and the acceptable ones among them over
// all n positions, staged through shared memory, and offers the candidate to
// a grid-wide minimum if good >= target * early.  Floats are ordered through
// their bit patterns (negative values with the magnitude bits flipped), so
// the minimum is an integer atomicMin.
constexpr int kTauThreads = 256, kTauTile = 2048;

__device__ __forceinline__ int float_key(float f) {
    const int b = __float_as_int(f);
    return b >= 0 ? b : b ^ 0x7fffffff;
}
__device__ __forceinline__ float key_float(int k) { return __int_as_float(k >= 0 ? k : k ^ 0x7fffffff); }

__global__ void k_tau_init(int* scratch) {
    if (threadIdx.x == 0) {
        scratch[0] = float_key(INFINITY);
        scratch[1] = 0;
    }
}

__global__ void __launch_bounds__(kTauThreads) k_select_tau(const float* conf, int stride, const int32_t* member,
                                                             int n, double target, float* tau, int* scratch) {
    __shared__ float sc[kTauTile];
    __shared__ unsigned char sg[kTauTile];
    __shared__ int is_last;
    const int64_t n_cand = (int64_t)n + 1;
    const int64_t per_pass = (int64_t)gridDim.x * blockDim.x;
    for (int64_t base = 0; base < n_cand; base += per_pass) {
        const int64_t ci = base + (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
        const bool have = ci < n_cand;
        const float cand = !have ? INFINITY : (ci == 0 ? -INFINITY : conf[(ci - 1) * stride]);
        int early = 0, good = 0;
        for (int i0 = 0; i0 < n; i0 += kTauTile) {
            const int len = min(kTauTile, n - i0);
            __syncthreads();
            for (int i = threadIdx.x; i < len; i += blockDim.x) {
                sc[i] = conf[(int64_t)(i0 + i) * stride];
                sg[i] = member[i0 + i] != 0;
            }
            __syncthreads();
            for (int i = 0; i < len; ++i) {
                const int e = sc[i] > cand;
                early += e;
                good += e & sg[i];
            }
        }
        if (have && early > 0 && (double)good >= target * (double)early) atomicMin(&scratch[0], float_key(cand));
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        __threadfence();
        is_last = atomicAdd(&scratch[1], 1) == (int)gridDim.x - 1;
    }
    __syncthreads();
    if (is_last && threadIdx.x == 0) {
        __threadfence();
        *tau = key_float(atomicAdd(&scratch[0], 0));
    }
}

cudaError_t launch_select_tau(const float* conf, int stride, const int32_t* member, int n, double target, float* tau,
                              int* scratch, int n_sm, cudaStream_t s) {
    const int64_t want = ((int64_t)n + 1 + kTauThreads - 1) / kTauThreads;
    const int grid = (int)std::min<int64_t>(want, (int64_t)4 * std::max(n_sm, 1));
    k_tau_init<<<1, 32, 0, s>>>(scratch);
    k_select_tau<<<grid, kTauThreads, 0, s>>>(conf, stride, member, n, target, tau, scratch);
    return cudaGetLastError();
}

// ------------------------------------------------------------------ launchers

template <typename... KArgs, typename... Args>
static cudaError_t launch_k(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, bool pdl, cudaStream_t s,
                            Args... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl ? 1 : 0;
    return cudaLaunchKernelEx(&cfg, kern, args...);
}

static size_t g_smem = 0;

size_t gemv_smem_bytes(int kmax) {
    return ((size_t)((kmax + 3) & ~3) * 2 + (size_t)kSlotTiles * kWarps * 32) * sizeof(float);
}

cudaError_t configure_kernels(int kmax) {
    if (gemv_smem_bytes(kmax) > g_smem) g_smem = gemv_smem_bytes(kmax);
    int dev = 0, optin = 0;
    cudaError_t e;
    if ((e = cudaGetDevice(&dev))) return e;
    if ((e = cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev))) return e;
    cudaFuncAttributes fa;
    // each kernel may use the opt-in maximum less its own static shared memory
#define EE_SMEM(k)                                                                                   \
    if ((e = cudaFuncGetAttributes(&fa, k))) return e;                                                \
    if ((e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize,                     \
                                  optin - (int)fa.sharedSizeBytes)))                                  \
        return e;
    EE_SMEM(k_qkv<true>) EE_SMEM(k_qkv<false>) EE_SMEM(k_kvfill<true>) EE_SMEM(k_kvfill<false>)
    EE_SMEM(k_oproj<true>) EE_SMEM(k_oproj<false>) EE_SMEM(k_gateup<true>) EE_SMEM(k_gateup<false>)
    EE_SMEM(k_down<true>) EE_SMEM(k_down<false>) EE_SMEM(k_readout<true>) EE_SMEM(k_readout<false>)
    EE_SMEM(k_vocab) EE_SMEM(k_vocab_rowmajor)
    if ((e = cudaFuncSetAttribute(k_attn_cluster<64>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1))) return e;
    if ((e = cudaFuncSetAttribute(k_attn_cluster<128>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1))) return e;
    EE_SMEM(k_attn_cluster<64>) EE_SMEM(k_attn_cluster<128>)
#undef EE_SMEM
    return cudaSuccess;
}

// x (K floats, padded to 16 bytes) + tile partials [+ the first layer's embedding row].
static size_t smem_for(int k, int extra = 0) {
    return ((size_t)((k + 3) & ~3) + (size_t)kSlotTiles * kWarps * 32 + (size_t)extra) * sizeof(float);
}

// Dynamic shared memory of a GEMV launch: x, tile partials, `extra` floats
// and, in whole-tile mode, the staged tile (32 rows x K bf16).
static size_t gemv_smem(int K, int extra, bool whole) {
    return smem_for(K, extra) + (whole ? (size_t)64 * K : 0);
}

cudaError_t launch_qkv(const DevModel& m, int layer, int first, int grid, bool whole, bool pdl, cudaStream_t s) {
    const size_t sm = gemv_smem(m.d, m.d, whole);
    if (whole) return launch_k(k_qkv<true>, dim3(grid), dim3(kGemvThreads), sm, pdl, s, m, layer, first);
    return launch_k(k_qkv<false>, dim3(grid), dim3(kGemvThreads), sm, pdl, s, m, layer, first);
}
cudaError_t launch_kvfill(const DevModel& m, int exit_layer, int grid_x, bool whole, bool pdl, cudaStream_t s) {
    const dim3 grid(grid_x, m.L - exit_layer);
    const size_t sm = gemv_smem(m.d, 0, whole);
    if (whole) return launch_k(k_kvfill<true>, grid, dim3(kGemvThreads), sm, pdl, s, m, exit_layer);
    return launch_k(k_kvfill<false>, grid, dim3(kGemvThreads), sm, pdl, s, m, exit_layer);
}
cudaError_t launch_record_exit(const DevModel& m, int exit_layer, bool pdl, cudaStream_t s) {
    return launch_k(k_record_exit, dim3((m.d + 255) / 256), dim3(256), 0, pdl, s, m, exit_layer);
}
size_t fill_pending_smem(int d) {
    return 4 * (size_t)(((d + 3) & ~3) + 8 * 32 + kFillThreads + 4) + 2 * 32 * (size_t)d;
}
cudaError_t configure_fill_pending(int d) {
    return cudaFuncSetAttribute(k_fill_pending, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)fill_pending_smem(d));
}
cudaError_t launch_fill_pending(const DevModel& m, int j0, int j1, bool pdl, cudaStream_t s) {
    if (j1 <= j0) return cudaSuccess;
    const dim3 grid((unsigned)((2LL * m.KH * m.D + 31) / 32), (unsigned)(j1 - j0));
    return launch_k(k_fill_pending, grid, dim3(kFillThreads), fill_pending_smem(m.d), pdl, s, m, j0);
}
cudaError_t launch_oproj(const DevModel& m, int layer, int grid, bool whole, bool pdl, cudaStream_t s) {
    const size_t sm = gemv_smem(m.A * m.D, 0, whole);
    if (whole) return launch_k(k_oproj<true>, dim3(grid), dim3(kGemvThreads), sm, pdl, s, m, layer);
    return launch_k(k_oproj<false>, dim3(grid), dim3(kGemvThreads), sm, pdl, s, m, layer);
}
cudaError_t launch_gateup(const DevModel& m, int layer, int grid, bool whole, bool pdl, cudaStream_t s) {
    const size_t sm = gemv_smem(m.d, 0, whole);
    if (whole) return launch_k(k_gateup<true>, dim3(grid), dim3(kGemvThreads), sm, pdl, s, m, layer);
    return launch_k(k_gateup<false>, dim3(grid), dim3(kGemvThreads), sm, pdl, s, m, layer);
}
cudaError_t launch_down(const DevModel& m, int layer, int grid, bool whole, bool pdl, cudaStream_t s) {
    const size_t sm = gemv_smem(m.F, 0, whole);
    if (whole) return launch_k(k_down<true>, dim3(grid), dim3(kGemvThreads), sm, pdl, s, m, layer);
    return launch_k(k_down<false>, dim3(grid), dim3(kGemvThreads), sm, pdl, s, m, layer);
}
cudaError_t launch_readout(const DevModel& m, int r, int grid, bool whole, bool pdl, cudaStream_t s) {
    const size_t sm = gemv_smem(m.d, 0, whole);
    if (whole) return launch_k(k_readout<true>, dim3(grid), dim3(kGemvThreads), sm, pdl, s, m, r);
    return launch_k(k_readout<false>, dim3(grid), dim3(kGemvThreads), sm, pdl, s, m, r);
}
cudaError_t launch_vocab(const VocabArgs& v, int grid, bool pdl, cudaStream_t s) {
    // x, then (LM head) the chunk partials of one row's logit
    const size_t smem = ((size_t)((v.d + 3) & ~3) + (size_t)(v.d / 8)) * sizeof(float);
    if (v.tiled) return launch_k(k_vocab, dim3(grid), dim3(kGemvThreads), smem, pdl, s, v);
    return launch_k(k_vocab_rowmajor, dim3(grid), dim3(kGemvThreads), smem, pdl, s, v);
}
cudaError_t launch_attention(const AttnArgs& a, int head_dim, bool pdl, cudaStream_t s) {
    const dim3 grid(kAttnMaxSplits, a.KH);
    if (head_dim == 64) return launch_k(k_attention<64>, grid, dim3(kAttnThreads), 0, pdl, s, a);
    if (head_dim == 128) return launch_k(k_attention<128>, grid, dim3(kAttnThreads), 0, pdl, s, a);
    return cudaErrorInvalidValue;
}
cudaError_t launch_attention_cluster(const AttnArgs& a, int head_dim, int cluster, bool pdl, cudaStream_t s) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(cluster, a.KH);
    cfg.blockDim = dim3(kAttnThreads);
    cfg.dynamicSmemBytes = head_dim == 64 ? AttnSmem<64>::bytes : AttnSmem<128>::bytes;
    cfg.stream = s;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = cluster;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl ? 2 : 1;
    if (head_dim == 64) return cudaLaunchKernelEx(&cfg, k_attn_cluster<64>, a);
    if (head_dim == 128) return cudaLaunchKernelEx(&cfg, k_attn_cluster<128>, a);
    return cudaErrorInvalidValue;
}
int attention_cluster_size(int head_dim, int n_kv_heads) {
    for (int cl : {16, 8}) {
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(cl, n_kv_heads);
        cfg.blockDim = dim3(kAttnThreads);
        cfg.dynamicSmemBytes = head_dim == 64 ? AttnSmem<64>::bytes : AttnSmem<128>::bytes;
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeClusterDimension;
        attr[0].val.clusterDim.x = cl;
        attr[0].val.clusterDim.y = 1;
        attr[0].val.clusterDim.z = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        int n = 0;
        const cudaError_t e = head_dim == 64 ? cudaOccupancyMaxActiveClusters(&n, k_attn_cluster<64>, &cfg)
                                             : cudaOccupancyMaxActiveClusters(&n, k_attn_cluster<128>, &cfg);
        if (e == cudaSuccess && n >= 1) return cl;
        cudaGetLastError();
    }
    return 8;
}
cudaError_t launch_step_end(const DevModel& m, int has_cond, cudaGraphConditionalHandle cond, bool pdl,
                            cudaStream_t s) {
    return launch_k(k_step_end, dim3(1), dim3(32), 0, pdl, s, m, has_cond, cond);
}
cudaError_t launch_prefill_advance(const DevModel& m, int has_cond, cudaGraphConditionalHandle cond, bool pdl,
                                   cudaStream_t s) {
    return launch_k(k_prefill_advance, dim3(1), dim3(32), 0, pdl, s, m, has_cond, cond);
}
cudaError_t launch_prefill_end(const DevModel& m, bool pdl, cudaStream_t s) {
    return launch_k(k_prefill_end, dim3(1), dim3(32), 0, pdl, s, m);
}
cudaError_t launch_set_inputs(Ctl* c, const CtlInputs& in, cudaStream_t s) {
    return launch_k(k_set_inputs, dim3(1), dim3(32), 0, false, s, c, in);
}

}  // namespace ee
