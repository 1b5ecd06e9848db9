// Persistent layer-segment kernel for sm_103a: layers [j0, j1) of one decode
// step in a single launch.
//
// Each step of a layer is the paper's decoder layer (§2; App. C): RMSNorm,
// Q/K/V projection with RoPE and the KV append, grouped-query attention over
// the paged cache, output projection with the residual add, RMSNorm, the
// gated feed-forward (SiLU(W_g x) * W_u x) and the down projection with the
// residual add.  The arithmetic is the same as the per-kernel path in
// ee_kernels.cu; the difference is how bytes move.
//
// One CTA per SM.  Warp 8 is the producer: its lane 0 walks the CTA's whole
// work list for the segment -- its share of every weight matrix, cut into
// 16 KB chunks of 32 rows x 256 columns of the tile-packed layout, and the
// key/value pages of its attention unit -- and streams each chunk into a
// shared-memory ring with cp.async.bulk, completing on an mbarrier.  Weights
// and the cache entries of earlier positions do not depend on the step, so
// the producer runs ahead of the data dependencies and HBM stays busy while
// the consumers wait for one.  Warps 0..7 consume the ring in the same order.
//
// Phases hand results to each other through global memory: a phase writes
// per-tile partial sums ([tile][slot][32], one slot per CTA that covered part
// of the tile), bumps a completion counter with a release, and the next
// phase's CTAs acquire the counter once every CTA has bumped it and rebuild
// exactly the inputs they need by summing the slots in slot order (the
// result does not depend on timing).  The residual stream is never updated
// in place inside the segment: h_in of layer j lives in hbuf[j & 1] and
// h_out = h_in + (O-projection slots) + (down slots), rebuilt by whoever
// reads it; the last phase writes h_out of the last layer to the model's h.
//
// Every wait is bounded: after kStallNs the waiting thread sets kErrStall in
// the control block and the CTA winds down (the producer first waits, again
// with a bound, for the copies it still has in flight).  Co-residency of all
// CTAs, which the cross-CTA waits rely on, comes from a cooperative launch.
#include <cuda_bf16.h>
#include <math.h>

#include <algorithm>

#include "ee_internal.h"

namespace ee {
namespace {

constexpr int kCW = kSegConsumerWarps;
constexpr int kCT = 32 * kCW;              // consumer threads
constexpr int kColsPerChunk = kSegChunk / (2 * kTileRows);  // 256
constexpr unsigned long long kStallNs = 2000000000ull;     // 2 s

enum { kPhQKV = 0, kPhAttn = 1, kPhO = 2, kPhGU = 3, kPhDn = 4, kPhases = 5 };

__device__ __forceinline__ float bf(uint16_t b) { return __uint_as_float((uint32_t)b << 16); }
__device__ __forceinline__ float bflo(uint32_t v) { return __uint_as_float(v << 16); }
__device__ __forceinline__ float bfhi(uint32_t v) { return __uint_as_float(v & 0xffff0000u); }
__device__ __forceinline__ uint16_t tobf(float f) { return __bfloat16_as_ushort(__float2bfloat16_rn(f)); }
__device__ __forceinline__ float round_bf(float f) { return bf(tobf(f)); }

__device__ __forceinline__ unsigned long long now_ns() {
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}
__device__ __forceinline__ uint32_t saddr(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }

// ---------------------------------------------------------------- mbarriers
__device__ __forceinline__ void mb_init(uint64_t* b, int n) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(saddr(b)), "r"(n) : "memory");
}
__device__ __forceinline__ bool mb_test(uint64_t* b, int parity) {
    uint32_t ok;
    asm volatile(
        "{ .reg .pred p; mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2; selp.u32 %0, 1, 0, p; }"
        : "=r"(ok)
        : "r"(saddr(b)), "r"(parity)
        : "memory");
    return ok != 0;
}
// Wait for the phase of parity `parity` to complete; false after the time
// limit or once another thread has flagged a stall.
__device__ __forceinline__ bool mb_wait(uint64_t* b, int parity, const volatile int* err) {
    if (mb_test(b, parity)) return true;
    const unsigned long long t0 = now_ns();
    for (unsigned it = 1;; ++it) {
        if (mb_test(b, parity)) return true;
        if ((it & 63) == 0 && ((*err & kErrStall) || now_ns() - t0 > kStallNs)) return false;
    }
}
__device__ __forceinline__ void mb_arrive(uint64_t* b) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(saddr(b)) : "memory");
}
__device__ __forceinline__ void mb_expect_tx(uint64_t* b, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(saddr(b)), "r"(bytes) : "memory");
}
// Bulk copy global -> this CTA's shared memory, completing on `bar`.  The
// weights are read once per step: evict-first in L2.
__device__ __forceinline__ void bulk_load(void* dst, const void* src, uint32_t bytes, uint64_t* bar, uint64_t pol) {
    asm volatile(
        "cp.async.bulk.shared::cta.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], %4;" ::"r"(
            saddr(dst)),
        "l"(src), "r"(bytes), "r"(saddr(bar)), "l"(pol)
        : "memory");
}
__device__ __forceinline__ uint64_t evict_first() {
    uint64_t pol;
    asm("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
    return pol;
}
__device__ __forceinline__ uint64_t evict_normal() {
    uint64_t pol;
    asm("createpolicy.fractional.L2::evict_normal.b64 %0, 1.0;" : "=l"(pol));
    return pol;
}

// Barrier of the consumer warps only (the producer never joins it).
__device__ __forceinline__ void csync() { asm volatile("bar.sync 1, %0;" ::"r"(kCT) : "memory"); }

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
    for (int o = 16; o; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}
__device__ __forceinline__ float dot8(const uint4 w, const float* x) {
    const float4 a = *reinterpret_cast<const float4*>(x);
    const float4 b = *reinterpret_cast<const float4*>(x + 4);
    float s = bflo(w.x) * a.x;
    s = fmaf(bfhi(w.x), a.y, s);
    s = fmaf(bflo(w.y), a.z, s);
    s = fmaf(bfhi(w.y), a.w, s);
    s = fmaf(bflo(w.z), b.x, s);
    s = fmaf(bfhi(w.z), b.y, s);
    s = fmaf(bflo(w.w), b.z, s);
    s = fmaf(bfhi(w.w), b.w, s);
    return s;
}

// ------------------------------------------------------------ work geometry
// Matrix mt of layer j as ring items: item i = (tile i / nc, chunk i % nc).
// Items are split into contiguous ranges over Ge = min(G, N) CTAs.
struct Items {
    int N, Ge, lo, hi, nc, K, n_tiles;
};
__device__ __forceinline__ Items items_of(const SegPlan& p, int mt, int cta) {
    Items it;
    it.nc = p.n_chunks[mt];
    it.K = p.K[mt];
    it.n_tiles = p.n_tiles[mt];
    it.N = it.n_tiles * it.nc;
    it.Ge = min(p.G, it.N);
    if (cta < it.Ge) {
        it.lo = (int)((int64_t)cta * it.N / it.Ge);
        it.hi = (int)((int64_t)(cta + 1) * it.N / it.Ge);
    } else {
        it.lo = it.hi = 0;
    }
    return it;
}
// The CTA whose range holds item i.
__device__ __forceinline__ int item_owner(const Items& it, int i) {
    return (int)(((int64_t)(i + 1) * it.Ge - 1) / it.N);
}
__device__ __forceinline__ int tile_slots(const Items& it, int t) {
    return item_owner(it, t * it.nc + it.nc - 1) - item_owner(it, t * it.nc) + 1;
}
// Sum of the slots of row `lane` of tile t (slot order, so deterministic).
__device__ __forceinline__ float slot_sum(const float* part, const Items& it, int t, int lane) {
    const int ns = tile_slots(it, t);
    const float* q = part + (int64_t)t * it.nc * 32 + lane;
    float s = 0.f;
    for (int k = 0; k < ns; ++k) s += q[k * 32];
    return s;
}
__device__ __forceinline__ uint32_t chunk_bytes(const Items& it, int c) {
    return (uint32_t)min(kColsPerChunk, it.K - c * kColsPerChunk) * (2 * kTileRows);
}

__device__ __forceinline__ const uint8_t* layer_bytes(const DevModel& m, int j, int64_t off) {
    return reinterpret_cast<const uint8_t*>(m.layers + (int64_t)j * m.layer_stride + off);
}
__device__ __forceinline__ const uint8_t* mat_base(const DevModel& m, int j, int mt) {
    const int64_t off = mt == 0 ? m.off_wqkv : mt == 1 ? m.off_wo : mt == 2 ? m.off_wgu : m.off_wd;
    return layer_bytes(m, j, off);
}

// Attention work of one step: kv head g, split s covers logical pages
// [s * pps, min((s + 1) * pps, n_pages)).  Unit u = g * splits + s runs on
// CTA u * G / U.
struct AttnGeo {
    int T, n_pages, pps, splits, U;
};
__device__ __forceinline__ AttnGeo attn_geo(const DevModel& m, const SegPlan& p, int pos) {
    AttnGeo a;
    a.T = pos + 1;
    a.n_pages = (a.T + m.page_size - 1) / m.page_size;
    const int cap = max(1, min(kSegMaxSplits, p.G / m.KH));
    a.pps = (a.n_pages + cap - 1) / cap;
    a.splits = (a.n_pages + a.pps - 1) / a.pps;
    a.U = m.KH * a.splits;
    return a;
}
// Attention unit of this CTA, or -1.
__device__ __forceinline__ int attn_unit(const AttnGeo& a, int G, int cta) {
    // u * G / U == cta  <=>  u = ceil(cta * U / G) when that u maps back to cta
    const int u = (int)(((int64_t)cta * a.U + G - 1) / G);
    if (u < a.U && (int)((int64_t)u * G / a.U) == cta) return u;
    return -1;
}

// ------------------------------------------------------------ shared memory
struct Smem {
    uint8_t* ring;      // stages x kSegChunk
    uint64_t* full;     // [stages]
    uint64_t* empty;    // [stages]
    float* xs;          // [d] normalised input of Q/K/V and gate/up
    float* hs;          // [d] residual
    float* xc;          // [256] input columns of an O-projection or down chunk
    float* red;         // [2][kCW][32]
    float* qa;          // [group][D] rotated queries of the attention unit
    float* kv;          // [2][D] k, v of the step's position (bf16 values)
    float* sc;          // [group][pps * page_size] scores, then probabilities
    float* ml;          // [group][2] max, sum
};
__device__ __forceinline__ Smem carve(uint8_t* base, const DevModel& m, const SegPlan& p) {
    Smem s;
    uint8_t* q = base;
    s.ring = q;
    q += (size_t)p.stages * kSegChunk;
    s.full = reinterpret_cast<uint64_t*>(q);
    q += 8 * p.stages;
    s.empty = reinterpret_cast<uint64_t*>(q);
    q += 8 * p.stages;
    float* f = reinterpret_cast<float*>(q);
    s.xs = f;
    f += (m.d + 3) & ~3;
    s.hs = f;
    f += (m.d + 3) & ~3;
    s.xc = f;
    f += kColsPerChunk;
    s.red = f;
    f += 2 * kCW * 32;
    const int grp = m.A / m.KH;
    s.qa = f;
    f += grp * m.D;
    s.kv = f;
    f += 2 * m.D;
    s.sc = f;
    f += grp * p.max_pps * m.page_size;
    s.ml = f;
    return s;
}

// ------------------------------------------------------------ the producer
struct Producer {
    const Smem& s;
    int stages;
    long long n;  // chunks issued
    uint64_t pol_w, pol_kv;
    const volatile int* err;
    bool ok = true;
    __device__ Producer(const Smem& sm, int st, const volatile int* e)
        : s(sm), stages(st), n(0), pol_w(evict_first()), pol_kv(evict_normal()), err(e) {}
    __device__ __forceinline__ void push(const void* src, uint32_t bytes, uint64_t pol) {
        if (!ok) return;
        const int st = (int)(n % stages);
        if (n >= stages && !mb_wait(&s.empty[st], (int)(((n / stages) - 1) & 1), err)) {
            atomicOr((int*)err, kErrStall);
            ok = false;
            return;
        }
        mb_expect_tx(&s.full[st], bytes);
        bulk_load(s.ring + (size_t)st * kSegChunk, src, bytes, &s.full[st], pol);
        ++n;
    }
    // Before leaving: every issued copy has landed (the consumers normally
    // see to that; after a stall they may not have).
    __device__ void drain() {
        for (long long i = max(0ll, n - stages); i < n; ++i)
            mb_wait(&s.full[i % stages], (int)((i / stages) & 1), err);
    }
};

// ------------------------------------------------------------ the consumers
struct Consumer {
    const Smem& s;
    int stages;
    long long n;
    volatile int* err;
    bool ok = true;
    __device__ Consumer(const Smem& sm, int st, volatile int* e) : s(sm), stages(st), n(0), err(e) {}
    __device__ __forceinline__ const uint8_t* acquire() {
        const int st = (int)(n % stages);
        if (ok && !mb_wait(&s.full[st], (int)((n / stages) & 1), err)) {
            atomicOr((int*)err, kErrStall);
            ok = false;
        }
        return s.ring + (size_t)st * kSegChunk;
    }
    __device__ __forceinline__ void release() {
        __syncwarp();
        if ((threadIdx.x & 31) == 0) mb_arrive(&s.empty[n % stages]);
        ++n;
    }
};

// Wait (one thread) until counter >= target, then sync the consumers.  False
// on a stall (flagged in the control block).
__device__ __forceinline__ bool wait_count(const unsigned* cnt, unsigned target, volatile int* err) {
    __shared__ int ok_s;
    if (threadIdx.x == 0) {
        int ok = 1;
        unsigned v;
        asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(cnt) : "memory");
        if (v < target) {
            const unsigned long long t0 = now_ns();
            for (unsigned it = 1;; ++it) {
                asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(cnt) : "memory");
                if (v >= target) break;
                if ((it & 15) == 0 && ((*err & kErrStall) || now_ns() - t0 > kStallNs)) {
                    atomicOr((int*)err, kErrStall);
                    ok = 0;
                    break;
                }
            }
        }
        ok_s = ok;
    }
    csync();
    return ok_s != 0;
}
// All consumer threads' global writes, then one release increment.
__device__ __forceinline__ void signal_count(unsigned* cnt) {
    __threadfence();
    csync();
    if (threadIdx.x == 0) asm volatile("red.release.gpu.global.add.u32 [%0], 1;" ::"l"(cnt) : "memory");
}

// RMSNorm of hs (d values) times gain g into xs (consumer threads).
__device__ __forceinline__ void rmsnorm_sm(const float* hs, const uint16_t* g, int d, float eps, float* xs,
                                           float* red) {
    const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
    float ss = 0.f;
    for (int i = threadIdx.x; i < d; i += kCT) ss = fmaf(hs[i], hs[i], ss);
    ss = warp_sum(ss);
    if (l == 0) red[w] = ss;
    csync();
    float t = l < kCW ? red[l] : 0.f;
    t = warp_sum(t);
    const float inv = 1.0f / sqrtf(t / (float)d + eps);
    for (int i = threadIdx.x; i < d; i += kCT) xs[i] = hs[i] * inv * bf(g[i]);
    csync();
}

// Stream this CTA's items of one matrix against x, writing tile partial
// slots.  xfn(c) returns the 256 input columns of chunk c (it may rebuild
// them into shared memory; every consumer thread calls it).
template <class XFn>
__device__ __forceinline__ void gemv_items(Consumer& cs, const Items& it, int cta, float* part, float* red, XFn xfn) {
    const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
    float acc = 0.f;
    int rb = 0;
    for (int i = it.lo; i < it.hi; ++i) {
        const int t = i / it.nc, c = i - t * it.nc;
        const float* x = xfn(c);
        const uint4* buf = reinterpret_cast<const uint4*>(cs.acquire());
        const int ccn = (int)(chunk_bytes(it, c) / 512);
        if (cs.ok)
            for (int cc = w; cc < ccn; cc += kCW) acc += dot8(buf[cc * 32 + lane], x + cc * 8);
        cs.release();
        if (i + 1 == it.hi || c + 1 == it.nc) {
            float* r = red + rb * kCW * 32;
            r[w * 32 + lane] = acc;
            acc = 0.f;
            csync();
            if (w == 0) {
                float sum = 0.f;
#pragma unroll
                for (int k = 0; k < kCW; ++k) sum += r[k * 32 + lane];
                const int slot = cta - item_owner(it, t * it.nc);
                part[((int64_t)t * it.nc + slot) * 32 + lane] = sum;
            }
            rb ^= 1;
        }
    }
}

// Residual rebuild: hs = hbuf_prev + O slots + down slots of layer jp (or a
// plain copy of `src`).
__device__ __forceinline__ void rebuild_h(const DevModel& m, const SegPlan& p, const float* hin, bool add_parts,
                                          float* hs) {
    const Items io = items_of(p, 1, 0), idn = items_of(p, 3, 0);
    for (int i = threadIdx.x; i < m.d; i += kCT) {
        float v = hin[i];
        if (add_parts) {
            v += slot_sum(p.part[1], io, i >> 5, i & 31);
            v += slot_sum(p.part[3], idn, i >> 5, i & 31);
        }
        hs[i] = v;
    }
}

}  // namespace

__global__ void __launch_bounds__(kSegThreads, 1) k_layers(DevModel m, SegPlan p, int j0, int j1, int first) {
    extern __shared__ __align__(128) uint8_t seg_smem[];
    const Smem s = carve(seg_smem, m, p);
    const int cta = blockIdx.x, G = p.G;
    volatile int* err = &m.ctl->err;
    const int half = m.D >> 1, grp = m.A / m.KH;
    const int nq = m.A * half, nk = m.KH * half;

    if (threadIdx.x == 0) {
        for (int i = 0; i < p.stages; ++i) {
            mb_init(&s.full[i], 1);
            mb_init(&s.empty[i], kCW);
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    __syncthreads();

    Ctl* c = m.ctl;
    const int pos = c->pos;
    const bool pos_ok = pos >= 0 && pos < m.max_ctx;
    const AttnGeo ag = attn_geo(m, p, pos_ok ? pos : 0);
    const int unit = attn_unit(ag, G, cta);
    const int rpc = p.rows_per_kv_chunk, cpp = m.page_size / rpc;

    // ---------------------------------------------------------- producer
    if (threadIdx.x >= kCT) {
        if (threadIdx.x != kCT || !pos_ok) return;
        Producer pr(s, p.stages, err);
        for (int j = j0; j < j1 && pr.ok; ++j) {
            for (int mt = 0; mt < 4; ++mt) {
                const Items it = items_of(p, mt, cta);
                const uint8_t* W = mat_base(m, j, mt);
                for (int i = it.lo; i < it.hi; ++i) {
                    const int t = i / it.nc, ch = i - t * it.nc;
                    pr.push(W + (int64_t)t * kTileRows * it.K * 2 + (int64_t)ch * kSegChunk, chunk_bytes(it, ch),
                            pr.pol_w);
                }
                if (mt == 0 && unit >= 0) {
                    const int g = unit / ag.splits, sp = unit - g * ag.splits;
                    const int pg0 = sp * ag.pps, pg1 = min(ag.n_pages, pg0 + ag.pps);
                    const uint16_t* pools[2] = {m.kpool + (int64_t)j * m.kv_layer_stride,
                                                m.vpool + (int64_t)j * m.kv_layer_stride};
                    for (int kvi = 0; kvi < 2; ++kvi)
                        for (int pg = pg0; pg < pg1; ++pg) {
                            const int phys = m.page_table[pg];
                            for (int q = 0; q < cpp; ++q)
                                pr.push(pools[kvi] + (((int64_t)phys * m.KH + g) * m.page_size + q * rpc) * m.D,
                                        (uint32_t)(rpc * m.D * 2), pr.pol_kv);
                        }
                }
            }
        }
        pr.drain();
        return;
    }

    // ---------------------------------------------------------- consumers
    const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (!pos_ok) {
        if (cta == 0 && threadIdx.x == 0) atomicOr(&c->err, kErrPosition);
        return;
    }
    Consumer cs(s, p.stages, err);
    unsigned* sync = p.sync;
    const float2* cs_row = m.rope + (int64_t)pos * half;
    const float scale = 1.0f / sqrtf((float)m.D);
    const int slice0 = (int)((int64_t)cta * m.d / G), slice1 = (int)((int64_t)(cta + 1) * m.d / G);

    if (first && cta == 0 && threadIdx.x == 0) {
        c->exit_readout = -1;
        c->n_evaluated = 0;
        c->full_token = -1;
    }

    for (int j = j0; j < j1; ++j) {
        const int li = j - j0;
        unsigned* cnt = sync + li * kPhases;
        const uint16_t* lw = m.layers + (int64_t)j * m.layer_stride;

        // ---------------- Q/K/V: residual in, RMSNorm, projection slots
        if (j > j0 && !wait_count(cnt - kPhases + kPhDn, G, err)) return;
        float* hin = p.hbuf + (j & 1) * m.d;
        if (j == j0 && first) {
            int tok = c->in_tok;
            if (tok < 0 || tok >= m.V) {
                if (cta == 0 && threadIdx.x == 0) atomicOr(&c->err, kErrTokenRange);
                tok = 0;
            }
            const uint16_t* e = m.embed + (int64_t)tok * m.d;
            for (int i = threadIdx.x; i < m.d; i += kCT) s.hs[i] = bf(e[i]);
        } else if (j == j0) {
            rebuild_h(m, p, m.h, false, s.hs);
        } else {
            rebuild_h(m, p, p.hbuf + ((j - 1) & 1) * m.d, true, s.hs);
        }
        csync();
        for (int i = slice0 + threadIdx.x; i < slice1; i += kCT) hin[i] = s.hs[i];
        rmsnorm_sm(s.hs, lw + m.off_gattn, m.d, m.eps, s.xs, s.red);
        {
            const Items it = items_of(p, 0, cta);
            gemv_items(cs, it, cta, p.part[0], s.red, [&](int ch) { return s.xs + ch * kColsPerChunk; });
        }
        signal_count(cnt + kPhQKV);

        // ---------------- attention unit (if this CTA has one)
        if (unit >= 0) {
            const int g = unit / ag.splits, sp = unit - g * ag.splits;
            const int pg0 = sp * ag.pps, pg1 = min(ag.n_pages, pg0 + ag.pps);
            const int p0 = pg0 * m.page_size, p1 = min(ag.T, pg1 * m.page_size);
            const int npos = p1 - p0;
            if (!wait_count(cnt + kPhQKV, G, err)) return;
            // rebuild q (rotated), k and v of the step's position for group g
            const Items iq = items_of(p, 0, 0);
            const uint16_t* bias = m.qkv_bias ? lw + m.off_bqkv : nullptr;
            for (int e = threadIdx.x; e < (grp + 2) * half; e += kCT) {
                const int hh = e / half, i = e - hh * half;
                int u;
                if (hh < grp)
                    u = (g * grp + hh) * half + i;
                else if (hh == grp)
                    u = nq + g * half + i;
                else
                    u = nq + nk + g * half + i;
                const int t = u >> 4, l0 = (u & 15) * 2;
                float r0 = slot_sum(p.part[0], iq, t, l0), r1 = slot_sum(p.part[0], iq, t, l0 + 1);
                if (bias) {
                    r0 += bf(bias[2 * u]);
                    r1 += bf(bias[2 * u + 1]);
                }
                if (hh <= grp) {
                    const float2 cz = cs_row[i];
                    const float a0 = r0 * cz.x - r1 * cz.y, a1 = r0 * cz.y + r1 * cz.x;
                    if (hh < grp) {
                        s.qa[hh * m.D + i] = a0 * scale;
                        s.qa[hh * m.D + i + half] = a1 * scale;
                    } else {
                        s.kv[i] = round_bf(a0);
                        s.kv[i + half] = round_bf(a1);
                    }
                } else {
                    s.kv[m.D + i] = round_bf(r0);
                    s.kv[m.D + i + half] = round_bf(r1);
                }
            }
            csync();
            if (sp == 0) {  // the cache entry of this position, for later steps
                const int64_t off = (int64_t)j * m.kv_layer_stride +
                                    (((int64_t)m.page_table[pos / m.page_size] * m.KH + g) * m.page_size +
                                     pos % m.page_size) *
                                        m.D;
                for (int i = threadIdx.x; i < m.D; i += kCT) {
                    m.kpool[off + i] = tobf(s.kv[i]);
                    m.vpool[off + i] = tobf(s.kv[m.D + i]);
                }
                if (g == 0 && threadIdx.x == 0) m.kv_src[(int64_t)j * m.max_ctx + pos] = 1;
            }
            // scores: warp per position, lane per D/32 dimensions
            const int dpl = m.D >> 5;  // 2 or 4
            float qr[kSegMaxGroup][4];
#pragma unroll
            for (int hh = 0; hh < kSegMaxGroup; ++hh)
#pragma unroll
                for (int k = 0; k < 4; ++k) qr[hh][k] = (hh < grp && k < dpl) ? s.qa[hh * m.D + lane * dpl + k] : 0.f;
            const int spc = p.max_pps * m.page_size;  // score row stride
            for (int pg = pg0; pg < pg1; ++pg)
                for (int q = 0; q < cpp; ++q) {
                    const uint16_t* kb = reinterpret_cast<const uint16_t*>(cs.acquire());
                    const int base = pg * m.page_size + q * rpc;
                    for (int r = w; r < rpc; r += kCW) {
                        const int ps = base + r;
                        if (ps >= p1) break;
                        float kd[4];
#pragma unroll
                        for (int k = 0; k < 4; ++k)
                            kd[k] = k < dpl ? (ps == pos ? s.kv[lane * dpl + k] : bf(kb[r * m.D + lane * dpl + k])) : 0.f;
#pragma unroll
                        for (int hh = 0; hh < kSegMaxGroup; ++hh) {
                            if (hh >= grp) break;
                            float d = 0.f;
#pragma unroll
                            for (int k = 0; k < 4; ++k) d = fmaf(qr[hh][k], kd[k], d);
                            d = warp_sum(d);
                            if (lane == 0) s.sc[hh * spc + (ps - p0)] = d;
                        }
                    }
                    cs.release();
                }
            csync();
            for (int hh = w; hh < grp; hh += kCW) {
                float mx = -INFINITY;
                for (int k = lane; k < npos; k += 32) mx = fmaxf(mx, s.sc[hh * spc + k]);
                mx = warp_max(mx);
                float sum = 0.f;
                for (int k = lane; k < npos; k += 32) {
                    const float e = expf(s.sc[hh * spc + k] - mx);
                    s.sc[hh * spc + k] = e;
                    sum += e;
                }
                sum = warp_sum(sum);
                if (lane == 0) {
                    s.ml[2 * hh] = mx;
                    s.ml[2 * hh + 1] = sum;
                }
            }
            csync();
            // P V: warp per head, lane per D/32 dimensions
            float oacc[4] = {0.f, 0.f, 0.f, 0.f};
            for (int pg = pg0; pg < pg1; ++pg)
                for (int q = 0; q < cpp; ++q) {
                    const uint16_t* vb = reinterpret_cast<const uint16_t*>(cs.acquire());
                    const int base = pg * m.page_size + q * rpc;
                    if (w < grp && cs.ok)
                        for (int r = 0; r < rpc; ++r) {
                            const int ps = base + r;
                            if (ps >= p1) break;
                            const float pr = s.sc[w * spc + (ps - p0)];
#pragma unroll
                            for (int k = 0; k < 4; ++k)
                                if (k < dpl)
                                    oacc[k] = fmaf(pr, ps == pos ? s.kv[m.D + lane * dpl + k]
                                                                 : bf(vb[r * m.D + lane * dpl + k]),
                                                   oacc[k]);
                        }
                    cs.release();
                }
            if (w < grp) {
                float* dst = p.attn_part + ((int64_t)(g * grp + w) * kAttnMaxSplits + sp) * (m.D + 2);
#pragma unroll
                for (int k = 0; k < 4; ++k)
                    if (k < dpl) dst[lane * dpl + k] = oacc[k];
                if (lane == 0) {
                    dst[m.D] = s.ml[2 * w];
                    dst[m.D + 1] = s.ml[2 * w + 1];
                }
            }
        }
        signal_count(cnt + kPhAttn);

        // ---------------- O-projection slots (input: merged attention output)
        if (!wait_count(cnt + kPhAttn, G, err)) return;
        {
            const Items it = items_of(p, 1, cta);
            gemv_items(cs, it, cta, p.part[1], s.red, [&](int ch) {
                // columns [256 ch, 256 ch + 256) of o: merge the splits of each head
                csync();  // the previous chunk's readers of xc are done
                const int c0 = ch * kColsPerChunk, nc = min(kColsPerChunk, m.A * m.D - c0);
                for (int e = threadIdx.x; e < nc; e += kCT) {
                    const int col = c0 + e, h = col / m.D, dd = col - h * m.D;
                    const float* src = p.attn_part + (int64_t)h * kAttnMaxSplits * (m.D + 2);
                    float mx = -INFINITY;
                    for (int k = 0; k < ag.splits; ++k) mx = fmaxf(mx, src[k * (m.D + 2) + m.D]);
                    float num = 0.f, den = 0.f;
                    for (int k = 0; k < ag.splits; ++k) {
                        const float* q = src + k * (m.D + 2);
                        const float wgt = expf(q[m.D] - mx);
                        num = fmaf(wgt, q[dd], num);
                        den = fmaf(wgt, q[m.D + 1], den);
                    }
                    s.xc[e] = num / den;
                }
                csync();
                return (const float*)s.xc;
            });
        }
        signal_count(cnt + kPhO);

        // ---------------- gate/up slots (input: RMSNorm of the mid residual)
        if (!wait_count(cnt + kPhO, G, err)) return;
        {
            const Items io = items_of(p, 1, 0);
            for (int i = threadIdx.x; i < m.d; i += kCT) s.hs[i] = hin[i] + slot_sum(p.part[1], io, i >> 5, i & 31);
            csync();
            rmsnorm_sm(s.hs, lw + m.off_gmlp, m.d, m.eps, s.xs, s.red);
            const Items it = items_of(p, 2, cta);
            gemv_items(cs, it, cta, p.part[2], s.red, [&](int ch) { return s.xs + ch * kColsPerChunk; });
        }
        signal_count(cnt + kPhGU);

        // ---------------- down slots (input: SiLU(gate) * up)
        if (!wait_count(cnt + kPhGU, G, err)) return;
        {
            const Items ig = items_of(p, 2, 0);
            const Items it = items_of(p, 3, cta);
            gemv_items(cs, it, cta, p.part[3], s.red, [&](int ch) {
                csync();  // the previous chunk's readers of xc are done
                const int c0 = ch * kColsPerChunk, nc = min(kColsPerChunk, m.F - c0);
                for (int e = threadIdx.x; e < nc; e += kCT) {
                    const int f = c0 + e, t = f >> 4, l0 = (f & 15) * 2;
                    const float gt = slot_sum(p.part[2], ig, t, l0), up = slot_sum(p.part[2], ig, t, l0 + 1);
                    s.xc[e] = gt / (1.0f + expf(-gt)) * up;
                }
                csync();
                return (const float*)s.xc;
            });
        }
        signal_count(cnt + kPhDn);
    }

    // ---------------- the segment's output residual, then the exit ticket
    if (!wait_count(sync + (j1 - 1 - j0) * kPhases + kPhDn, G, err)) return;
    {
        const Items io = items_of(p, 1, 0), idn = items_of(p, 3, 0);
        const float* hin = p.hbuf + ((j1 - 1) & 1) * m.d;
        for (int i = slice0 + threadIdx.x; i < slice1; i += kCT)
            m.h[i] = hin[i] + slot_sum(p.part[1], io, i >> 5, i & 31) + slot_sum(p.part[3], idn, i >> 5, i & 31);
    }
    __threadfence();
    csync();
    if (threadIdx.x == 0) {
        unsigned* ticket = sync + (j1 - j0) * kPhases;
        const unsigned prev = atomicAdd(ticket, 1u);
        if (prev == (unsigned)G - 1) {  // every CTA is past its last wait: reset for the next launch
            for (int i = 0; i <= (j1 - j0) * kPhases; ++i) sync[i] = 0;
            __threadfence();
        }
    }
}

bool seg_plan(const DevModel& m, int n_sm, SegPlan& p) {
    p.G = n_sm;
    const int grp = m.A / m.KH;
    if (m.A % m.KH || grp > kSegMaxGroup || (m.D != 64 && m.D != 128)) return false;
    const int Ks[4] = {m.d, m.A * m.D, m.d, m.F};
    const int64_t rows[4] = {(int64_t)(m.A + 2 * m.KH) * m.D, m.d, 2LL * m.F, m.d};
    for (int i = 0; i < 4; ++i) {
        if (Ks[i] % 8) return false;
        p.K[i] = Ks[i];
        p.n_tiles[i] = (int)tile_count(rows[i]);
        p.n_chunks[i] = (Ks[i] + kColsPerChunk - 1) / kColsPerChunk;
    }
    p.rows_per_kv_chunk = std::min(m.page_size, kSegChunk / (2 * m.D));
    if (m.page_size % p.rows_per_kv_chunk) return false;
    const int cap = std::max(1, std::min(kSegMaxSplits, p.G / m.KH));
    const int np_max = (m.max_ctx + m.page_size - 1) / m.page_size;
    p.max_pps = std::max(1, (np_max + cap - 1) / cap);
    const size_t floats = 2 * (size_t)((m.d + 3) & ~3) + kColsPerChunk + 2 * kCW * 32 + (size_t)grp * m.D +
                          2 * (size_t)m.D + (size_t)grp * p.max_pps * m.page_size + 2 * (size_t)grp;
    const size_t fixed = floats * 4 + 256;
    const size_t budget = 227 * 1024;
    if (fixed + 4 * (size_t)(kSegChunk + 16) > budget) return false;
    p.stages = (int)std::min<size_t>(16, (budget - fixed) / (kSegChunk + 16));
    p.smem = (size_t)p.stages * (kSegChunk + 16) + floats * 4;
    return true;
}

cudaError_t configure_layers(size_t smem) {
    return cudaFuncSetAttribute(k_layers, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
}

int layers_blocks_per_sm(size_t smem) {
    int n = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, k_layers, kSegThreads, smem) != cudaSuccess) return 0;
    return n;
}

cudaError_t launch_layers(const DevModel& m, const SegPlan& p, int j0, int j1, int first, cudaStream_t s) {
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = dim3(p.G);
    cfg.blockDim = dim3(kSegThreads);
    cfg.dynamicSmemBytes = p.smem;
    cfg.stream = s;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeCooperative;
    at[0].val.cooperative = 1;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, k_layers, m, p, j0, j1, first);
}

}  // namespace ee
