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
// 32 KB chunks of 32 rows x 512 columns of the tile-packed layout, and the
// key/value pages of its attention unit -- and streams each chunk into a
// shared-memory ring with cp.async.bulk, completing on an mbarrier.  Weights
// and the cache entries of earlier positions do not depend on the step, so
// the producer runs ahead of the data dependencies and HBM stays busy while
// the consumers wait for one.  Warps 0..7 consume the ring in the same order.
//
// Phases hand results to each other through global memory as tagged
// values (see "tagged values" below): every float one CTA hands to another
// travels in a 64-bit word beside its layer's tag, and the reader loads
// until the tags are the expected ones, so there are no phase counters and
// no fences.  Q/K/V and gate/up are split by whole 32-row tiles, so each
// tile's epilogue (bias, RoPE and the KV append; SiLU(gate) * up) runs in
// the CTA that owns it.  The O and down projections have few, long rows:
// they are split into (tile, 512-column chunk) items over all CTAs, each
// writing the partial sums of its tiles into slots; the residual is rebuilt
// by its readers from the slots in slot order (no dependence on timing).  The
// attention of kv head g over the step's positions is split over up to 64
// CTAs by pages (scores on the tensor cores); the O items merge the splits
// (flash-decoding combine).
//
// Every wait is bounded: after kStallCycles the waiting thread sets kErrStall
// in the control block, later waits return at once and the launch ends (the
// producer first waits, again with a bound, for the copies it still has in
// flight).  Co-residency of all CTAs, which the cross-CTA waits rely on,
// comes from a cooperative launch.
//
// The same ring feeds k_vocab_ring, the vocabulary pass of the default path.
#include <cuda_bf16.h>
#include <math.h>

#include <algorithm>

#include "ee_internal.h"
#include "ee_vocab.cuh"

namespace ee {
namespace {

constexpr int kCW = kSegConsumerWarps;
constexpr int kCT = 32 * kCW;              // consumer threads
constexpr int kColsPerChunk = kSegChunk / (2 * kTileRows);  // 512
constexpr int kCCPerWarp = (kColsPerChunk / 8 + kCW - 1) / kCW;  // 16-byte column chunks a warp takes per stage
// Wait bounds are in SM clock cycles (kSegStallCycles, kSegCheckCycles;
// clock64 is cheap to read, the error word in global memory is not, so a
// waiting thread looks at it only once per check interval).


__device__ __forceinline__ float bf(uint16_t b) { return __uint_as_float((uint32_t)b << 16); }
__device__ __forceinline__ float bflo(uint32_t v) { return __uint_as_float(v << 16); }
__device__ __forceinline__ float bfhi(uint32_t v) { return __uint_as_float(v & 0xffff0000u); }
__device__ __forceinline__ uint16_t tobf(float f) { return __bfloat16_as_ushort(__float2bfloat16_rn(f)); }

__device__ __forceinline__ long long cycles() { return clock64(); }
// The error word a wait watches and its bounds (cycles).
struct Waits {
    volatile int* err;
    long long stall, check;
};
// Bookkeeping of a bounded wait: true once the wait has run out of time or
// another thread has flagged a stall.
struct Bound {
    long long t0, tc;
    __device__ __forceinline__ Bound() : t0(cycles()), tc(t0) {}
    __device__ __forceinline__ bool expired(const Waits& w) {
        const long long t = cycles();
        if (t - tc < w.check) return false;
        tc = t;
        return (*w.err & kErrStall) || t - t0 > w.stall;
    }
};
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
__device__ __forceinline__ bool mb_wait(uint64_t* b, int parity, const Waits& w) {
    if (mb_test(b, parity)) return true;
    Bound bd;
    for (unsigned it = 1;; ++it) {
        if (mb_test(b, parity)) return true;
        if ((it & 15) == 0 && bd.expired(w)) return false;
    }
}
// Wait for a bulk copy issued earlier to land, whatever the error word says
// (a CTA must not exit with copies into its shared memory in flight; issued
// copies always land), bounded by `deadline` on the SM clock.
__device__ __forceinline__ void mb_wait_landed(uint64_t* b, int parity, long long deadline) {
    while (!mb_test(b, parity) && cycles() < deadline) {
    }
}
// Non-blocking test with a sleeping back-off, for the producer: it waits
// for ring space while the consumers work, and must not compete with them
// for issue slots or the shared-memory pipe.
__device__ __forceinline__ bool mb_probe(uint64_t* b, int parity) {
    uint32_t ok;
    asm volatile(
        "{ .reg .pred p; mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2; selp.u32 %0, 1, 0, p; }"
        : "=r"(ok)
        : "r"(saddr(b)), "r"(parity)
        : "memory");
    return ok != 0;
}
__device__ __forceinline__ bool mb_wait_sleep(uint64_t* b, int parity, const Waits& w) {
    if (mb_probe(b, parity)) return true;
    Bound bd;
    for (unsigned it = 1;; ++it) {
        __nanosleep(32);
        if (mb_probe(b, parity)) return true;
        if ((it & 15) == 0 && bd.expired(w)) return false;
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

// Explicit shared-memory loads (32-bit shared-window addresses).
__device__ __forceinline__ uint4 lds128(uint32_t a) {
    uint4 v;
    asm volatile("ld.shared.v4.u32 {%0,%1,%2,%3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(a));
    return v;
}
__device__ __forceinline__ float4 lds128f(uint32_t a) {
    float4 v;
    asm volatile("ld.shared.v4.f32 {%0,%1,%2,%3}, [%4];" : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w) : "r"(a));
    return v;
}
__device__ __forceinline__ uint2 lds64(uint32_t a) {
    uint2 v;
    asm volatile("ld.shared.v2.u32 {%0,%1}, [%2];" : "=r"(v.x), "=r"(v.y) : "r"(a));
    return v;
}
__device__ __forceinline__ uint32_t lds32(uint32_t a) {
    uint32_t v;
    asm volatile("ld.shared.u32 %0, [%1];" : "=r"(v) : "r"(a));
    return v;
}

__device__ __forceinline__ void sts64(uint32_t a, uint32_t x, uint32_t y) {
    asm volatile("st.shared.v2.b32 [%0], {%1, %2};" ::"r"(a), "r"(x), "r"(y) : "memory");
}
// Two floats as bf16 (round to nearest even), the first in the low half.
__device__ __forceinline__ uint32_t pack_bf16x2(float a, float b) {
    return (uint32_t)tobf(a) | ((uint32_t)tobf(b) << 16);
}
// x0, x1 as three packed bf16 parts: high = bf16(x), middle = bf16(x -
// high), low = bf16(x - high - middle).  Both differences are exact in fp32
// and the low part holds what is left, so high + middle + low = x.
__device__ __forceinline__ void split3_bf16x2(float x0, float x1, uint32_t& hi, uint32_t& mid, uint32_t& lo) {
    const uint16_t h0 = tobf(x0), h1 = tobf(x1);
    const float r0 = x0 - bf(h0), r1 = x1 - bf(h1);
    const uint16_t m0 = tobf(r0), m1 = tobf(r1);
    hi = (uint32_t)h0 | ((uint32_t)h1 << 16);
    mid = (uint32_t)m0 | ((uint32_t)m1 << 16);
    lo = pack_bf16x2(r0 - bf(m0), r1 - bf(m1));
}
// d += A B for one m16n8k16 tile: bf16 A (4 registers, row-major
// fragment), bf16 B (2 registers, column-major fragment), fp32 accumulators.
__device__ __forceinline__ void mma_bf16(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3, uint32_t b0,
                                         uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
        "{%0, %1, %2, %3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
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
__device__ __forceinline__ float dot8s(const uint4 w, uint32_t xa) {
    const float4 a = lds128f(xa);
    const float4 b = lds128f(xa + 16);
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
// Dot products of one ring stage for one warp: lane = row of the tile, the
// warp's 16-byte column chunks are w, w + kCW, ... (stage byte address `wl`
// already offset by lane * 16 + w * 512, input address `xl` by w * 32).
// Full stages take the branch-free path with every chunk's product an
// independent chain; a ragged last stage of a row checks each chunk.
template <int CC>
__device__ __forceinline__ float stage_dot(uint32_t wl, uint32_t xl, int cc_first, int ccn) {
    if (cc_first + (CC - 1) * kSegConsumerWarps < ccn) {
        uint4 wv[CC];
#pragma unroll
        for (int u = 0; u < CC; ++u) wv[u] = lds128(wl + u * kSegConsumerWarps * 512);
        float a[CC];
#pragma unroll
        for (int u = 0; u < CC; ++u) {
            const float4 x0 = lds128f(xl + u * kSegConsumerWarps * 32);
            const float4 x1 = lds128f(xl + u * kSegConsumerWarps * 32 + 16);
            float p0 = bflo(wv[u].x) * x0.x, p1 = bfhi(wv[u].x) * x0.y;
            p0 = fmaf(bflo(wv[u].y), x0.z, p0);
            p1 = fmaf(bfhi(wv[u].y), x0.w, p1);
            p0 = fmaf(bflo(wv[u].z), x1.x, p0);
            p1 = fmaf(bfhi(wv[u].z), x1.y, p1);
            p0 = fmaf(bflo(wv[u].w), x1.z, p0);
            p1 = fmaf(bfhi(wv[u].w), x1.w, p1);
            a[u] = p0 + p1;
        }
        float t = 0.f;
#pragma unroll
        for (int u = 0; u < CC; ++u) t += a[u];
        return t;
    }
    float t = 0.f;
    for (int u = 0; cc_first + u * kSegConsumerWarps < ccn; ++u)
        t += dot8s(lds128(wl + u * kSegConsumerWarps * 512), xl + u * kSegConsumerWarps * 32);
    return t;
}


// ------------------------------------------------------------ work geometry
// Q/K/V and gate/up are split by whole 32-row tiles: rank r < Ge =
// min(G, n_tiles) owns tiles [r n / Ge, (r + 1) n / Ge) and runs on CTA
// r G / Ge, so each of those phases finishes its rows in one CTA and applies
// its epilogue there.  The O and down projections (few rows, long rows) are
// split into (tile, 512-column chunk) items over all CTAs.  An O item writes
// its chunk's partial sums to slot [tile][chunk][32] (chunk 0 also carries
// the residual entering the layer), so the mid residual is the sum of a
// tile's O slots; a down item adds into its CTA's slot [tile][slot][32].
__device__ __forceinline__ void whole_tiles(int n_t, int G, int cta, int& t0, int& t1) {
    const int Ge = min(G, n_t);
    const int r = (int)(((int64_t)cta * Ge + G - 1) / G);
    if (r < Ge && (int)((int64_t)r * G / Ge) == cta) {
        t0 = (int)((int64_t)r * n_t / Ge);
        t1 = (int)((int64_t)(r + 1) * n_t / Ge);
    } else {
        t0 = t1 = 0;
    }
}
struct Items {
    int N, Ge, lo, hi, nc, K;
};
__device__ __forceinline__ Items items_for(const SegPlan& p, int mt, int cta) {
    Items it;
    it.nc = p.n_chunks[mt];
    it.K = p.K[mt];
    it.N = p.n_tiles[mt] * it.nc;
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
__device__ __forceinline__ uint32_t chunk_bytes(int K, int c) {
    return (uint32_t)min(kColsPerChunk, K - c * kColsPerChunk) * (2 * kTileRows);
}
__device__ __forceinline__ const uint8_t* mat_base(const DevModel& m, int j, int mt) {
    const int64_t off = mt == 0 ? m.off_wqkv : mt == 1 ? m.off_wo : mt == 2 ? m.off_wgu : m.off_wd;
    return reinterpret_cast<const uint8_t*>(m.layers + (int64_t)j * m.layer_stride + off);
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
__device__ __forceinline__ int attn_unit(const AttnGeo& a, int G, int cta) {
    const int u = (int)(((int64_t)cta * a.U + G - 1) / G);
    if (u < a.U && (int)((int64_t)u * G / a.U) == cta) return u;
    return -1;
}

// ------------------------------------------------------------ shared memory
struct Smem {
    uint8_t* ring;      // stages x kSegChunk
    uint64_t* full;     // [stages]
    uint64_t* empty;    // [stages]
    float* xs;          // [max(d, A D)] input vector of a whole-tile phase
    float* xa;          // [max items][512] staged input columns of the O / down items, then
                        // [max items][32] residual rows of the O items of chunk 0
    float2* rope;       // [D/2] (cos, sin) of the step's position
    float* red;         // [2][kCW][32], then [kCW] sums of squares of the RMSNorm
    float* qa;          // [group][D] scaled queries of the attention unit
    float* kv;          // [2][D] k, v of the step's position
    float* sc;          // [group][pps * page_size] scores, then probabilities
    float* ml;          // [group][2] max, sum
    uint8_t* nsd;       // [down tiles] slots per down tile
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
    f += (max(m.d, m.A * m.D) + 3) & ~3;
    s.xa = f;
    f += p.max_items * (kColsPerChunk + 32);
    s.rope = reinterpret_cast<float2*>(f);
    f += m.D;
    s.red = f;
    f += 2 * kCW * 32 + kCW;
    const int grp = m.A / m.KH;
    s.qa = f;
    f += grp * m.D;
    s.kv = f;
    f += 2 * m.D;
    s.sc = f;
    f += grp * p.max_pps * m.page_size;
    s.ml = f;
    f += 2 * grp;
    s.nsd = reinterpret_cast<uint8_t*>(f);
    return s;
}

// ------------------------------------------------------------ the producer
// Ring positions advance by one stage per chunk; (stage, parity) pairs are
// kept incrementally (no division in the per-chunk path).
struct RingPos {
    int st = 0, ph = 0;
    __device__ __forceinline__ void next(int stages) {
        if (++st == stages) {
            st = 0;
            ph ^= 1;
        }
    }
};
struct Producer {
    const Smem& s;
    int stages, inflight;
    long long n;   // chunks issued
    RingPos head;  // stage of the next chunk
    RingPos tail;  // stage of chunk n - inflight (once n >= inflight)
    uint64_t pol_w, pol_kv;
    Waits wt;
    bool ok = true;
    __device__ Producer(const Smem& sm, int st, int infl, const Waits& w)
        : s(sm), stages(st), inflight(infl), n(0), pol_w(evict_first()), pol_kv(evict_normal()), wt(w) {}
    __device__ __forceinline__ void push(const void* src, uint32_t bytes, uint64_t pol) {
        if (!ok) return;
        // at most `inflight` copies outstanding: the ring still runs up to
        // `stages` chunks ahead, but the copies queued in HBM stay few
        if (n >= inflight) {
            if (!mb_wait_sleep(&s.full[tail.st], tail.ph, wt)) {
                atomicOr((int*)wt.err, kErrStall);
                ok = false;
                return;
            }
            tail.next(stages);
        }
        // the stage is free once the consumers released its previous chunk
        if (n >= stages && !mb_wait_sleep(&s.empty[head.st], head.ph ^ 1, wt)) {
            atomicOr((int*)wt.err, kErrStall);
            ok = false;
            return;
        }
        mb_expect_tx(&s.full[head.st], bytes);
        bulk_load(s.ring + (size_t)head.st * kSegChunk, src, bytes, &s.full[head.st], pol);
        head.next(stages);
        ++n;
    }
    // Before leaving: every issued copy has landed (the consumers normally
    // see to that; after a stall they may not have).  Walks back over the
    // last min(n, stages) chunks, whose copies are the only ones that can
    // still be in flight (chunk n lands before chunk n + stages is issued).
    __device__ void drain() {
        RingPos q = head;
        const long long deadline = cycles() + kSegStallCycles;
        for (long long i = 0; i < min(n, (long long)stages); ++i) {
            if (--q.st < 0) {
                q.st = stages - 1;
                q.ph ^= 1;
            }
            mb_wait_landed(&s.full[q.st], q.ph, deadline);
        }
    }
};

// ------------------------------------------------------------ the consumers
struct Consumer {
    const Smem& s;
    int stages;
    RingPos pos;
    Waits wt;
    bool ok = true;
    __device__ Consumer(const Smem& sm, int st, const Waits& w) : s(sm), stages(st), wt(w) {}
    __device__ __forceinline__ const uint4* acquire() {
        if (ok && !mb_wait(&s.full[pos.st], pos.ph, wt)) {
            atomicOr((int*)wt.err, kErrStall);
            ok = false;
        }
        return reinterpret_cast<const uint4*>(s.ring + (size_t)pos.st * kSegChunk);
    }
    __device__ __forceinline__ void release() {
        __syncwarp();
        if ((threadIdx.x & 31) == 0) mb_arrive(&s.empty[pos.st]);
        pos.next(stages);
    }
};

// ------------------------------------------------------------ tagged values
// A value one CTA hands to another within a launch is a Tagged word: the
// float's bits in the low half, its layer's tag in the high half, 0x80000000
// | (seq mod 2^31), seq counting the layers run since the context was reset
// (over all launches).  Writers store the word with one 64-bit relaxed store
// and neither fence nor count; readers load it with 64-bit relaxed loads
// until the tag is the expected one.  A 64-bit aligned word is observed
// whole, so value and tag arrive together, and the value keeps all 32 bits
// (a NaN or an infinity too).  Every word a layer reads is written by every
// layer (the O slots by every other layer, into the buffer of seq's parity),
// so before it receives the value of seq it holds the one of seq - 1 or
// seq - 2, whose tags differ; attention partials of splits a launch does not
// use are set to 0, which is no tag, as is every word after a reset.  The
// readers of a word are done with it before it is written again: every later
// write depends, through the values it is computed from, on all of them.
__device__ __forceinline__ uint32_t seq_tag(unsigned seq) { return 0x80000000u | (seq & 0x7fffffffu); }
__device__ __forceinline__ void st_tagged(Tagged* p, float v, uint32_t tag) {
    const unsigned long long b = (unsigned long long)__float_as_uint(v) | ((unsigned long long)tag << 32);
    asm volatile("st.relaxed.gpu.global.b64 [%0], %1;" ::"l"(p), "l"(b) : "memory");
}
__device__ __forceinline__ void st_zero(Tagged* p) {
    asm volatile("st.relaxed.gpu.global.b64 [%0], %1;" ::"l"(p), "l"(0ull) : "memory");
}
__device__ __forceinline__ unsigned long long ld_strong(const Tagged* p) {
    unsigned long long r;
    asm volatile("ld.relaxed.gpu.global.b64 %0, [%1];" : "=l"(r) : "l"(p) : "memory");
    return r;
}
// Two consecutive words (p 16-byte aligned): each 64-bit element is observed whole.
__device__ __forceinline__ void ld_strong2(const Tagged* p, unsigned long long& a, unsigned long long& b) {
    asm volatile("ld.relaxed.gpu.global.v2.b64 {%0, %1}, [%2];" : "=l"(a), "=l"(b) : "l"(p) : "memory");
}
__device__ __forceinline__ float untag(unsigned long long b) { return __uint_as_float((uint32_t)b); }
__device__ __forceinline__ uint32_t tag_of(unsigned long long b) { return (uint32_t)(b >> 32); }
// Four consecutive words (p 16-byte aligned) as a float4; a tag other than
// `tag` sets bits in bad.
__device__ __forceinline__ float4 load4(const Tagged* p, uint32_t tag, uint32_t& bad) {
    unsigned long long w0, w1, w2, w3;
    ld_strong2(p, w0, w1);
    ld_strong2(p + 2, w2, w3);
    bad |= (tag_of(w0) ^ tag) | (tag_of(w1) ^ tag) | (tag_of(w2) ^ tag) | (tag_of(w3) ^ tag);
    return make_float4(untag(w0), untag(w1), untag(w2), untag(w3));
}

// One thread's bounded waits for tagged values.  After a wait has run out
// (kErrStall set) the later ones return zeros at once, so the launch still
// ends; the host reports the stall.
struct Poll {
    Waits wt;
    bool failed;
    __device__ explicit Poll(const Waits& w) : wt(w), failed(false) {}
    __device__ __forceinline__ float wait1(const Tagged* p, uint32_t tag) {
        if (!failed) {
            Bound bd;
            for (;;) {
                const unsigned long long b = ld_strong(p);
                if (tag_of(b) == tag) return untag(b);
                if (bd.expired(wt)) break;
            }
            atomicOr((int*)wt.err, kErrStall);
            failed = true;
        }
        return 0.f;
    }
    // Between two rounds of loads of values not all written yet: false once
    // the wait has run out (kErrStall set; the caller keeps what it has).
    __device__ __forceinline__ bool again(Bound& bd) {
        if (failed) return false;
        if (!bd.expired(wt)) return true;
        atomicOr((int*)wt.err, kErrStall);
        failed = true;
        return false;
    }
    // One thread waits until the word at p carries `tag` (loads a little
    // apart), then the consumer warps sync.  p is one of the phase's inputs:
    // once it has arrived the others mostly have too, so the gather that
    // follows finds them written and few threads poll.
    __device__ __forceinline__ void probe(const Tagged* p, uint32_t tag) {
        if (threadIdx.x == 0) (void)get(p, tag);
        csync();
    }
    __device__ __forceinline__ float get(const Tagged* p, uint32_t tag) {
        const unsigned long long b = ld_strong(p);
        return tag_of(b) == tag ? untag(b) : wait1(p, tag);
    }
};


// Reload the elements of a gather round whose tags were not yet all the
// expected ones, every such element's loads issued together, until none is
// left (or the wait has run out).
template <int U, class F>
__device__ __forceinline__ void retry(Poll& pl, int b, float4 (&v)[U], uint32_t (&bad)[U], F f) {
    uint32_t any = 0;
#pragma unroll
    for (int e = 0; e < U; ++e) any |= bad[e];
    if (!any) return;
    Bound bd;
    while (pl.again(bd)) {
        any = 0;
#pragma unroll
        for (int e = 0; e < U; ++e)
            if (bad[e]) {
                bad[e] = 0;
                v[e] = f(4 * (b + e * kCT), bad[e]);
                any |= bad[e];
            }
        if (!any) return;
    }
}

// dst[i..i+3] = f(i) for i < n (n and dst 4-aligned), U float4 per thread
// per round with all their loads issued before any store.  f(i, bad) loads
// once and ORs a nonzero value into bad if a tag was not yet the expected
// one; such elements are loaded again (retry).
template <int U, class F>
__device__ __forceinline__ void gather4(float* dst, int n, Poll& pl, F f) {
    const int n4 = n >> 2;
    float4* d4 = reinterpret_cast<float4*>(dst);
    for (int b = threadIdx.x; b < n4; b += U * kCT) {
        float4 v[U];
        uint32_t bad[U];
#pragma unroll
        for (int e = 0; e < U; ++e) {
            bad[e] = 0;
            v[e] = (b + e * kCT < n4) ? f(4 * (b + e * kCT), bad[e]) : make_float4(0.f, 0.f, 0.f, 0.f);
        }
        retry<U>(pl, b, v, bad, f);
#pragma unroll
        for (int e = 0; e < U; ++e)
            if (b + e * kCT < n4) d4[b + e * kCT] = v[e];
    }
}
__device__ __forceinline__ float4 f4add(float4 a, float4 b) {
    return make_float4(a.x + b.x, a.y + b.y, a.z + b.z, a.w + b.w);
}
__device__ __forceinline__ float4 ldg4(const float* p) { return *reinterpret_cast<const float4*>(p); }
// a + the four tagged values at p, noting a tag mismatch in bad
__device__ __forceinline__ float4 add_tagged(float4 a, const Tagged* p, uint32_t tag, uint32_t& bad) {
    return f4add(a, load4(p, tag, bad));
}
__device__ __forceinline__ float4 bf4(const uint16_t* p) {
    const uint2 u = *reinterpret_cast<const uint2*>(p);
    return make_float4(bflo(u.x), bfhi(u.x), bflo(u.y), bfhi(u.y));
}

// RMSNorm folded into the gather of its input: xs = h * g (d values, h
// from f four at a time, g the bf16 gain in global memory) and the return
// value 1 / sqrt(mean(h^2) + eps), the
// factor the projection's epilogue applies to each row's dot product
// (W (h * g) / rms = W (RMSNorm(h) * g)).  One consumer barrier; nss: [kCW]
// floats of shared memory not otherwise in use until the next call.
template <int U, class F>
__device__ __forceinline__ float gather_norm(float* xs, const uint16_t* g, int d, float eps, float* nss, Poll& pl, F f) {
    const int n4 = d >> 2;
    float4* x4 = reinterpret_cast<float4*>(xs);
    float ss = 0.f;
    for (int b = threadIdx.x; b < n4; b += U * kCT) {
        float4 v[U];
        uint32_t bad[U];
        uint2 gg[U];  // the gain (global, read-only), loaded with the values
#pragma unroll
        for (int e = 0; e < U; ++e) {
            bad[e] = 0;
            const bool in = b + e * kCT < n4;
            gg[e] = in ? __ldg(reinterpret_cast<const uint2*>(g) + (b + e * kCT)) : make_uint2(0u, 0u);
            v[e] = in ? f(4 * (b + e * kCT), bad[e]) : make_float4(0.f, 0.f, 0.f, 0.f);
        }
        retry<U>(pl, b, v, bad, f);
#pragma unroll
        for (int e = 0; e < U; ++e) {
            const int k = b + e * kCT;
            if (k < n4) {
                ss = fmaf(v[e].x, v[e].x, ss);
                ss = fmaf(v[e].y, v[e].y, ss);
                ss = fmaf(v[e].z, v[e].z, ss);
                ss = fmaf(v[e].w, v[e].w, ss);
                const uint2 gu = gg[e];
                x4[k] = make_float4(v[e].x * bflo(gu.x), v[e].y * bfhi(gu.x), v[e].z * bflo(gu.y), v[e].w * bfhi(gu.y));
            }
        }
    }
    ss = warp_sum(ss);
    if ((threadIdx.x & 31) == 0) nss[threadIdx.x >> 5] = ss;
    csync();
    float t = 0.f;
#pragma unroll
    for (int k = 0; k < kCW; ++k) t += nss[k];
    return 1.0f / sqrtf(t / (float)d + eps);
}

// Whole tiles [t0, t1) of a matrix with rows of length K against x (all K
// columns in shared memory).  epi(t, s) runs in warp 0 with lane = row of
// the tile and s its complete dot product.
template <class Epi>
__device__ __forceinline__ void tile_gemv(Consumer& cs, int t0, int t1, int K, int nc, const float* x, float* red,
                                          int& rb, Epi epi) {
    const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
    for (int t = t0; t < t1; ++t) {
        float acc = 0.f;
        for (int c = 0; c < nc; ++c) {
            const uint32_t buf = saddr(cs.acquire()) + lane * 16 + w * 512;
            const int ccn = (int)(chunk_bytes(K, c) / 512);
            const uint32_t xc = saddr(x + c * kColsPerChunk) + w * 32;
            if (cs.ok) acc += stage_dot<kCCPerWarp>(buf, xc, w, ccn);
            cs.release();
        }
        float* r = red + rb * kCW * 32;
        r[w * 32 + lane] = acc;
        csync();
        if (w == 0) {
            float sum = 0.f;
#pragma unroll
            for (int k = 0; k < kCW; ++k) sum += r[k * 32 + lane];
            epi(t, sum);
        }
        rb ^= 1;
    }
}

// Residual entering layer j at row i: the embedding (first layer of a step),
// the model's h (first layer of a later segment), or the sum of the previous
// layer's down slots (slot 0 of each tile carries that layer's mid residual),
// tagged with that layer's tag.
struct ResidIn {
    const SegPlan* p;
    const uint16_t* emb;  // embedding row, or null
    const float* src;     // m.h, or null for the slot sums
    const uint8_t* nsd;
    uint32_t tag;         // the previous layer's tag
    __device__ __forceinline__ float operator()(int i, Poll& pl) const {
        if (emb) return bf(emb[i]);
        if (src) return src[i];
        const int t = i >> 5, l = i & 31, ns = nsd[t];
        const Tagged* qd = p->dpart + (int64_t)t * p->n_chunks[3] * 32 + l;
        float v = 0.f;
        for (int k = 0; k < ns; ++k) v += pl.get(qd + k * 32, tag);
        return v;
    }
    // rows i..i+3 (i a multiple of 4, same tile): one load per slot
    __device__ __forceinline__ float4 four(int i, uint32_t& bad) const {
        if (emb) return bf4(emb + i);
        if (src) return ldg4(src + i);
        const int t = i >> 5, l = i & 31, ns = nsd[t];
        const Tagged* qd = p->dpart + (int64_t)t * p->n_chunks[3] * 32 + l;
        float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int k = 0; k < kSegMaxSlots; ++k)
            if (k < ns) v = add_tagged(v, qd + k * 32, tag, bad);
        return v;
    }
};
// O slots of layer seq: two buffers, alternating by layer (a chunk-0 O item
// reads the previous layer's slots while the other items of its tile write
// this layer's).
__device__ __forceinline__ Tagged* opart_of(const SegPlan& p, unsigned seq) {
    return p.opart + (int64_t)(seq & 1u) * p.n_tiles[1] * p.n_chunks[1] * 32;
}
// Mid residual (after the attention block) at rows i..i+3: the sum of the O
// slots, tagged with this layer's tag.
__device__ __forceinline__ float4 resid_mid4(const SegPlan& p, const Tagged* opart, int i, uint32_t tag,
                                             uint32_t& bad) {
    const int t = i >> 5, nco = p.n_chunks[1];
    const Tagged* qo = opart + (int64_t)t * nco * 32 + (i & 31);
    float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int k = 0; k < kSegMaxSlots; ++k)
        if (k < nco) v = add_tagged(v, qo + k * 32, tag, bad);
    return v;
}

}  // namespace

__global__ void __launch_bounds__(kSegThreads, 1) k_layers(DevModel m, SegPlan p, int j0, int j1, int first) {
    extern __shared__ __align__(128) uint8_t seg_smem[];
    const Smem s = carve(seg_smem, m, p);
    const int cta = blockIdx.x, G = p.G;
    const Waits wt{&m.ctl->err, p.stall_cycles, p.check_cycles};
    const int half = m.D >> 1, grp = m.A / m.KH;
    const int AD = m.A * m.D;

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
    int tq0, tq1, tg0, tg1;
    whole_tiles(p.n_tiles[0], G, cta, tq0, tq1);
    whole_tiles(p.n_tiles[2], G, cta, tg0, tg1);
    const Items io = items_for(p, 1, cta);
    const Items idn = items_for(p, 3, cta);

    // ---------------------------------------------------------- producer
    if (threadIdx.x >= kCT) {
        if (threadIdx.x != kCT || !pos_ok) return;
        Producer pr(s, p.stages, min(p.stages, p.inflight), wt);
        // The CTA's chunk list, layer by layer: its Q/K/V tiles, its
        // attention unit's K then V pages, its O items, its gate/up tiles,
        // its down items.
        const int nc0 = p.n_chunks[0], nc2 = p.n_chunks[2];
        int pg0 = 0, pg1 = 0, g = 0;
        if (unit >= 0) {
            g = unit / ag.splits;
            const int sp = unit - g * ag.splits;
            pg0 = sp * ag.pps;
            pg1 = min(ag.n_pages, pg0 + ag.pps);
        }
        const int nq = (tq1 - tq0) * nc0, nkv = 2 * (pg1 - pg0) * cpp, no = io.hi - io.lo;
        const int ng = (tg1 - tg0) * nc2, nd = idn.hi - idn.lo;
        const int per = nq + nkv + no + ng + nd;
        const long long total = (long long)per * (j1 - j0);
        auto chunk = [&](long long n, const void*& src, uint32_t& bytes) -> bool {  // true: a cache page
            const int j = j0 + (int)(n / per);
            int r = (int)(n - (long long)(j - j0) * per);
            if (r < nq) {
                const int t = tq0 + r / nc0, ch = r - (r / nc0) * nc0;
                src = mat_base(m, j, 0) + (int64_t)t * kTileRows * p.K[0] * 2 + (int64_t)ch * kSegChunk;
                bytes = chunk_bytes(p.K[0], ch);
                return false;
            }
            r -= nq;
            if (r < nkv) {
                const int per_kv = (pg1 - pg0) * cpp, kvi = r / per_kv, r2 = r - kvi * per_kv;
                const int pg = pg0 + r2 / cpp, q = r2 - (r2 / cpp) * cpp;
                const uint16_t* pool = (kvi ? m.vpool : m.kpool) + (int64_t)j * m.kv_layer_stride;
                src = pool + (((int64_t)m.page_table[pg] * m.KH + g) * m.page_size + q * rpc) * m.D;
                bytes = (uint32_t)(rpc * m.D * 2);
                return true;
            }
            r -= nkv;
            if (r < no) {
                const int i = io.lo + r, t = i / io.nc, ch = i - t * io.nc;
                src = mat_base(m, j, 1) + (int64_t)t * kTileRows * io.K * 2 + (int64_t)ch * kSegChunk;
                bytes = chunk_bytes(io.K, ch);
                return false;
            }
            r -= no;
            if (r < ng) {
                const int t = tg0 + r / nc2, ch = r - (r / nc2) * nc2;
                src = mat_base(m, j, 2) + (int64_t)t * kTileRows * p.K[2] * 2 + (int64_t)ch * kSegChunk;
                bytes = chunk_bytes(p.K[2], ch);
                return false;
            }
            r -= ng;
            const int i = idn.lo + r, t = i / idn.nc, ch = i - t * idn.nc;
            src = mat_base(m, j, 3) + (int64_t)t * kTileRows * idn.K * 2 + (int64_t)ch * kSegChunk;
            bytes = chunk_bytes(idn.K, ch);
            return false;
        };
        for (long long n = 0; n < total && pr.ok; ++n) {
            const void* src;
            uint32_t bytes;
            const bool kv = chunk(n, src, bytes);
            pr.push(src, bytes, kv ? pr.pol_kv : pr.pol_w);
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
    Consumer cs(s, p.stages, wt);
    Poll pl(wt);
    unsigned* sync = p.sync;
    const int64_t last_dn_slot = (int64_t)(p.n_tiles[3] - 1) * p.n_chunks[3];  // first slot of the last down tile
    const unsigned seq0 = sync[1];  // layers run since the context was reset
    for (int i = threadIdx.x; i < half; i += kCT) s.rope[i] = m.rope[(int64_t)pos * half + i];
    const float2* cs_row = s.rope;
    const float scale = 1.0f / sqrtf((float)m.D);
    const int slice0 = (int)((int64_t)cta * m.d / G), slice1 = (int)((int64_t)(cta + 1) * m.d / G);
    const int nq = m.A * half, nk = m.KH * half;
    const int64_t kvo_pos = ((int64_t)m.page_table[pos / m.page_size] * m.KH * m.page_size + pos % m.page_size) * m.D;
    {   // slots of each down tile
        Items all = items_for(p, 3, 0);
        for (int t = threadIdx.x; t < p.n_tiles[3]; t += kCT)
            s.nsd[t] = (uint8_t)(item_owner(all, t * all.nc + all.nc - 1) - item_owner(all, t * all.nc) + 1);
    }
    int tok = c->in_tok;
    if (first) {
        if (tok < 0 || tok >= m.V) {
            if (cta == 0 && threadIdx.x == 0) atomicOr(&c->err, kErrTokenRange);
            tok = 0;
        }
        if (cta == 0 && threadIdx.x == 0) {
            c->exit_readout = -1;
            c->n_evaluated = 0;
            c->full_token = -1;
            c->nucleus_member = -1;
        }
    }
    {   // attention partials of the splits this launch does not use: 0 (no
        // tag), so a later launch that uses them again cannot take an old value
        const int per_head = max(0, p.max_splits - ag.splits) * (m.D + 4);
        const int64_t n = (int64_t)m.A * per_head;
        for (int64_t e = (int64_t)cta * kCT + threadIdx.x; e < n; e += (int64_t)G * kCT) {
            const int h = (int)(e / per_head), r = (int)(e - (int64_t)h * per_head);
            st_zero(p.attn_part + ((int64_t)h * kSegMaxSplits + ag.splits) * (m.D + 4) + r);
        }
    }
    csync();
    int rb = 0;

    for (int j = j0; j < j1; ++j) {
        const unsigned seq = seq0 + (unsigned)(j - j0);
        const uint32_t tag = seq_tag(seq);
        const uint16_t* lw = m.layers + (int64_t)j * m.layer_stride;
        Tagged* op_cur = opart_of(p, seq);
        const ResidIn rin{&p, (j == j0 && first) ? m.embed + (int64_t)tok * m.d : nullptr, j == j0 ? m.h : nullptr,
                          s.nsd, seq_tag(seq - 1)};
        // The RMSNorm gains the next gathers read (this layer's MLP gain, the
        // next layer's attention gain, or after the last layer the final gain
        // the vocabulary pass reads): into L2 now, so that those gathers do
        // not wait on HBM.  A few CTAs issue them, one 128-byte line per lane.
        if (cta < 2 && w == 1) {
            const uint16_t* gsrc = cta == 0 ? lw + m.off_gmlp
                                            : (j + 1 < m.L ? m.layers + (int64_t)(j + 1) * m.layer_stride + m.off_gattn
                                                           : m.g_final);
            for (int b = lane * 64; b < m.d; b += 32 * 64)
                asm volatile("prefetch.global.L2 [%0];" ::"l"(gsrc + b));
        }

        // ---------------- Q/K/V tiles: RMSNorm, projection, bias, RoPE, KV append
        if (tq1 > tq0) {
            if (j > j0)
                pl.probe(p.dpart + (last_dn_slot + s.nsd[p.n_tiles[3] - 1] - 1) * 32 + 31, seq_tag(seq - 1));
            else
                csync();
            const float inv = gather_norm<2>(s.xs, lw + m.off_gattn, m.d, m.eps, s.red + 2 * kCW * 32, pl,
                                          [&](int i, uint32_t& bad) { return rin.four(i, bad); });
            const uint16_t* bias = m.qkv_bias ? lw + m.off_bqkv : nullptr;
            uint16_t* kdst = m.kpool + (int64_t)j * m.kv_layer_stride + kvo_pos;
            uint16_t* vdst = m.vpool + (int64_t)j * m.kv_layer_stride + kvo_pos;
            tile_gemv(cs, tq0, tq1, p.K[0], p.n_chunks[0], s.xs, s.red, rb, [&](int t, float v) {
                const int odd = lane & 1;
                const int u = t * 16 + (lane >> 1);
                v *= inv;
                if (bias) v += bf(bias[2 * u + odd]);
                const float other = __shfl_xor_sync(0xffffffffu, v, 1);
                const float r0 = odd ? other : v, r1 = odd ? v : other;
                // q, and the step's k and v as the cache holds them (bf16), go to
                // the attention units tagged; k and v also go to the cache
                if (u < nq) {
                    const int h = u / half, i = u - h * half;
                    const float2 cz = cs_row[i];
                    if (!odd)
                        st_tagged(p.q + h * m.D + i, r0 * cz.x - r1 * cz.y, tag);
                    else
                        st_tagged(p.q + h * m.D + i + half, r0 * cz.y + r1 * cz.x, tag);
                } else if (u < nq + nk) {
                    const int g = (u - nq) / half, i = (u - nq) - g * half;
                    const float2 cz = cs_row[i];
                    uint16_t* k = kdst + (int64_t)g * m.page_size * m.D;
                    const int at = odd ? i + half : i;
                    const uint16_t kb = tobf(odd ? r0 * cz.y + r1 * cz.x : r0 * cz.x - r1 * cz.y);
                    k[at] = kb;
                    st_tagged(p.kvn + g * m.D + at, bf(kb), tag);
                } else if (u < nq + 2 * nk) {
                    const int g = (u - nq - nk) / half, i = (u - nq - nk) - g * half;
                    uint16_t* v2 = vdst + (int64_t)g * m.page_size * m.D;
                    const int at = odd ? i + half : i;
                    const uint16_t vb = tobf(odd ? r1 : r0);
                    v2[at] = vb;
                    st_tagged(p.kvn + (m.KH + g) * m.D + at, bf(vb), tag);
                }
            });
        }
        if (cta == 0 && threadIdx.x == 0) m.kv_src[(int64_t)j * m.max_ctx + pos] = 1;

        // ---------------- attention unit (if this CTA has one)
        if (unit >= 0) {
            const int g = unit / ag.splits, sp = unit - g * ag.splits;
            const int pg0 = sp * ag.pps, pg1 = min(ag.n_pages, pg0 + ag.pps);
            const int p0 = pg0 * m.page_size, p1 = min(ag.T, pg1 * m.page_size);
            const int npos = p1 - p0;
            pl.probe(p.kvn + (m.KH + g + 1) * m.D - 1, tag);  // the last value of this group's v
            const Tagged* qsrc = p.q + (int64_t)g * grp * m.D;
            const Tagged* kt = p.kvn + (int64_t)g * m.D;
            const Tagged* vt = p.kvn + (int64_t)(m.KH + g) * m.D;
            // the group's scaled queries, then k and v, in one round (s.kv follows s.qa)
            const int nqa = grp * m.D;
            gather4<1>(s.qa, nqa + 2 * m.D, pl, [&](int i, uint32_t& bad) {
                if (i >= nqa) {
                    const int e = i - nqa;
                    return load4(e < m.D ? kt + e : vt + e - m.D, tag, bad);
                }
                const float4 q = load4(qsrc + i, tag, bad);
                return make_float4(q.x * scale, q.y * scale, q.z * scale, q.w * scale);
            });
            csync();
            // Scores on the tensor cores: S[h][r] = q_h . k_r as mma m16n8k16
            // (bf16 operands, fp32 accumulation) with B = 8 cached keys and A
            // the group's queries split into three bf16 parts (high + middle +
            // low = q exactly): one product with the high parts in rows 0..7
            // and the middle parts in rows 8..15, a second with the low parts
            // in rows 0..7 (rows 8..15 zero), into the same accumulators.  The
            // bf16 products are exact in fp32.  A lane loads 8 consecutive
            // dimensions of one key row (16 bytes, no bank conflicts beyond the
            // row stride's); the product's k index runs over the dimensions in
            // the same permuted order in A and B.  Row g of the result holds
            // head g's high- and low-part dot products, row g + 8 its
            // middle-part one.
            const int spc = p.max_pps * m.page_size;  // score row stride
            const int npair = m.D >> 5;               // pairs of k16 steps (32 dimensions)
            const int g8 = lane >> 2, t4 = lane & 3;
            // The group's queries as three bf16 parts, converted once into
            // rows padded to 16 bytes past D (xs is free here: seg_plan checks
            // it holds 3 grp (D + 8) bf16), so that the fragment loads of 8
            // heads at one column fall in different banks.
            {
                const int qrow = m.D + 8;
                uint16_t* qhs = reinterpret_cast<uint16_t*>(s.xs);
                for (int e = threadIdx.x; e < nqa / 4; e += kCT) {
                    const float4 q4 = lds128f(saddr(s.qa + 4 * e));
                    const int h = (4 * e) / m.D, c = 4 * e - h * m.D;
                    uint32_t h01, m01, l01, h23, m23, l23;
                    split3_bf16x2(q4.x, q4.y, h01, m01, l01);
                    split3_bf16x2(q4.z, q4.w, h23, m23, l23);
                    sts64(saddr(qhs + h * qrow + c), h01, h23);
                    sts64(saddr(qhs + (grp + h) * qrow + c), m01, m23);
                    sts64(saddr(qhs + (2 * grp + h) * qrow + c), l01, l23);
                }
                csync();
            }
            // [pair][word]: dimensions pair*32 + 8 t4 .. +7 of query g8 (the
            // low parts stay in shared memory: qlo_at, read with each product)
            uint32_t qhi[4][4], qmid[4][4];
            const bool qrow_ok = g8 < grp;
            const uint32_t qlo_at =
                saddr(reinterpret_cast<const uint16_t*>(s.xs) + (2 * grp + (qrow_ok ? g8 : 0)) * (m.D + 8) + 8 * t4);
#pragma unroll
            for (int pr = 0; pr < 4; ++pr) {
                if (pr < npair && qrow_ok) {
                    const uint16_t* qhs = reinterpret_cast<const uint16_t*>(s.xs) + g8 * (m.D + 8) + pr * 32 + 8 * t4;
                    const uint4 a = lds128(saddr(qhs)), b = lds128(saddr(qhs + grp * (m.D + 8)));
                    qhi[pr][0] = a.x, qhi[pr][1] = a.y, qhi[pr][2] = a.z, qhi[pr][3] = a.w;
                    qmid[pr][0] = b.x, qmid[pr][1] = b.y, qmid[pr][2] = b.z, qmid[pr][3] = b.w;
                } else {
#pragma unroll
                    for (int wd = 0; wd < 4; ++wd) qhi[pr][wd] = qmid[pr][wd] = 0u;
                }
            }
            for (int pg = pg0; pg < pg1; ++pg)
                for (int q = 0; q < cpp; ++q) {
                    const uint32_t kst = saddr(cs.acquire());
                    const int base = pg * m.page_size + q * rpc;
                    const int nr = min(rpc, p1 - base);
                    if (cs.ok) {
                        for (int nt = w; nt * 8 < nr; nt += kCW) {
                            const int r0 = nt * 8, own = pos - base;
                            if (own >= r0 && own < r0 + 8) {
                                // the ring holds the cache's stale copy of the step's
                                // own row: write the new k over it (bf16, exact)
                                for (int e = lane; e < (m.D >> 2); e += 32) {
                                    const float4 kk = lds128f(saddr(s.kv + 4 * e));
                                    sts64(kst + own * m.D * 2 + 8 * e, pack_bf16x2(kk.x, kk.y), pack_bf16x2(kk.z, kk.w));
                                }
                                __syncwarp();
                            }
                            const uint32_t krow = kst + (r0 + g8) * m.D * 2 + 16 * t4;
                            float acc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
                            for (int pr = 0; pr < 4; ++pr) {
                                if (pr < npair) {
                                    const uint4 kw = lds128(krow + pr * 64);
                                    mma_bf16(acc, qhi[pr][0], qmid[pr][0], qhi[pr][1], qmid[pr][1], kw.x, kw.y);
                                    mma_bf16(acc, qhi[pr][2], qmid[pr][2], qhi[pr][3], qmid[pr][3], kw.z, kw.w);
                                    uint4 lo = lds128(qlo_at + pr * 64);
                                    if (!qrow_ok) lo = make_uint4(0u, 0u, 0u, 0u);
                                    mma_bf16(acc, lo.x, 0u, lo.y, 0u, kw.x, kw.y);
                                    mma_bf16(acc, lo.z, 0u, lo.w, 0u, kw.z, kw.w);
                                }
                            }
                            const int ra = r0 + 2 * t4;
                            if (g8 < grp) {
                                float* sr = s.sc + g8 * spc + (base - p0);
                                if (ra < nr) sr[ra] = acc[0] + acc[2];
                                if (ra + 1 < nr) sr[ra + 1] = acc[1] + acc[3];
                            }
                        }
                    }
                    // generic writes to the stage (the fixed row) before the
                    // producer's next bulk copy into it
                    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
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
            // P V: warp w takes head group hg = w / npq (hpg heads) and the
            // positions r = w mod npq (mod npq); lane = dpl dimensions.  Each V
            // row is read once per head group.  The npq partial sums per head
            // meet in shared memory (xs and xa, contiguous and free here) and are
            // added in order.
            const int dpl = m.D >> 5;  // 2 or 4
            const int hgn = grp > 4 ? 2 : 1, hpg = (grp + hgn - 1) / hgn;
            const int avail = ((max(m.d, AD) + 3) & ~3) + p.max_items * (kColsPerChunk + 32);
            int npq = kCW / hgn;
            while (npq > 1 && npq * grp * m.D > avail) npq >>= 1;
            const int hg = w / npq, pq = w - hg * npq;
            const bool pv = hg < hgn;
            float vvt[4];  // the step's own v (this lane's dimensions)
            if (dpl == 4) {
                const float4 t = lds128f(saddr(s.kv + m.D + lane * 4));
                vvt[0] = t.x, vvt[1] = t.y, vvt[2] = t.z, vvt[3] = t.w;
            } else {
                const float2 t = *reinterpret_cast<const float2*>(s.kv + m.D + lane * 2);
                vvt[0] = t.x, vvt[1] = t.y, vvt[2] = vvt[3] = 0.f;
            }
            float acc[4][4];
#pragma unroll
            for (int hh = 0; hh < 4; ++hh)
#pragma unroll
                for (int k = 0; k < 4; ++k) acc[hh][k] = 0.f;
            for (int pg = pg0; pg < pg1; ++pg)
                for (int q = 0; q < cpp; ++q) {
                    const uint32_t vb = saddr(cs.acquire()) + lane * dpl * 2;
                    const int base = pg * m.page_size + q * rpc;
                    const int nr = min(rpc, p1 - base);
                    if (pv && cs.ok) {
                        const float* pr0 = s.sc + (hg * hpg) * spc + (base - p0);
#pragma unroll 4
                        for (int r = pq; r < nr; r += npq) {
                            float v[4];
                            if (dpl == 4) {
                                const uint2 u = lds64(vb + r * m.D * 2);
                                v[0] = bflo(u.x), v[1] = bfhi(u.x), v[2] = bflo(u.y), v[3] = bfhi(u.y);
                            } else {
                                const uint32_t u = lds32(vb + r * m.D * 2);
                                v[0] = bflo(u), v[1] = bfhi(u), v[2] = v[3] = 0.f;
                            }
                            const bool own = base + r == pos;  // the ring's copy of this row is stale
#pragma unroll
                            for (int k = 0; k < 4; ++k) v[k] = own ? vvt[k] : v[k];
#pragma unroll
                            for (int hh = 0; hh < 4; ++hh) {
                                if (hh < hpg && hg * hpg + hh < grp) {
                                    const float pr = pr0[hh * spc + r];
#pragma unroll
                                    for (int k = 0; k < 4; ++k) acc[hh][k] = fmaf(pr, v[k], acc[hh][k]);
                                }
                            }
                        }
                    }
                    cs.release();
                }
            float* part = s.xs;  // [grp][npq][D]
            if (pv) {
#pragma unroll
                for (int hh = 0; hh < 4; ++hh) {
                    const int h = hg * hpg + hh;
                    if (hh < hpg && h < grp) {
                        float* dst = part + (h * npq + pq) * m.D + lane * dpl;
#pragma unroll
                        for (int k = 0; k < 4; ++k)
                            if (k < dpl) dst[k] = acc[hh][k];
                    }
                }
            }
            csync();
            {
                const int d4 = m.D >> 2;
                for (int e = threadIdx.x; e < grp * d4; e += kCT) {
                    const int h = e / d4, c = 4 * (e - h * d4);
                    float4 sum = make_float4(0.f, 0.f, 0.f, 0.f);
                    for (int k = 0; k < npq; ++k) sum = f4add(sum, *reinterpret_cast<const float4*>(part + (h * npq + k) * m.D + c));
                    Tagged* dst = p.attn_part + ((int64_t)(g * grp + h) * kSegMaxSplits + sp) * (m.D + 4) + c;
                    st_tagged(dst, sum.x, tag);
                    st_tagged(dst + 1, sum.y, tag);
                    st_tagged(dst + 2, sum.z, tag);
                    st_tagged(dst + 3, sum.w, tag);
                }
                if (threadIdx.x < grp) {
                    Tagged* dst = p.attn_part + ((int64_t)(g * grp + threadIdx.x) * kSegMaxSplits + sp) * (m.D + 4) + m.D;
                    st_tagged(dst, s.ml[2 * threadIdx.x], tag);
                    st_tagged(dst + 1, s.ml[2 * threadIdx.x + 1], tag);
                }
            }
        }

        // ---------------- O items: merge the attention splits of the chunk's heads,
        // project, write the chunk's slot (chunk 0 adds the residual)
        if (io.hi > io.lo) {
            const int ns = ag.splits;
            const int nit = io.hi - io.lo, ncol = nit * kColsPerChunk;
            const int hpc = kColsPerChunk / m.D;  // heads per chunk
            float* rows = s.xa + ncol;
            // The residual rows a chunk-0 item's slot carries: the previous
            // layer's (or the segment's input), complete since this layer's
            // Q/K/V phase read them, so gathered before the wait below.
            for (int it = w; it < nit; it += kCW) {
                const int i = io.lo + it, t = i / io.nc;
                if (lane < 8) {
                    const int row = t * 32 + 4 * lane;
                    float4 r = make_float4(0.f, 0.f, 0.f, 0.f);
                    if (i - t * io.nc == 0 && row < m.d) {
                        uint32_t bad = 0;
                        r = rin.four(row, bad);
                        if (bad) {
                            Bound bd;
                            while (pl.again(bd)) {
                                bad = 0;
                                r = rin.four(row, bad);
                                if (!bad) break;
                            }
                        }
                    }
                    reinterpret_cast<float4*>(rows + it * 32)[lane] = r;
                }
            }
            {   // the last split's maximum of the first item's first head
                const int h0 = min(m.A - 1, (io.lo % io.nc) * hpc);
                pl.probe(p.attn_part + ((int64_t)h0 * kSegMaxSplits + ns - 1) * (m.D + 4) + m.D, tag);
            }
            // D / 64 warps per (item, head), each over 64 columns: the head's
            // split statistics (lane = split) and this lane's two columns of
            // every split's partial o in one round of loads (up to kB splits),
            // then o = sum_s w_s o_s / sum_s w_s l_s with w_s = exp(m_s - max m).
            const int wph = m.D >> 6;
            for (int wi = w; wi < nit * hpc * wph; wi += kCW) {
                const int it = wi / (hpc * wph), r = wi - it * hpc * wph, hc = r / wph, c0 = (r - hc * wph) * 64;
                const int h = ((io.lo + it) % io.nc) * hpc + hc;
                float2* dst = reinterpret_cast<float2*>(s.xa + it * kColsPerChunk + hc * m.D + c0) + lane;
                if (h >= m.A) {
                    *dst = make_float2(0.f, 0.f);
                    continue;
                }
                const Tagged* base = p.attn_part + (int64_t)h * kSegMaxSplits * (m.D + 4);
                const Tagged* st = base + lane * (m.D + 4) + m.D;
                const Tagged* oc = base + c0 + 2 * lane;
                constexpr int kB = 8;
                // lane l holds the statistics of splits l and l + 32
                float mk = -INFINITY, lk = 0.f, mk2 = -INFINITY, lk2 = 0.f;
                float2 ob[kB];
                Bound bd;
                for (;;) {  // one round of loads, again until every lane has its values
                    uint32_t bad = 0;
                    if (lane < ns) {
                        unsigned long long a, b;
                        ld_strong2(st, a, b);
                        bad |= (tag_of(a) ^ tag) | (tag_of(b) ^ tag);
                        mk = untag(a);
                        lk = untag(b);
                    }
                    if (lane + 32 < ns) {
                        unsigned long long a, b;
                        ld_strong2(st + 32 * (m.D + 4), a, b);
                        bad |= (tag_of(a) ^ tag) | (tag_of(b) ^ tag);
                        mk2 = untag(a);
                        lk2 = untag(b);
                    }
#pragma unroll
                    for (int u = 0; u < kB; ++u) {
                        ob[u] = make_float2(0.f, 0.f);
                        if (u < ns) {
                            unsigned long long a, b;
                            ld_strong2(oc + u * (m.D + 4), a, b);
                            bad |= (tag_of(a) ^ tag) | (tag_of(b) ^ tag);
                            ob[u] = make_float2(untag(a), untag(b));
                        }
                    }
                    if (!__any_sync(0xffffffffu, bad != 0)) break;
                    const bool more = pl.again(bd);
                    if (!__all_sync(0xffffffffu, more)) break;
                }
                const float mx = warp_max(fmaxf(mk, mk2));
                const float wk = lane < ns ? expf(mk - mx) : 0.f;
                const float wk2 = lane + 32 < ns ? expf(mk2 - mx) : 0.f;
                const float dn = warp_sum(wk * lk + wk2 * lk2);
                float2 num = make_float2(0.f, 0.f);
                for (int k0 = 0; k0 < ns; k0 += kB) {
                    if (k0 > 0) {  // the next splits (their statistics are in hand)
                        Bound bd2;
                        for (;;) {
                            uint32_t bad = 0;
#pragma unroll
                            for (int u = 0; u < kB; ++u) {
                                ob[u] = make_float2(0.f, 0.f);
                                if (k0 + u < ns) {
                                    unsigned long long a, b;
                                    ld_strong2(oc + (k0 + u) * (m.D + 4), a, b);
                                    bad |= (tag_of(a) ^ tag) | (tag_of(b) ^ tag);
                                    ob[u] = make_float2(untag(a), untag(b));
                                }
                            }
                            if (!__any_sync(0xffffffffu, bad != 0)) break;
                            const bool more = pl.again(bd2);
                            if (!__all_sync(0xffffffffu, more)) break;
                        }
                    }
#pragma unroll
                    for (int u = 0; u < kB; ++u) {
                        const float wu = __shfl_sync(0xffffffffu, k0 + u < 32 ? wk : wk2, (k0 + u) & 31);
                        if (k0 + u < ns) {
                            num.x = fmaf(wu, ob[u].x, num.x);
                            num.y = fmaf(wu, ob[u].y, num.y);
                        }
                    }
                }
                const float inv = 1.0f / dn;
                *dst = make_float2(num.x * inv, num.y * inv);
            }
            csync();
            for (int i = io.lo; i < io.hi; ++i) {
                const int t = i / io.nc, ch = i - t * io.nc;
                const uint32_t buf = saddr(cs.acquire()) + lane * 16 + w * 512;
                const int ccn = (int)(chunk_bytes(io.K, ch) / 512);
                const uint32_t x = saddr(s.xa + (i - io.lo) * kColsPerChunk) + w * 32;
                const float acc = cs.ok ? stage_dot<kCCPerWarp>(buf, x, w, ccn) : 0.f;
                cs.release();
                float* r = s.red + rb * kCW * 32;
                r[w * 32 + lane] = acc;
                csync();
                if (w == 0) {
                    float sum = ch == 0 ? rows[(i - io.lo) * 32 + lane] : 0.f;
#pragma unroll
                    for (int k = 0; k < kCW; ++k) sum += r[k * 32 + lane];
                    st_tagged(op_cur + ((int64_t)t * io.nc + ch) * 32 + lane, sum, tag);
                }
                rb ^= 1;
            }
        }

        // ---------------- gate/up tiles: RMSNorm of the mid residual, SwiGLU
        if (tg1 > tg0) {
            pl.probe(op_cur + ((int64_t)p.n_tiles[1] * p.n_chunks[1] - 1) * 32 + 31, tag);  // the last O slot
            const float inv = gather_norm<2>(s.xs, lw + m.off_gmlp, m.d, m.eps, s.red + 2 * kCW * 32, pl,
                                          [&](int i, uint32_t& bad) { return resid_mid4(p, op_cur, i, tag, bad); });
            tile_gemv(cs, tg0, tg1, p.K[2], p.n_chunks[2], s.xs, s.red, rb, [&](int t, float v) {
                v *= inv;
                const float up = __shfl_xor_sync(0xffffffffu, v, 1);
                const int f = t * 16 + (lane >> 1);
                if (!(lane & 1) && f < m.F) st_tagged(p.a + f, v / (1.0f + expf(-v)) * up, tag);
            });
        }

        // ---------------- down items: partial slots of h_out (slot 0 of a tile
        // adds the tile's mid residual rows, so the slots sum to h_out)
        if (idn.hi > idn.lo) {
            // the mid residual rows of the tiles whose first item is this
            // CTA's (the O slots are complete: this CTA's gate/up gather read
            // them), gathered before the wait for the SwiGLU products
            float* hm = s.xa + (idn.hi - idn.lo) * kColsPerChunk;  // [items][32]
            for (int it = w; it < idn.hi - idn.lo; it += kCW) {
                const int i = idn.lo + it, t = i / idn.nc;
                if (lane < 8 && i - t * idn.nc == 0) {
                    uint32_t bad = 0;
                    float4 r = resid_mid4(p, op_cur, t * 32 + 4 * lane, tag, bad);
                    if (bad) {
                        Bound bd;
                        while (pl.again(bd)) {
                            bad = 0;
                            r = resid_mid4(p, op_cur, t * 32 + 4 * lane, tag, bad);
                            if (!bad) break;
                        }
                    }
                    reinterpret_cast<float4*>(hm + it * 32)[lane] = r;
                }
            }
            pl.probe(p.a + (idn.lo % idn.nc) * kColsPerChunk, tag);  // the first product this CTA reads
            gather4<4>(s.xa, (idn.hi - idn.lo) * kColsPerChunk, pl, [&](int e, uint32_t& bad) {
                const int i = idn.lo + e / kColsPerChunk, col = e % kColsPerChunk;
                const int ch = i % idn.nc, f = ch * kColsPerChunk + col;
                return f < m.F ? load4(p.a + f, tag, bad) : make_float4(0.f, 0.f, 0.f, 0.f);
            });
            csync();
            float acc = 0.f;
            for (int i = idn.lo; i < idn.hi; ++i) {
                const int t = i / idn.nc, ch = i - t * idn.nc;
                const uint32_t buf = saddr(cs.acquire()) + lane * 16 + w * 512;
                const int ccn = (int)(chunk_bytes(idn.K, ch) / 512);
                const uint32_t x = saddr(s.xa + (i - idn.lo) * kColsPerChunk) + w * 32;
                if (cs.ok) acc += stage_dot<kCCPerWarp>(buf, x, w, ccn);
                cs.release();
                if (i + 1 == idn.hi || ch + 1 == idn.nc) {
                    float* r = s.red + rb * kCW * 32;
                    r[w * 32 + lane] = acc;
                    acc = 0.f;
                    csync();
                    if (w == 0) {
                        const int slot = cta - item_owner(idn, t * idn.nc);
                        float sum = slot == 0 ? hm[(t * idn.nc - idn.lo) * 32 + lane] : 0.f;
#pragma unroll
                        for (int k = 0; k < kCW; ++k) sum += r[k * 32 + lane];
                        st_tagged(p.dpart + ((int64_t)t * idn.nc + slot) * 32 + lane, sum, tag);
                    }
                    rb ^= 1;
                }
            }
        }
    }

    // ---------------- the segment's output residual, then the exit ticket
    {
        const unsigned last = seq0 + (unsigned)(j1 - j0 - 1);
        pl.probe(p.dpart + (last_dn_slot + s.nsd[p.n_tiles[3] - 1] - 1) * 32 + 31, seq_tag(last));
        const ResidIn rout{&p, nullptr, nullptr, s.nsd, seq_tag(last)};
        for (int i = slice0 + threadIdx.x; i < slice1; i += kCT) m.h[i] = rout(i, pl);  // slice: scalar
    }
    // the exit ticket: once every CTA has taken it, no CTA reads the launch
    // count any more and the last one advances it for the next launch
    csync();
    if (threadIdx.x == 0) {
        const unsigned prev = atomicAdd(&sync[0], 1u);
        if (prev == (unsigned)G - 1) {
            sync[0] = 0;
            sync[1] = seq0 + (unsigned)(j1 - j0);
        }
    }
}

namespace {

__device__ __forceinline__ void vr_pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void vr_pdl_launch() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

// The vocabulary pass fed through the shared-memory ring: z = RMSNorm(x) *
// gain, l = U z over the tile-packed unembedding, with the online softmax
// statistics of every row (and, for the LM head with nucleus tracking, the
// mass above readout 0's token), finished like the streaming pass.  One CTA
// per SM owns whole 32-row tiles; warp 8's lane 0 streams the tiles' 32 KB
// chunks with cp.async.bulk (it needs nothing from the previous kernel, so it
// starts before the programmatic wait), warps 0..7 take the dot products.
__global__ void __launch_bounds__(kSegThreads, 1) k_vocab_ring(VocabArgs v, int stages) {
    extern __shared__ __align__(128) uint8_t vr_smem[];
    __shared__ int err_local;  // the stall word when there is no control block
    __shared__ float lx_s;
    Smem s{};
    s.ring = vr_smem;
    s.full = reinterpret_cast<uint64_t*>(vr_smem + (size_t)stages * kSegChunk);
    s.empty = s.full + stages;
    float* xs = reinterpret_cast<float*>(s.empty + stages);
    float* red = xs + ((v.d + 3) & ~3);      // [2][kCW][32], then [kCW] norm partials
    float* part = red + 2 * kCW * 32 + kCW;  // [d / 8] partial dot products of one row
    const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        err_local = 0;
        for (int i = 0; i < stages; ++i) {
            mb_init(&s.full[i], 1);
            mb_init(&s.empty[i], kCW);
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    __syncthreads();
    const Waits wt{v.ctl ? &v.ctl->err : &err_local, kSegStallCycles, kSegCheckCycles};
    const int n_tiles = (v.V + kTileRows - 1) / kTileRows, nc = (v.d + kColsPerChunk - 1) / kColsPerChunk;
    int t0, t1;
    whole_tiles(n_tiles, gridDim.x, blockIdx.x, t0, t1);
    const uint8_t* U = reinterpret_cast<const uint8_t*>(v.U);

    if (threadIdx.x >= kCT) {  // producer
        if (threadIdx.x != kCT) return;
        Producer pr(s, stages, stages, wt);
        for (int t = t0; t < t1 && pr.ok; ++t)
            for (int c = 0; c < nc; ++c)
                pr.push(U + (int64_t)t * kTileRows * v.d * 2 + (int64_t)c * kSegChunk, chunk_bytes(v.d, c), pr.pol_w);
        pr.drain();
        return;
    }

    Consumer cs(s, stages, wt);
    vr_pdl_wait();
    vr_pdl_launch();
    // RMSNorm(x) * gain
    float ss = 0.f;
    for (int i = threadIdx.x; i < v.d; i += kCT) ss = fmaf(v.x[i], v.x[i], ss);
    ss = warp_sum(ss);
    if (lane == 0) red[2 * kCW * 32 + w] = ss;
    csync();
    float tot = 0.f;
#pragma unroll
    for (int k = 0; k < kCW; ++k) tot += red[2 * kCW * 32 + k];
    const float inv = 1.0f / sqrtf(tot / (float)v.d + v.eps);
    for (int i = threadIdx.x; i < v.d; i += kCT) xs[i] = v.x[i] * inv * bf(v.gain[i]);
    csync();
    // nucleus tracking: the logit of readout 0's token, then the mass above it
    const bool nucleus = v.mode == 2 && v.ctl->nucleus_on && v.ctl->n_evaluated > 0;
    int nx = -1;
    float lx = INFINITY;
    if (nucleus) {
        nx = v.ctl->readout_token[0];
        if (nx < 0 || nx >= v.V) nx = 0;  // the readout pass flags an out-of-range token
        const int Rc = v.d >> 3, tx = nx >> 5, lx_lane = nx & 31;
        const uint4* W = reinterpret_cast<const uint4*>(v.U);
        for (int c = threadIdx.x; c < Rc; c += kCT) {
            const uint4 wv = __ldg(W + ((int64_t)tx * Rc + c) * 32 + lx_lane);
            part[c] = dot8s(wv, saddr(xs + 8 * c));
        }
        csync();
        if (threadIdx.x == 0) {
            float acc = 0.f;
            for (int c = 0; c < Rc; ++c) acc += part[c];
            lx_s = acc;
        }
        csync();
        lx = lx_s;
    }
    const bool keep = v.logits && (!v.logits_if_dbg || (v.ctl && v.ctl->dbg));
    SoftStats st;
    int rb = 0;
    for (int t = t0; t < t1; ++t) {
        float acc = 0.f;
        for (int c = 0; c < nc; ++c) {
            const uint32_t buf = saddr(cs.acquire()) + lane * 16 + w * 512;
            const int ccn = (int)(chunk_bytes(v.d, c) / 512);
            const uint32_t xc = saddr(xs + c * kColsPerChunk) + w * 32;
            if (cs.ok) acc += stage_dot<kCCPerWarp>(buf, xc, w, ccn);
            cs.release();
        }
        float* r = red + rb * kCW * 32;
        r[w * 32 + lane] = acc;
        csync();
        if (w == 0) {
            float sum = 0.f;
#pragma unroll
            for (int k = 0; k < kCW; ++k) sum += r[k * 32 + lane];
            const int row = t * kTileRows + lane;
            if (row < v.V) {
                if (keep) v.logits[row] = sum;
                st.add(sum, row, lx, nx);
            }
        }
        rb ^= 1;
    }
    vocab_finish(v, st, nucleus, kCW, [] { csync(); });
}

}  // namespace

bool vocab_ring_plan(int d, int n_sm, VocabRing& vr) {
    if (d % 8 || d <= 0 || n_sm <= 0) return false;
    const size_t fixed = (size_t)(((d + 3) & ~3) + 2 * kCW * 32 + kCW + d / 8) * 4 + 1024;
    const size_t budget = 227 * 1024;
    if (fixed + 4 * (size_t)(kSegChunk + 16) > budget) return false;
    vr.G = n_sm;
    vr.stages = (int)std::min<size_t>(16, (budget - fixed) / (kSegChunk + 16));
    vr.smem = (size_t)vr.stages * (kSegChunk + 16) + fixed - 1024;
    return true;
}

cudaError_t configure_vocab_ring(size_t smem) {
    return cudaFuncSetAttribute(k_vocab_ring, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
}

cudaError_t launch_vocab_ring(const VocabArgs& v, const VocabRing& vr, bool pdl, cudaStream_t s) {
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = dim3(vr.G);
    cfg.blockDim = dim3(kSegThreads);
    cfg.dynamicSmemBytes = vr.smem;
    cfg.stream = s;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = at;
    cfg.numAttrs = pdl ? 1 : 0;
    return cudaLaunchKernelEx(&cfg, k_vocab_ring, v, vr.stages);
}

bool seg_plan(const DevModel& m, int n_sm, SegPlan& p) {
    p.G = n_sm;
    const int grp = m.A / m.KH;
    if (m.A % m.KH || grp > kSegMaxGroup || (m.D != 64 && m.D != 128) || m.A > 32 * kCW) return false;
    const int Ks[4] = {m.d, m.A * m.D, m.d, m.F};
    const int64_t rows[4] = {(int64_t)(m.A + 2 * m.KH) * m.D, m.d, 2LL * m.F, m.d};
    for (int i = 0; i < 4; ++i) {
        if (Ks[i] % 8) return false;
        p.K[i] = Ks[i];
        p.n_tiles[i] = (int)tile_count(rows[i]);
        p.n_chunks[i] = (Ks[i] + kColsPerChunk - 1) / kColsPerChunk;
    }
    // O and down items: chunks per O tile and slots per down tile within
    // kSegMaxSlots; items per CTA size the staging buffer
    if (p.n_chunks[1] > kSegMaxSlots) return false;
    const int64_t N = (int64_t)p.n_tiles[3] * p.n_chunks[3];
    const int64_t Ge = std::min<int64_t>(p.G, N);
    const int64_t No = (int64_t)p.n_tiles[1] * p.n_chunks[1], Geo = std::min<int64_t>(p.G, No);
    p.max_items = (int)std::max((N + Ge - 1) / Ge, (No + Geo - 1) / Geo);
    for (int64_t t = 0; t < p.n_tiles[3]; ++t) {
        const int64_t a = ((t * p.n_chunks[3] + 1) * Ge - 1) / N, b = (((t + 1) * p.n_chunks[3]) * Ge - 1) / N;
        if (b - a + 1 > kSegMaxSlots) return false;
    }
    p.rows_per_kv_chunk = std::min(m.page_size, kSegChunk / (2 * m.D));
    if (m.page_size % p.rows_per_kv_chunk) return false;
    const int cap = std::max(1, std::min(kSegMaxSplits, p.G / m.KH));
    const int np_max = (m.max_ctx + m.page_size - 1) / m.page_size;
    p.max_pps = std::max(1, (np_max + cap - 1) / cap);
    p.max_splits = std::min(cap, np_max);
    // xs, xa, rope, red (+ norm partials), qa, kv, sc, ml (the carve above)
    const size_t floats = (size_t)((std::max(m.d, m.A * m.D) + 3) & ~3) + (size_t)p.max_items * (kColsPerChunk + 32) +
                          (size_t)m.D + 2 * kCW * 32 + kCW + (size_t)grp * m.D + 2 * (size_t)m.D +
                          (size_t)grp * p.max_pps * m.page_size + 2 * (size_t)grp;
    const size_t fixed = floats * 4 + (size_t)p.n_tiles[3] + 256;
    const size_t budget = 227 * 1024;
    if (fixed + 4 * (size_t)(kSegChunk + 16) > budget) return false;
    // the attention unit's three bf16 parts of the group's queries fit in xs
    if ((size_t)3 * grp * (m.D + 8) * 2 > (size_t)4 * ((std::max(m.d, m.A * m.D) + 3) & ~3)) return false;
    p.stages = (int)std::min<size_t>(16, (budget - fixed) / (kSegChunk + 16));
    p.smem = (size_t)p.stages * (kSegChunk + 16) + floats * 4 + (size_t)p.n_tiles[3];
    p.inflight = p.stages;
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
