// Online softmax statistics and the end of the vocabulary pass, shared by
// the streaming vocabulary kernel and the ring-fed one.
#ifndef EE_VOCAB_CUH_
#define EE_VOCAB_CUH_

#include <math.h>

#include "ee_internal.h"

namespace ee {

// Online softmax statistics of a set of logits (Section 2 confidence and
// the Section 10 alternatives), all from one pass:
//   m  = max l,  s = sum exp(l - m),  t = sum exp(l - m) (l - m),
//   m2 = the second largest logit (m again if the maximum is tied),
//   a  = lowest index attaining m,
//   g  = sum exp(l - m) over the rows other than x with l > l_x (the
//        tokens more probable than a given token x; 0 when x = -1).
// Then p_max = 1/s, margin = (1 - exp(m2 - m))/s, negative entropy =
// sum p log p = t/s - log s, and the probability above x is g/s.
struct SoftStats {
    float m, s, t, m2, g;
    int a;
    __device__ __forceinline__ SoftStats() : m(-INFINITY), s(0.f), t(0.f), m2(-INFINITY), g(0.f), a(0x7fffffff) {}
    __device__ __forceinline__ void add(float l, int row, float lx = INFINITY, int x = -1) {
        const bool above = l > lx && row != x;
        if (s == 0.f) {
            m = l;
            s = 1.f;
            t = 0.f;
            g = above ? 1.f : 0.f;
            a = row;
        } else if (l > m) {
            const float dl = m - l, e = expf(dl);
            t = e * (t + dl * s);
            s = s * e + 1.0f;
            g = above ? fmaf(g, e, 1.0f) : g * e;
            m2 = m;
            m = l;
            a = row;
        } else {
            const float dl = l - m, e = expf(dl);
            s += e;
            t = fmaf(e, dl, t);
            if (above) g += e;
            if (l > m2) m2 = l;
        }
    }
    // Merge another set (its indices all differ from this one's).
    __device__ __forceinline__ void merge(const SoftStats& o) {
        if (o.s == 0.f) return;
        if (s == 0.f) {
            *this = o;
            return;
        }
        const float M = fmaxf(m, o.m);
        const float ea = expf(m - M), eb = expf(o.m - M);
        t = ea * (t + (m - M) * s) + eb * (o.t + (o.m - M) * o.s);
        s = s * ea + o.s * eb;
        g = g * ea + o.g * eb;
        m2 = fmaxf(fminf(m, o.m), fmaxf(m2, o.m2));
        a = m > o.m ? a : (o.m > m ? o.a : min(a, o.a));
        m = M;
    }
};

__device__ __forceinline__ SoftStats shfl_down_stats(const SoftStats& x, int o) {
    SoftStats y;
    y.m = __shfl_down_sync(0xffffffffu, x.m, o);
    y.s = __shfl_down_sync(0xffffffffu, x.s, o);
    y.t = __shfl_down_sync(0xffffffffu, x.t, o);
    y.m2 = __shfl_down_sync(0xffffffffu, x.m2, o);
    y.g = __shfl_down_sync(0xffffffffu, x.g, o);
    y.a = __shfl_down_sync(0xffffffffu, x.a, o);
    return y;
}

// Warp-wide merge; lane 0 ends with the merge of all lanes in lane order.
__device__ __forceinline__ void warp_merge_stats(SoftStats& st) {
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const SoftStats y = shfl_down_stats(st, o);
        if (((threadIdx.x & 31) & ((o << 1) - 1)) == 0) st.merge(y);
    }
}

// Running statistics of one lane's rows.
using LaneStats = SoftStats;

// After the vocabulary pass: merge the per-lane statistics of the CTA, then
// (last CTA) of the grid; turn them into the confidence signals and, for a
// readout, the gate decision signal > tau, which also selects the graph's
// branch.  The signal is the top-1 probability (Section 2) or, by the
// context's choice, the margin or the negative entropy (Section 10).  With
// nucleus tracking on, the LM head also reports whether readout 0's token
// lies in the full model's nucleus (Section 2 acceptance): the probability
// of the strictly more probable tokens stays below the nucleus share.
// nwarps: the warps that call it (all of the CTA's threads up to nwarps * 32);
// sync: a barrier over exactly those threads.
template <class Sync>
__device__ __forceinline__ void vocab_finish(const VocabArgs& v, LaneStats st, bool nucleus, int nwarps, Sync sync) {
    __shared__ float sm_m[32], sm_s[32], sm_t[32], sm_m2[32], sm_g[32];
    __shared__ int sm_a[32];
    __shared__ int is_last;
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    warp_merge_stats(st);
    if (lane == 0) {
        sm_m[w] = st.m;
        sm_s[w] = st.s;
        sm_t[w] = st.t;
        sm_m2[w] = st.m2;
        sm_g[w] = st.g;
        sm_a[w] = st.a;
    }
    sync();
    if (w == 0) {
        const int nw = nwarps;
        SoftStats x;
        if (lane < nw) {
            x.m = sm_m[lane];
            x.s = sm_s[lane];
            x.t = sm_t[lane];
            x.m2 = sm_m2[lane];
            x.g = sm_g[lane];
            x.a = sm_a[lane];
        }
        warp_merge_stats(x);
        if (lane == 0) {
            float* q = v.part + blockIdx.x * 8;
            q[0] = x.m;
            q[1] = x.s;
            q[2] = x.t;
            q[3] = x.m2;
            reinterpret_cast<int*>(q)[4] = x.a;
            q[5] = x.g;
            __threadfence();
            is_last = atomicAdd(v.ticket, 1) == (int)gridDim.x - 1;
        }
    }
    sync();
    if (!is_last || w != 0) return;
    __threadfence();
    SoftStats x;
    for (int b = lane; b < (int)gridDim.x; b += 32) {
        const float* q = v.part + b * 8;
        SoftStats y;
        y.m = __ldcg(q + 0);
        y.s = __ldcg(q + 1);
        y.t = __ldcg(q + 2);
        y.m2 = __ldcg(q + 3);
        y.a = __ldcg(reinterpret_cast<const int*>(q) + 4);
        y.g = __ldcg(q + 5);
        x.merge(y);
    }
    warp_merge_stats(x);
    if (lane != 0) return;
    *v.ticket = 0;
    const int a = x.a;
    const float p = 1.0f / x.s;
    const float margin = (1.0f - expf(x.m2 - x.m)) / x.s;
    const float negent = x.t / x.s - logf(x.s);
    if (v.mode == 0) {
        *v.out_token = a;
        if (v.out_p) *v.out_p = p;
        if (v.out_sig) {
            v.out_sig[0] = p;
            v.out_sig[1] = margin;
            v.out_sig[2] = negent;
        }
        return;
    }
    Ctl* c = v.ctl;
    const int kind = c->conf_kind;
    const float sig = kind == EE_CONF_MARGIN ? margin : (kind == EE_CONF_NEGENT ? negent : p);
    if (!(sig == sig) || !(p == p) || a < 0 || a >= v.V) atomicOr(&c->err, kErrNanConfidence);
    if (v.mode == 1) {
        const int r = v.r;
        const int f = c->sched ? (int)c->sched[c->step] : c->force;
        const int pass = sig > c->tau[r] ? 1 : 0;
        c->conf[r] = sig;
        c->readout_token[r] = a;
        c->gate_pass[r] = pass;
        c->n_evaluated = r + 1;
        const int take = (f == EE_FREE) ? pass : (f == EE_FORCE_EXIT_AT(r) ? 1 : 0);
        if (take) {
            c->exit_readout = r;
            c->token = a;
        }
        if (v.has_cond) cudaGraphSetConditional(v.cond, take);
    } else {
        c->token = a;
        c->full_token = a;
        c->full_conf = sig;
        c->exit_readout = -1;
        if (nucleus) {
            const float mass = x.g / x.s;
            c->nucleus_mass = mass;
            c->nucleus_member = mass < c->nucleus_p ? 1 : 0;
        }
    }
}

}  // namespace ee

#endif  // EE_VOCAB_CUH_
