// Host engine of libee: workspace layout, weight repack and upload, CUDA graph
// construction, and the extern "C" entry points declared in include/ee.h.
//
// One decode step is one CUDA graph launch.  The graph holds layers 1..k, the
// readout's affine map and vocabulary pass, and an IF/ELSE conditional node
// whose condition the vocabulary pass sets on the device from p > tau: the
// THEN body fills the skipped layers' KV entries, the ELSE body runs the next
// segment of layers (and, with several readouts, the next readout and its own
// conditional node, nested) down to the LM head.  ee_decode_n wraps the step
// in a WHILE conditional node, so n steps run from one launch with the token
// fed back in device memory and no host round trip.
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <string>
#include <thread>
#include <vector>

#include "ee.h"
#include "ee_internal.h"

using namespace ee;

namespace {

thread_local std::string g_err = "";

int fail(int code, const std::string& msg) {
    g_err = msg;
    return code;
}

#define EE_CK(call)                                                                                 \
    do {                                                                                            \
        cudaError_t e_ = (call);                                                                    \
        if (e_ != cudaSuccess) return fail(EE_ECUDA, std::string(#call) + ": " + cudaGetErrorString(e_)); \
    } while (0)

#define EE_TRY(call)             \
    do {                         \
        int rc_ = (call);        \
        if (rc_ != EE_OK) return rc_; \
    } while (0)

constexpr size_t kAlign = 256;
constexpr int kMaxGemvCtas = 1024;
constexpr int kMaxVocabCtas = 1024;
constexpr int kCaptureDepth = kMaxReadouts + 3;

size_t align_up(size_t x, size_t a = kAlign) { return (x + a - 1) / a * a; }
int64_t align_elems(int64_t x) { return (x + 127) / 128 * 128; }  // 256 bytes of bf16

// Byte offsets of every region of the workspace.
struct Layout {
    size_t ctl, rope, layers, embed, lm_head, g_final, ro_w[kMaxReadouts], ro_b[kMaxReadouts];
    size_t kpool, vpool, page_table, kv_src, h_exit, exit_at, repass_pos, h, q, o, a, y, hk, logits_ro, logits_final;
    size_t gemv_part, gemv_ticket, attn_part, attn_ticket, vocab_part, vocab_ticket;
    size_t seg_dpart, seg_opart, seg_q, seg_kvn, seg_a, seg_attn, seg_sync, seg_end;
    size_t rows_H, rows_x3, rows_Q, rows_part, rows_pos;
    size_t prompt, sched, out_tok, out_exit, out_conf, out_conf_all, out_member, out_mass, tau_scratch, total;
    int64_t layer_stride, off_wqkv, off_bqkv, off_gattn, off_wo, off_gmlp, off_wgu, off_wd;
    int64_t n_units_qkv, kv_layer_stride, gemv_ticket_stride, rows_part_floats;
    int n_pages, rows_ldx;
};

int check_config(const ee_model_config* c) {
    if (!c) return fail(EE_EINVAL, "config is NULL");
    if (c->n_layers <= 0 || c->d_model <= 0 || c->n_heads <= 0 || c->n_kv_heads <= 0 || c->ffn_dim <= 0 ||
        c->vocab <= 1 || c->max_ctx <= 0)
        return fail(EE_EINVAL, "config: sizes must be positive");
    if (c->head_dim != 64 && c->head_dim != 128) return fail(EE_EINVAL, "config: head_dim must be 64 or 128");
    if (c->n_heads % c->n_kv_heads || c->n_heads / c->n_kv_heads > 8)
        return fail(EE_EINVAL, "config: n_heads must be a multiple of n_kv_heads, group <= 8");
    if (c->d_model % 8 || c->ffn_dim % 8 || (c->n_heads * c->head_dim) % 8)
        return fail(EE_EINVAL, "config: d_model, ffn_dim and n_heads*head_dim must be multiples of 8");
    if (c->d_model < 256 || c->ffn_dim < 256 || c->n_heads * c->head_dim < 256)
        return fail(EE_EINVAL, "config: rows shorter than 256 elements are not supported");
    if (c->page_size < 16 || c->page_size > 256 || (c->page_size & (c->page_size - 1)))
        return fail(EE_EINVAL, "config: page_size must be a power of two in [16, 256]");
    if (c->max_readouts < 0 || c->max_readouts > kMaxReadouts) return fail(EE_EINVAL, "config: max_readouts");
    if (!(c->rms_eps >= 0.f) || !(c->rope_base > 0.f)) return fail(EE_EINVAL, "config: rms_eps / rope_base");
    return EE_OK;
}

Layout make_layout(const ee_model_config& c) {
    Layout l{};
    const int64_t d = c.d_model, A = c.n_heads, KH = c.n_kv_heads, D = c.head_dim, F = c.ffn_dim, V = c.vocab;
    const int64_t L = c.n_layers, R = std::max(1, c.max_readouts);
    l.n_units_qkv = (A + 2 * KH) * D / 2;
    int64_t o = 0;
    l.off_wqkv = o;
    o += align_elems(tiled_elems(l.n_units_qkv * 2, d));
    l.off_bqkv = o;
    o += align_elems(l.n_units_qkv * 2);
    l.off_gattn = o;
    o += align_elems(d);
    l.off_wo = o;
    o += align_elems(tiled_elems(d, A * D));
    l.off_gmlp = o;
    o += align_elems(d);
    l.off_wgu = o;
    o += align_elems(tiled_elems(2 * F, d));
    l.off_wd = o;
    o += align_elems(tiled_elems(d, F));
    l.layer_stride = o;
    l.n_pages = (c.max_ctx + c.page_size - 1) / c.page_size;
    l.kv_layer_stride = (int64_t)l.n_pages * KH * c.page_size * D;
    l.gemv_ticket_stride = align_elems(std::max<int64_t>({tile_count(2 * l.n_units_qkv), tile_count(d),
                                                         tile_count(2 * F)}));

    size_t b = 0;
    auto take = [&](size_t bytes) {
        const size_t at = b;
        b = align_up(b + bytes);
        return at;
    };
    l.ctl = take(sizeof(Ctl));
    l.rope = take(sizeof(float2) * (size_t)c.max_ctx * (D / 2));
    l.layers = take(2 * (size_t)l.layer_stride * L);
    l.embed = take(2 * (size_t)V * d);
    l.lm_head = take(2 * (size_t)tiled_elems(V, d));
    l.g_final = take(2 * (size_t)d);
    for (int r = 0; r < kMaxReadouts; ++r) {
        if (r < c.max_readouts) {
            l.ro_w[r] = take(2 * (size_t)tiled_elems(d, d));
            l.ro_b[r] = take(2 * (size_t)d);
        } else {
            l.ro_w[r] = l.ro_b[r] = 0;
        }
    }
    l.kpool = take(2 * (size_t)l.kv_layer_stride * L);
    l.vpool = take(2 * (size_t)l.kv_layer_stride * L);
    l.page_table = take(4 * (size_t)l.n_pages);
    l.kv_src = take((size_t)L * c.max_ctx);
    l.h_exit = take(4 * (size_t)c.max_ctx * d);
    l.exit_at = take(2 * (size_t)c.max_ctx);
    l.repass_pos = take(4 * ((size_t)c.max_ctx + 1));
    l.h = take(4 * (size_t)d);
    l.q = take(4 * (size_t)A * D);
    l.o = take(4 * (size_t)A * D);
    l.a = take(4 * (size_t)F);
    l.y = take(4 * (size_t)R * d);
    l.hk = take(4 * (size_t)R * d);
    l.logits_ro = take(4 * (size_t)R * V);
    l.logits_final = take(4 * (size_t)V);
    l.gemv_part = take(4 * (size_t)(kMaxGemvCtas + L) * 2 * kTileRows);
    l.gemv_ticket = take(4 * (size_t)l.gemv_ticket_stride * L);
    l.attn_part = take(4 * (size_t)A * kAttnMaxSplits * (D + 2));
    l.attn_ticket = take(4 * (size_t)KH);
    l.vocab_part = take(4 * (size_t)kMaxVocabCtas * 8);
    l.vocab_ticket = take(4);
    // persistent layer kernel: down-projection partials, mid residual, counters
    {
        const int64_t cols = kSegChunk / (2 * kTileRows);  // columns per ring chunk
        l.seg_dpart = take(sizeof(Tagged) * (size_t)tile_count(d) * ((F + cols - 1) / cols) * kTileRows);
        l.seg_opart = take(2 * sizeof(Tagged) * (size_t)tile_count(d) * ((A * D + cols - 1) / cols) * kTileRows);
    }
    l.seg_q = take(sizeof(Tagged) * (size_t)A * D);
    l.seg_kvn = take(sizeof(Tagged) * 2 * (size_t)KH * D);
    l.seg_a = take(sizeof(Tagged) * (size_t)F);
    l.seg_attn = take(sizeof(Tagged) * (size_t)A * kSegMaxSplits * (D + 4));
    l.seg_sync = take(4 * 8);
    l.seg_end = b;
    // multi-position layer pass (prompt and re-pass batches)
    l.rows_ldx = (int)((std::max({d, F, A * D}) + 63) / 64 * 64);
    l.rows_part_floats = rows_part_floats((int)d, (int)A, (int)KH, (int)D, (int)F);
    l.rows_H = take(4 * (size_t)kRowsMax * d);
    l.rows_x3 = take(2 * 3 * (size_t)kRowsMax * l.rows_ldx);
    l.rows_Q = take(4 * (size_t)kRowsMax * A * D);
    l.rows_part = take(4 * (size_t)l.rows_part_floats);
    l.rows_pos = take(4 * (size_t)kRowsMax);
    l.prompt = take(4 * (size_t)c.max_ctx);
    l.sched = take((size_t)c.max_ctx);
    l.out_tok = take(4 * (size_t)c.max_ctx);
    l.out_exit = take(4 * (size_t)c.max_ctx);
    l.out_conf = take(4 * (size_t)c.max_ctx);
    l.out_conf_all = take(4 * (size_t)c.max_ctx * R);
    l.out_member = take(4 * (size_t)c.max_ctx);
    l.out_mass = take(4 * (size_t)c.max_ctx);
    l.tau_scratch = take(8);
    l.total = b;
    return l;
}

// Copy rows (nullptr = zero padding) of K bf16 values into the tiled layout:
// element (row, k) goes to ((row / 32 * K / 8 + k / 8) * 32 + row % 32) * 8 + k % 8.
void pack_tiles(uint16_t* dst, const std::vector<const uint16_t*>& rows, int64_t K) {
    const int64_t n_tiles = tile_count((int64_t)rows.size()), Rc = K / 8;
    auto work = [&](int64_t t0, int64_t t1) {
        for (int64_t t = t0; t < t1; ++t)
            for (int r = 0; r < kTileRows; ++r) {
                const int64_t row = t * kTileRows + r;
                const uint16_t* src = row < (int64_t)rows.size() ? rows[row] : nullptr;
                for (int64_t cc = 0; cc < Rc; ++cc) {
                    uint16_t* o = dst + ((t * Rc + cc) * kTileRows + r) * 8;
                    if (src)
                        std::memcpy(o, src + cc * 8, 16);
                    else
                        std::memset(o, 0, 16);
                }
            }
    };
    const int nt = (int)std::max(1u, std::min(16u, std::thread::hardware_concurrency()));
    std::vector<std::thread> pool;
    for (int i = 0; i < nt; ++i) pool.emplace_back(work, n_tiles * i / nt, n_tiles * (i + 1) / nt);
    for (auto& th : pool) th.join();
}

std::vector<const uint16_t*> row_ptrs(const uint16_t* base, int64_t n_rows, int64_t K) {
    std::vector<const uint16_t*> v(n_rows);
    for (int64_t i = 0; i < n_rows; ++i) v[i] = base + i * K;
    return v;
}

}  // namespace

int ee::set_last_error(int code, const char* msg) { return fail(code, msg); }

struct ee_ctx {
    ee_model_config cfg{};
    Layout lay{};
    cudaStream_t stream = nullptr;
    cudaStream_t cap[kCaptureDepth] = {};
    char* ws = nullptr;
    bool own_ws = false;
    int device = 0, n_sm = 0;
    DevModel dm{};
    Ctl* d_ctl = nullptr;
    Ctl* h_ctl = nullptr;  // pinned mirror
    int n_readouts = 0;
    int ro_layer[kMaxReadouts] = {};
    bool weights = false, started = false, prefilled = false;
    int pos = 0;
    bool use_graphs = true, use_pdl = true;
    bool seg_ok = false, use_persistent = true;  // persistent layer kernel supported / chosen
    SegPlan seg{};
    bool vring_ok = false;  // ring-fed vocabulary pass supported (used with the persistent layers)
    VocabRing vring{};
    bool use_rows = false;  // EE_OPT_ROWS: prompt and re-pass in batches of positions
    bool lazy_fill = false; // EE_OPT_LAZY_FILL: skipped layers' entries filled by the next step that runs them
    RowsBuf rows{};
    int dbg = 0;
    int conf_kind = EE_CONF_PMAX;  // signal the gates compare with tau
    int repass_period = 0;         // EE_OPT_REPASS: re-pass every this many decode steps (0 = off)
    int repass_from = 0;           // first position the periodic re-pass has not covered
    int nucleus_permille = 0;      // EE_OPT_NUCLEUS: nucleus share in 1/1000, 0 = off
    cudaGraphExec_t g_step = nullptr, g_n = nullptr, g_prefill = nullptr;
    int grid_gemv = 0, grid_vocab = 0;
    int attn_cluster = 8;  // CTAs per key-value head in the attention kernel
};

namespace {

void drop_graphs(ee_ctx* c) {
    for (cudaGraphExec_t* g : {&c->g_step, &c->g_n, &c->g_prefill})
        if (*g) {
            cudaGraphExecDestroy(*g);
            *g = nullptr;
        }
}

// Matrices whose tiles are at most this many bytes, and that have no more
// tiles than the GEMV grid, run one CTA per tile with the tile staged in
// shared memory before the kernel waits on its predecessor.
constexpr int64_t kWholeTileBytes = 144 * 1024;

bool gemv_whole(const ee_ctx* c, int64_t rows, int64_t K) {
    return tile_count(rows) <= c->grid_gemv && 2 * kTileRows * K <= kWholeTileBytes;
}

// Grid of a tiled GEMV launch over `rows` rows of length K: two CTAs per SM,
// or one per tile for small matrices, fewer when each warp would get less
// than one 512-byte item, but enough that no CTA touches more than
// kGemvSlotTiles tiles.
int gemv_grid(const ee_ctx* c, int64_t rows, int64_t K) {
    const int64_t tiles = tile_count(rows), items = tiles * (K / 8);
    if (gemv_whole(c, rows, K)) return (int)tiles;
    int64_t g = std::min<int64_t>(c->grid_gemv, std::max<int64_t>(1, items / (kGemvThreads / 32)));
    const int64_t need = (tiles + kGemvSlotTiles - 3) / (kGemvSlotTiles - 2);
    return (int)std::max<int64_t>(g, need);
}

AttnArgs attn_args(const ee_ctx* c, int j) {
    const DevModel& m = c->dm;
    AttnArgs a{};
    a.q = m.q;
    a.kp = m.kpool + (int64_t)j * m.kv_layer_stride;
    a.vp = m.vpool + (int64_t)j * m.kv_layer_stride;
    a.page_table = m.page_table;
    a.ctl = m.ctl;
    a.T = 0;
    a.A = m.A;
    a.KH = m.KH;
    a.page_size = m.page_size;
    a.out = m.o;
    a.part = m.attn_part;
    a.ticket = m.attn_ticket;
    return a;
}

VocabArgs vocab_args(const ee_ctx* c, int mode, int r, int has_cond, cudaGraphConditionalHandle cond) {
    const DevModel& m = c->dm;
    VocabArgs v{};
    v.x = mode == 1 ? m.y + (int64_t)r * m.d : m.h;
    v.gain = m.g_final;
    v.U = m.lm_head;
    v.tiled = 1;
    v.V = m.V;
    v.d = m.d;
    v.eps = m.eps;
    v.logits = mode == 1 ? m.logits_ro + (int64_t)r * m.V : m.logits_final;
    v.logits_if_dbg = 1;
    v.part = m.vocab_part;
    v.ticket = m.vocab_ticket;
    v.mode = mode;
    v.r = r;
    v.ctl = m.ctl;
    v.has_cond = has_cond;
    v.cond = cond;
    return v;
}

// Layers [j0, j1) of one step on stream s.  `pdl` is the attribute for the
// first launch (false at the start of a graph body).
int enqueue_layers(ee_ctx* c, cudaStream_t s, int j0, int j1, bool& pdl) {
    const DevModel& m = c->dm;
    const int64_t d = m.d, F = m.F, AD = (int64_t)m.A * m.D;
    const int64_t nqkv = c->lay.n_units_qkv * 2;
    const int gq = gemv_grid(c, nqkv, d), go = gemv_grid(c, d, AD), gu = gemv_grid(c, 2 * F, d),
              gd = gemv_grid(c, d, F);
    const bool wq = gemv_whole(c, nqkv, d), wo = gemv_whole(c, d, AD), wu = gemv_whole(c, 2 * F, d),
               wd = gemv_whole(c, d, F);
    if (c->seg_ok && c->use_persistent && j1 > j0) {
        EE_CK(launch_layers(m, c->seg, j0, j1, j0 == 0 ? 1 : 0, s));
        pdl = c->use_pdl;
        return EE_OK;
    }
    for (int j = j0; j < j1; ++j) {
        EE_CK(launch_qkv(m, j, j == 0 ? 1 : 0, gq, wq, pdl, s));
        pdl = c->use_pdl;
        EE_CK(launch_attention_cluster(attn_args(c, j), m.D, c->attn_cluster, pdl, s));
        EE_CK(launch_oproj(m, j, go, wo, pdl, s));
        EE_CK(launch_gateup(m, j, gu, wu, pdl, s));
        EE_CK(launch_down(m, j, gd, wd, pdl, s));
    }
    return EE_OK;
}

// The vocabulary pass: ring-fed alongside the persistent layer kernel,
// streaming otherwise.
cudaError_t enqueue_vocab(const ee_ctx* c, const VocabArgs& v, bool pdl, cudaStream_t s) {
    if (c->use_persistent && c->seg_ok && c->vring_ok) return launch_vocab_ring(v, c->vring, pdl, s);
    return launch_vocab(v, c->grid_vocab, pdl, s);
}

int enqueue_readout(ee_ctx* c, cudaStream_t s, int r, int has_cond, cudaGraphConditionalHandle cond, bool& pdl) {
    const DevModel& m = c->dm;
    EE_CK(launch_readout(m, r, gemv_grid(c, m.d, m.d), gemv_whole(c, m.d, m.d), pdl, s));
    pdl = c->use_pdl;
    EE_CK(enqueue_vocab(c, vocab_args(c, 1, r, has_cond, cond), pdl, s));
    return EE_OK;
}

int enqueue_head(ee_ctx* c, cudaStream_t s, bool& pdl) {
    EE_CK(enqueue_vocab(c, vocab_args(c, 2, 0, 0, 0), pdl, s));
    pdl = c->use_pdl;
    return EE_OK;
}

// CTAs per layer of the KV fill: the SMs shared between the filled layers.
int fill_grid_x(const ee_ctx* c, int n_layers) {
    const int64_t rows = 2LL * c->dm.KH * c->dm.D;
    const int g = gemv_grid(c, rows, c->dm.d);
    const int need = (int)((tile_count(rows) + kGemvSlotTiles - 3) / (kGemvSlotTiles - 2));
    return std::max(need, std::min(g, (c->grid_gemv + n_layers - 1) / n_layers));
}

int enqueue_fill(ee_ctx* c, cudaStream_t s, int exit_layer, bool pdl) {
    const DevModel& m = c->dm;
    if (exit_layer >= m.L) return EE_OK;
    const int nl = m.L - exit_layer;
    const int64_t rows = 2LL * m.KH * m.D;
    const int gx = fill_grid_x(c, nl);
    EE_CK(launch_kvfill(m, exit_layer, gx, gx == tile_count(rows) && gemv_whole(c, rows, m.d), pdl, s));
    return EE_OK;
}

// Add a conditional node at the current capture point of stream s.
int add_conditional(cudaStream_t s, cudaGraphConditionalHandle h, cudaGraphConditionalNodeType type,
                    unsigned size, cudaGraph_t* bodies) {
    cudaStreamCaptureStatus st;
    cudaGraph_t g;
    const cudaGraphNode_t* deps = nullptr;
    size_t nd = 0;
    EE_CK(cudaStreamGetCaptureInfo(s, &st, nullptr, &g, &deps, nullptr, &nd));
    if (st != cudaStreamCaptureStatusActive) return fail(EE_ECUDA, "stream is not capturing");
    cudaGraphNodeParams p{};
    p.type = cudaGraphNodeTypeConditional;
    p.conditional.handle = h;
    p.conditional.type = type;
    p.conditional.size = size;
    cudaGraphNode_t node;
    EE_CK(cudaGraphAddNode(&node, g, deps, nullptr, nd, &p));
    for (unsigned i = 0; i < size; ++i) bodies[i] = p.conditional.phGraph_out[i];
    EE_CK(cudaStreamUpdateCaptureDependencies(s, &node, nullptr, 1, cudaStreamSetCaptureDependencies));
    return EE_OK;
}

int current_capture_graph(cudaStream_t s, cudaGraph_t* g) {
    cudaStreamCaptureStatus st;
    EE_CK(cudaStreamGetCaptureInfo(s, &st, nullptr, g, nullptr, nullptr, nullptr));
    if (st != cudaStreamCaptureStatusActive) return fail(EE_ECUDA, "stream is not capturing");
    return EE_OK;
}

// Capture layers j0.. of a step with readout r next, into the graph being
// captured on c->cap[depth].
int capture_segment(ee_ctx* c, int depth, int j0, int r) {
    if (depth + 1 >= kCaptureDepth) return fail(EE_EINVAL, "too many nested readouts");
    cudaStream_t s = c->cap[depth];
    const int L = c->cfg.n_layers;
    const int j1 = r < c->n_readouts ? c->ro_layer[r] : L;
    bool pdl = false;
    if (c->lazy_fill && j0 > 0) EE_CK(launch_fill_pending(c->dm, j0, j1, false, s));
    EE_TRY(enqueue_layers(c, s, j0, j1, pdl));
    if (r >= c->n_readouts) return enqueue_head(c, s, pdl);
    cudaGraph_t g;
    EE_TRY(current_capture_graph(s, &g));
    cudaGraphConditionalHandle h;
    EE_CK(cudaGraphConditionalHandleCreate(&h, g, 0, 0));
    EE_TRY(enqueue_readout(c, s, r, 1, h, pdl));
    cudaGraph_t bodies[2];
    EE_TRY(add_conditional(s, h, cudaGraphCondTypeIf, 2, bodies));
    cudaStream_t s2 = c->cap[depth + 1];
    // THEN: exit at layer j1, fill the layers above it
    EE_CK(cudaStreamBeginCaptureToGraph(s2, bodies[0], nullptr, nullptr, 0, cudaStreamCaptureModeRelaxed));
    int rc = EE_OK;
    if (j1 < L) {
        if (c->lazy_fill) {
            const cudaError_t e2 = launch_record_exit(c->dm, j1, false, s2);
            if (e2 != cudaSuccess) rc = fail(EE_ECUDA, cudaGetErrorString(e2));
        } else {
            rc = enqueue_fill(c, s2, j1, false);
        }
    }
    cudaGraph_t tmp;
    cudaError_t e = cudaStreamEndCapture(s2, &tmp);
    if (rc != EE_OK) return rc;
    EE_CK(e);
    if (j1 >= L) {
        cudaGraphNode_t empty;
        EE_CK(cudaGraphAddEmptyNode(&empty, bodies[0], nullptr, 0));
    }
    // ELSE: continue to the next readout or the LM head
    EE_CK(cudaStreamBeginCaptureToGraph(s2, bodies[1], nullptr, nullptr, 0, cudaStreamCaptureModeRelaxed));
    rc = capture_segment(c, depth + 1, j1, r + 1);
    e = cudaStreamEndCapture(s2, &tmp);
    if (rc != EE_OK) return rc;
    EE_CK(e);
    return EE_OK;
}

int instantiate(cudaGraph_t g, cudaGraphExec_t* out) {
    cudaError_t e = cudaGraphInstantiate(out, g, 0);
    cudaGraphDestroy(g);
    EE_CK(e);
    return EE_OK;
}

int build_step_graph(ee_ctx* c) {
    cudaStream_t s = c->cap[0];
    EE_CK(cudaStreamBeginCapture(s, cudaStreamCaptureModeRelaxed));
    int rc = capture_segment(c, 0, 0, 0);
    if (rc == EE_OK) {
        cudaError_t e = launch_step_end(c->dm, 0, 0, false, s);
        if (e != cudaSuccess) rc = fail(EE_ECUDA, std::string("step_end: ") + cudaGetErrorString(e));
    }
    cudaGraph_t g = nullptr;
    cudaError_t e = cudaStreamEndCapture(s, &g);
    if (rc != EE_OK) {
        if (g) cudaGraphDestroy(g);
        return rc;
    }
    EE_CK(e);
    return instantiate(g, &c->g_step);
}

// A graph holding one WHILE conditional node whose body is captured by
// `fill_body` on c->cap[1]; the body's last kernel sets the condition.
// Optional `tail` work is captured after the loop on c->cap[0].
template <class Body, class Tail>
int build_while_graph(ee_ctx* c, cudaGraphExec_t* out, Body fill_body, Tail tail) {
    cudaGraph_t g = nullptr;
    EE_CK(cudaGraphCreate(&g, 0));
    int rc = EE_OK;
    do {
        cudaGraphConditionalHandle h;
        cudaError_t e = cudaGraphConditionalHandleCreate(&h, g, 1, cudaGraphCondAssignDefault);
        if (e != cudaSuccess) {
            rc = fail(EE_ECUDA, std::string("while handle: ") + cudaGetErrorString(e));
            break;
        }
        cudaGraphNodeParams p{};
        p.type = cudaGraphNodeTypeConditional;
        p.conditional.handle = h;
        p.conditional.type = cudaGraphCondTypeWhile;
        p.conditional.size = 1;
        cudaGraphNode_t loop;
        e = cudaGraphAddNode(&loop, g, nullptr, nullptr, 0, &p);
        if (e != cudaSuccess) {
            rc = fail(EE_ECUDA, std::string("while node: ") + cudaGetErrorString(e));
            break;
        }
        cudaGraph_t body = p.conditional.phGraph_out[0];
        cudaStream_t s1 = c->cap[1];
        e = cudaStreamBeginCaptureToGraph(s1, body, nullptr, nullptr, 0, cudaStreamCaptureModeRelaxed);
        if (e != cudaSuccess) {
            rc = fail(EE_ECUDA, std::string("body capture: ") + cudaGetErrorString(e));
            break;
        }
        rc = fill_body(s1, h);
        cudaGraph_t tmp = nullptr;
        e = cudaStreamEndCapture(s1, &tmp);
        if (rc == EE_OK && e != cudaSuccess) rc = fail(EE_ECUDA, std::string("body end: ") + cudaGetErrorString(e));
        if (rc != EE_OK) break;
        cudaStream_t s0 = c->cap[0];
        e = cudaStreamBeginCaptureToGraph(s0, g, &loop, nullptr, 1, cudaStreamCaptureModeRelaxed);
        if (e != cudaSuccess) {
            rc = fail(EE_ECUDA, std::string("tail capture: ") + cudaGetErrorString(e));
            break;
        }
        rc = tail(s0);
        e = cudaStreamEndCapture(s0, &tmp);
        if (rc == EE_OK && e != cudaSuccess) rc = fail(EE_ECUDA, std::string("tail end: ") + cudaGetErrorString(e));
    } while (0);
    if (rc != EE_OK) {
        cudaGraphDestroy(g);
        return rc;
    }
    return instantiate(g, out);
}

// n gated steps: WHILE { step body; step_end sets (step < n_steps) }.
int build_loop_graph(ee_ctx* c) {
    return build_while_graph(
        c, &c->g_n,
        [c](cudaStream_t s1, cudaGraphConditionalHandle h) -> int {
            EE_TRY(capture_segment(c, 1, 0, 0));
            EE_CK(launch_step_end(c->dm, 1, h, false, s1));
            return EE_OK;
        },
        [](cudaStream_t) -> int { return EE_OK; });
}

// Prefill: WHILE { all layers at the prompt position; advance }, then the LM
// head on the last position and the hand-over of its token.
int build_prefill_graph(ee_ctx* c) {
    return build_while_graph(
        c, &c->g_prefill,
        [c](cudaStream_t s1, cudaGraphConditionalHandle h) -> int {
            bool pdl = false;
            EE_TRY(enqueue_layers(c, s1, 0, c->cfg.n_layers, pdl));
            EE_CK(launch_prefill_advance(c->dm, 1, h, c->use_pdl, s1));
            return EE_OK;
        },
        [c](cudaStream_t s0) -> int {
            bool pdl = false;
            EE_TRY(enqueue_head(c, s0, pdl));
            EE_CK(launch_prefill_end(c->dm, c->use_pdl, s0));
            return EE_OK;
        });
}

int ensure_graphs(ee_ctx* c) {
    if (!c->g_step) EE_TRY(build_step_graph(c));
    if (!c->g_n) EE_TRY(build_loop_graph(c));
    if (!c->g_prefill) EE_TRY(build_prefill_graph(c));
    return EE_OK;
}

int fetch_ctl(ee_ctx* c) {
    EE_CK(cudaMemcpyAsync(c->h_ctl, c->d_ctl, sizeof(Ctl), cudaMemcpyDeviceToHost, c->stream));
    EE_CK(cudaStreamSynchronize(c->stream));
    return EE_OK;
}

int device_error(const ee_ctx* c) {
    const int e = c->h_ctl->err;
    if (!e) return EE_OK;
    std::string m = "device error:";
    if (e & kErrNanConfidence) m += " non-finite confidence;";
    if (e & kErrTokenRange) m += " token out of range;";
    if (e & kErrPosition) m += " position beyond max_ctx;";
    if (e & kErrStall) m += " a wait of the persistent layer kernel timed out (call ee_reset);";
    return fail(EE_EDEVICE, m);
}

CtlInputs base_inputs(const ee_ctx* c, const float* taus) {
    CtlInputs in{};
    in.set_token = 0;
    in.n_steps = 1;
    in.dbg = c->dbg;
    in.conf_kind = c->conf_kind;
    in.nucleus_on = c->nucleus_permille > 0 && c->n_readouts > 0;
    in.nucleus_p = (float)c->nucleus_permille / 1000.0f;
    for (int r = 0; r < kMaxReadouts; ++r) in.tau[r] = (taus && r < c->n_readouts) ? taus[r] : 2.0f;
    return in;
}

// The re-pass through the multi-position layer pass: batches of kRowsMax
// positions in position order (a batch's attention reads the entries earlier
// batches re-passed), the rows of a batch ordered by the layer they start at.
// The final residual of the last position is left in m.h.
int rows_repass(ee_ctx* c, const std::vector<int32_t>& todo, const std::vector<int32_t>& from) {
    cudaStream_t s = c->stream;
    const DevModel& m = c->dm;
    const int n = (int)todo.size();
    std::vector<int32_t> pos(n);
    std::vector<int> start(n);
    int last_row = 0;
    for (int b0 = 0; b0 < n; b0 += kRowsMax) {
        const int M = std::min(kRowsMax, n - b0);
        std::vector<int> idx(M);
        for (int i = 0; i < M; ++i) idx[i] = b0 + i;
        std::stable_sort(idx.begin(), idx.end(), [&](int a, int b) { return from[a] < from[b]; });
        for (int i = 0; i < M; ++i) {
            pos[b0 + i] = todo[idx[i]];
            start[b0 + i] = from[idx[i]];
            if (idx[i] == n - 1) last_row = i;
        }
    }
    int32_t* d_pos = (int32_t*)(c->ws + c->lay.repass_pos);
    EE_CK(cudaMemcpy(d_pos, pos.data(), 4 * (size_t)n, cudaMemcpyHostToDevice));  // the stream is idle
    for (int b0 = 0; b0 < n; b0 += kRowsMax) {
        const int M = std::min(kRowsMax, n - b0);
        const bool last = b0 + M == n;
        const int t_max = *std::max_element(pos.begin() + b0, pos.begin() + b0 + M) + 1;
        EE_CK(rows_pass(m, c->rows, start.data() + b0, M, d_pos + b0, nullptr, 0, t_max, !last, s));
    }
    EE_CK(cudaMemcpyAsync(m.h, c->rows.H + (int64_t)last_row * m.d, 4 * (size_t)m.d, cudaMemcpyDeviceToDevice, s));
    EE_TRY(fetch_ctl(c));
    return device_error(c);
}

// The prompt in batches of kRowsMax positions through the multi-position
// layer pass (only the last batch runs the last layer past its cache
// entries), then the LM head on the last position's final residual.
int rows_prefill(ee_ctx* c, const int32_t* d_prompt, int n) {
    cudaStream_t s = c->stream;
    const DevModel& m = c->dm;
    const std::vector<int> start(kRowsMax, 0);
    int last_row = 0;
    for (int b0 = 0; b0 < n; b0 += kRowsMax) {
        const int M = std::min(kRowsMax, n - b0);
        EE_CK(rows_pass(m, c->rows, start.data(), M, c->rows.pos, d_prompt + b0, b0, b0 + M, b0 + M < n, s));
        last_row = M - 1;
    }
    EE_CK(cudaMemcpyAsync(m.h, c->rows.H + (int64_t)last_row * m.d, 4 * (size_t)m.d, cudaMemcpyDeviceToDevice, s));
    EE_CK(launch_rows_prefill_done(m, n, s));
    bool pdl = false;
    EE_TRY(enqueue_head(c, s, pdl));
    EE_CK(launch_prefill_end(m, false, s));
    return EE_OK;
}

// Fill every entry the deferred fill left pending (all layers, positions
// below the decode position); afterwards nothing below it is pending.
int flush_pending(ee_ctx* c) {
    const DevModel& m = c->dm;
    EE_CK(launch_fill_pending(m, 1, m.L, false, c->stream));
    EE_CK(cudaMemcpyAsync(&c->d_ctl->pend_lo, &c->d_ctl->pos, 4, cudaMemcpyDeviceToDevice, c->stream));
    return EE_OK;
}

// Section 11's full-depth re-pass over positions [t0, t1) (t1 <= pos): each
// position whose upper layers still hold filled entries runs them again from
// the residual it exited with (h_exit), in position order, through the same
// layer kernels as a decode step; the control block's position is pointed at
// each one in turn and restored at the end.  Synchronous.
int repass_range(ee_ctx* c, int t0, int t1, int* n_done) {
    cudaStream_t s = c->stream;
    const DevModel& m = c->dm;
    const int L = m.L, W = t1 - t0;
    if (n_done) *n_done = 0;
    if (W <= 0) return EE_OK;
    if (c->lazy_fill) EE_TRY(flush_pending(c));  // the re-pass finds exited positions by their fills
    EE_CK(cudaStreamSynchronize(s));
    std::vector<int16_t> ex(W);
    std::vector<int8_t> src((size_t)L * W);
    EE_CK(cudaMemcpy(ex.data(), m.exit_at + t0, 2 * (size_t)W, cudaMemcpyDeviceToHost));
    EE_CK(cudaMemcpy2D(src.data(), (size_t)W, m.kv_src + t0, (size_t)m.max_ctx, (size_t)W, (size_t)L,
                       cudaMemcpyDeviceToHost));
    std::vector<int32_t> todo, from;
    for (int i = 0; i < W; ++i) {
        const int k = ex[i];
        if (k >= 1 && k < L && src[(size_t)k * W + i] == 2) {
            todo.push_back(t0 + i);
            from.push_back(k);
        }
    }
    if (todo.empty()) return EE_OK;
    if (c->use_rows) {
        EE_TRY(rows_repass(c, todo, from));
        if (n_done) *n_done = (int)todo.size();
        return EE_OK;
    }
    int32_t* d_pos = (int32_t*)(c->ws + c->lay.repass_pos);  // the positions, then the decode position
    std::vector<int32_t> pos_list(todo);
    pos_list.push_back(c->pos);
    EE_CK(cudaMemcpy(d_pos, pos_list.data(), 4 * pos_list.size(), cudaMemcpyHostToDevice));
    for (size_t i = 0; i < todo.size(); ++i) {
        EE_CK(cudaMemcpyAsync(m.h, m.h_exit + (int64_t)todo[i] * m.d, 4 * (size_t)m.d, cudaMemcpyDeviceToDevice, s));
        EE_CK(cudaMemcpyAsync(&c->d_ctl->pos, d_pos + i, 4, cudaMemcpyDeviceToDevice, s));
        bool pdl = false;
        EE_TRY(enqueue_layers(c, s, from[i], L, pdl));
    }
    EE_CK(cudaMemcpyAsync(&c->d_ctl->pos, d_pos + todo.size(), 4, cudaMemcpyDeviceToDevice, s));
    EE_TRY(fetch_ctl(c));
    EE_TRY(device_error(c));
    if (n_done) *n_done = (int)todo.size();
    return EE_OK;
}

// Direct launches with the branch taken on the host (EE_OPT_GRAPHS = 0).
int eager_step(ee_ctx* c) {
    cudaStream_t s = c->stream;
    const DevModel& m = c->dm;
    bool pdl = false;
    int j0 = 0;
    for (int r = 0; r <= c->n_readouts; ++r) {
        const int j1 = r < c->n_readouts ? c->ro_layer[r] : m.L;
        if (c->lazy_fill && j0 > 0) EE_CK(launch_fill_pending(m, j0, j1, false, s));
        EE_TRY(enqueue_layers(c, s, j0, j1, pdl));
        if (r == c->n_readouts) {
            EE_TRY(enqueue_head(c, s, pdl));
            break;
        }
        EE_TRY(enqueue_readout(c, s, r, 0, 0, pdl));
        EE_TRY(fetch_ctl(c));
        pdl = false;
        if (c->h_ctl->exit_readout == r) {
            if (j1 < m.L && c->lazy_fill)
                EE_CK(launch_record_exit(m, j1, false, s));
            else
                EE_TRY(enqueue_fill(c, s, j1, false));
            break;
        }
        j0 = j1;
    }
    EE_CK(launch_step_end(m, 0, 0, false, s));
    return EE_OK;
}

}  // namespace

// ======================================================================
// extern "C" entry points
// ======================================================================

extern "C" {

const char* ee_last_error(void) { return g_err.c_str(); }

int ee_workspace_bytes(const ee_model_config* cfg, size_t* bytes) {
    EE_TRY(check_config(cfg));
    if (!bytes) return fail(EE_EINVAL, "bytes is NULL");
    *bytes = make_layout(*cfg).total;
    return EE_OK;
}

int ee_create(const ee_model_config* cfg, void* d_workspace, size_t workspace_bytes, void* stream, ee_ctx** out) {
    EE_TRY(check_config(cfg));
    if (!out) return fail(EE_EINVAL, "out is NULL");
    *out = nullptr;
    if (d_workspace && ((uintptr_t)d_workspace % kAlign)) return fail(EE_EINVAL, "workspace not 256-byte aligned");
    ee_ctx* c = new ee_ctx();
    c->cfg = *cfg;
    c->lay = make_layout(*cfg);
    c->stream = (cudaStream_t)stream;
    auto bail = [&](int rc) {
        ee_destroy(c);
        return rc;
    };
    if (cudaGetDevice(&c->device) != cudaSuccess) return bail(fail(EE_ECUDA, "no CUDA device"));
    cudaDeviceGetAttribute(&c->n_sm, cudaDevAttrMultiProcessorCount, c->device);
    c->grid_gemv = std::min(2 * c->n_sm, kMaxGemvCtas);  // two 512-thread CTAs per SM
    c->grid_vocab = std::min(2 * c->n_sm, kMaxVocabCtas);
    c->attn_cluster = 0;  // chosen after the kernels are configured
    if (d_workspace) {
        if (workspace_bytes < c->lay.total) return bail(fail(EE_ENOMEM, "workspace too small"));
        c->ws = (char*)d_workspace;
    } else {
        if (cudaMalloc(&c->ws, c->lay.total) != cudaSuccess) {
            c->ws = nullptr;
            return bail(fail(EE_ENOMEM, "cudaMalloc of the workspace failed"));
        }
        c->own_ws = true;
    }
    for (int i = 0; i < kCaptureDepth; ++i)
        if (cudaStreamCreateWithFlags(&c->cap[i], cudaStreamNonBlocking) != cudaSuccess)
            return bail(fail(EE_ECUDA, "stream creation failed"));
    if (cudaMallocHost(&c->h_ctl, sizeof(Ctl)) != cudaSuccess) return bail(fail(EE_ENOMEM, "pinned alloc failed"));
    const Layout& l = c->lay;
    char* w = c->ws;
    DevModel& m = c->dm;
    m.L = cfg->n_layers;
    m.d = cfg->d_model;
    m.A = cfg->n_heads;
    m.KH = cfg->n_kv_heads;
    m.D = cfg->head_dim;
    m.F = cfg->ffn_dim;
    m.V = cfg->vocab;
    m.max_ctx = cfg->max_ctx;
    m.page_size = cfg->page_size;
    m.n_pages = l.n_pages;
    m.qkv_bias = cfg->qkv_bias;
    m.n_readouts = 0;
    m.eps = cfg->rms_eps;
    m.layers = (const uint16_t*)(w + l.layers);
    m.layer_stride = l.layer_stride;
    m.off_wqkv = l.off_wqkv;
    m.off_bqkv = l.off_bqkv;
    m.off_gattn = l.off_gattn;
    m.off_wo = l.off_wo;
    m.off_gmlp = l.off_gmlp;
    m.off_wgu = l.off_wgu;
    m.off_wd = l.off_wd;
    m.embed = (const uint16_t*)(w + l.embed);
    m.lm_head = (const uint16_t*)(w + l.lm_head);
    m.g_final = (const uint16_t*)(w + l.g_final);
    for (int r = 0; r < cfg->max_readouts; ++r) {
        m.ro_w[r] = (const uint16_t*)(w + l.ro_w[r]);
        m.ro_b[r] = (const uint16_t*)(w + l.ro_b[r]);
    }
    m.rope = (const float2*)(w + l.rope);
    m.kpool = (uint16_t*)(w + l.kpool);
    m.vpool = (uint16_t*)(w + l.vpool);
    m.kv_layer_stride = l.kv_layer_stride;
    m.page_table = (const int32_t*)(w + l.page_table);
    m.kv_src = (int8_t*)(w + l.kv_src);
    m.h_exit = (float*)(w + l.h_exit);
    m.exit_at = (int16_t*)(w + l.exit_at);
    m.h = (float*)(w + l.h);
    m.q = (float*)(w + l.q);
    m.o = (float*)(w + l.o);
    m.a = (float*)(w + l.a);
    m.y = (float*)(w + l.y);
    m.hk = (float*)(w + l.hk);
    m.logits_ro = (float*)(w + l.logits_ro);
    m.logits_final = (float*)(w + l.logits_final);
    m.gemv_part = (float*)(w + l.gemv_part);
    m.gemv_ticket = (unsigned*)(w + l.gemv_ticket);
    m.gemv_ticket_stride = l.gemv_ticket_stride;
    m.attn_part = (float*)(w + l.attn_part);
    m.attn_ticket = (int*)(w + l.attn_ticket);
    m.vocab_part = (float*)(w + l.vocab_part);
    m.vocab_ticket = (int*)(w + l.vocab_ticket);
    m.ctl = (Ctl*)(w + l.ctl);
    c->d_ctl = m.ctl;
    c->rows.H = (float*)(w + l.rows_H);
    c->rows.x3 = (uint16_t*)(w + l.rows_x3);
    c->rows.Q = (float*)(w + l.rows_Q);
    c->rows.part = (float*)(w + l.rows_part);
    c->rows.pos = (int32_t*)(w + l.rows_pos);
    c->rows.part_floats = l.rows_part_floats;
    c->rows.ldx = l.rows_ldx;
    c->rows.n_sm = c->n_sm;
    c->rows.err = &c->d_ctl->err;
    // prompts and re-passes in batches on the tcgen05 tensor cores where available
    c->rows.umma = umma_available() ? 1 : 0;
    c->use_rows = c->rows.umma == 1;

    const int kmax = std::max({2 * m.d, m.A * m.D, m.F});
    if (configure_kernels(kmax) != cudaSuccess || configure_fill_pending(m.d) != cudaSuccess ||
        configure_rows() != cudaSuccess)
        return bail(fail(EE_ECUDA, "kernel configuration failed"));
    c->attn_cluster = attention_cluster_size(m.D, m.KH);
    if (seg_plan(m, c->n_sm, c->seg) && configure_layers(c->seg.smem) == cudaSuccess &&
        layers_blocks_per_sm(c->seg.smem) >= 1) {
        c->seg.dpart = (Tagged*)(w + l.seg_dpart);
        c->seg.opart = (Tagged*)(w + l.seg_opart);
        c->seg.attn_part = (Tagged*)(w + l.seg_attn);
        c->seg.q = (Tagged*)(w + l.seg_q);
        c->seg.kvn = (Tagged*)(w + l.seg_kvn);
        c->seg.a = (Tagged*)(w + l.seg_a);
        c->seg.sync = (unsigned*)(w + l.seg_sync);
        c->seg.stall_cycles = kSegStallCycles;
        c->seg.check_cycles = kSegCheckCycles;
        c->seg_ok = true;
    }
    if (vocab_ring_plan(m.d, c->n_sm, c->vring) && configure_vocab_ring(c->vring.smem) == cudaSuccess)
        c->vring_ok = c->vring.G <= kMaxVocabCtas;
    cudaGetLastError();

    // RoPE table: angle t * base^(-2i/D) in double, cos/sin rounded to fp32.
    std::vector<float2> rope((size_t)m.max_ctx * (m.D / 2));
    for (int t = 0; t < m.max_ctx; ++t)
        for (int i = 0; i < m.D / 2; ++i) {
            const double ang = (double)t * std::pow((double)cfg->rope_base, -2.0 * i / (double)m.D);
            rope[(size_t)t * (m.D / 2) + i] = make_float2((float)std::cos(ang), (float)std::sin(ang));
        }
    if (cudaMemcpy(w + l.rope, rope.data(), rope.size() * sizeof(float2), cudaMemcpyHostToDevice) != cudaSuccess)
        return bail(fail(EE_ECUDA, "rope upload failed"));
    std::vector<int32_t> pt(l.n_pages);
    for (int i = 0; i < l.n_pages; ++i) pt[i] = i;
    if (cudaMemcpy(w + l.page_table, pt.data(), pt.size() * 4, cudaMemcpyHostToDevice) != cudaSuccess)
        return bail(fail(EE_ECUDA, "page table upload failed"));
    // zero the arrival counters (kernels return them to zero after use)
    if (cudaMemset(w + l.gemv_ticket, 0, 4 * (size_t)l.gemv_ticket_stride * m.L) != cudaSuccess ||
        cudaMemset(w + l.attn_ticket, 0, 4 * (size_t)m.KH) != cudaSuccess ||
        cudaMemset(w + l.vocab_ticket, 0, 4) != cudaSuccess)
        return bail(fail(EE_ECUDA, "memset failed"));
    *out = c;
    int rc = ee_reset(c);
    if (rc != EE_OK) {
        *out = nullptr;
        return bail(rc);
    }
    return EE_OK;
}

int ee_destroy(ee_ctx* c) {
    if (!c) return EE_OK;
    if (c->stream || c->ws) cudaStreamSynchronize(c->stream);
    drop_graphs(c);
    for (int i = 0; i < kCaptureDepth; ++i)
        if (c->cap[i]) cudaStreamDestroy(c->cap[i]);
    if (c->h_ctl) cudaFreeHost(c->h_ctl);
    if (c->own_ws && c->ws) cudaFree(c->ws);
    delete c;
    return EE_OK;
}

int ee_load_weights(ee_ctx* c, const ee_host_weights* w) {
    if (!c || !w) return fail(EE_EINVAL, "NULL argument");
    const ee_model_config& cf = c->cfg;
    const int L = cf.n_layers;
    const int64_t d = cf.d_model, A = cf.n_heads, KH = cf.n_kv_heads, D = cf.head_dim, F = cf.ffn_dim,
                  V = cf.vocab;
    if (!w->embed || !w->final_norm || (!cf.tied_embedding && !w->lm_head) || !w->attn_norm || !w->wq || !w->wk ||
        !w->wv || !w->wo || !w->mlp_norm || !w->wg || !w->wu || !w->wd)
        return fail(EE_EINVAL, "missing weight array");
    if (cf.qkv_bias && (!w->bq || !w->bk || !w->bv)) return fail(EE_EINVAL, "missing bias array");
    for (int j = 0; j < L; ++j)
        if (!w->attn_norm[j] || !w->wq[j] || !w->wk[j] || !w->wv[j] || !w->wo[j] || !w->mlp_norm[j] || !w->wg[j] ||
            !w->wu[j] || !w->wd[j] || (cf.qkv_bias && (!w->bq[j] || !w->bk[j] || !w->bv[j])))
            return fail(EE_EINVAL, "missing per-layer weight");
    const Layout& l = c->lay;
    uint16_t* stage = nullptr;
    EE_CK(cudaMallocHost(&stage, 2 * (size_t)l.layer_stride));
    std::memset(stage, 0, 2 * (size_t)l.layer_stride);
    int rc = EE_OK;
    const int64_t half = D / 2;
    for (int j = 0; j < L && rc == EE_OK; ++j) {
        // Q/K/V: 16 units per tile, a unit being the row pair (i, i + D/2) of
        // one head (first row on the even lane); Q heads, then K, then V.
        std::vector<const uint16_t*> rows;
        uint16_t* bqkv = stage + l.off_bqkv;
        int64_t u = 0;
        const uint16_t* mats[3] = {w->wq[j], w->wk[j], w->wv[j]};
        const uint16_t* bias[3] = {cf.qkv_bias ? w->bq[j] : nullptr, cf.qkv_bias ? w->bk[j] : nullptr,
                                   cf.qkv_bias ? w->bv[j] : nullptr};
        const int64_t heads[3] = {A, KH, KH};
        for (int t = 0; t < 3; ++t)
            for (int64_t h = 0; h < heads[t]; ++h)
                for (int64_t i = 0; i < half; ++i, ++u) {
                    const int64_t r0 = h * D + i, r1 = h * D + i + half;
                    rows.push_back(mats[t] + r0 * d);
                    rows.push_back(mats[t] + r1 * d);
                    if (bias[t]) {
                        bqkv[u * 2 + 0] = bias[t][r0];
                        bqkv[u * 2 + 1] = bias[t][r1];
                    }
                }
        pack_tiles(stage + l.off_wqkv, rows, d);
        std::memcpy(stage + l.off_gattn, w->attn_norm[j], 2 * (size_t)d);
        pack_tiles(stage + l.off_wo, row_ptrs(w->wo[j], d, A * D), A * D);
        std::memcpy(stage + l.off_gmlp, w->mlp_norm[j], 2 * (size_t)d);
        // gate/up: 16 units per tile, unit i = (W_g row i, W_u row i)
        rows.clear();
        for (int64_t i = 0; i < F; ++i) {
            rows.push_back(w->wg[j] + i * d);
            rows.push_back(w->wu[j] + i * d);
        }
        pack_tiles(stage + l.off_wgu, rows, d);
        pack_tiles(stage + l.off_wd, row_ptrs(w->wd[j], d, F), F);
        cudaError_t e = cudaMemcpy(c->ws + l.layers + 2 * (size_t)l.layer_stride * j, stage,
                                   2 * (size_t)l.layer_stride, cudaMemcpyHostToDevice);
        if (e != cudaSuccess) rc = fail(EE_ECUDA, std::string("layer upload: ") + cudaGetErrorString(e));
    }
    cudaFreeHost(stage);
    if (rc != EE_OK) return rc;
    EE_CK(cudaMemcpy(c->ws + l.embed, w->embed, 2 * (size_t)V * d, cudaMemcpyHostToDevice));
    {
        std::vector<uint16_t> tiled((size_t)tiled_elems(V, d));
        pack_tiles(tiled.data(), row_ptrs(cf.tied_embedding ? w->embed : w->lm_head, V, d), d);
        EE_CK(cudaMemcpy(c->ws + l.lm_head, tiled.data(), 2 * tiled.size(), cudaMemcpyHostToDevice));
    }
    EE_CK(cudaMemcpy(c->ws + l.g_final, w->final_norm, 2 * (size_t)d, cudaMemcpyHostToDevice));
    c->weights = true;
    drop_graphs(c);
    return EE_OK;
}

int ee_add_readout(ee_ctx* c, int layer, const uint16_t* wr, const uint16_t* br, int* readout_id) {
    if (!c || !wr || !br) return fail(EE_EINVAL, "NULL argument");
    if (c->started) return fail(EE_ESTATE, "readouts must be added before the first prefill");
    if (c->n_readouts >= c->cfg.max_readouts) return fail(EE_EINVAL, "max_readouts reached");
    if (layer < 1 || layer > c->cfg.n_layers) return fail(EE_EINVAL, "readout layer outside [1, n_layers]");
    if (c->n_readouts > 0 && layer <= c->ro_layer[c->n_readouts - 1])
        return fail(EE_EINVAL, "readouts must be added in increasing layer order");
    const int r = c->n_readouts;
    const size_t d = c->cfg.d_model;
    std::vector<uint16_t> tiled((size_t)tiled_elems(d, d));
    pack_tiles(tiled.data(), row_ptrs(wr, d, d), d);
    EE_CK(cudaMemcpy(c->ws + c->lay.ro_w[r], tiled.data(), 2 * tiled.size(), cudaMemcpyHostToDevice));
    EE_CK(cudaMemcpy(c->ws + c->lay.ro_b[r], br, 2 * d, cudaMemcpyHostToDevice));
    c->ro_layer[r] = layer;
    c->dm.ro_layer[r] = layer;
    c->n_readouts = r + 1;
    c->dm.n_readouts = r + 1;
    drop_graphs(c);
    if (readout_id) *readout_id = r;
    return EE_OK;
}

int ee_set_page_table(ee_ctx* c, const int32_t* pages, int n_pages) {
    if (!c || !pages) return fail(EE_EINVAL, "NULL argument");
    if (n_pages != c->lay.n_pages) return fail(EE_EINVAL, "page table must cover every logical page");
    if (c->prefilled) return fail(EE_ESTATE, "page table can only change between reset and prefill");
    std::vector<char> seen(n_pages, 0);
    for (int i = 0; i < n_pages; ++i) {
        if (pages[i] < 0 || pages[i] >= n_pages || seen[pages[i]]) return fail(EE_EINVAL, "not a permutation");
        seen[pages[i]] = 1;
    }
    EE_CK(cudaMemcpyAsync(c->ws + c->lay.page_table, pages, 4 * (size_t)n_pages, cudaMemcpyHostToDevice, c->stream));
    EE_CK(cudaStreamSynchronize(c->stream));
    return EE_OK;
}

int ee_reset(ee_ctx* c) {
    if (!c) return fail(EE_EINVAL, "NULL context");
    EE_CK(cudaStreamSynchronize(c->stream));
    std::memset(c->h_ctl, 0, sizeof(Ctl));
    c->h_ctl->exit_readout = -1;
    c->h_ctl->full_token = -1;
    c->h_ctl->max_ctx = c->cfg.max_ctx;
    EE_CK(cudaMemcpyAsync(c->d_ctl, c->h_ctl, sizeof(Ctl), cudaMemcpyHostToDevice, c->stream));
    EE_CK(cudaMemsetAsync(c->ws + c->lay.kv_src, 0, (size_t)c->cfg.n_layers * c->cfg.max_ctx, c->stream));
    EE_CK(cudaMemsetAsync(c->ws + c->lay.exit_at, 0, 2 * (size_t)c->cfg.max_ctx, c->stream));
    // the persistent layer kernel's exchange buffers (tags 0: never valid),
    // exit ticket and launch count
    EE_CK(cudaMemsetAsync(c->ws + c->lay.seg_dpart, 0, c->lay.seg_end - c->lay.seg_dpart, c->stream));
    EE_CK(cudaStreamSynchronize(c->stream));
    c->pos = 0;
    c->repass_from = 0;
    c->prefilled = false;
    return EE_OK;
}

int ee_set_option(ee_ctx* c, int option, int value) {
    if (!c) return fail(EE_EINVAL, "NULL context");
    switch (option) {
        case EE_OPT_GRAPHS:
            c->use_graphs = value != 0;
            return EE_OK;
        case EE_OPT_PDL:
            if (c->use_pdl != (value != 0)) drop_graphs(c);
            c->use_pdl = value != 0;
            return EE_OK;
        case EE_OPT_DEBUG_LOGITS:
            c->dbg = value != 0;
            return EE_OK;
        case EE_OPT_CONFIDENCE:
            if (value < EE_CONF_PMAX || value > EE_CONF_NEGENT) return fail(EE_EINVAL, "unknown confidence signal");
            c->conf_kind = value;
            return EE_OK;
        case EE_OPT_REPASS:
            if (value < 0) return fail(EE_EINVAL, "re-pass period must be >= 0");
            c->repass_period = value;
            c->repass_from = c->pos;
            return EE_OK;
        case EE_OPT_NUCLEUS:
            if (value < 0 || value > 1000) return fail(EE_EINVAL, "nucleus share must be 0..1000 per mille");
            c->nucleus_permille = value;
            return EE_OK;
        case EE_OPT_ROWS:
            if (value < 0 || value > 2) return fail(EE_EINVAL, "EE_OPT_ROWS takes 0, 1 or 2");
            if (value == 1 && !umma_available())
                return fail(EE_EINVAL, "the tcgen05 projections are not available on this device");
            c->use_rows = value != 0;
            c->rows.umma = value == 1 ? 1 : 0;
            return EE_OK;
        case EE_OPT_LAZY_FILL:
            if (c->lazy_fill == (value != 0)) return EE_OK;
            if (c->lazy_fill && c->prefilled) {  // off: fill what is pending first
                EE_TRY(flush_pending(c));
                EE_CK(cudaStreamSynchronize(c->stream));
            }
            drop_graphs(c);
            c->lazy_fill = value != 0;
            return EE_OK;
        case EE_OPT_WAIT_LIMIT:
            if (value < 0) return fail(EE_EINVAL, "wait limit must be >= 0");
            drop_graphs(c);
            c->seg.stall_cycles = value ? (long long)value : kSegStallCycles;
            c->seg.check_cycles = value ? std::max(1LL, (long long)value / 4) : kSegCheckCycles;
            return EE_OK;
        case EE_OPT_PERSISTENT:
            if (value && !c->seg_ok) return fail(EE_EINVAL, "the persistent layer kernel does not support this shape");
            if (c->use_persistent != (value != 0)) drop_graphs(c);
            c->use_persistent = value != 0;
            return EE_OK;
        default:
            return fail(EE_EINVAL, "unknown option");
    }
}

int ee_prefill(ee_ctx* c, const int32_t* ids, int n, int32_t* first_token) {
    if (!c || !ids) return fail(EE_EINVAL, "NULL argument");
    if (!c->weights) return fail(EE_ESTATE, "weights not loaded");
    if (c->prefilled || c->pos != 0) return fail(EE_ESTATE, "prefill needs a fresh or reset context");
    if (n <= 0) return fail(EE_EINVAL, "empty prompt");
    if (n > c->cfg.max_ctx) return fail(EE_ERANGE, "prompt longer than max_ctx");
    for (int i = 0; i < n; ++i)
        if (ids[i] < 0 || ids[i] >= c->cfg.vocab) return fail(EE_EINVAL, "prompt token out of range");
    c->started = true;
    cudaStream_t s = c->stream;
    int32_t* d_prompt = (int32_t*)(c->ws + c->lay.prompt);
    EE_CK(cudaMemcpyAsync(d_prompt, ids, 4 * (size_t)n, cudaMemcpyHostToDevice, s));
    CtlInputs in = base_inputs(c, nullptr);
    in.set_token = 1;
    in.in_tok = ids[0];
    in.prefill_n = n;
    in.prompt = d_prompt;
    EE_CK(launch_set_inputs(c->d_ctl, in, s));
    if (c->use_rows) {
        EE_TRY(rows_prefill(c, d_prompt, n));
    } else if (c->use_graphs) {
        EE_TRY(ensure_graphs(c));
        EE_CK(cudaGraphLaunch(c->g_prefill, s));
    } else {
        for (int i = 0; i < n; ++i) {
            bool pdl = false;
            EE_TRY(enqueue_layers(c, s, 0, c->cfg.n_layers, pdl));
            EE_CK(launch_prefill_advance(c->dm, 0, 0, false, s));
        }
        bool pdl = false;
        EE_TRY(enqueue_head(c, s, pdl));
        EE_CK(launch_prefill_end(c->dm, false, s));
    }
    EE_TRY(fetch_ctl(c));
    EE_TRY(device_error(c));
    c->pos = c->h_ctl->pos;
    if (c->pos != n) return fail(EE_EDEVICE, "prefill ended at an unexpected position");
    c->prefilled = true;
    c->repass_from = n;
    if (first_token) *first_token = c->h_ctl->token;
    return EE_OK;
}

int ee_decode_step(ee_ctx* c, int32_t input_token, const float* taus, int force, ee_step_result* out) {
    if (!c || !out) return fail(EE_EINVAL, "NULL argument");
    if (!c->prefilled) return fail(EE_ESTATE, "decode before prefill");
    if (input_token < -1 || input_token >= c->cfg.vocab) return fail(EE_EINVAL, "input token out of range");
    if (c->n_readouts > 0 && !taus) return fail(EE_EINVAL, "taus is NULL");
    if (force < 0 || force > 1 + c->n_readouts) return fail(EE_EINVAL, "bad force value");
    if (c->pos + 1 > c->cfg.max_ctx) return fail(EE_ERANGE, "position would pass max_ctx");
    cudaStream_t s = c->stream;
    CtlInputs in = base_inputs(c, taus);
    in.set_token = input_token >= 0;
    in.in_tok = input_token;
    in.force = force;
    EE_CK(launch_set_inputs(c->d_ctl, in, s));
    if (c->use_graphs) {
        EE_TRY(ensure_graphs(c));
        EE_CK(cudaGraphLaunch(c->g_step, s));
    } else {
        EE_TRY(eager_step(c));
    }
    EE_TRY(fetch_ctl(c));
    EE_TRY(device_error(c));
    const Ctl* h = c->h_ctl;
    std::memset(out, 0, sizeof(*out));
    out->token = h->token;
    out->exit_readout = h->exit_readout;
    out->exited = h->exit_readout >= 0;
    out->exit_layer = h->exit_readout >= 0 ? c->ro_layer[h->exit_readout] : c->cfg.n_layers;
    out->n_evaluated = h->n_evaluated;
    out->full_token = h->exit_readout >= 0 ? -1 : h->full_token;
    for (int r = 0; r < h->n_evaluated && r < kMaxReadouts; ++r) {
        out->gate_pass[r] = h->gate_pass[r];
        out->readout_token[r] = h->readout_token[r];
        out->confidence[r] = h->conf[r];
    }
    out->full_confidence = h->exit_readout >= 0 ? 0.f : h->full_conf;
    out->nucleus_member = in.nucleus_on && h->exit_readout < 0 ? h->nucleus_member : -1;
    out->nucleus_mass = out->nucleus_member >= 0 ? h->nucleus_mass : 0.f;
    c->pos = h->pos;
    return EE_OK;
}

int ee_decode_n(ee_ctx* c, int n, int32_t input_token, const float* taus, const int8_t* force_schedule,
                int32_t* tokens, int32_t* exit_readout, float* confidence, int where) {
    if (!c) return fail(EE_EINVAL, "NULL context");
    if (!c->prefilled) return fail(EE_ESTATE, "decode before prefill");
    if (n <= 0) return fail(EE_EINVAL, "n must be positive");
    if (input_token < -1 || input_token >= c->cfg.vocab) return fail(EE_EINVAL, "input token out of range");
    if (c->n_readouts > 0 && !taus) return fail(EE_EINVAL, "taus is NULL");
    if (where != EE_HOST && where != EE_DEVICE) return fail(EE_EINVAL, "where must be EE_HOST or EE_DEVICE");
    if (c->pos + n > c->cfg.max_ctx) return fail(EE_ERANGE, "steps would pass max_ctx");
    if (force_schedule)
        for (int i = 0; i < n; ++i)
            if (force_schedule[i] < 0 || force_schedule[i] > 1 + c->n_readouts)
                return fail(EE_EINVAL, "bad force schedule entry");
    cudaStream_t s = c->stream;
    int8_t* d_sched = (int8_t*)(c->ws + c->lay.sched);
    if (force_schedule) EE_CK(cudaMemcpyAsync(d_sched, force_schedule, (size_t)n, cudaMemcpyHostToDevice, s));
    int32_t* d_tok = (int32_t*)(c->ws + c->lay.out_tok);
    int32_t* d_exit = (int32_t*)(c->ws + c->lay.out_exit);
    float* d_conf = (float*)(c->ws + c->lay.out_conf);
    int32_t* o_tok = where == EE_DEVICE ? tokens : (tokens ? d_tok : nullptr);
    int32_t* o_exit = where == EE_DEVICE ? exit_readout : (exit_readout ? d_exit : nullptr);
    float* o_conf = where == EE_DEVICE ? confidence : (confidence ? d_conf : nullptr);
    // In runs of steps; with a re-pass period, each run ends where the next
    // periodic re-pass (Section 11) falls due.
    for (int done = 0; done < n;) {
        int len = n - done;
        if (c->repass_period > 0) len = std::min(len, std::max(1, c->repass_from + c->repass_period - c->pos));
        CtlInputs in = base_inputs(c, taus);
        in.set_token = done == 0 && input_token >= 0;
        in.in_tok = input_token;
        in.force = EE_FREE;
        in.n_steps = len;
        in.sched = force_schedule ? d_sched + done : nullptr;
        in.out_tokens = o_tok ? o_tok + done : nullptr;
        in.out_exit = o_exit ? o_exit + done : nullptr;
        in.out_conf = o_conf ? o_conf + done : nullptr;
        EE_CK(launch_set_inputs(c->d_ctl, in, s));
        if (c->use_graphs) {
            EE_TRY(ensure_graphs(c));
            EE_CK(cudaGraphLaunch(c->g_n, s));
        } else {
            for (int i = 0; i < len; ++i) EE_TRY(eager_step(c));
        }
        c->pos += len;
        done += len;
        if (c->repass_period > 0 && c->pos - c->repass_from >= c->repass_period) {
            EE_TRY(repass_range(c, c->repass_from, c->pos, nullptr));
            c->repass_from = c->pos;
        }
    }
    if (where == EE_HOST) {
        if (tokens) EE_CK(cudaMemcpyAsync(tokens, d_tok, 4 * (size_t)n, cudaMemcpyDeviceToHost, s));
        if (exit_readout) EE_CK(cudaMemcpyAsync(exit_readout, d_exit, 4 * (size_t)n, cudaMemcpyDeviceToHost, s));
        if (confidence) EE_CK(cudaMemcpyAsync(confidence, d_conf, 4 * (size_t)n, cudaMemcpyDeviceToHost, s));
        EE_TRY(fetch_ctl(c));
        EE_TRY(device_error(c));
        if (c->h_ctl->pos != c->pos) return fail(EE_EDEVICE, "device position out of step with the host");
    }
    return EE_OK;
}

int ee_calibrate(ee_ctx* c, const int32_t* ids, int n, float p_nuc, float* conf, int32_t* member, float* mass,
                 int where) {
    if (!c || !ids) return fail(EE_EINVAL, "NULL argument");
    if (!c->prefilled) return fail(EE_ESTATE, "calibration before prefill");
    if (c->n_readouts < 1) return fail(EE_ESTATE, "calibration needs a readout");
    if (n <= 0) return fail(EE_EINVAL, "n must be positive");
    if (!(p_nuc > 0.0f && p_nuc <= 1.0f)) return fail(EE_EINVAL, "p_nuc must lie in (0, 1]");
    if (where != EE_HOST && where != EE_DEVICE) return fail(EE_EINVAL, "where must be EE_HOST or EE_DEVICE");
    if (c->pos + n > c->cfg.max_ctx) return fail(EE_ERANGE, "steps would pass max_ctx");
    const int R = c->n_readouts;
    cudaStream_t s = c->stream;
    int32_t* d_ids = (int32_t*)(c->ws + c->lay.prompt);
    if (where == EE_HOST) {
        for (int i = 0; i < n; ++i)
            if (ids[i] < 0 || ids[i] >= c->cfg.vocab) return fail(EE_EINVAL, "token id out of range");
        EE_CK(cudaMemcpyAsync(d_ids, ids, 4 * (size_t)n, cudaMemcpyHostToDevice, s));
    } else {
        EE_CK(cudaMemcpyAsync(d_ids, ids, 4 * (size_t)n, cudaMemcpyDeviceToDevice, s));
    }
    float taus[kMaxReadouts];
    for (int r = 0; r < kMaxReadouts; ++r) taus[r] = 2.0f;
    CtlInputs in = base_inputs(c, taus);
    in.force = EE_FORCE_FULL;
    in.n_steps = n;
    in.set_token = 0;
    in.forced_in = d_ids;
    in.nucleus_on = 1;
    in.nucleus_p = p_nuc;
    float* d_conf = (float*)(c->ws + c->lay.out_conf_all);
    int32_t* d_member = (int32_t*)(c->ws + c->lay.out_member);
    float* d_mass = (float*)(c->ws + c->lay.out_mass);
    if (where == EE_DEVICE) {
        in.out_conf_all = conf;
        in.out_member = member;
        in.out_mass = mass;
    } else {
        in.out_conf_all = conf ? d_conf : nullptr;
        in.out_member = member ? d_member : nullptr;
        in.out_mass = mass ? d_mass : nullptr;
    }
    EE_CK(launch_set_inputs(c->d_ctl, in, s));
    // step 0's input: ids[0], read on the device
    EE_CK(cudaMemcpyAsync(&c->d_ctl->in_tok, d_ids, 4, cudaMemcpyDeviceToDevice, s));
    if (c->use_graphs) {
        EE_TRY(ensure_graphs(c));
        EE_CK(cudaGraphLaunch(c->g_n, s));
    } else {
        for (int i = 0; i < n; ++i) EE_TRY(eager_step(c));
    }
    c->pos += n;
    if (where == EE_HOST) {
        if (conf) EE_CK(cudaMemcpyAsync(conf, d_conf, 4 * (size_t)n * R, cudaMemcpyDeviceToHost, s));
        if (member) EE_CK(cudaMemcpyAsync(member, d_member, 4 * (size_t)n, cudaMemcpyDeviceToHost, s));
        if (mass) EE_CK(cudaMemcpyAsync(mass, d_mass, 4 * (size_t)n, cudaMemcpyDeviceToHost, s));
        EE_TRY(fetch_ctl(c));
        EE_TRY(device_error(c));
        if (c->h_ctl->pos != c->pos) return fail(EE_EDEVICE, "device position out of step with the host");
    }
    return EE_OK;
}

int ee_repass(ee_ctx* c, int32_t t0, int32_t t1, int32_t* n_repassed) {
    if (!c) return fail(EE_EINVAL, "NULL context");
    if (!c->prefilled) return fail(EE_ESTATE, "re-pass before prefill");
    if (t0 < 0 || t1 < t0 || t1 > c->pos) return fail(EE_ERANGE, "re-pass range outside [0, position]");
    int n = 0;
    EE_TRY(repass_range(c, t0, t1, &n));
    if (n_repassed) *n_repassed = n;
    return EE_OK;
}

int ee_flush_fills(ee_ctx* c) {
    if (!c) return fail(EE_EINVAL, "NULL context");
    if (!c->prefilled) return EE_OK;
    EE_TRY(flush_pending(c));
    EE_TRY(fetch_ctl(c));
    return device_error(c);
}

int ee_sync(ee_ctx* c) {
    if (!c) return fail(EE_EINVAL, "NULL context");
    EE_TRY(fetch_ctl(c));
    return device_error(c);
}

int ee_get_stats(ee_ctx* c, ee_stats* out) {
    if (!c || !out) return fail(EE_EINVAL, "NULL argument");
    EE_TRY(fetch_ctl(c));
    std::memset(out, 0, sizeof(*out));
    out->steps = c->h_ctl->steps;
    out->full_steps = c->h_ctl->full_steps;
    for (int r = 0; r < kMaxReadouts; ++r) out->exits[r] = c->h_ctl->exits[r];
    return EE_OK;
}

int ee_position(ee_ctx* c, int32_t* pos) {
    if (!c || !pos) return fail(EE_EINVAL, "NULL argument");
    *pos = c->pos;
    return EE_OK;
}

int ee_debug_read(ee_ctx* c, int what, int layer, int pos, void* host_dst, size_t bytes) {
    if (!c || !host_dst) return fail(EE_EINVAL, "NULL argument");
    const ee_model_config& cf = c->cfg;
    const size_t d = cf.d_model, V = cf.vocab, kd = (size_t)cf.n_kv_heads * cf.head_dim;
    const Layout& l = c->lay;
    EE_CK(cudaStreamSynchronize(c->stream));
    auto rd = [&](size_t off, size_t n) -> int {
        if (bytes != n) return fail(EE_EINVAL, "byte count does not match the requested item");
        EE_CK(cudaMemcpy(host_dst, c->ws + off, n, cudaMemcpyDeviceToHost));
        return EE_OK;
    };
    switch (what) {
        case EE_DBG_HIDDEN_READOUT:
            if (layer < 0 || layer >= c->n_readouts) return fail(EE_EINVAL, "bad readout index");
            return rd(l.hk + 4 * d * layer, 4 * d);
        case EE_DBG_READOUT_Y:
            if (layer < 0 || layer >= c->n_readouts) return fail(EE_EINVAL, "bad readout index");
            return rd(l.y + 4 * d * layer, 4 * d);
        case EE_DBG_HIDDEN_FINAL:
            return rd(l.h, 4 * d);
        case EE_DBG_READOUT_LOGITS:
            if (layer < 0 || layer >= c->n_readouts) return fail(EE_EINVAL, "bad readout index");
            return rd(l.logits_ro + 4 * V * layer, 4 * V);
        case EE_DBG_FINAL_LOGITS:
            return rd(l.logits_final, 4 * V);
        case EE_DBG_KV:
        case EE_DBG_KV_SRC: {
            if (layer < 0 || layer >= cf.n_layers || pos < 0 || pos >= cf.max_ctx)
                return fail(EE_EINVAL, "bad layer or position");
            if (what == EE_DBG_KV_SRC) return rd(l.kv_src + (size_t)layer * cf.max_ctx + pos, 1);
            if (bytes != 2 * 2 * kd) return fail(EE_EINVAL, "byte count does not match the requested item");
            int32_t page;
            EE_CK(cudaMemcpy(&page, c->ws + l.page_table + 4 * (size_t)(pos / cf.page_size), 4, cudaMemcpyDeviceToHost));
            const int slot = pos % cf.page_size;
            uint16_t* dst = (uint16_t*)host_dst;
            for (int g = 0; g < cf.n_kv_heads; ++g) {
                const size_t off = 2 * ((size_t)layer * l.kv_layer_stride +
                                        (((size_t)page * cf.n_kv_heads + g) * cf.page_size + slot) * cf.head_dim);
                EE_CK(cudaMemcpy(dst + g * cf.head_dim, c->ws + l.kpool + off, 2 * (size_t)cf.head_dim,
                                 cudaMemcpyDeviceToHost));
                EE_CK(cudaMemcpy(dst + kd + g * cf.head_dim, c->ws + l.vpool + off, 2 * (size_t)cf.head_dim,
                                 cudaMemcpyDeviceToHost));
            }
            return EE_OK;
        }
        default:
            return fail(EE_EINVAL, "unknown debug item");
    }
}

int ee_profile_kernels(ee_ctx* c, int iters, float* ms_out) {
    if (!c || !ms_out || iters <= 0) return fail(EE_EINVAL, "bad argument");
    if (!c->prefilled || c->n_readouts == 0) return fail(EE_ESTATE, "needs a prefilled context with a readout");
    if (c->pos >= c->cfg.max_ctx) return fail(EE_ERANGE, "no free position to profile at");
    const DevModel& m = c->dm;
    cudaStream_t s = c->stream;
    const int L = m.L;
    const int64_t d = m.d, F = m.F, AD = (int64_t)m.A * m.D;
    const int gq = gemv_grid(c, c->lay.n_units_qkv * 2, d), go = gemv_grid(c, d, AD);
    const int gu = gemv_grid(c, 2 * F, d), gd = gemv_grid(c, d, F), gr = gemv_grid(c, d, d);
    char* scratch = c->ws + c->lay.out_tok;  // int32 token + float p of the standalone vocab mode
    VocabArgs va = vocab_args(c, 2, 0, 0, 0);
    va.mode = 0;
    va.logits = nullptr;
    va.out_token = (int32_t*)scratch;
    va.out_p = (float*)(scratch + 4);
    cudaEvent_t e0, e1;
    EE_CK(cudaEventCreate(&e0));
    EE_CK(cudaEventCreate(&e1));
    int rc = EE_OK;
    for (int k = 0; k < EE_NUM_KERNELS && rc == EE_OK; ++k) {
        auto one = [&](int i) -> cudaError_t {
            const int j = i % L;
            switch (k) {
                case EE_KERNEL_QKV: return launch_qkv(m, j, 0, gq, gemv_whole(c, c->lay.n_units_qkv * 2, d), false, s);
                case EE_KERNEL_ATTN: return launch_attention_cluster(attn_args(c, j), m.D, c->attn_cluster, false, s);
                case EE_KERNEL_OPROJ: return launch_oproj(m, j, go, gemv_whole(c, d, AD), false, s);
                case EE_KERNEL_GATEUP: return launch_gateup(m, j, gu, gemv_whole(c, 2 * F, d), false, s);
                case EE_KERNEL_DOWN: return launch_down(m, j, gd, gemv_whole(c, d, F), false, s);
                case EE_KERNEL_READOUT:
                    return launch_readout(m, i % c->n_readouts, gr, gemv_whole(c, d, d), false, s);
                case EE_KERNEL_VOCAB: return enqueue_vocab(c, va, false, s);
                case EE_KERNEL_LAYERS:
                    if (!c->seg_ok) return cudaSuccess;
                    return launch_layers(m, c->seg, 0, c->ro_layer[0], 0, s);
                default: {
                    const int e = c->ro_layer[0];
                    if (e >= L) return cudaSuccess;
                    const int64_t rows = 2LL * m.KH * m.D;
                    const int gx = fill_grid_x(c, L - e);
                    return launch_kvfill(m, e, gx, gx == tile_count(rows) && gemv_whole(c, rows, m.d), false, s);
                }
            }
        };
        cudaError_t e = one(0);  // warm the launch path
        if (e == cudaSuccess) e = cudaEventRecord(e0, s);
        for (int i = 0; i < iters && e == cudaSuccess; ++i) e = one(i + 1);
        if (e == cudaSuccess) e = cudaEventRecord(e1, s);
        if (e == cudaSuccess) e = cudaEventSynchronize(e1);
        float ms = 0.f;
        if (e == cudaSuccess) e = cudaEventElapsedTime(&ms, e0, e1);
        if (e != cudaSuccess) rc = fail(EE_ECUDA, std::string("profile: ") + cudaGetErrorString(e));
        ms_out[k] = ms / iters;
    }
    cudaEventDestroy(e0);
    cudaEventDestroy(e1);
    return rc;
}

// ---------------------------------------------------------------- standalone ops

int ee_attention_scratch_bytes(int n_heads, int n_kv_heads, int head_dim, size_t* bytes) {
    if (!bytes || n_heads <= 0 || n_kv_heads <= 0 || (head_dim != 64 && head_dim != 128)) return fail(EE_EINVAL, "bad shape");
    *bytes = align_up(4 * (size_t)n_heads * kAttnMaxSplits * (head_dim + 2)) + align_up(4 * (size_t)n_kv_heads);
    return EE_OK;
}

int ee_attention_decode(const float* q, const uint16_t* k_pages, const uint16_t* v_pages, const int32_t* page_table,
                        int T, int n_heads, int n_kv_heads, int head_dim, int page_size, void* scratch,
                        size_t scratch_bytes, float* out, void* stream) {
    size_t need = 0;
    EE_TRY(ee_attention_scratch_bytes(n_heads, n_kv_heads, head_dim, &need));
    if (!q || !k_pages || !v_pages || !page_table || !scratch || !out) return fail(EE_EINVAL, "NULL argument");
    if (T <= 0) return fail(EE_EINVAL, "T must be positive");
    if (n_heads % n_kv_heads || n_heads / n_kv_heads > 8) return fail(EE_EINVAL, "bad head grouping");
    if (page_size <= 0) return fail(EE_EINVAL, "bad page size");
    if (scratch_bytes < need) return fail(EE_ENOMEM, "scratch too small");
    cudaStream_t s = (cudaStream_t)stream;
    char* sc = (char*)scratch;
    AttnArgs a{};
    a.q = q;
    a.kp = k_pages;
    a.vp = v_pages;
    a.page_table = page_table;
    a.ctl = nullptr;
    a.T = T;
    a.A = n_heads;
    a.KH = n_kv_heads;
    a.page_size = page_size;
    a.out = out;
    a.part = (float*)sc;
    a.ticket = (int*)(sc + align_up(4 * (size_t)n_heads * kAttnMaxSplits * (head_dim + 2)));
    EE_CK(cudaMemsetAsync(a.ticket, 0, 4 * (size_t)n_kv_heads, s));
    EE_CK(launch_attention(a, head_dim, false, s));
    return EE_OK;
}

int ee_vocab_scratch_bytes(int vocab, int d_model, size_t* bytes) {
    if (!bytes || vocab <= 1 || d_model < 256 || d_model % 8) return fail(EE_EINVAL, "bad shape");
    *bytes = align_up(4 * (size_t)kMaxVocabCtas * 8) + align_up(4);
    return EE_OK;
}

namespace {
int vocab_standalone(const float* x, const uint16_t* gain, const uint16_t* U, int vocab, int d_model, float eps,
                     void* scratch, size_t scratch_bytes, int32_t* out_token, float* out_p, float* out_sig,
                     float* logits, void* stream) {
    size_t need = 0;
    EE_TRY(ee_vocab_scratch_bytes(vocab, d_model, &need));
    if (!x || !gain || !U || !scratch || !out_token || (!out_p && !out_sig)) return fail(EE_EINVAL, "NULL argument");
    if (scratch_bytes < need) return fail(EE_ENOMEM, "scratch too small");
    int dev = 0, nsm = 0;
    EE_CK(cudaGetDevice(&dev));
    EE_CK(cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev));
    if (configure_kernels(d_model) != cudaSuccess) return fail(EE_ECUDA, "kernel configuration failed");
    cudaStream_t s = (cudaStream_t)stream;
    char* sc = (char*)scratch;
    VocabArgs v{};
    v.x = x;
    v.gain = gain;
    v.U = U;
    v.tiled = 0;
    v.V = vocab;
    v.d = d_model;
    v.eps = eps;
    v.logits = logits;
    v.logits_if_dbg = 0;
    v.part = (float*)sc;
    v.ticket = (int*)(sc + align_up(4 * (size_t)kMaxVocabCtas * 8));
    v.mode = 0;
    v.out_token = out_token;
    v.out_p = out_p;
    v.out_sig = out_sig;
    EE_CK(cudaMemsetAsync(v.ticket, 0, 4, s));
    EE_CK(launch_vocab(v, std::min(nsm, kMaxVocabCtas), false, s));
    return EE_OK;
}
}  // namespace

int ee_vocab_confidence(const float* x, const uint16_t* gain, const uint16_t* U, int vocab, int d_model, float eps,
                        void* scratch, size_t scratch_bytes, int32_t* out_token, float* out_p, float* logits,
                        void* stream) {
    if (!out_p) return fail(EE_EINVAL, "NULL argument");
    return vocab_standalone(x, gain, U, vocab, d_model, eps, scratch, scratch_bytes, out_token, out_p, nullptr,
                            logits, stream);
}

int ee_vocab_signals(const float* x, const uint16_t* gain, const uint16_t* U, int vocab, int d_model, float eps,
                     void* scratch, size_t scratch_bytes, int32_t* out_token, float* out_signals, float* logits,
                     void* stream) {
    if (!out_signals) return fail(EE_EINVAL, "NULL argument");
    return vocab_standalone(x, gain, U, vocab, d_model, eps, scratch, scratch_bytes, out_token, nullptr,
                            out_signals, logits, stream);
}

int ee_select_tau(const float* conf, int conf_stride, const int32_t* member, int n, float target, float* tau,
                  void* scratch, void* stream) {
    if (!conf || !member || !tau || !scratch) return fail(EE_EINVAL, "NULL argument");
    if (n < 1 || conf_stride < 1) return fail(EE_EINVAL, "n and conf_stride must be positive");
    if (!(target >= 0.0f && target <= 1.0f)) return fail(EE_EINVAL, "target must lie in [0, 1]");
    int dev = 0, nsm = 0;
    EE_CK(cudaGetDevice(&dev));
    EE_CK(cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev));
    EE_CK(launch_select_tau(conf, conf_stride, member, n, (double)target, tau, (int*)scratch, nsm,
                            (cudaStream_t)stream));
    return EE_OK;
}

}  // extern "C"
