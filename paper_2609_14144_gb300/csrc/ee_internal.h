// Internal structures shared by the sm_103a kernels (ee_kernels.cu) and the
// host engine (ee_engine.cu).  Not part of the public ABI.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "ee.h"

namespace ee {

constexpr int kMaxReadouts = EE_MAX_READOUTS;
constexpr int kGemvThreads = 512;   // 16 warps per CTA in the streaming GEMVs
constexpr int kAttnThreads = 256;   // 8 warps per CTA in split-K attention
constexpr int kAttnMinRows = 32;    // positions per attention split (at least)
constexpr int kAttnMaxSplits = 128; // splits per key-value head (at most)

// Bits of the device error word.
constexpr int kErrNanConfidence = 1;
constexpr int kErrTokenRange = 2;
constexpr int kErrPosition = 4;
constexpr int kErrShape = 8;  // a GEMV CTA would touch more tiles than it can hold
constexpr int kErrStall = 16; // a wait of the persistent layer kernel ran out of time

// Device-resident control block: everything a step reads or writes that is
// not a tensor, so one captured graph serves every step, tau and force.
struct Ctl {
    int32_t pos;          // position of the step's input token
    int32_t in_tok;       // input token of the next step
    int32_t force;        // EE_FREE / EE_FORCE_FULL / EE_FORCE_EXIT_AT(r)
    int32_t step;         // step index inside one ee_decode_n call
    int32_t n_steps;      // steps requested by ee_decode_n
    int32_t err;          // device error word (kErr* bits)
    int32_t dbg;          // 1: keep readout / final logits
    int32_t exit_readout; // readout that emitted this step, -1 = full depth
    int32_t token;        // emitted token of the last step
    int32_t full_token;   // LM head token of the last full step, else -1
    int32_t n_evaluated;  // readouts evaluated this step
    int32_t prefill_n;    // prompt length of the running prefill
    int32_t prefill_i;    // prompt index of the running prefill
    int32_t max_ctx;
    int32_t conf_kind;    // EE_CONF_*: the signal the gates compare with tau
    int32_t nucleus_on;   // 1: full steps check readout 0's token against the LM head's nucleus
    int32_t gate_pass[kMaxReadouts];
    int32_t readout_token[kMaxReadouts];
    float conf[kMaxReadouts];
    float tau[kMaxReadouts];
    float full_conf;
    float nucleus_p;        // share of probability the nucleus holds
    float nucleus_mass;     // LM head probability of the tokens above readout 0's token
    int32_t nucleus_member; // readout 0's token in the nucleus (1/0), -1 when not computed
    long long steps, full_steps, exits[kMaxReadouts];
    int32_t* out_tokens;   // per-step outputs of ee_decode_n (may be null)
    int32_t* out_exit;
    float* out_conf;
    const int8_t* sched;   // per-step force values (may be null)
    const int32_t* prompt; // prompt ids of the running prefill
    float* out_conf_all;   // [n_steps][n_readouts] every readout's signal (may be null)
    int32_t* out_member;   // [n_steps] nucleus_member per step (may be null)
    float* out_mass;       // [n_steps] nucleus_mass per step (may be null)
    const int32_t* forced_in; // [n_steps] teacher-forced inputs (null: the emitted token is fed back)
    int32_t pend_lo;          // positions below have no deferred (pending) KV entries
    int32_t pad_;
};

static_assert(sizeof(Ctl) == 368, "control block size is part of the host read-back accounting");

// Device pointers and shape, passed by value to every kernel.
struct DevModel {
    int L, d, A, KH, D, F, V, max_ctx, page_size, n_pages, qkv_bias, n_readouts;
    float eps;
    // Packed per-layer weights: layer j starts at layers + j * layer_stride.
    const uint16_t* layers;
    int64_t layer_stride;
    int64_t off_wqkv, off_bqkv, off_gattn, off_wo, off_gmlp, off_wgu, off_wd;
    const uint16_t* embed;
    const uint16_t* lm_head;
    const uint16_t* g_final;
    const uint16_t* ro_w[kMaxReadouts];
    const uint16_t* ro_b[kMaxReadouts];
    int ro_layer[kMaxReadouts];
    const float2* rope;           // [max_ctx][D/2] (cos, sin)
    uint16_t* kpool;              // [L][n_pages][KH][page_size][D]
    uint16_t* vpool;
    int64_t kv_layer_stride;      // elements per layer in a pool
    const int32_t* page_table;    // [n_pages]
    int8_t* kv_src;               // [L][max_ctx]
    float* h_exit;                // [max_ctx][d] residual each position exited with
    int16_t* exit_at;             // [max_ctx] first filled layer of an exited position
    float* h;                     // residual stream [d]
    float* q;                     // rotated queries [A*D]
    float* o;                     // attention output [A*D]
    float* a;                     // SwiGLU product [F]
    float* y;                     // readout outputs [R][d]
    float* hk;                    // residual seen by each readout [R][d]
    float* logits_ro;             // [R][V] (debug)
    float* logits_final;          // [V] (debug)
    float* gemv_part;             // cross-CTA tile partials: [CTA slot][2][32]
    unsigned* gemv_ticket;        // per-tile arrival counters
    int64_t gemv_ticket_stride;   // counters per fill layer in gemv_ticket
    float* attn_part;             // [A][kAttnMaxSplits][D + 2]
    int* attn_ticket;             // [KH]
    float* vocab_part;            // [grid][8]
    int* vocab_ticket;            // [1]
    Ctl* ctl;
};

// Arguments of the split-K attention kernel (engine and standalone op).
struct AttnArgs {
    const float* q;
    const uint16_t* kp;       // pool of this layer: [n_pages][KH][page_size][D]
    const uint16_t* vp;
    const int32_t* page_table;
    const Ctl* ctl;           // if set, T = ctl->pos + 1
    int T;
    int A, KH, page_size;
    float* out;
    float* part;
    int* ticket;
};

// Arguments of the vocabulary pass (readout / LM head / standalone).
struct VocabArgs {
    const float* x;           // residual-space input [d]
    const uint16_t* gain;     // final RMSNorm gain [d]
    const uint16_t* U;        // [V, d], tiled (engine) or row-major (standalone)
    int tiled;
    int V, d;
    float eps;
    float* logits;            // optional [V]
    int logits_if_dbg;        // write logits only when ctl->dbg is set
    float* part;
    int* ticket;
    int mode;                 // 0 standalone, 1 readout r, 2 LM head
    int r;
    Ctl* ctl;
    int32_t* out_token;
    float* out_p;
    float* out_sig;           // standalone: [3] p_max, margin, negative entropy (may be null)
    int has_cond;
    cudaGraphConditionalHandle cond;
};

// Per-call inputs of a graph launch.
struct CtlInputs {
    int set_token, in_tok, force, n_steps, dbg, prefill_n, conf_kind, nucleus_on;
    float nucleus_p;
    float tau[kMaxReadouts];
    const int8_t* sched;
    int32_t* out_tokens;
    int32_t* out_exit;
    float* out_conf;
    const int32_t* prompt;
    float* out_conf_all;
    int32_t* out_member;
    float* out_mass;
    const int32_t* forced_in;
};

// Launch helpers (ee_kernels.cu).  Each enqueues one kernel on `s`;
// `pdl` adds the programmatic-stream-serialisation attribute.
// `whole`: one CTA per tile, the tile staged in shared memory before the wait.
cudaError_t launch_qkv(const DevModel& m, int layer, int first, int grid, bool whole, bool pdl, cudaStream_t s);
cudaError_t launch_attention(const AttnArgs& a, int head_dim, bool pdl, cudaStream_t s);
// The engine's attention: one thread-block cluster of `cluster` CTAs per kv head.
cudaError_t launch_attention_cluster(const AttnArgs& a, int head_dim, int cluster, bool pdl, cudaStream_t s);
// Largest cluster size (16 or 8) the attention kernel can be resident with.
int attention_cluster_size(int head_dim, int n_kv_heads);
cudaError_t launch_oproj(const DevModel& m, int layer, int grid, bool whole, bool pdl, cudaStream_t s);
cudaError_t launch_gateup(const DevModel& m, int layer, int grid, bool whole, bool pdl, cudaStream_t s);
cudaError_t launch_down(const DevModel& m, int layer, int grid, bool whole, bool pdl, cudaStream_t s);
cudaError_t launch_readout(const DevModel& m, int r, int grid, bool whole, bool pdl, cudaStream_t s);
cudaError_t launch_vocab(const VocabArgs& v, int grid, bool pdl, cudaStream_t s);
cudaError_t launch_kvfill(const DevModel& m, int exit_layer, int grid_x, bool whole, bool pdl, cudaStream_t s);
// Deferred fill (EE_OPT_LAZY_FILL): an exit step only records its residual
// and exit layer; before a later step runs layers [j0, j1) every pending
// entry of those layers is filled (one read of their key/value weights).
cudaError_t launch_record_exit(const DevModel& m, int exit_layer, bool pdl, cudaStream_t s);
size_t fill_pending_smem(int d);
cudaError_t configure_fill_pending(int d);
cudaError_t launch_fill_pending(const DevModel& m, int j0, int j1, bool pdl, cudaStream_t s);
cudaError_t launch_step_end(const DevModel& m, int has_cond, cudaGraphConditionalHandle cond, bool pdl,
                            cudaStream_t s);
cudaError_t launch_prefill_advance(const DevModel& m, int has_cond, cudaGraphConditionalHandle cond, bool pdl,
                                   cudaStream_t s);
cudaError_t launch_prefill_end(const DevModel& m, bool pdl, cudaStream_t s);
cudaError_t launch_set_inputs(Ctl* c, const CtlInputs& in, cudaStream_t s);
// Section 4, step four threshold selection over n (confidence, acceptable)
// pairs; scratch: 2 device ints.
cudaError_t launch_select_tau(const float* conf, int stride, const int32_t* member, int n, double target, float* tau,
                              int* scratch, int n_sm, cudaStream_t s);

// Persistent layer-segment kernel (ee_persist.cu): one CTA per SM, warps
// 0..7 consume a shared-memory ring that warp 8 fills with cp.async.bulk.
constexpr int kSegConsumerWarps = 8;
constexpr int kSegThreads = 32 * (kSegConsumerWarps + 1);
constexpr int kSegChunk = 32768;   // bytes per ring stage: 32 rows x 512 bf16 columns
constexpr int kSegMaxSplits = 64;  // attention splits per kv head (at most; the O merge's lanes hold two each)
constexpr int kSegMaxGroup = 8;    // query heads per kv head (at most)
constexpr int kSegMaxSlots = 8;    // CTAs sharing one down tile, chunks of one O tile (at most)
// A value handed from one CTA to another inside a launch of the persistent
// layer kernel: the float's bits in the low word and its layer's tag in the
// high word, stored and loaded as one 64-bit word (observed whole).
using Tagged = unsigned long long;
// Bounds of the persistent kernel's waits, in SM clock cycles: a wait gives
// up after `stall` cycles; a waiting thread looks at the error word once
// every `check` cycles.
constexpr long long kSegStallCycles = 4000000000ll;  // about 2 s
constexpr long long kSegCheckCycles = 2000000ll;     // about 1 ms
struct SegPlan {
    int G;                  // CTAs (one per SM)
    int stages;             // ring stages
    int inflight;           // ring chunks a producer keeps in flight (at most)
    int max_pps;            // attention pages per split (at most)
    int max_splits;         // attention splits per kv head any step can use (at most)
    int rows_per_kv_chunk;  // cache positions per ring chunk
    int max_items;          // O / down-projection items per CTA (at most)
    int n_tiles[4], n_chunks[4], K[4];  // Q/K/V, O, gate/up, down
    // Values handed between CTAs, each a Tagged word (zero after ee_reset):
    Tagged* dpart;          // down-projection partials [tile][n_chunks][32]
    Tagged* opart;          // O-projection chunk partials [2][tile][n_chunks][32] (by the layer count's parity)
    Tagged* attn_part;      // [A][kSegMaxSplits][D + 4]: unnormalised o, max, sum per split
    Tagged* q;              // [A D] rotated queries
    Tagged* kvn;            // [2][KH D] the step's k and v (bf16 values)
    Tagged* a;              // [F] SwiGLU product
    unsigned* sync;         // [0] exit ticket (zero between launches), [1] layers run since ee_reset
    size_t smem;            // dynamic shared memory per CTA
    long long stall_cycles; // wait bounds (kSegStallCycles, kSegCheckCycles unless a test lowers them)
    long long check_cycles;
};
// Geometry and shared-memory plan for `m` on n_sm SMs (pointers left
// unset); false if the shape is outside what the kernel supports.
bool seg_plan(const DevModel& m, int n_sm, SegPlan& p);
cudaError_t configure_layers(size_t smem);
int layers_blocks_per_sm(size_t smem);
// Layers [j0, j1) of the step at ctl->pos; `first`: layer j0 takes the
// embedding of ctl->in_tok.  A cooperative launch of p.G CTAs.
cudaError_t launch_layers(const DevModel& m, const SegPlan& p, int j0, int j1, int first, cudaStream_t s);

// The vocabulary pass fed through a shared-memory ring (ee_persist.cu): one
// CTA per SM, same arguments and results as launch_vocab with a tiled U.
struct VocabRing {
    int G = 0, stages = 0;
    size_t smem = 0;
};
bool vocab_ring_plan(int d, int n_sm, VocabRing& vr);
cudaError_t configure_vocab_ring(size_t smem);
cudaError_t launch_vocab_ring(const VocabArgs& v, const VocabRing& vr, bool pdl, cudaStream_t s);

// Multi-position layer pass (ee_rows.cu): the prompt and the re-pass run
// each layer over up to kRowsMax positions at once, every weight byte read
// once per batch.  Products are tensor-core mma of the bf16 weights with the
// fp32 activations split into three bf16 parts (high, middle, low).
constexpr int kRowsMax = 256;            // positions per batch (the tcgen05 products' largest N)
// Row stride of a batch's activation parts: M rounded up to 16.
__host__ __device__ constexpr int x3_rows(int M) { return (M + 15) & ~15; }
constexpr int kRowsTargetUnits = 2432;   // (tile, K split) units a projection aims for: 152 SMs x 16 warps
struct RowsBuf {
    float* H;           // [kRowsMax][d] residual of each row
    uint16_t* x3;       // next product's input as three bf16 parts (high, x - high, the rest),
                        // chunk-major: [ldx / 8][3][x3_rows(M)][8] for a batch of M rows
    float* Q;           // [kRowsMax][A D] rotated queries
    float* part;        // split partials [S][M][n_rows padded to 32]
    int32_t* pos;       // [kRowsMax] positions of a prompt batch
    int64_t part_floats;
    int ldx;
    int umma;           // 1: projections on the tcgen05 tensor cores (ee_umma.cu), 0: warp-level mma
    int n_sm;
    int* err;           // device error word
};
// Shared-memory attributes of the multi-position pass's kernels.
cudaError_t configure_rows();
// Splits along K of an n_tiles x K projection for a batch of M rows.
int rows_splits(int64_t n_tiles, int K, int M);
// Floats of the partial buffer every batch size fits in.
int64_t rows_part_floats(int d, int A, int KH, int D, int F);
// Run layers over M rows at the device positions d_pos (ascending layer
// start): row i starts at layer start[i] (host, non-decreasing).  With ids,
// rows take the embedding of ids[i] and positions pos_base + i (written to
// d_pos); otherwise each row starts from h_exit at its position.  t_max:
// the largest position of the batch + 1.  kv_only: the last layer stops
// after its cache entries.
cudaError_t rows_pass(const DevModel& m, const RowsBuf& b, const int* start, int M, int32_t* d_pos,
                      const int32_t* ids, int pos_base, int t_max, bool kv_only, cudaStream_t s);
// tcgen05 projections of the multi-position pass (ee_umma.cu): available on
// this device (tensor-map encoding and the kernel's shared memory), the K
// splits for n_sm SMs, and one projection into part[S][M][Np] (the layout of
// the warp-level path).
bool umma_available();
int umma_splits(int64_t n_tiles, int K, int n_sm);
cudaError_t launch_mm_umma(const uint16_t* W, int64_t n_rows, int K, const uint16_t* x3, int M, int S, float* part,
                           int Np, int* err, cudaStream_t s);
// After a batched prompt: the control block as the per-position prefill
// leaves it before its LM head (position n).
cudaError_t launch_rows_prefill_done(const DevModel& m, int n, cudaStream_t s);

// Record `msg` as the calling thread's last error and return `code`.
int set_last_error(int code, const char* msg);

// Dynamic shared memory each GEMV kernel asks for, given the largest K.
size_t gemv_smem_bytes(int kmax);
cudaError_t configure_kernels(int kmax);

// Geometry of the tiled weight layout (rows grouped by 32, see ee_kernels.cu).
constexpr int kTileRows = 32;
constexpr int kGemvSlotTiles = 8;   // tiles one GEMV CTA may touch
constexpr int kGemvMaxSmem = 227 * 1024;  // dynamic shared memory a GEMV CTA may use
inline int64_t tile_count(int64_t rows) { return (rows + kTileRows - 1) / kTileRows; }
inline int64_t tiled_elems(int64_t rows, int64_t K) { return tile_count(rows) * kTileRows * K; }

}  // namespace ee
