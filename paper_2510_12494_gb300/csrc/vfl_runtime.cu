// Host runtime of libvfl: context, workspace layout, channel rings, the
// per-phase enqueue logic and the exported C ABI (include/vfl.h).
//
// Mapping to the paper (arxiv 2510.12494):
//  - Sec. 3 / Eq. 1-2: split forward, loss, cut-layer gradient exchange, SGD.
//  - Algorithm 1: vfl_passive_forward = publisher phase, vfl_active_step =
//    subscriber phase, vfl_passive_backward = backward phase.
//  - Sec. 4.1 channels keyed by batch id with bounded buffers: here HBM rings of
//    S+1 slots with a header {k, batch, version}, written by the kernel that
//    writes the payload last and checked by the first kernel that reads it; a
//    CUDA event per publish orders the subscriber's stream after the publisher's.
//  - App. D (Assumption 4, theorem): the gradient applied at step k was
//    computed with weights of version k - tau(k); updates apply in step order.
//    Each party keeps its S+1 most recent weight versions in a ring.
//  - Sec. 4.1 waiting deadline / buffer overflow: a dropped step trains nothing
//    (both parties copy version k to k+1) and hands its batch to the next step.
//  - Sec. 4.1 / Eq. 5 (ps_dt0 > 0): one replica of each party's parameters per
//    worker, each worker's steps chained on its own stream pair, the replicas
//    averaged after the epochs Eq. 5 selects.
#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <limits>
#include <map>
#include <utility>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <string>
#include <vector>

#include "vfl_fused.cuh"
#include "vfl_kernels.cuh"
#include "vfl_tc.cuh"

using namespace vfl;

namespace {

constexpr int kMaxWorkers = 16;
constexpr int kMaxSlots = 16;
constexpr int kEvPool = 64;
constexpr int kMaxIoSlots = kMaxSlots + kMaxWorkers + 2;   // staging ring: S + W + 2 slots
constexpr int kLossCap = 4096;
constexpr int kInfoRing = 64;   // per-step host records (batch, drop) of the steps in flight

thread_local std::string g_global_err;

// Kernel classes for launch accounting and per-class CUDA-event timing.
enum KClass : int {
    K_SIMT_FWD, K_SIMT_DX, K_SIMT_DW, K_TC_FWD, K_TC_DX, K_TC_DW,
    K_LOSS, K_DP, K_MASK, K_SGD, K_HEADER, K_CAST,
    K_FUSED_PFWD, K_FUSED_ACTIVE, K_FUSED_PBWD, K_FUSED_UPDATE, K_HEAD, K_PS_AVG, K_TC_DW_SGD, K_TC_CHAIN, K_NCLASS
};
const char* const kClassNames[K_NCLASS] = {
    "gemm_simt_fwd", "gemm_simt_dx", "gemm_simt_dw", "gemm_tc_fwd", "gemm_tc_dx", "gemm_tc_dw",
    "loss", "dp_clip_noise", "relu_mask", "sgd", "channel_header", "cast",
    "fused_passive_fwd", "fused_active_step", "fused_passive_bwd", "fused_update", "head_loss",
    "ps_average", "gemm_tc_dw_sgd", "gemm_tc_chain"};

struct ProfRec {
    int cls;
    double flops, bytes;
    cudaEvent_t e0, e1;
};
struct ProfAgg {
    long long n = 0;
    double ms = 0, flops = 0, bytes = 0;
};

inline long long ld8(long long x) { return (x + 7) / 8 * 8; }
// Row stride of the bf16 dataset and weight copies: whole 128-byte lines, so that every row the tensor-core
// GEMMs load with TMA starts on a line (rows that straddle lines cost the loads about a third more).
inline long long ld64(long long x) { return (x + 63) / 64 * 64; }

struct Layer {
    int party = 0, idx = 0, in = 0, out = 0;
    long long in_ld = 0;                  // leading dim of the compute copy of W
    float* W = nullptr;                   // fp32 master [out, in]
    float* b = nullptr;                   // fp32 master [out]
    float* Wr[kMaxWorkers] = {};          // parameter-server mode: replica w's master (Wr[0] = W)
    float* br[kMaxWorkers] = {};
    void* cW[kMaxSlots] = {};             // version copies [out, in_ld], compute dtype
    float* cb[kMaxSlots] = {};            // version copies of b, fp32
    float* pW[kMaxWorkers] = {};          // split-K partial dW [nsplit][out*in]
    float* pb[kMaxWorkers] = {};          // partial db [nsplit][out]
    int nsplit = 1;                       // weight-gradient partials
    int nsplit_b = 1;                     // bias-gradient partials
    int kchunk = 0;
    bool tc_dw = false;                   // dW, db on the tensor-core cluster kernel (one reduced partial)
    bool sgd_in_dw = false;               // ... which also applies this layer's SGD step
    float* dw_ws[kMaxWorkers] = {};       // ... and exchanges its partial tiles through this workspace
    long long dw_ws_floats = 0;
};

// Bump allocator over the caller's workspace (dry run when base == nullptr).
struct Carver {
    char* base;
    unsigned long long off = 0;
    explicit Carver(void* b) : base(static_cast<char*>(b)) {}
    void* take(unsigned long long bytes) {
        off = (off + 255) / 256 * 256;
        void* p = base ? base + off : nullptr;
        off += bytes;
        return p;
    }
};

}  // namespace

struct vfl_ctx {
    vfl_config cfg{};
    long long n_rows = 0;
    int S1 = 1;                 // slots = staleness + 1 (parameter-server mode: one per worker)
    int W = 1;                  // workers per party
    int esz = 4;                // bytes per compute element
    int bf16 = 0;
    int nb = 1;                 // steps per epoch
    std::string err;
    long long launches = 0;
    bool broken = false;

    std::vector<Layer> P, A, T;   // passive bottom, active bottom, top

    // device buffers
    void* Xp = nullptr; void* Xa = nullptr; int* Y = nullptr;
    long long ldxp = 0, ldxa = 0;
    float* stage_p = nullptr;                    // fp32 rows on their way into the dataset (vfl_load_data)
    float* stage_a = nullptr;
    std::vector<void*> act_p[kMaxSlots];          // per slot, per passive layer [B, ld8(out)]
    std::vector<void*> dpre_p[kMaxWorkers];       // per worker, per passive layer
    std::vector<void*> act_a[kMaxWorkers], dpre_a[kMaxWorkers];
    std::vector<void*> act_t[kMaxWorkers], dpre_t[kMaxWorkers];  // top hidden layers
    float* logits[kMaxWorkers] = {};
    float* ds[kMaxWorkers] = {};
    float* dzp32[kMaxWorkers] = {};
    void* grad[kMaxSlots] = {};
    void* emb_pub[kMaxSlots] = {};      // DP on the embedding: the published (noisy) payload per slot
    float* emb_c[kMaxSlots] = {};       // and its per-row clip factors [B], for the passive backward
    ChannelHeader* emb_hdr = nullptr;   // [S1]
    ChannelHeader* grad_hdr = nullptr;  // [S1]
    float* losses = nullptr;            // [kLossCap]
    int* status = nullptr;
    float* scratch_f32 = nullptr;       // for taps [B * max width]
    unsigned long long ws_bytes = 0;

    // fused one-launch-per-phase path (narrow fp32 models)
    bool fused = false;
    int f_act_ld = 0, f_wp = 0, f_wa = 0;       // smem row stride, weight-stage floats per party
    float* f_rowloss[kMaxWorkers] = {};         // per worker: per-row loss [B]
    float* f_zpc[kMaxWorkers] = {};             // per worker: z^p rows consumed by the step [B, ld8(e_p)]

    // parameter-server mode (Sec. 4.1, Eq. 5): replicas per worker, averaged per Eq. 5
    bool psmode = false;
    PsAvgLayer* ps_tab = nullptr;               // device table: P's layers, then A's, then T's
    long long ps_total[2] = {};                 // flat parameter counts: passive, active (f_a and g)
    cudaEvent_t ev_pavg[kEvPool] = {}, ev_aavg[kEvPool] = {};   // per aggregation step: averaging done

    // bf16 path: weight-gradient kernels that also apply the SGD step (one worker stream per party)
    bool sgd_in_dw = false;

    // bf16 path: g's output layer and the loss in one launch (narrow output over a narrow hidden layer)
    bool head = false;
    bool chain = false;                           // bf16 bottom models forward as one layer-chain launch
    int* h_counter = nullptr;                   // per worker: blocks finished
    float* h_blk_loss[kMaxWorkers] = {};        // per worker: per-block loss sums

    // streams / events
    cudaStream_t ps[kMaxWorkers] = {};
    cudaStream_t as[kMaxWorkers] = {};
    cudaEvent_t ev_pver[kEvPool] = {}, ev_aver[kEvPool] = {}, ev_emb[kEvPool] = {}, ev_grad[kEvPool] = {};

    // host-resident data (vfl_bind_host_data): each step reads its rows into slot k mod io_R of a
    // device staging ring on the caller's I/O stream; the loss kernels also write the host ring
    bool hio = false;
    const float* h_xp = nullptr;                // device views of the bound arrays (fp32 features)
    const float* h_xa = nullptr;
    const void* hv_xp = nullptr;                // the same views, any feature dtype
    const void* hv_xa = nullptr;
    const int32_t* h_y = nullptr;
    int h_esz = 4;                              // element bytes of the bound features (4 fp32, 2 bf16,
                                                // 0 bit-packed words)
    // page-locked host rows already in the slot layout (the compute dtype, no padding columns): staged by
    // the copy engines from these host addresses instead of by a kernel
    bool h_copy = false;
    const char* hc_xp = nullptr;
    const char* hc_xa = nullptr;
    const int32_t* hc_y = nullptr;
    float* h_loss = nullptr;
    long long h_loss_cap = 0;
    int io_R = 0;
    void* io_xp[kMaxIoSlots] = {};
    void* io_xa[kMaxIoSlots] = {};
    int* io_y[kMaxIoSlots] = {};
    cudaStream_t io = nullptr;
    cudaEvent_t ev_staged[kEvPool] = {};

    // per-launch timing (vfl_profile)
    bool prof_on = false;
    std::vector<ProfRec> prof;
    std::vector<cudaEvent_t> ev_spare;
    ProfAgg agg[K_NCLASS];

    // host-side ordering state
    long long n_fwd = 0, n_act = 0, n_bwd = 0;
    long long n_drops = 0;                      // dropped steps among those published
    long long x_emb = 0, x_grad = 0;            // payload bytes published through the two channels
    long long step_id[kInfoRing];               // per step k (slot k mod kInfoRing): its index,
    long long step_batch[kInfoRing];            // batch id,
    long long step_trained[kInfoRing];          // batches trained before it,
    unsigned char step_drop[kInfoRing] = {};    // dropped (waiting deadline)
    int fwd_version[kMaxSlots] = {};
    long long slot_step_p[kMaxSlots];
    long long grad_step[kMaxSlots];
    long long last_act_step[kMaxWorkers];
    bool started = false;
    // every weight version <= ordered_floor is already ordered before all further work on the
    // context's streams (the context was idle, or a graph replay ended with every stream waiting on
    // it), so waits on the events that produced those versions are skipped -- those events may have
    // been recorded inside a graph capture, where they cannot be waited on from outside
    long long ordered_floor = -1;

    // graph capture of the fused path: the kernel node of each (phase, step), so that the edges a
    // consumer only needs at a later point of its run become programmatic (see vfl_graph_capture)
    bool capturing = false;
    bool direct_pdl = true;     // programmatic launches outside graphs (VFL_DISABLE_DIRECT_PDL turns them off)
    // uniform dependency order (vfl_set_order): every step waits for the previous step's updates and is
    // published after the previous backward, whatever its staleness, so that windows of steps have one
    // graph shape (vfl_graph_update); the arithmetic, with its stale versions, is unchanged
    bool uniform = false;
    // vfl_train_epoch in the uniform order: one epoch graph per first worker, updated in place every epoch
    vfl_graph* epoch_graph[kMaxWorkers] = {};
    std::map<std::pair<int, long long>, cudaGraphNode_t> cap_nodes;

    vfl_status fail(vfl_status st, const char* fmt, ...) {
        char buf[512];
        va_list ap;
        va_start(ap, fmt);
        vsnprintf(buf, sizeof buf, fmt, ap);
        va_end(ap);
        err = buf;
        if (st == VFL_E_CUDA) broken = true;
        return st;
    }
    vfl_status cuda(cudaError_t e, const char* what, int line) {
        return fail(VFL_E_CUDA, "%s failed (line %d): %s", what, line, cudaGetErrorString(e));
    }
    // Batch of step k: (k - drops before k) mod nb, recorded when the step is published.
    long long batch_of(long long k) const {
        const int i = (int)(k % kInfoRing);
        return step_id[i] == k ? step_batch[i] : (k - n_drops) % nb;
    }
    bool dropped(long long k) const {
        const int i = (int)(k % kInfoRing);
        return step_id[i] == k && step_drop[i];
    }
    int batch_rows(long long k, long long* r0) const {
        const long long j = batch_of(k);
        *r0 = j * cfg.batch;
        return (int)std::min<long long>(cfg.batch, n_rows - *r0);
    }
};

// Host-side ordering state of a context (saved around graph capture).
struct HostState {
    long long n_fwd, n_act, n_bwd, n_drops, x_emb, x_grad;
    long long step_id[kInfoRing], step_batch[kInfoRing], step_trained[kInfoRing];
    unsigned char step_drop[kInfoRing];
    int fwd_version[kMaxSlots];
    long long slot_step_p[kMaxSlots], grad_step[kMaxSlots], last_act_step[kMaxWorkers];
    bool started;
    long long launches;
};

static HostState save_state(const vfl_ctx* c) {
    HostState h;
    h.n_fwd = c->n_fwd;
    h.n_act = c->n_act;
    h.n_bwd = c->n_bwd;
    h.n_drops = c->n_drops;
    h.x_emb = c->x_emb;
    h.x_grad = c->x_grad;
    std::memcpy(h.step_id, c->step_id, sizeof h.step_id);
    std::memcpy(h.step_batch, c->step_batch, sizeof h.step_batch);
    std::memcpy(h.step_trained, c->step_trained, sizeof h.step_trained);
    std::memcpy(h.step_drop, c->step_drop, sizeof h.step_drop);
    std::memcpy(h.fwd_version, c->fwd_version, sizeof h.fwd_version);
    std::memcpy(h.slot_step_p, c->slot_step_p, sizeof h.slot_step_p);
    std::memcpy(h.grad_step, c->grad_step, sizeof h.grad_step);
    std::memcpy(h.last_act_step, c->last_act_step, sizeof h.last_act_step);
    h.started = c->started;
    h.launches = c->launches;
    return h;
}

static void load_state(vfl_ctx* c, const HostState& h) {
    c->n_fwd = h.n_fwd;
    c->n_act = h.n_act;
    c->n_bwd = h.n_bwd;
    c->n_drops = h.n_drops;
    c->x_emb = h.x_emb;
    c->x_grad = h.x_grad;
    std::memcpy(c->step_id, h.step_id, sizeof h.step_id);
    std::memcpy(c->step_batch, h.step_batch, sizeof h.step_batch);
    std::memcpy(c->step_trained, h.step_trained, sizeof h.step_trained);
    std::memcpy(c->step_drop, h.step_drop, sizeof h.step_drop);
    std::memcpy(c->fwd_version, h.fwd_version, sizeof h.fwd_version);
    std::memcpy(c->slot_step_p, h.slot_step_p, sizeof h.slot_step_p);
    std::memcpy(c->grad_step, h.grad_step, sizeof h.grad_step);
    std::memcpy(c->last_act_step, h.last_act_step, sizeof h.last_act_step);
    c->started = h.started;
    c->launches = h.launches;
}

struct vfl_graph {
    vfl_ctx* ctx;
    cudaGraphExec_t exec;
    long long k0, n;
    long long drops0;          // drop count the captured steps' batches start from
    HostState after;           // host state once the captured steps have run
    long long launches;        // kernels per replay
    bool hio;                  // captured with host data bound (its copies are part of the graph)
    cudaEvent_t fork, join[2 * kMaxWorkers + 1];
};

#define TRY(x)                          \
    do {                                \
        vfl_status st_ = (x);           \
        if (st_ != VFL_OK) return st_;  \
    } while (0)

#define CK(call)                                                     \
    do {                                                             \
        cudaError_t e_ = (call);                                     \
        if (e_ != cudaSuccess) return ctx->cuda(e_, #call, __LINE__); \
    } while (0)

namespace {

cudaEvent_t spare_event(vfl_ctx* ctx) {
    if (!ctx->ev_spare.empty()) {
        cudaEvent_t e = ctx->ev_spare.back();
        ctx->ev_spare.pop_back();
        return e;
    }
    cudaEvent_t e = nullptr;
    if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
    return e;
}

// Opens a profiled launch: records the start event when profiling is on.
// Under stream capture the record is made external, so that it becomes a graph node recording
// the event when the graph runs (a plain record would only order the capture's streams); outside
// a capture the flag is not accepted.  A failed record is cleared from the last-error state (it
// must not fail the launch it brackets) and drops the timing record.
bool prof_record(cudaEvent_t e, cudaStream_t s) {
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    if (cudaStreamIsCapturing(s, &cs) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    const unsigned flags = cs == cudaStreamCaptureStatusActive ? cudaEventRecordExternal : cudaEventRecordDefault;
    if (cudaEventRecordWithFlags(e, s, flags) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    return true;
}

bool prof_begin(vfl_ctx* ctx, ProfRec* r, int cls, double flops, double bytes, cudaStream_t s) {
    ++ctx->launches;
    if (!ctx->prof_on) return false;
    r->cls = cls;
    r->flops = flops;
    r->bytes = bytes;
    r->e0 = spare_event(ctx);
    r->e1 = spare_event(ctx);
    if (!r->e0 || !r->e1) return false;
    return prof_record(r->e0, s);
}

void prof_end(vfl_ctx* ctx, ProfRec* r, bool on, cudaStream_t s) {
    if (!on) return;
    if (prof_record(r->e1, s)) ctx->prof.push_back(*r);
}

}  // namespace

// Launch `call` (returning cudaError_t) on stream s as kernel class cls with
// the given algorithmic flops / bytes.
#define PLAUNCH(cls, flops, bytes, s, call)                              \
    do {                                                                 \
        ProfRec pr_;                                                     \
        const bool on_ = prof_begin(ctx, &pr_, (cls), (flops), (bytes), (s)); \
        cudaError_t e_ = (call);                                         \
        if (e_ != cudaSuccess) return ctx->cuda(e_, #call, __LINE__);    \
        prof_end(ctx, &pr_, on_, (s));                                   \
    } while (0)

namespace {

vfl_status check_config(const vfl_config* c, long long n_rows, std::string* why) {
    char buf[256];
    auto bad = [&](const char* m) { *why = m; return VFL_E_INVAL; };
    if (!c) return bad("null config");
    if (n_rows < 1) return bad("n_rows must be >= 1");
    if (c->d_passive < 1 || c->d_active < 1) return bad("feature dims must be >= 1");
    if (c->n_passive < 1 || c->n_passive > VFL_MAX_LAYERS || c->n_active < 1 || c->n_active > VFL_MAX_LAYERS ||
        c->n_top < 1 || c->n_top > VFL_MAX_LAYERS)
        return bad("layer counts must be in [1, 8]");
    for (int i = 0; i < c->n_passive; ++i) if (c->passive_out[i] < 1) return bad("passive width < 1");
    for (int i = 0; i < c->n_active; ++i) if (c->active_out[i] < 1) return bad("active width < 1");
    for (int i = 0; i < c->n_top; ++i) if (c->top_out[i] < 1) return bad("top width < 1");
    const int n_out = c->top_out[c->n_top - 1];
    if (c->loss == VFL_LOSS_BCE) {
        if (n_out != 1) return bad("BCE needs n_out == 1");
    } else if (c->loss == VFL_LOSS_CE) {
        if (n_out < 2) return bad("CE needs n_out >= 2");
    } else {
        return bad("unknown loss");
    }
    if (c->dtype != VFL_FP32 && c->dtype != VFL_BF16) return bad("unknown dtype");
    if (c->batch < 1) return bad("batch must be >= 1");
    if (c->staleness < 0 || c->staleness + 1 > kMaxSlots) return bad("staleness must be in [0, 15]");
    if (c->workers < 1 || c->workers > kMaxWorkers) return bad("workers must be in [1, 16]");
    if (c->staleness + 1 + c->workers + 2 > kEvPool) return bad("staleness + workers too large");
    if (!(c->lr >= 0.f)) return bad("lr must be >= 0");
    if (c->dp_clip < 0.f || c->dp_sigma < 0.f) return bad("dp_clip / dp_sigma must be >= 0");
    if (c->dp_target != VFL_DP_GRAD && c->dp_target != VFL_DP_EMB) return bad("unknown dp_target");
    if (c->ps_dt0 < 0) return bad("ps_dt0 must be >= 0");
    if (c->ps_dt0 > 0 && c->staleness != 0)
        return bad("the parameter-server mode reads each replica's latest version: staleness must be 0");
    if (c->n_active + c->n_top > kMaxSgdLayers || c->n_passive > kMaxSgdLayers) return bad("too many layers");
    (void)buf;
    return VFL_OK;
}

// Split-K factor of a weight-gradient GEMM reducing over B rows.
void choose_split(Layer& L, int B) {
    const long long tiles = (long long)((L.out + 63) / 64) * ((L.in + 63) / 64);
    long long ns = std::max<long long>(1, 2 * 152 / std::max<long long>(1, tiles));
    ns = std::min<long long>(ns, std::max(1, B / 64));
    ns = std::min<long long>(ns, 32);
    L.kchunk = (int)(((B + ns - 1) / ns + 15) / 16 * 16);
    L.nsplit = (B + L.kchunk - 1) / L.kchunk;
}

// The fused path serves fp32 models whose every width fits one shared-memory
// row tile, without DP.
bool fused_eligible(const vfl_config& c) {
    if (c.dtype != VFL_FP32 || (c.dp_clip > 0.f && c.dp_target != VFL_DP_EMB)) return false;
    if (c.d_passive > kFusedMaxWidth || c.d_active > kFusedMaxWidth) return false;
    for (int i = 0; i < c.n_passive; ++i) if (c.passive_out[i] > kFusedMaxWidth) return false;
    for (int i = 0; i < c.n_active; ++i) if (c.active_out[i] > kFusedMaxWidth) return false;
    for (int i = 0; i < c.n_top; ++i) if (c.top_out[i] > kFusedMaxWidth) return false;
    if (c.active_out[c.n_active - 1] + c.passive_out[c.n_passive - 1] > kFusedMaxWidth) return false;
    if (c.n_active + c.n_top > kFusedMaxLayers) return false;
    // z^p lands in the top's input tile after z^a's 8-column blocks, by 16-byte copies
    if (c.active_out[c.n_active - 1] % 8 != 0 || c.passive_out[c.n_passive - 1] % 4 != 0) return false;
    return true;
}

// The bf16 path folds g's output layer and the loss into one kernel when g has a hidden layer
// of at most kHeadMaxK (a multiple of 8) units and at most kHeadMaxOut outputs.
bool head_eligible(const vfl_config& c) {
    if (c.dtype != VFL_BF16 || c.n_top < 2) return false;
    const int K = c.top_out[c.n_top - 2], n_out = c.top_out[c.n_top - 1];
    return n_out <= kHeadMaxOut && K >= 8 && K <= kHeadMaxK && K % 8 == 0;
}

// Shared-memory layout of the weights one fused launch stages: layers
// [w_from, n) get W and b.  Returns the floats used.
int fused_weight_layout(FusedLayerArgs* L, int n, int w_from) {
    int off = 0;
    for (int l = 0; l < n; ++l) {
        L[l].ws_ld = fused_w_stride(L[l].in_ld);
        L[l].ws_off = -1;
        if (l >= w_from) {
            L[l].ws_off = off;
            off += (int)fused_layer_floats(L[l].out, L[l].in_ld);
        }
    }
    return off;
}

void build_layers(vfl_ctx* ctx) {
    const vfl_config& c = ctx->cfg;
    auto mk = [&](std::vector<Layer>& v, int party, int n, const int32_t* outs, int d_in) {
        v.clear();
        for (int l = 0; l < n; ++l) {
            Layer L;
            L.party = party;
            L.idx = l;
            L.in = d_in;
            L.out = outs[l];
            L.in_ld = c.dtype == VFL_BF16 ? ld64(d_in) : ld8(d_in);
            choose_split(L, c.batch);
            L.nsplit_b = L.nsplit;
            if (ctx->fused) {
                L.nsplit = 1;
                L.kchunk = c.batch;
            }
            v.push_back(L);
            d_in = outs[l];
        }
    };
    mk(ctx->P, 0, c.n_passive, c.passive_out, c.d_passive);
    mk(ctx->A, 1, c.n_active, c.active_out, c.d_active);
    mk(ctx->T, 2, c.n_top, c.top_out, c.active_out[c.n_active - 1] + c.passive_out[c.n_passive - 1]);
    if (c.dtype == VFL_BF16) {
        const int ea = ctx->A.back().out;
        for (auto* v : {&ctx->P, &ctx->A, &ctx->T})
            for (size_t l = 0; l < v->size(); ++l) {
                Layer& L = (*v)[l];
                const bool last_top = v == &ctx->T && l + 1 == v->size();
                const bool concat = v == &ctx->T && l == 0;
                if (!last_top && tc_shape_dw(L.out, L.in, concat, ea)) {
                    // the cluster kernel reduces the batch: one gradient, its bias column sums and, with one
                    // worker stream per party, the SGD step (a step's first such kernel waits for the party's
                    // previous update; with several workers that wait would hold every weight-gradient kernel
                    // of the step back, so there the SGD stays a separate launch behind them)
                    L.tc_dw = true;
                    tc_choose_split(L.out, L.in, c.batch, &L.nsplit, &L.kchunk);
                    L.nsplit_b = 1;
                    L.sgd_in_dw = ctx->W == 1;
                    ctx->sgd_in_dw = ctx->sgd_in_dw || L.sgd_in_dw;
                }
            }
    }
    if (ctx->fused) {
        int maxw = std::max(c.d_passive, c.d_active);
        ctx->f_wp = ctx->f_wa = 0;
        for (const Layer& L : ctx->P) maxw = std::max(maxw, std::max(L.in, L.out));
        for (auto* v : {&ctx->A, &ctx->T})
            for (const Layer& L : *v) maxw = std::max(maxw, std::max(L.in, L.out));
        ctx->f_act_ld = fused_act_stride(ld8(maxw));
        // staged weights per launch (row-major W): every layer of f_p for the forward, every layer of
        // f_a and g for the active step, f_p's layers after the first for the backward
        long long w_pf = 0, w_pb = 0, w_a = 0;
        for (size_t l = 0; l < ctx->P.size(); ++l) {
            const long long w = fused_layer_floats(ctx->P[l].out, ctx->P[l].in_ld);
            w_pf += w;
            if (l > 0) w_pb += w;
        }
        for (auto* v : {&ctx->A, &ctx->T})
            for (const Layer& L : *v) w_a += fused_layer_floats(L.out, L.in_ld);
        ctx->f_wp = (int)std::max(w_pf, w_pb);
        ctx->f_wa = (int)w_a;
        const size_t sa = fused_smem_active(ctx->f_wa, ctx->f_act_ld, (int)ctx->A.size(), (int)ctx->T.size());
        const size_t sp = fused_smem_pbwd((int)w_pb, ctx->f_act_ld, (int)ctx->P.size());
        const size_t sf = fused_smem_fwd((int)w_pf, ctx->f_act_ld);
        if (std::max(sa, std::max(sp, sf)) > kFusedMaxSmem) ctx->fused = false;
    }
    if (ctx->head) {
        // one dW / db partial per block of kHeadRows rows, summed by the SGD kernel in block order
        Layer& H = ctx->T.back();
        H.nsplit = H.nsplit_b = head_blocks(c.batch);
        H.kchunk = kHeadRows;
        H.tc_dw = H.sgd_in_dw = false;
    }
}

// Lay out every device buffer; with base == nullptr only measures.
unsigned long long carve_all(vfl_ctx* ctx, void* base) {
    Carver cv(base);
    const vfl_config& c = ctx->cfg;
    const int es = ctx->esz;
    const long long B = c.batch;
    ctx->ldxp = ctx->bf16 ? ld64(c.d_passive) : ld8(c.d_passive);
    ctx->ldxa = ctx->bf16 ? ld64(c.d_active) : ld8(c.d_active);
    ctx->Xp = cv.take((unsigned long long)ctx->n_rows * ctx->ldxp * es);
    ctx->Xa = cv.take((unsigned long long)ctx->n_rows * ctx->ldxa * es);
    ctx->Y = static_cast<int*>(cv.take((unsigned long long)ctx->n_rows * 4));
    ctx->stage_p = static_cast<float*>(cv.take(B * c.d_passive * 4ull));
    ctx->stage_a = static_cast<float*>(cv.take(B * c.d_active * 4ull));
    for (std::vector<Layer>* v : {&ctx->P, &ctx->A, &ctx->T}) {
        for (Layer& L : *v) {
            L.W = static_cast<float*>(cv.take((unsigned long long)L.out * L.in * 4));
            L.b = static_cast<float*>(cv.take((unsigned long long)L.out * 4));
            L.Wr[0] = L.W;
            L.br[0] = L.b;
            for (int w = 1; ctx->psmode && w < ctx->W; ++w) {
                L.Wr[w] = static_cast<float*>(cv.take((unsigned long long)L.out * L.in * 4));
                L.br[w] = static_cast<float*>(cv.take((unsigned long long)L.out * 4));
            }
            for (int s = 0; s < ctx->S1; ++s) {
                L.cW[s] = cv.take((unsigned long long)L.out * L.in_ld * es);
                L.cb[s] = static_cast<float*>(cv.take((unsigned long long)L.out * 4));
            }
            for (int w = 0; w < ctx->W; ++w) {
                L.pW[w] = static_cast<float*>(cv.take((unsigned long long)L.nsplit * L.out * L.in * 4));
                L.pb[w] = static_cast<float*>(cv.take((unsigned long long)L.nsplit_b * L.out * 4));
                if (L.tc_dw) {
                    L.dw_ws_floats = tc_dw_ws_floats(L.out, L.in, ctx->cfg.batch);
                    L.dw_ws[w] = static_cast<float*>(cv.take((unsigned long long)L.dw_ws_floats * 4));
                }
            }
        }
    }
    for (int s = 0; s < ctx->S1; ++s) {
        ctx->act_p[s].clear();
        for (const Layer& L : ctx->P) ctx->act_p[s].push_back(cv.take(B * ld8(L.out) * es));
        ctx->grad[s] = cv.take(B * ld8(ctx->P.back().out) * es);
        if (c.dp_clip > 0.f && c.dp_target == VFL_DP_EMB) {
            ctx->emb_pub[s] = cv.take(B * ld8(ctx->P.back().out) * es);
            ctx->emb_c[s] = static_cast<float*>(cv.take(B * 4ull));
        }
    }
    const int n_out = ctx->T.back().out;
    for (int w = 0; w < ctx->W; ++w) {
        ctx->dpre_p[w].clear();
        for (const Layer& L : ctx->P) ctx->dpre_p[w].push_back(cv.take(B * ld8(L.out) * es));
        ctx->act_a[w].clear();
        ctx->dpre_a[w].clear();
        for (const Layer& L : ctx->A) {
            ctx->act_a[w].push_back(cv.take(B * ld8(L.out) * es));
            ctx->dpre_a[w].push_back(cv.take(B * ld8(L.out) * es));
        }
        ctx->act_t[w].clear();
        ctx->dpre_t[w].clear();
        for (size_t l = 0; l + 1 < ctx->T.size(); ++l) {
            ctx->act_t[w].push_back(cv.take(B * ld8(ctx->T[l].out) * es));
            ctx->dpre_t[w].push_back(cv.take(B * ld8(ctx->T[l].out) * es));
        }
        ctx->logits[w] = static_cast<float*>(cv.take(B * n_out * 4ull));
        ctx->ds[w] = static_cast<float*>(cv.take(B * n_out * 4ull));
        ctx->dzp32[w] = static_cast<float*>(cv.take(B * ld8(ctx->P.back().out) * 4ull));
    }
    ctx->emb_hdr = static_cast<ChannelHeader*>(cv.take(sizeof(ChannelHeader) * ctx->S1));
    ctx->grad_hdr = static_cast<ChannelHeader*>(cv.take(sizeof(ChannelHeader) * ctx->S1));
    ctx->losses = static_cast<float*>(cv.take(kLossCap * 4ull));
    if (ctx->psmode)
        ctx->ps_tab = static_cast<PsAvgLayer*>(
            cv.take(sizeof(PsAvgLayer) * (ctx->P.size() + ctx->A.size() + ctx->T.size())));
    ctx->status = static_cast<int*>(cv.take(256));
    // scratch for taps and version reads/writes: a [B, widest] activation or a whole weight matrix
    long long maxw = std::max<long long>(c.d_passive, c.d_active);
    long long maxwt = 0;
    for (auto* v : {&ctx->P, &ctx->A, &ctx->T})
        for (const Layer& L : *v) {
            maxw = std::max<long long>(maxw, std::max(L.out, L.in));
            maxwt = std::max<long long>(maxwt, (long long)L.out * L.in_ld);
        }
    ctx->scratch_f32 = static_cast<float*>(cv.take(std::max(B * ld8(maxw), maxwt) * 4ull));
    if (ctx->fused) {
        for (int w = 0; w < ctx->W; ++w) {
            ctx->f_rowloss[w] = static_cast<float*>(cv.take(B * 4ull));
            ctx->f_zpc[w] = static_cast<float*>(cv.take(B * ld8(ctx->P.back().out) * 4ull));
        }
    }
    // staging ring of host-resident data: slot k mod io_R holds step k's rows
    ctx->io_R = c.staleness + ctx->W + 2;
    for (int r = 0; r < ctx->io_R; ++r) {
        ctx->io_xp[r] = cv.take(B * ctx->ldxp * es);
        ctx->io_xa[r] = cv.take(B * ctx->ldxa * es);
        ctx->io_y[r] = static_cast<int*>(cv.take(B * 4ull));
    }
    if (ctx->head) {
        ctx->h_counter = static_cast<int*>(cv.take(kMaxWorkers * sizeof(int)));
        for (int w = 0; w < ctx->W; ++w)
            ctx->h_blk_loss[w] = static_cast<float*>(cv.take(head_blocks(B) * 4ull));
    }
    return cv.off + 256;
}

inline cudaStream_t pstream(vfl_ctx* ctx, long long k) { return ctx->ps[k % ctx->W]; }

// DP on the published embedding (App. C) rather than on its gradient
inline bool emb_dp(const vfl_ctx* ctx) { return ctx->cfg.dp_clip > 0.f && ctx->cfg.dp_target == VFL_DP_EMB; }

// ---- parameter-server mode (Sec. 4.1, Eq. 5) ------------------------------------------------
// Synchronization interval after epoch t (1-based), Eq. 5:
// Delta T_t = ceil(Delta T_0 / 2 * tanh(2 t / Delta T_0 - 2) + Delta T_0 / 2).
long long ps_interval(long long t, int dt0) {
    const double h = dt0 / 2.0;
    const long long v = (long long)std::ceil(h * std::tanh(2.0 * (double)t / dt0 - 2.0) + h);
    return std::max<long long>(1, v);
}
// Whether the replicas are averaged right after step e: e ends epoch t and t mod Delta T_t == 0
// (with one worker the mean is the replica itself and nothing is launched).
// Epochs count trained batches: with drops, epoch t ends at the step that trains batch nb-1 for the
// t-th time.
bool ps_agg_at(const vfl_ctx* ctx, long long e) {
    if (!ctx->psmode || ctx->W < 2 || e < 0 || ctx->dropped(e) || ctx->batch_of(e) != ctx->nb - 1) return false;
    const long long t = ctx->step_trained[e % kInfoRing] / ctx->nb + 1;
    return t % ps_interval(t, ctx->cfg.ps_dt0) == 0;
}
// The latest averaging step a < k that step k must follow (a >= k - W: older ones are ordered
// through the worker's own stream), or -1.
long long ps_last_agg(const vfl_ctx* ctx, long long k) {
    for (long long e = k - 1; e >= 0 && e >= k - ctx->W; --e)
        if (ps_agg_at(ctx, e)) return e;
    return -1;
}
// Passive updates that must be enqueued before step k's publisher: its worker's previous step, and
// the averaging it follows.
long long ps_need_bwd(const vfl_ctx* ctx, long long k) {
    return std::max(k - ctx->W + 1, ps_last_agg(ctx, k) + 1);
}
// Replica and version slot step k's worker reads and updates (the single master and ring otherwise).
inline int ps_rep(const vfl_ctx* ctx, long long k) { return ctx->psmode ? (int)(k % ctx->W) : 0; }
inline int new_version_slot(const vfl_ctx* ctx, long long k) {
    return ctx->psmode ? (int)(k % ctx->W) : (int)((k + 1) % ctx->S1);
}

// Rows of step k (first row r0): the staging ring's slot when host data is bound, else the
// device-resident dataset.  Both have the same row strides.
inline const void* xp_rows(const vfl_ctx* ctx, long long k, long long r0) {
    return ctx->hio ? ctx->io_xp[k % ctx->io_R] : static_cast<const char*>(ctx->Xp) + r0 * ctx->ldxp * ctx->esz;
}
inline const void* xa_rows(const vfl_ctx* ctx, long long k, long long r0) {
    return ctx->hio ? ctx->io_xa[k % ctx->io_R] : static_cast<const char*>(ctx->Xa) + r0 * ctx->ldxa * ctx->esz;
}
inline const int* y_rows(const vfl_ctx* ctx, long long k, long long r0) {
    return ctx->hio ? ctx->io_y[k % ctx->io_R] : ctx->Y + r0;
}
// Where the kernel that computes step k's mean loss also writes it: the bound host ring, if any.
inline float* loss_host(const vfl_ctx* ctx, long long k) {
    return ctx->hio && ctx->h_loss ? ctx->h_loss + k % ctx->h_loss_cap : nullptr;
}
inline cudaStream_t astream(vfl_ctx* ctx, long long k) { return ctx->as[k % ctx->W]; }

// ---- GEMM helpers ---------------------------------------------------------
GemmArgs gemm_base(int mode, int M, int N, int K) {
    GemmArgs g;
    std::memset(&g, 0, sizeof g);
    g.mode = mode;
    g.M = M;
    g.N = N;
    g.K = K;
    g.n_split = N;
    return g;
}

// Y[rows, out] = act(X W^T + b); X may be [X1 | X2] split at column ka.
vfl_status linear_fwd(vfl_ctx* ctx, const Layer& L, int slot, const void* X, long long ldx, const void* X2,
                      long long ldx2, int ka, int rows, void* Y, long long ldy, bool relu, bool y_f32,
                      cudaStream_t s, const HeaderOps* hdr = nullptr) {
    const int in_bf = ctx->bf16;
    const double flops = 2.0 * rows * L.out * L.in;
    const double bytes = ((double)rows * L.in + (double)L.out * L.in) * ctx->esz +
                         (double)rows * L.out * (y_f32 ? 4 : ctx->esz) + L.out * 4.0;
    if (in_bf && tc_supported_fwd(L.in, L.out, X2 != nullptr, ka, y_f32)) {
        TcGemm t = {};
        t.mode = GEMM_FWD;
        t.M = rows; t.N = L.out; t.K = L.in;
        t.A = X; t.lda = ldx; t.A2 = X2; t.lda2 = ldx2; t.ka = X2 ? ka : L.in;
        t.B = L.cW[slot]; t.ldb = L.in_ld;
        t.bias = L.cb[slot]; t.relu = relu;
        t.C = Y; t.ldc = ldy;
        t.err = ctx->status;
        if (hdr) t.hdr = *hdr;
        PLAUNCH(K_TC_FWD, flops, bytes, s, launch_tc_gemm(t, s));
        return VFL_OK;
    }
    GemmArgs g = gemm_base(GEMM_FWD, rows, L.out, L.in);
    g.A = X; g.a_rs = ldx; g.a_cs = 1;
    if (X2) { g.A2 = X2; g.a2_rs = ldx2; g.ka = ka; }
    g.B = L.cW[slot]; g.b_rs = L.in_ld; g.b_cs = 1;
    g.bias = L.cb[slot];
    g.relu = relu ? 1 : 0;
    g.C = Y; g.ldc = ldy; g.c_bf16 = y_f32 ? 0 : in_bf;
    if (hdr) g.hdr = *hdr;
    PLAUNCH(K_SIMT_FWD, flops, bytes, s, launch_gemm_simt(g, in_bf, in_bf, in_bf, 1, s));
    return VFL_OK;
}

// Partial dW, db of layer L for the step on worker w:
//   dW[out, in] = dpre^T X, dpre [rows, out] (leading dim ldd, fp32 when dpre_f32).
//   X may be [X1 | X2] split at column ka (then two GEMMs write the two column blocks).
// On the tensor-core cluster kernel (L.tc_dw) the one reduced dW and db land in the partial buffers, and
// with L.sgd_in_dw the same kernel applies the SGD step to replica `rep` and writes version slot `new_slot`
// (the caller orders it after update k-1 of the party: wait_update_order before the step's first such kernel).
vfl_status linear_dw(vfl_ctx* ctx, const Layer& L, int w, const void* dpre, long long ldd, bool dpre_f32,
                     const void* X, long long ldx, const void* X2, long long ldx2, int ka, int rows, cudaStream_t s,
                     int rep = 0, int new_slot = 0) {
    const int bf = ctx->bf16;
    const int a_bf = dpre_f32 ? 0 : bf;
    const double flops = 2.0 * rows * L.out * L.in;
    if (L.tc_dw && !dpre_f32) {
        if (!tc_available()) return ctx->fail(VFL_E_CUDA, "tensor-core weight gradient: no tensor-map encoder");
        TcGemm t = {};
        t.mode = GEMM_DW;
        t.M = L.out; t.N = L.in; t.K = rows;
        t.A = dpre; t.lda = ldd;
        t.B = X; t.ldb = ldx; t.B2 = X2; t.ldb2 = ldx2; t.kb = X2 ? ka : L.in;
        t.P = L.pW[w]; t.ldc = L.in;
        t.Pb = L.pb[w];
        t.ws = L.dw_ws[w]; t.ws_floats = L.dw_ws_floats;
        if (L.sgd_in_dw) {
            t.Wm = L.Wr[rep]; t.bm = L.br[rep];
            t.cW = L.cW[new_slot]; t.cw_ld = L.in_ld; t.cb = L.cb[new_slot];
            t.lr = ctx->cfg.lr;
        }
        t.err = ctx->status;
        // D and X once, dW and db written; with the SGD the masters read and written and the copies written
        const double np_ = (double)L.out * L.in + L.out;
        const double bytes = (double)rows * L.out * ctx->esz + (double)rows * L.in * ctx->esz + np_ * 4 +
                             (L.sgd_in_dw ? np_ * 8 + (double)L.out * L.in * ctx->esz + L.out * 4.0 : 0.0);
        PLAUNCH(L.sgd_in_dw ? K_TC_DW_SGD : K_TC_DW, flops + (L.sgd_in_dw ? 2.0 * np_ : 0.0), bytes, s,
                launch_tc_gemm(t, s));
        return VFL_OK;
    }
    const double bytes = (double)rows * L.out * (dpre_f32 ? 4 : ctx->esz) + (double)rows * L.in * ctx->esz +
                         (double)L.nsplit * ((double)L.out * L.in + L.out) * 4;
    const int n1 = X2 ? ka : L.in;
    GemmArgs g = gemm_base(GEMM_DW, L.out, n1, rows);
    g.A = dpre; g.a_rs = 1; g.a_cs = ldd;
    g.B = X; g.b_rs = 1; g.b_cs = ldx;
    g.P = L.pW[w]; g.p_stride = (long long)L.out * L.in; g.ldc = L.in;
    g.Pb = L.pb[w]; g.pb_stride = L.out;
    g.kchunk = L.kchunk;
    const double f1 = X2 ? flops * n1 / L.in : flops, b1 = X2 ? bytes * n1 / L.in : bytes;
    PLAUNCH(K_SIMT_DW, f1, b1, s, launch_gemm_simt(g, a_bf, bf, bf, L.nsplit, s));
    if (X2) {
        GemmArgs g2 = gemm_base(GEMM_DW, L.out, L.in - ka, rows);
        g2.A = dpre; g2.a_rs = 1; g2.a_cs = ldd;
        g2.B = X2; g2.b_rs = 1; g2.b_cs = ldx2;
        g2.P = L.pW[w] + ka; g2.p_stride = (long long)L.out * L.in; g2.ldc = L.in;
        g2.Pb = nullptr;
        g2.kchunk = L.kchunk;
        PLAUNCH(K_SIMT_DW, flops - f1, bytes - b1, s, launch_gemm_simt(g2, a_bf, bf, bf, L.nsplit, s));
    }
    return VFL_OK;
}

// dX[rows, in] = dpre W (W of version slot), columns < n_split -> C (masked by
// mask1 > 0), the rest -> C2 (masked by mask2 when given).
vfl_status linear_dx(vfl_ctx* ctx, const Layer& L, int slot, const void* dpre, long long ldd, bool dpre_f32,
                     int rows, void* C, long long ldc, const void* mask1, int n_split, void* C2, long long ldc2,
                     bool c2_f32, const void* mask2, cudaStream_t s, const HeaderOps* hdr = nullptr) {
    const int bf = ctx->bf16;
    const double flops = 2.0 * rows * L.out * L.in;
    const double bytes = (double)rows * L.out * (dpre_f32 ? 4 : ctx->esz) + (double)L.out * L.in * ctx->esz +
                         (double)rows * L.in * ctx->esz * 2;
    if (bf && !dpre_f32 && tc_supported_dx(L.in, L.out, n_split, c2_f32)) {
        TcGemm t = {};
        t.mode = GEMM_DX;
        t.M = rows; t.N = L.in; t.K = L.out;
        t.A = dpre; t.lda = ldd;
        t.B = L.cW[slot]; t.ldb = L.in_ld;
        t.C = C; t.ldc = ldc; t.mask1 = mask1;
        t.n_split = n_split; t.C2 = C2; t.ldc2 = ldc2; t.mask2 = mask2;
        t.c2_f32 = c2_f32 ? 1 : 0;
        t.err = ctx->status;
        if (hdr) t.hdr = *hdr;
        PLAUNCH(K_TC_DX, flops, bytes, s, launch_tc_gemm(t, s));
        return VFL_OK;
    }
    GemmArgs g = gemm_base(GEMM_DX, rows, L.in, L.out);
    g.A = dpre; g.a_rs = ldd; g.a_cs = 1;
    g.B = L.cW[slot]; g.b_rs = 1; g.b_cs = L.in_ld;
    g.C = C; g.ldc = ldc; g.c_bf16 = bf;
    g.mask1 = mask1; g.mask1_ld = ldc;
    g.n_split = n_split;
    g.C2 = C2; g.ldc2 = ldc2; g.c2_bf16 = c2_f32 ? 0 : bf;
    g.mask2 = mask2; g.mask2_ld = ldc2;
    if (hdr) g.hdr = *hdr;
    PLAUNCH(K_SIMT_DX, flops, bytes, s, launch_gemm_simt(g, dpre_f32 ? 0 : bf, bf, bf, 1, s));
    return VFL_OK;
}

vfl_status sgd(vfl_ctx* ctx, std::vector<Layer>* a, std::vector<Layer>* b, int w, int rep, int new_slot,
               cudaStream_t s) {
    SgdArgs args;
    std::memset(&args, 0, sizeof args);
    long long off = 0;
    int n = 0;
    for (std::vector<Layer>* v : {a, b}) {
        if (!v) continue;
        for (Layer& L : *v) {
            if (L.sgd_in_dw) continue;
            SgdLayer& d = args.L[n++];
            d.W = L.Wr[rep]; d.b = L.br[rep];
            d.pW = L.pW[w]; d.pb = L.pb[w];
            d.pW_stride = (long long)L.out * L.in;
            d.pb_stride = L.out;
            d.nsplit = L.nsplit;
            d.nsplit_b = L.nsplit_b;
            d.out = L.out; d.in = L.in; d.in_ld = L.in_ld;
            d.cW = L.cW[new_slot]; d.cb = L.cb[new_slot];
            d.begin = off;
            off += (long long)L.out * L.in + L.out;
        }
    }
    if (n == 0) return VFL_OK;
    args.n_layers = n;
    args.total = off;
    args.lr = ctx->cfg.lr;
    args.c_bf16 = ctx->bf16;
    double bytes = 0;
    for (int i = 0; i < n; ++i) {
        const SgdLayer& d = args.L[i];
        const double np_ = (double)d.out * d.in + d.out;
        bytes += np_ * 8.0 + 4.0 * ((double)d.out * d.in * d.nsplit + (double)d.out * d.nsplit_b) +
                 (double)d.out * d.in * ctx->esz + d.out * 4.0;
    }
    PLAUNCH(K_SGD, 2.0 * off, bytes, s, launch_sgd(args, s));
    return VFL_OK;
}

vfl_status wait_ev(vfl_ctx* ctx, cudaStream_t s, cudaEvent_t e) {
    CK(cudaStreamWaitEvent(s, e, 0));
    return VFL_OK;
}


// Fused-path phases whose kernel nodes a capture records.
enum CapPhase : int { CAP_PFWD, CAP_ACTIVE, CAP_AUPD, CAP_PBWD, CAP_PUPD };

// Under stream capture (and without per-launch timing, whose event nodes would sit in between),
// remember the kernel node just captured on stream s as phase `ph` of step k.
void note_node(vfl_ctx* ctx, int ph, long long k, cudaStream_t s) {
    if (!ctx->capturing || ctx->prof_on) return;
    cudaStreamCaptureStatus st;
    const cudaGraphNode_t* deps = nullptr;
    size_t n = 0;
    if (cudaStreamGetCaptureInfo(s, &st, nullptr, nullptr, &deps, nullptr, &n) == cudaSuccess &&
        st == cudaStreamCaptureStatusActive && n == 1)
        ctx->cap_nodes[{ph, k}] = deps[0];
    else
        cudaGetLastError();
}

// ---- fused path -------------------------------------------------------------
// Direct enqueue (not captured, not timed per launch) gives the fused kernels the programmatic
// dependencies a captured graph gets as edges: the passive forward and the active step record their
// channel events programmatically, and each update launches behind its row kernel on the same stream.
inline bool use_direct_pdl(const vfl_ctx* ctx) { return ctx->direct_pdl && !ctx->capturing && !ctx->prof_on; }

FusedLayerArgs fused_layer(const Layer& L, int vslot, void* Y, long long ldy, void* D, long long ldd) {
    FusedLayerArgs f;
    std::memset(&f, 0, sizeof f);
    f.in = L.in;
    f.out = L.out;
    f.fmap = fused_gemm_map((L.in + 7) / 8, (L.out + 7) / 8);
    f.dmap = fused_gemm_map((L.out + 7) / 8, (L.in + 7) / 8);
    f.in_ld = L.in_ld;
    f.out_ld = ld8(L.out);
    f.W = static_cast<const float*>(L.cW[vslot]);
    f.b = L.cb[vslot];
    f.Y = static_cast<float*>(Y);
    f.ldy = ldy;
    f.D = static_cast<float*>(D);
    f.ldd = ldd;
    return f;
}

// Update of layer L from its d(pre) rows D and input rows [X | X2] (X2 from column xsplit on).
FusedUpdLayer fused_upd_layer(const Layer& L, int new_slot, int rep, int w, const void* D, long long ldd,
                              const void* X, long long ldx, const void* X2, long long ldx2, int xsplit) {
    FusedUpdLayer u;
    std::memset(&u, 0, sizeof u);
    u.out = L.out;
    u.in = L.in;
    u.in_ld = L.in_ld;
    u.D = static_cast<const float*>(D);
    u.ldd = ldd;
    u.X = static_cast<const float*>(X);
    u.ldx = ldx;
    u.X2 = static_cast<const float*>(X2 ? X2 : X);
    u.ldx2 = X2 ? ldx2 : ldx;
    u.xsplit = X2 ? xsplit : L.in;
    u.Wm = L.Wr[rep];
    u.bm = L.br[rep];
    u.Wc = static_cast<float*>(L.cW[new_slot]);
    u.bc = L.cb[new_slot];
    u.gW = L.pW[w];
    u.gb = L.pb[w];
    return u;
}

// 2 rows in out FLOPs per layer for each of: forward, input gradient (all layers
// but the first unless dx_first), weight gradient.
double fused_flops(const std::vector<Layer>& v, int rows, bool fwd, bool dx, bool dx_first, bool dw) {
    double f = 0;
    for (size_t l = 0; l < v.size(); ++l) {
        const double mn = 2.0 * rows * v[l].in * v[l].out;
        if (fwd) f += mn;
        if (dx && (dx_first || l > 0)) f += mn;
        if (dw) f += mn;
    }
    return f;
}

vfl_status launch_update(vfl_ctx* ctx, FusedUpdArgs& u, int rows, cudaStream_t s) {
    u.ntiles = fused_update_tiles(u.L, u.nl);
    u.rows = rows;
    u.lr = ctx->cfg.lr;
    // algorithmic: dW = D^T X per layer; D and X read once, 16 B per parameter
    // (master read + write, gradient and new copy written)
    double flops = 0, bytes = 0;
    for (int l = 0; l < u.nl; ++l) {
        const FusedUpdLayer& L = u.L[l];
        flops += 2.0 * rows * L.out * L.in;
        bytes += (double)rows * (L.out + L.in) * 4 + ((double)L.out * L.in + L.out) * 16;
    }
    if (u.loss_out) bytes += rows * 4.0 + 4;
    LaunchOpt o;
    o.serialize = use_direct_pdl(ctx) ? 1 : 0;   // behind its row kernel on the same stream
    PLAUNCH(K_FUSED_UPDATE, flops, bytes, s, launch_fused_update(u, s, o));
    return VFL_OK;
}

vfl_status fused_passive_forward(vfl_ctx* ctx, long long k, long long v, int slot, int vslot, int rows,
                                 const float* X, int w, cudaStream_t s) {
    FusedChainArgs a;
    std::memset(&a, 0, sizeof a);
    a.nl = (int)ctx->P.size();
    for (int l = 0; l < a.nl; ++l)
        a.L[l] = fused_layer(ctx->P[l], vslot, ctx->act_p[slot][l], ld8(ctx->P[l].out), nullptr, 0);
    a.x = X;
    a.ldx = ctx->ldxp;
    a.rows = rows;
    a.act_ld = ctx->f_act_ld;
    a.w_floats = fused_weight_layout(a.L, a.nl, 0);
    a.hdr = ctx->emb_hdr + slot;
    if (emb_dp(ctx)) {
        a.dp_out = static_cast<float*>(ctx->emb_pub[slot]);
        a.ld_dp = ld8(ctx->P.back().out);
        a.dp_scale = ctx->emb_c[slot];
        a.dp_clip = ctx->cfg.dp_clip;
        a.dp_sigma = ctx->cfg.dp_sigma;
        a.dp_seed = ctx->cfg.dp_seed;
    }
    a.k = k;
    a.batch = (int)ctx->batch_of(k);
    a.version = (int)v;
    // algorithmic bytes: the batch's features in, the saved activations out, one read of the weights
    double bytes = (double)rows * ctx->cfg.d_passive * 4;
    for (const Layer& L : ctx->P) bytes += (double)rows * L.out * 4 + ((double)L.out * L.in + L.out) * 4;
    LaunchOpt o;
    if (use_direct_pdl(ctx)) o.pevent = ctx->ev_emb[k % kEvPool];
    PLAUNCH(K_FUSED_PFWD, fused_flops(ctx->P, rows, true, false, false, false), bytes, s,
            launch_fused_passive_fwd(a, s, o));
    return VFL_OK;
}

// Active party, row-parallel part: forward, loss, input gradients, dz^p published.
vfl_status fused_active_step(vfl_ctx* ctx, long long k, long long v, int slot, int vslot, int rows,
                             const float* Xa, int w, cudaStream_t s) {
    FusedStepArgs a;
    std::memset(&a, 0, sizeof a);
    const int La = (int)ctx->A.size(), Lt = (int)ctx->T.size();
    const int n_out = ctx->T.back().out;
    for (int l = 0; l < La; ++l) {
        const Layer& L = ctx->A[l];
        a.L[l] = fused_layer(L, vslot, ctx->act_a[w][l], ld8(L.out), ctx->dpre_a[w][l], ld8(L.out));
    }
    for (int l = 0; l < Lt; ++l) {
        const Layer& L = ctx->T[l];
        const bool last = l == Lt - 1;
        a.L[La + l] = fused_layer(L, vslot, last ? (void*)ctx->logits[w] : ctx->act_t[w][l], last ? n_out : ld8(L.out),
                                  last ? (void*)ctx->ds[w] : ctx->dpre_t[w][l], last ? n_out : ld8(L.out));
    }
    const int ep = ctx->P.back().out;
    a.na = La;
    a.nt = Lt;
    a.rows = rows;
    a.act_ld = ctx->f_act_ld;
    a.w_floats = fused_weight_layout(a.L, La + Lt, 0);
    a.x = Xa;
    a.ldx = ctx->ldxa;
    long long r0;
    ctx->batch_rows(k, &r0);
    a.y = y_rows(ctx, k, r0);
    a.loss = ctx->cfg.loss;
    a.zp = static_cast<const float*>(emb_dp(ctx) ? ctx->emb_pub[slot] : ctx->act_p[slot].back());
    a.ldzp = ld8(ep);
    a.zpc = ctx->f_zpc[w];
    a.ldzpc = ld8(ep);
    a.gradp = static_cast<float*>(ctx->grad[slot]);
    a.ldgp = ld8(ep);
    a.rowloss = ctx->f_rowloss[w];
    a.chk_hdr = ctx->emb_hdr + slot;
    a.pub_hdr = ctx->grad_hdr + slot;
    a.k = k;
    a.batch = (int)ctx->batch_of(k);
    a.version = (int)v;
    a.status = ctx->status;
    const double flops = fused_flops(ctx->A, rows, true, true, false, false) + fused_flops(ctx->T, rows, true, true, true, false);
    // algorithmic bytes: x^a, labels and z^p in; every layer's output and
    // d(pre-activation) out, z^p's copy and dz^p out; every weight read once
    double bytes = (double)rows * (ctx->cfg.d_active + 3.0 * ep + 2) * 4;
    for (auto* vv : {&ctx->A, &ctx->T})
        for (const Layer& L : *vv) bytes += (double)rows * L.out * 8 + ((double)L.out * L.in + L.out) * 4;
    LaunchOpt o;
    if (use_direct_pdl(ctx)) o.pevent = ctx->ev_grad[k % kEvPool];
    PLAUNCH(K_FUSED_ACTIVE, flops, bytes, s, launch_fused_active(a, s, o));
    return VFL_OK;
}

// Active party's weight gradients of f_a and g, and SGD to version k+1.
vfl_status fused_active_update(vfl_ctx* ctx, long long k, int rows, const float* Xa, int w, cudaStream_t s) {
    FusedUpdArgs u;
    std::memset(&u, 0, sizeof u);
    const int La = (int)ctx->A.size(), Lt = (int)ctx->T.size();
    const int new_slot = new_version_slot(ctx, k), rp = ps_rep(ctx, k);
    const int n_out = ctx->T.back().out;
    const int ea = ctx->A.back().out, ep = ctx->P.back().out;
    int n = 0;
    for (int l = 0; l < La; ++l) {
        const Layer& L = ctx->A[l];
        const void* X = l == 0 ? (const void*)Xa : ctx->act_a[w][l - 1];
        const long long ldx = l == 0 ? ctx->ldxa : ld8(ctx->A[l - 1].out);
        u.L[n++] = fused_upd_layer(L, new_slot, rp, w, ctx->dpre_a[w][l], ld8(L.out), X, ldx, nullptr, 0, 0);
    }
    u.L[0].x_early = 1;   // x^a's rows: every other input comes from the active step's row kernel
    for (int l = 0; l < Lt; ++l) {
        const Layer& L = ctx->T[l];
        const bool last = l == Lt - 1;
        const void* D = last ? (const void*)ctx->ds[w] : ctx->dpre_t[w][l];
        const long long ldd = last ? n_out : ld8(L.out);
        if (l == 0)
            u.L[n++] = fused_upd_layer(L, new_slot, rp, w, D, ldd, ctx->act_a[w][La - 1], ld8(ea), ctx->f_zpc[w],
                                       ld8(ep), ea);
        else
            u.L[n++] = fused_upd_layer(L, new_slot, rp, w, D, ldd, ctx->act_t[w][l - 1], ld8(ctx->T[l - 1].out),
                                       nullptr, 0, 0);
    }
    u.nl = n;
    u.rowloss = ctx->f_rowloss[w];
    u.loss_out = ctx->losses + (k % kLossCap);
    u.loss_host = loss_host(ctx, k);
    return launch_update(ctx, u, rows, s);
}

// Passive party, row-parallel part of the backward phase: d(pre) of every layer of f_p.
vfl_status fused_passive_backward(vfl_ctx* ctx, long long k, int slot, int vslot, int rows, int w, cudaStream_t s) {
    FusedStepArgs a;
    std::memset(&a, 0, sizeof a);
    const int Lp = (int)ctx->P.size();
    for (int l = 0; l < Lp; ++l) {
        const Layer& L = ctx->P[l];
        a.L[l] = fused_layer(L, vslot, ctx->act_p[slot][l], ld8(L.out), ctx->dpre_p[w][l], ld8(L.out));
    }
    a.na = Lp;
    a.nt = 0;
    a.rows = rows;
    a.act_ld = ctx->f_act_ld;
    a.w_floats = fused_weight_layout(a.L, Lp, 1);
    a.gradp = static_cast<float*>(ctx->grad[slot]);
    a.ldgp = ld8(ctx->P.back().out);
    a.chk_hdr = ctx->grad_hdr + slot;
    a.k = k;
    a.status = ctx->status;
    a.rowscale = emb_dp(ctx) ? ctx->emb_c[slot] : nullptr;
    // algorithmic bytes: dz^p and the saved activations in, every d(pre) out, weights after the first read once
    double bytes = (double)rows * ctx->P.back().out * 4;
    for (size_t l = 0; l < ctx->P.size(); ++l) {
        const Layer& L = ctx->P[l];
        bytes += (double)rows * L.out * 8;
        if (l > 0) bytes += ((double)L.out * L.in + L.out) * 4;
    }
    PLAUNCH(K_FUSED_PBWD, fused_flops(ctx->P, rows, false, true, false, false), bytes, s,
            launch_fused_passive_bwd(a, s));
    return VFL_OK;
}

// Passive party's weight gradients of f_p and SGD to version k+1.
vfl_status fused_passive_update(vfl_ctx* ctx, long long k, int slot, int rows, const float* Xp, int w,
                                cudaStream_t s) {
    FusedUpdArgs u;
    std::memset(&u, 0, sizeof u);
    const int Lp = (int)ctx->P.size();
    const int new_slot = new_version_slot(ctx, k), rp = ps_rep(ctx, k);
    for (int l = 0; l < Lp; ++l) {
        const Layer& L = ctx->P[l];
        const void* X = l == 0 ? (const void*)Xp : ctx->act_p[slot][l - 1];
        const long long ldx = l == 0 ? ctx->ldxp : ld8(ctx->P[l - 1].out);
        u.L[l] = fused_upd_layer(L, new_slot, rp, w, ctx->dpre_p[w][l], ld8(L.out), X, ldx, nullptr, 0, 0);
        u.L[l].x_early = 1;   // x^p's rows and the forward's activations: only D comes from the backward
    }
    u.nl = Lp;
    return launch_update(ctx, u, rows, s);
}

// ---- host-resident data ----------------------------------------------------
// Read step k's rows from the bound (mapped) host arrays into its staging slot on the I/O stream, after
// the last step that used the slot (k - io_R: its passive and active updates are its last reads
// of the rows); the step's phases wait for ev_staged.  io_R > S, so that step is always enqueued.
vfl_status stage_step(vfl_ctx* ctx, long long k) {
    const vfl_config& c = ctx->cfg;
    long long r0;
    const int rows = ctx->batch_rows(k, &r0);
    const int slot = (int)(k % ctx->io_R);
    cudaStream_t s = ctx->io;
    const long long prev = k - ctx->io_R;
    if (prev >= 0 && prev + 1 > ctx->ordered_floor) {
        TRY(wait_ev(ctx, s, ctx->ev_pver[(prev + 1) % kEvPool]));
        TRY(wait_ev(ctx, s, ctx->ev_aver[(prev + 1) % kEvPool]));
    }
    if (ctx->h_copy) {
        // rows already in the slot layout: three contiguous copies by the copy engines, which leave the
        // SMs to the steps' kernels
        const size_t bp = (size_t)c.d_passive * ctx->esz, ba = (size_t)c.d_active * ctx->esz;
        CK(cudaMemcpyAsync(ctx->io_xp[slot], ctx->hc_xp + r0 * bp, rows * bp, cudaMemcpyHostToDevice, s));
        CK(cudaMemcpyAsync(ctx->io_xa[slot], ctx->hc_xa + r0 * ba, rows * ba, cudaMemcpyHostToDevice, s));
        CK(cudaMemcpyAsync(ctx->io_y[slot], ctx->hc_y + r0, rows * sizeof(int32_t), cudaMemcpyHostToDevice, s));
    } else if (ctx->h_esz == 0) {
        // bit-packed binary rows: ceil(d / 32) words a row over the host link, expanded to 0 / 1 on the device
        const uint32_t* hp = static_cast<const uint32_t*>(ctx->hv_xp);
        const uint32_t* ha = static_cast<const uint32_t*>(ctx->hv_xa);
        const long long wp = (c.d_passive + 31) / 32, wa = (c.d_active + 31) / 32;
        PLAUNCH(K_CAST, 0, (double)rows * (wp + wa + 2) * 4 + (double)rows * (ctx->ldxp + ctx->ldxa) * ctx->esz, s,
                launch_stage_rows_bits(hp + r0 * wp, c.d_passive, ha + r0 * wa, c.d_active, ctx->h_y + r0, rows,
                                       ctx->io_xp[slot], ctx->ldxp, ctx->io_xa[slot], ctx->ldxa, ctx->io_y[slot],
                                       ctx->bf16, s));
    } else if (ctx->h_esz == 2) {
        // bf16 rows into the bf16 slot: half the bytes over the host link
        const uint16_t* hp = static_cast<const uint16_t*>(ctx->hv_xp);
        const uint16_t* ha = static_cast<const uint16_t*>(ctx->hv_xa);
        PLAUNCH(K_CAST, 0, (double)rows * (c.d_passive + c.d_active) * 2 * 2 + (double)rows * 8, s,
                launch_stage_rows_b16(hp + r0 * c.d_passive, c.d_passive, ha + r0 * c.d_active, c.d_active,
                                      ctx->h_y + r0, rows, ctx->io_xp[slot], ctx->ldxp, ctx->io_xa[slot], ctx->ldxa,
                                      ctx->io_y[slot], s));
    } else {
        PLAUNCH(K_CAST, 0, (double)rows * (c.d_passive + c.d_active + 1) * 4 + (double)rows * (ctx->ldxp + ctx->ldxa) * ctx->esz,
                s, launch_stage_rows(ctx->h_xp + r0 * c.d_passive, c.d_passive, ctx->h_xa + r0 * c.d_active, c.d_active,
                                     ctx->h_y + r0, rows, ctx->io_xp[slot], ctx->ldxp, ctx->io_xa[slot], ctx->ldxa,
                                     ctx->io_y[slot], ctx->bf16, s));
    }
    CK(cudaEventRecord(ctx->ev_staged[k % kEvPool], s));
    return VFL_OK;
}


// ---- parameter-server aggregation ---------------------------------------------
// After step e's update on its worker's stream s: wait for every other worker's latest update
// (steps e-W+1 .. e-1; workers that have not run yet still hold the initial replica), then replace
// the party's replicas by their mean.  The steps of the next W that read a replica wait for ev_*avg.
vfl_status ps_average(vfl_ctx* ctx, long long e, bool passive, cudaStream_t s) {
    cudaEvent_t* ev = passive ? ctx->ev_pver : ctx->ev_aver;
    for (long long j = std::max(0ll, e - ctx->W + 1); j < e; ++j)
        if (j + 1 > ctx->ordered_floor) TRY(wait_ev(ctx, s, ev[(j + 1) % kEvPool]));
    const int first = passive ? 0 : (int)ctx->P.size();
    const int n = passive ? (int)ctx->P.size() : (int)(ctx->A.size() + ctx->T.size());
    const long long total = ctx->ps_total[passive ? 0 : 1];
    // algorithmic bytes: every replica's master read and written, every compute copy written
    const double bytes = (double)total * ctx->W * (8.0 + ctx->esz);
    PLAUNCH(K_PS_AVG, (double)total * ctx->W, bytes, s,
            launch_ps_average(ctx->ps_tab + first, n, total, ctx->W, ctx->bf16, s));
    CK(cudaEventRecord((passive ? ctx->ev_pavg : ctx->ev_aavg)[e % kEvPool], s));
    return VFL_OK;
}

// Before step k's first launch on party stream s: in the parameter-server mode, wait for the
// averaging it follows (its replica's own chain is ordered by the stream); otherwise for the
// update that produced version v.
vfl_status wait_version(vfl_ctx* ctx, long long k, long long v, bool passive, cudaStream_t s) {
    if (ctx->psmode) {
        const long long a = ps_last_agg(ctx, k);
        if (a >= 0 && a + 1 > ctx->ordered_floor)
            TRY(wait_ev(ctx, s, (passive ? ctx->ev_pavg : ctx->ev_aavg)[a % kEvPool]));
        return VFL_OK;
    }
    if (ctx->uniform) v = k;   // version k exists only after every version before it
    if (v > 0 && v > ctx->ordered_floor) TRY(wait_ev(ctx, s, (passive ? ctx->ev_pver : ctx->ev_aver)[v % kEvPool]));
    return VFL_OK;
}

// Before step k's update on s: updates apply in step order (App. D); in the parameter-server mode
// the replica's previous update ran on the same stream.
vfl_status wait_update_order(vfl_ctx* ctx, long long k, bool passive, cudaStream_t s) {
    // in the uniform order the step's first launch on this stream already waited for update k-1
    if (ctx->psmode || ctx->uniform || k <= 0 || k <= ctx->ordered_floor) return VFL_OK;
    return wait_ev(ctx, s, (passive ? ctx->ev_pver : ctx->ev_aver)[k % kEvPool]);
}

// ---- the three phases ------------------------------------------------------
// Host record of step k at its publish: its batch (the next untrained one) and whether it is dropped.
void record_step(vfl_ctx* ctx, long long k, bool drop) {
    const int i = (int)(k % kInfoRing);
    ctx->step_id[i] = k;
    ctx->step_trained[i] = k - ctx->n_drops;
    ctx->step_batch[i] = (k - ctx->n_drops) % ctx->nb;
    ctx->step_drop[i] = drop ? 1 : 0;
    if (drop) ++ctx->n_drops;
}

// A dropped step's version k+1 = version k: copy the compute copies of one party's layers from
// slot k mod S1 to slot (k+1) mod S1 on s, after version k exists (the masters already hold it).
// With one slot, or one per worker (parameter-server mode), there is nothing to copy.
vfl_status copy_version_forward(vfl_ctx* ctx, long long k, bool passive, cudaStream_t s) {
    if (k > 0 && k > ctx->ordered_floor && !ctx->psmode)
        TRY(wait_ev(ctx, s, (passive ? ctx->ev_pver : ctx->ev_aver)[k % kEvPool]));
    const int from = (int)(k % ctx->S1), to = new_version_slot(ctx, k);
    if (from != to && !ctx->psmode)
        for (std::vector<Layer>* v : passive ? std::vector<std::vector<Layer>*>{&ctx->P}
                                             : std::vector<std::vector<Layer>*>{&ctx->A, &ctx->T})
            for (Layer& L : *v) {
                CK(cudaMemcpyAsync(L.cW[to], L.cW[from], (size_t)L.out * L.in_ld * ctx->esz, cudaMemcpyDeviceToDevice, s));
                CK(cudaMemcpyAsync(L.cb[to], L.cb[from], (size_t)L.out * 4, cudaMemcpyDeviceToDevice, s));
            }
    CK(cudaEventRecord((passive ? ctx->ev_pver : ctx->ev_aver)[(k + 1) % kEvPool], s));
    return VFL_OK;
}

// The subscriber's side of a dropped step (waiting deadline): no active work, the loss slot(s) NaN,
// the active version carried forward.
vfl_status do_drop_active(vfl_ctx* ctx, long long k) {
    cudaStream_t s = astream(ctx, k);
    PLAUNCH(K_LOSS, 0, 8, s, launch_mark_dropped(ctx->losses + (k % kLossCap), loss_host(ctx, k), s));
    TRY(copy_version_forward(ctx, k, false, s));
    ctx->n_act = k + 1;
    return VFL_OK;
}

// A bottom model's forward as one layer-chain launch when its shape allows (every layer 128 or 256 wide,
// 2-4 layers, an input of at most 256 features); *done = false when it does not (the caller runs the layers).
vfl_status chain_forward(vfl_ctx* ctx, const std::vector<Layer>& Ls, int vslot, const void* X, long long ldx,
                         int rows, void* const* Y, const HeaderOps* hdr, cudaStream_t s, bool* done) {
    *done = false;
    if (!ctx->chain || Ls.size() < 2 || Ls.size() > 4) return VFL_OK;
    int outs[4];
    for (size_t l = 0; l < Ls.size(); ++l) outs[l] = Ls[l].out;
    if (!tc_chain_supported((int)Ls.size(), Ls[0].in, outs)) return VFL_OK;
    TcChain t = {};
    t.L = (int)Ls.size();
    t.M = rows;
    t.K0 = Ls[0].in;
    t.X = X;
    t.ldx = ldx;
    double flops = 0.0, bytes = (double)rows * ldx * ctx->esz;
    for (int l = 0; l < t.L; ++l) {
        const Layer& L = Ls[l];
        t.W[l] = L.cW[vslot];
        t.ldw[l] = L.in_ld;
        t.out[l] = L.out;
        t.bias[l] = L.cb[vslot];
        t.Y[l] = Y[l];
        t.ldy[l] = ld8(L.out);
        flops += 2.0 * rows * L.out * L.in;
        bytes += ((double)L.out * L.in + (double)rows * L.out) * ctx->esz + L.out * 4.0;
    }
    t.err = ctx->status;
    if (hdr) t.hdr = *hdr;
    PLAUNCH(K_TC_CHAIN, flops, bytes, s, launch_tc_chain(t, s));
    *done = true;
    return VFL_OK;
}

vfl_status do_passive_forward(vfl_ctx* ctx, long long k, int tau_p, bool drop = false) {
    const vfl_config& c = ctx->cfg;
    if (k != ctx->n_fwd) return ctx->fail(VFL_E_STATE, "passive_forward(%lld): next publish is step %lld", k, ctx->n_fwd);
    if (tau_p < 0 || tau_p > c.staleness || tau_p > k)
        return ctx->fail(VFL_E_STATE, "passive_forward(%lld): tau_p=%d outside [0, min(k, S=%d)]", k, tau_p, c.staleness);
    const long long v = k - tau_p;
    const long long u = ctx->n_bwd;  // passive updates enqueued
    if (ctx->psmode) {
        if (u < ps_need_bwd(ctx, k))
            return ctx->fail(VFL_E_STATE, "passive_forward(%lld): the update or averaging its replica follows is not "
                             "enqueued yet (%lld updates)", k, u);
    } else if (v > u) {
        return ctx->fail(VFL_E_STATE, "passive_forward(%lld): passive version %lld not produced yet (%lld updates)", k, v, u);
    } else if (v < u - c.staleness) {
        return ctx->fail(VFL_E_STATE, "passive_forward(%lld): passive version %lld no longer stored", k, v);
    }
    record_step(ctx, k, drop);
    cudaStream_t s = pstream(ctx, k);
    const int slot = (int)(k % ctx->S1);
    const int vslot = (int)(v % ctx->S1);
    long long r0;
    const int rows = ctx->batch_rows(k, &r0);
    TRY(wait_version(ctx, k, v, true, s));
    if (ctx->hio) {
        TRY(stage_step(ctx, k));
        TRY(wait_ev(ctx, s, ctx->ev_staged[k % kEvPool]));
    }
    const void* X = xp_rows(ctx, k, r0);
    if (ctx->fused) {
        const bool pdl = use_direct_pdl(ctx);
        TRY(fused_passive_forward(ctx, k, v, slot, vslot, rows, static_cast<const float*>(X), (int)(k % ctx->W), s));
        note_node(ctx, CAP_PFWD, k, s);
        if (!pdl) CK(cudaEventRecord(ctx->ev_emb[k % kEvPool], s));
        ctx->fwd_version[slot] = (int)v;
        ctx->slot_step_p[slot] = k;
        ctx->x_emb += (long long)rows * ctx->P.back().out * ctx->esz;
        ctx->n_fwd = k + 1;
        ctx->started = true;
        return VFL_OK;
    }
    long long ldx = ctx->ldxp;
    // the embedding's header is published by the kernel that writes the payload last
    HeaderOps pub{};
    pub.pub = ctx->emb_hdr + slot;
    pub.k = k;
    pub.batch = (int)ctx->batch_of(k);
    pub.version = (int)v;
    bool chained = false;
    TRY(chain_forward(ctx, ctx->P, vslot, X, ldx, rows, ctx->act_p[slot].data(), emb_dp(ctx) ? nullptr : &pub, s,
                      &chained));
    if (!chained) {
        for (size_t l = 0; l < ctx->P.size(); ++l) {
            const Layer& L = ctx->P[l];
            void* Y = ctx->act_p[slot][l];
            const bool publish = l + 1 == ctx->P.size() && !emb_dp(ctx);
            TRY(linear_fwd(ctx, L, vslot, X, ldx, nullptr, 0, 0, rows, Y, ld8(L.out), true, false, s,
                           publish ? &pub : nullptr));
            X = Y;
            ldx = ld8(L.out);
        }
    }
    if (emb_dp(ctx)) {   // App. C: the published embedding is clipped and noised; z stays for the backward
        const int ep = ctx->P.back().out;
        PLAUNCH(K_DP, 0, (double)rows * ep * 2 * ctx->esz + rows * 4.0, s,
                launch_dp_emb(ctx->act_p[slot].back(), ld8(ep), ctx->bf16, ctx->emb_pub[slot], ctx->emb_c[slot], rows,
                              ep, c.dp_clip, c.dp_sigma, c.dp_seed, k, s));
        PLAUNCH(K_HEADER, 0, 16, s, launch_write_header(ctx->emb_hdr + slot, k, (int)ctx->batch_of(k), (int)v, s));
    }
    CK(cudaEventRecord(ctx->ev_emb[k % kEvPool], s));
    ctx->fwd_version[slot] = (int)v;
    ctx->slot_step_p[slot] = k;
    ctx->x_emb += (long long)rows * ctx->P.back().out * ctx->esz;
    ctx->n_fwd = k + 1;
    ctx->started = true;
    return VFL_OK;
}

vfl_status do_active_step(vfl_ctx* ctx, long long k, int tau_a) {
    const vfl_config& c = ctx->cfg;
    if (k != ctx->n_act) return ctx->fail(VFL_E_STATE, "active_step(%lld): next active step is %lld", k, ctx->n_act);
    if (k >= ctx->n_fwd) return ctx->fail(VFL_E_STATE, "active_step(%lld): embedding not published yet", k);
    if (ctx->dropped(k)) return do_drop_active(ctx, k);
    if (tau_a < 0 || tau_a > c.staleness || tau_a > k)
        return ctx->fail(VFL_E_STATE, "active_step(%lld): tau_a=%d outside [0, min(k, S=%d)]", k, tau_a, c.staleness);
    const long long v = k - tau_a;
    const int w = (int)(k % ctx->W);
    cudaStream_t s = astream(ctx, k);
    const int slot = (int)(k % ctx->S1);
    const int vslot = (int)(v % ctx->S1);
    long long r0;
    const int rows = ctx->batch_rows(k, &r0);
    const int La = (int)ctx->A.size(), Lt = (int)ctx->T.size(), Lp = (int)ctx->P.size();
    const int ea = ctx->A.back().out, ep = ctx->P.back().out;
    const int n_out = ctx->T.back().out;

    TRY(wait_version(ctx, k, v, false, s));
    // the per-layer path reads x^a's staged rows before it subscribes; the fused kernel launches behind the
    // publisher, which itself waited for the staging
    if (ctx->hio && !ctx->fused) TRY(wait_ev(ctx, s, ctx->ev_staged[k % kEvPool]));
    const void* Xa0 = xa_rows(ctx, k, r0);
    if (ctx->fused) {
        TRY(wait_ev(ctx, s, ctx->ev_emb[k % kEvPool]));
        const bool pdl = use_direct_pdl(ctx);
        TRY(fused_active_step(ctx, k, v, slot, vslot, rows, static_cast<const float*>(Xa0), w, s));
        note_node(ctx, CAP_ACTIVE, k, s);
        if (!pdl) CK(cudaEventRecord(ctx->ev_grad[k % kEvPool], s));
        // SGD on theta_1 in step order: version k+1 from version k
        TRY(wait_update_order(ctx, k, false, s));
        TRY(fused_active_update(ctx, k, rows, static_cast<const float*>(Xa0), w, s));
        note_node(ctx, CAP_AUPD, k, s);
        CK(cudaEventRecord(ctx->ev_aver[(k + 1) % kEvPool], s));
        if (ps_agg_at(ctx, k)) TRY(ps_average(ctx, k, false, s));
        ctx->grad_step[slot] = k;
        ctx->x_grad += (long long)rows * ep * ctx->esz;
        ctx->last_act_step[w] = k;
        ctx->n_act = k + 1;
        return VFL_OK;
    }
    // active bottom forward: z^a = f_a(x^a)
    const void* X = Xa0;
    long long ldx = ctx->ldxa;
    bool chained = false;
    TRY(chain_forward(ctx, ctx->A, vslot, X, ldx, rows, ctx->act_a[w].data(), nullptr, s, &chained));
    if (!chained) {
        for (int l = 0; l < La; ++l) {
            const Layer& L = ctx->A[l];
            TRY(linear_fwd(ctx, L, vslot, X, ldx, nullptr, 0, 0, rows, ctx->act_a[w][l], ld8(L.out), true, false, s));
            X = ctx->act_a[w][l];
            ldx = ld8(L.out);
        }
    }
    // subscribe: wait for the embedding of step k; the first kernel that reads it checks its header
    TRY(wait_ev(ctx, s, ctx->ev_emb[k % kEvPool]));
    HeaderOps sub{};
    sub.chk = ctx->emb_hdr + slot;
    sub.k = k;
    sub.status = ctx->status;
    const void* Za = ctx->act_a[w][La - 1];
    const void* Zp = emb_dp(ctx) ? ctx->emb_pub[slot] : ctx->act_p[slot][Lp - 1];
    // top forward on [z^a | z^p]; with the head kernel, g's output layer runs with the loss
    const int Lf = ctx->head ? Lt - 1 : Lt;
    for (int l = 0; l < Lf; ++l) {
        const Layer& L = ctx->T[l];
        const bool last = l == Lt - 1;
        void* Y = last ? (void*)ctx->logits[w] : ctx->act_t[w][l];
        const long long ldy = last ? n_out : ld8(L.out);
        if (l == 0)
            TRY(linear_fwd(ctx, L, vslot, Za, ld8(ea), Zp, ld8(ep), ea, rows, Y, ldy, !last, last, s, &sub));
        else
            TRY(linear_fwd(ctx, L, vslot, ctx->act_t[w][l - 1], ld8(ctx->T[l - 1].out), nullptr, 0, 0, rows, Y, ldy,
                           !last, last, s));
    }
    if (ctx->head) {
        // output layer, loss, d(logits), its dW / db partials and the hidden layer's d(pre-activation)
        const Layer& H = ctx->T[Lt - 1];
        HeadArgs h;
        std::memset(&h, 0, sizeof h);
        h.h = ctx->act_t[w][Lt - 2]; h.ldh = ld8(H.in);
        h.W = H.cW[vslot]; h.ldw = H.in_ld;
        h.b = H.cb[vslot];
        h.K = H.in; h.nout = n_out; h.rows = rows; h.loss = c.loss;
        h.y = y_rows(ctx, k, r0);
        h.logits = ctx->logits[w]; h.ds = ctx->ds[w];
        h.dh = ctx->dpre_t[w][Lt - 2]; h.lddh = ld8(H.in);
        h.pW = H.pW[w]; h.pw_stride = (long long)n_out * H.in;
        h.pb = H.pb[w]; h.pb_stride = n_out;
        h.nblk = H.nsplit;
        h.blk_loss = ctx->h_blk_loss[w];
        h.counter = ctx->h_counter + w;
        h.loss_out = ctx->losses + (k % kLossCap);
        h.loss_host = loss_host(ctx, k);
        const double hf = 2.0 * rows * n_out * H.in * 3.0;
        const double hb = (double)rows * H.in * ctx->esz * 2 + (double)n_out * H.in * ctx->esz +
                          (double)rows * (n_out * 8.0 + 4.0) + 4.0 * H.nsplit * ((double)n_out * H.in + n_out);
        PLAUNCH(K_HEAD, hf, hb, s, launch_head(h, s));
    } else {
        // loss and d(logits)
        PLAUNCH(K_LOSS, 0, (double)rows * n_out * 8 + rows * 4.0, s,
                launch_loss(ctx->logits[w], y_rows(ctx, k, r0), rows, n_out, c.loss, ctx->ds[w],
                            ctx->losses + (k % kLossCap), loss_host(ctx, k), s));
    }
    // top backward (the head kernel has done the output layer's part).  Each layer's input gradient runs
    // before its weight gradient: a weight-gradient kernel that applies the SGD step may write the version
    // slot the input gradient reads (tau_a = S), and the published gradient goes out first.
    const bool dp = c.dp_clip > 0.f && c.dp_target == VFL_DP_GRAD;
    const int rep = ps_rep(ctx, k), nslot = new_version_slot(ctx, k);
    // SGD in step order (App. D): the first weight-gradient kernel that applies it follows update k-1
    // (the input gradients and the published gradient before it do not wait)
    bool waited = false;
    auto dw_order = [&]() -> vfl_status {
        if (waited || !ctx->sgd_in_dw) return VFL_OK;
        waited = true;
        return wait_update_order(ctx, k, false, s);
    };
    for (int l = Lf - 1; l >= 0; --l) {
        const Layer& L = ctx->T[l];
        const bool last = l == Lt - 1;
        const void* dpre = last ? (const void*)ctx->ds[w] : ctx->dpre_t[w][l];
        const long long ldd = last ? n_out : ld8(L.out);
        if (l > 0) {
            const long long ldo = ld8(ctx->T[l - 1].out);
            TRY(linear_dx(ctx, L, vslot, dpre, ldd, last, rows, ctx->dpre_t[w][l - 1], ldo, ctx->act_t[w][l - 1],
                          L.in, nullptr, 0, false, nullptr, s));
            TRY(dw_order());
            TRY(linear_dw(ctx, L, w, dpre, ldd, last, ctx->act_t[w][l - 1], ld8(ctx->T[l - 1].out), nullptr, 0, 0,
                          rows, s, rep, nslot));
            continue;
        }
        // split: dz^a (masked -> dpre of the active cut layer), dz^p -> gradient channel (or fp32 for DP)
        // without DP this kernel writes the published gradient and its header
        void* C2 = dp ? (void*)ctx->dzp32[w] : ctx->grad[slot];
        HeaderOps gpub{};
        gpub.pub = ctx->grad_hdr + slot;
        gpub.k = k;
        gpub.batch = (int)ctx->batch_of(k);
        gpub.version = (int)v;
        TRY(linear_dx(ctx, L, vslot, dpre, ldd, last, rows, ctx->dpre_a[w][La - 1], ld8(ea), Za, ea, C2,
                      ld8(ep), dp, nullptr, s, dp ? nullptr : &gpub));
        if (dp) {
            PLAUNCH(K_DP, 0, (double)rows * ep * (4 + ctx->esz), s,
                    launch_dp(ctx->dzp32[w], ld8(ep), ctx->grad[slot], ld8(ep), ctx->bf16, rows, ep, c.dp_clip,
                              c.dp_sigma, c.dp_seed, k, s));
            PLAUNCH(K_HEADER, 0, 16, s,
                    launch_write_header(ctx->grad_hdr + slot, k, (int)ctx->batch_of(k), (int)v, s));
        }
        // publish the gradient
        CK(cudaEventRecord(ctx->ev_grad[k % kEvPool], s));
        ctx->grad_step[slot] = k;
        ctx->x_grad += (long long)rows * ep * ctx->esz;
        TRY(dw_order());
        TRY(linear_dw(ctx, L, w, dpre, ldd, last, Za, ld8(ea), Zp, ld8(ep), ea, rows, s, rep, nslot));
    }
    // active bottom backward
    for (int l = La - 1; l >= 0; --l) {
        const Layer& L = ctx->A[l];
        const void* Xin = l == 0 ? Xa0 : ctx->act_a[w][l - 1];
        const long long ldin = l == 0 ? ctx->ldxa : ld8(ctx->A[l - 1].out);
        if (l > 0) {
            const long long ldo = ld8(ctx->A[l - 1].out);
            TRY(linear_dx(ctx, L, vslot, ctx->dpre_a[w][l], ld8(L.out), false, rows, ctx->dpre_a[w][l - 1], ldo,
                          ctx->act_a[w][l - 1], L.in, nullptr, 0, false, nullptr, s));
        }
        TRY(dw_order());
        TRY(linear_dw(ctx, L, w, ctx->dpre_a[w][l], ld8(L.out), false, Xin, ldin, nullptr, 0, 0, rows, s, rep, nslot));
    }
    // SGD on theta_1 in step order: version k+1 from version k (the layers the weight-gradient kernels
    // did not update)
    if (!waited) TRY(wait_update_order(ctx, k, false, s));
    TRY(sgd(ctx, &ctx->A, &ctx->T, w, rep, nslot, s));
    CK(cudaEventRecord(ctx->ev_aver[(k + 1) % kEvPool], s));
    if (ps_agg_at(ctx, k)) TRY(ps_average(ctx, k, false, s));
    ctx->last_act_step[w] = k;
    ctx->n_act = k + 1;
    return VFL_OK;
}

vfl_status do_passive_backward(vfl_ctx* ctx, long long k) {
    if (k != ctx->n_bwd) return ctx->fail(VFL_E_STATE, "passive_backward(%lld): next backward is %lld", k, ctx->n_bwd);
    if (k >= ctx->n_act) return ctx->fail(VFL_E_STATE, "passive_backward(%lld): gradient not published yet", k);
    if (ctx->dropped(k)) {   // notified of the drop: no backward, the passive version carried forward
        TRY(copy_version_forward(ctx, k, true, pstream(ctx, k)));
        ctx->n_bwd = k + 1;
        return VFL_OK;
    }
    const int w = (int)(k % ctx->W);
    cudaStream_t s = pstream(ctx, k);
    const int slot = (int)(k % ctx->S1);
    const int vslot = ctx->fwd_version[slot] % ctx->S1;
    long long r0;
    const int rows = ctx->batch_rows(k, &r0);
    const int Lp = (int)ctx->P.size();
    const int ep = ctx->P.back().out;
    TRY(wait_ev(ctx, s, ctx->ev_grad[k % kEvPool]));
    if (ctx->fused) {
        const float* Xp = static_cast<const float*>(xp_rows(ctx, k, r0));
        TRY(fused_passive_backward(ctx, k, slot, vslot, rows, w, s));
        note_node(ctx, CAP_PBWD, k, s);
        // SGD on theta_2 in step order
        TRY(wait_update_order(ctx, k, true, s));
        TRY(fused_passive_update(ctx, k, slot, rows, Xp, w, s));
        note_node(ctx, CAP_PUPD, k, s);
        CK(cudaEventRecord(ctx->ev_pver[(k + 1) % kEvPool], s));
        if (ps_agg_at(ctx, k)) TRY(ps_average(ctx, k, true, s));
        ctx->n_bwd = k + 1;
        return VFL_OK;
    }
    // dpre of the cut layer = dLoss/dz^p * [z^p > 0]; with DP on the embedding the received gradient is
    // first scaled by the row's clip factor (straight-through backward of the mechanism); the kernel checks
    // the gradient's header
    HeaderOps sub{};
    sub.chk = ctx->grad_hdr + slot;
    sub.k = k;
    sub.status = ctx->status;
    PLAUNCH(K_MASK, 0, 3.0 * rows * ep * ctx->esz, s,
            launch_relu_mask(ctx->grad[slot], ctx->act_p[slot][Lp - 1], ctx->dpre_p[w][Lp - 1], ld8(ep), rows, ep,
                             ctx->bf16, emb_dp(ctx) ? ctx->emb_c[slot] : nullptr, sub, s));
    const void* Xp0 = xp_rows(ctx, k, r0);
    const int rep = ps_rep(ctx, k), nslot = new_version_slot(ctx, k);
    bool waited = false;
    for (int l = Lp - 1; l >= 0; --l) {
        const Layer& L = ctx->P[l];
        const void* Xin = l == 0 ? Xp0 : ctx->act_p[slot][l - 1];
        const long long ldin = l == 0 ? ctx->ldxp : ld8(ctx->P[l - 1].out);
        // the input gradient reads the version the forward used, which this step's SGD may overwrite
        if (l > 0) {
            const long long ldo = ld8(ctx->P[l - 1].out);
            TRY(linear_dx(ctx, L, vslot, ctx->dpre_p[w][l], ld8(L.out), false, rows, ctx->dpre_p[w][l - 1], ldo,
                          ctx->act_p[slot][l - 1], L.in, nullptr, 0, false, nullptr, s));
        }
        // SGD in step order (App. D): the first weight-gradient kernel that applies it follows update k-1
        if (ctx->sgd_in_dw && !waited) {
            waited = true;
            TRY(wait_update_order(ctx, k, true, s));
        }
        TRY(linear_dw(ctx, L, w, ctx->dpre_p[w][l], ld8(L.out), false, Xin, ldin, nullptr, 0, 0, rows, s, rep, nslot));
    }
    if (!waited) TRY(wait_update_order(ctx, k, true, s));
    TRY(sgd(ctx, &ctx->P, nullptr, w, rep, nslot, s));
    CK(cudaEventRecord(ctx->ev_pver[(k + 1) % kEvPool], s));
    if (ps_agg_at(ctx, k)) TRY(ps_average(ctx, k, true, s));
    ctx->n_bwd = k + 1;
    return VFL_OK;
}

vfl_status read_status(vfl_ctx* ctx) {
    int st = 0;
    CK(cudaMemcpy(&st, ctx->status, sizeof(int), cudaMemcpyDeviceToHost));
    if (st) {
        CK(cudaMemset(ctx->status, 0, sizeof(int)));
        if (st & ST_VERSION) return ctx->fail(VFL_E_VERSION, "a subscriber found a channel header of another step");
        if (st & ST_TIMEOUT) return ctx->fail(VFL_E_TIMEOUT, "a bounded channel wait gave up");
        if (st & ST_KERNEL_TIMEOUT)
            return ctx->fail(VFL_E_TIMEOUT, "a tensor-core GEMM gave up waiting on its pipeline");
    }
    return VFL_OK;
}

// Every stream the context enqueues on: the workers' (passive, active), then the I/O pair.
int ctx_streams(const vfl_ctx* ctx, cudaStream_t* out) {
    int n = 0;
    for (int w = 0; w < ctx->W; ++w) {
        out[n++] = ctx->ps[w];
        out[n++] = ctx->as[w];
    }
    if (ctx->hio) out[n++] = ctx->io;
    return n;
}
constexpr int kMaxStreams = 2 * kMaxWorkers + 1;

vfl_status sync_all(vfl_ctx* ctx) {
    cudaStream_t ss[kMaxStreams];
    const int n = ctx_streams(ctx, ss);
    for (int i = 0; i < n; ++i) CK(cudaStreamSynchronize(ss[i]));
    return read_status(ctx);
}

Layer* find_layer(vfl_ctx* ctx, int party, int layer) {
    std::vector<Layer>* v = party == 0 ? &ctx->P : party == 1 ? &ctx->A : party == 2 ? &ctx->T : nullptr;
    if (!v || layer < 0 || layer >= (int)v->size()) return nullptr;
    return &(*v)[layer];
}

}  // namespace

namespace vfl {
void set_global_error(const char* msg) { g_global_err = msg; }
}  // namespace vfl

namespace {
// Philox4x32-10 with counter (k lo, k hi, c2, c3) and key (seed lo, seed hi): the four output words.
void philox4(uint64_t seed, int64_t k, uint32_t c2, uint32_t c3, uint32_t out[4]) {
    uint32_t c[4] = {(uint32_t)(k & 0xFFFFFFFFu), (uint32_t)((uint64_t)k >> 32), c2, c3};
    uint32_t key[2] = {(uint32_t)(seed & 0xFFFFFFFFu), (uint32_t)(seed >> 32)};
    for (int r = 0; r < 10; ++r) {
        const uint64_t p0 = (uint64_t)0xD2511F53u * c[0];
        const uint64_t p1 = (uint64_t)0xCD9E8D57u * c[2];
        const uint32_t n0 = (uint32_t)(p1 >> 32) ^ c[1] ^ key[0];
        const uint32_t n2 = (uint32_t)(p0 >> 32) ^ c[3] ^ key[1];
        c[0] = n0;
        c[1] = (uint32_t)p1;
        c[2] = n2;
        c[3] = (uint32_t)p0;
        key[0] += 0x9E3779B9u;
        key[1] += 0xBB67AE85u;
    }
    for (int j = 0; j < 4; ++j) out[j] = c[j];
}
uint32_t philox_word0(uint64_t seed, int64_t k, uint32_t c2, uint32_t c3) {
    uint32_t w[4];
    philox4(seed, k, c2, c3, w);
    return w[0];
}
}  // namespace

// ============================================================================
// C ABI
// ============================================================================
extern "C" {

vfl_status vfl_workspace_bytes(const vfl_config* cfg, int64_t n_rows, uint64_t* bytes) {
    std::string why;
    if (!bytes) return VFL_E_INVAL;
    vfl_status st = check_config(cfg, n_rows, &why);
    if (st != VFL_OK) {
        g_global_err = why;
        return st;
    }
    vfl_ctx tmp;
    tmp.cfg = *cfg;
    tmp.n_rows = n_rows;
    tmp.psmode = cfg->ps_dt0 > 0;
    tmp.W = cfg->workers;
    tmp.S1 = tmp.psmode ? tmp.W : cfg->staleness + 1;
    tmp.bf16 = cfg->dtype == VFL_BF16;
    tmp.esz = tmp.bf16 ? 2 : 4;
    tmp.fused = fused_eligible(*cfg) && !getenv("VFL_DISABLE_FUSED");
    tmp.head = head_eligible(*cfg) && !getenv("VFL_DISABLE_HEAD");
    build_layers(&tmp);
    *bytes = carve_all(&tmp, nullptr);
    return VFL_OK;
}

vfl_status vfl_create(const vfl_config* cfg, int64_t n_rows, void* workspace, uint64_t workspace_bytes,
                      vfl_ctx** out) {
    if (!out) return VFL_E_INVAL;
    *out = nullptr;
    std::string why;
    vfl_status st = check_config(cfg, n_rows, &why);
    if (st != VFL_OK) {
        g_global_err = why;
        return st;
    }
    if (!workspace || (reinterpret_cast<uintptr_t>(workspace) & 255)) {
        g_global_err = "workspace must be a non-null, 256-byte aligned device pointer";
        return VFL_E_INVAL;
    }
    vfl_ctx* ctx = new vfl_ctx();
    ctx->cfg = *cfg;
    ctx->n_rows = n_rows;
    ctx->psmode = cfg->ps_dt0 > 0;
    ctx->W = cfg->workers;
    ctx->S1 = ctx->psmode ? ctx->W : cfg->staleness + 1;
    ctx->bf16 = cfg->dtype == VFL_BF16;
    ctx->esz = ctx->bf16 ? 2 : 4;
    ctx->nb = (int)((n_rows + cfg->batch - 1) / cfg->batch);
    for (int s = 0; s < kMaxSlots; ++s) ctx->slot_step_p[s] = ctx->grad_step[s] = -1;
    for (int w = 0; w < kMaxWorkers; ++w) ctx->last_act_step[w] = -1;
    for (int i = 0; i < kInfoRing; ++i) ctx->step_id[i] = -1;
    ctx->fused = fused_eligible(*cfg) && !getenv("VFL_DISABLE_FUSED");
    ctx->head = head_eligible(*cfg) && !getenv("VFL_DISABLE_HEAD");
    ctx->chain = cfg->dtype == VFL_BF16 && !ctx->fused && !getenv("VFL_DISABLE_CHAIN");
    ctx->direct_pdl = !getenv("VFL_DISABLE_DIRECT_PDL");
    build_layers(ctx);
    const unsigned long long need = carve_all(ctx, nullptr);
    if (workspace_bytes < need) {
        g_global_err = "workspace too small: need " + std::to_string(need) + " bytes";
        delete ctx;
        return VFL_E_OOM;
    }
    carve_all(ctx, workspace);
    ctx->ws_bytes = need;
    cudaError_t e = cudaSuccess;
    for (int i = 0; i < kEvPool && e == cudaSuccess; ++i) {
        e = cudaEventCreateWithFlags(&ctx->ev_pver[i], cudaEventDisableTiming);
        if (e == cudaSuccess) e = cudaEventCreateWithFlags(&ctx->ev_aver[i], cudaEventDisableTiming);
        if (e == cudaSuccess) e = cudaEventCreateWithFlags(&ctx->ev_emb[i], cudaEventDisableTiming);
        if (e == cudaSuccess) e = cudaEventCreateWithFlags(&ctx->ev_grad[i], cudaEventDisableTiming);
        if (e == cudaSuccess) e = cudaEventCreateWithFlags(&ctx->ev_staged[i], cudaEventDisableTiming);
        if (e == cudaSuccess && ctx->psmode) e = cudaEventCreateWithFlags(&ctx->ev_pavg[i], cudaEventDisableTiming);
        if (e == cudaSuccess && ctx->psmode) e = cudaEventCreateWithFlags(&ctx->ev_aavg[i], cudaEventDisableTiming);
    }
    if (e == cudaSuccess) e = cudaMemset(workspace, 0, need);
    if (e == cudaSuccess) e = cudaMemset(ctx->emb_hdr, 0xFF, sizeof(ChannelHeader) * ctx->S1);
    if (e == cudaSuccess) e = cudaMemset(ctx->grad_hdr, 0xFF, sizeof(ChannelHeader) * ctx->S1);
    if (e == cudaSuccess && ctx->psmode) {
        // the averaging kernel's layer table: per party, flat offsets from 0
        std::vector<PsAvgLayer> tab;
        for (std::vector<Layer>* v : {&ctx->P, &ctx->A, &ctx->T}) {
            long long& total = ctx->ps_total[v == &ctx->P ? 0 : 1];
            for (const Layer& L : *v) {
                PsAvgLayer t;
                std::memset(&t, 0, sizeof t);
                for (int w = 0; w < ctx->W; ++w) {
                    t.Wr[w] = L.Wr[w];
                    t.br[w] = L.br[w];
                    t.cW[w] = L.cW[w];
                    t.cb[w] = L.cb[w];
                }
                t.out = L.out;
                t.in = L.in;
                t.in_ld = L.in_ld;
                t.begin = total;
                total += (long long)L.out * L.in + L.out;
                tab.push_back(t);
            }
        }
        e = cudaMemcpy(ctx->ps_tab, tab.data(), sizeof(PsAvgLayer) * tab.size(), cudaMemcpyHostToDevice);
    }
    if (e == cudaSuccess) e = cudaDeviceSynchronize();
    if (e != cudaSuccess) {
        g_global_err = std::string("vfl_create: ") + cudaGetErrorString(e);
        vfl_destroy(ctx);
        return VFL_E_CUDA;
    }
    *out = ctx;
    return VFL_OK;
}

vfl_status vfl_destroy(vfl_ctx* ctx) {
    if (!ctx) return VFL_OK;
    if (!ctx->broken) {
        cudaStream_t ss[kMaxStreams];
        const int n = ctx_streams(ctx, ss);
        for (int i = 0; i < n; ++i) cudaStreamSynchronize(ss[i]);
    }
    for (vfl_graph*& g : ctx->epoch_graph) {
        vfl_graph_destroy(g);
        g = nullptr;
    }
    for (ProfRec& r : ctx->prof) {
        ctx->ev_spare.push_back(r.e0);
        ctx->ev_spare.push_back(r.e1);
    }
    for (cudaEvent_t e : ctx->ev_spare)
        if (e) cudaEventDestroy(e);
    for (int i = 0; i < kEvPool; ++i) {
        if (ctx->ev_pver[i]) cudaEventDestroy(ctx->ev_pver[i]);
        if (ctx->ev_aver[i]) cudaEventDestroy(ctx->ev_aver[i]);
        if (ctx->ev_emb[i]) cudaEventDestroy(ctx->ev_emb[i]);
        if (ctx->ev_grad[i]) cudaEventDestroy(ctx->ev_grad[i]);
        if (ctx->ev_staged[i]) cudaEventDestroy(ctx->ev_staged[i]);
        if (ctx->ev_pavg[i]) cudaEventDestroy(ctx->ev_pavg[i]);
        if (ctx->ev_aavg[i]) cudaEventDestroy(ctx->ev_aavg[i]);
    }
    delete ctx;
    return VFL_OK;
}

vfl_status vfl_set_streams(vfl_ctx* ctx, int32_t n, void* const* streams) {
    if (!ctx) return VFL_E_INVAL;
    if (ctx->broken) return VFL_E_CUDA;
    if (n != 2 * ctx->W || !streams) return ctx->fail(VFL_E_INVAL, "expected %d streams", 2 * ctx->W);
    TRY(sync_all(ctx));
    for (int w = 0; w < ctx->W; ++w) {
        ctx->ps[w] = static_cast<cudaStream_t>(streams[w]);
        ctx->as[w] = static_cast<cudaStream_t>(streams[ctx->W + w]);
    }
    return VFL_OK;
}

vfl_status vfl_load_data(vfl_ctx* ctx, const float* xp, const float* xa, const int32_t* y) {
    if (!ctx || !xp || !xa || !y) return ctx ? ctx->fail(VFL_E_INVAL, "null data pointer") : VFL_E_INVAL;
    if (ctx->broken) return VFL_E_CUDA;
    TRY(sync_all(ctx));
    const vfl_config& c = ctx->cfg;
    const int n_out = ctx->T.back().out;
    for (long long i = 0; i < ctx->n_rows; ++i) {
        const int v = y[i];
        if (v < 0 || v >= (c.loss == VFL_LOSS_BCE ? 2 : n_out))
            return ctx->fail(VFL_E_INVAL, "label %d at row %lld outside the label range", v, i);
    }
    cudaStream_t s = ctx->ps[0];
    for (long long r = 0; r < ctx->n_rows; r += c.batch) {
        const int n = (int)std::min<long long>(c.batch, ctx->n_rows - r);
        CK(cudaMemcpyAsync(ctx->stage_p, xp + r * c.d_passive, (size_t)n * c.d_passive * 4, cudaMemcpyHostToDevice, s));
        PLAUNCH(K_CAST, 0, 0, s, launch_cast_rows(ctx->stage_p, n, c.d_passive,
                                static_cast<char*>(ctx->Xp) + r * ctx->ldxp * ctx->esz, ctx->ldxp, ctx->bf16, s));
        CK(cudaMemcpyAsync(ctx->stage_a, xa + r * c.d_active, (size_t)n * c.d_active * 4, cudaMemcpyHostToDevice, s));
        PLAUNCH(K_CAST, 0, 0, s, launch_cast_rows(ctx->stage_a, n, c.d_active,
                                static_cast<char*>(ctx->Xa) + r * ctx->ldxa * ctx->esz, ctx->ldxa, ctx->bf16, s));
        CK(cudaStreamSynchronize(s));
    }
    CK(cudaMemcpy(ctx->Y, y, (size_t)ctx->n_rows * 4, cudaMemcpyHostToDevice));
    return VFL_OK;
}

namespace {
// The device-side address of host memory that kernels may read or write: page-locked memory
// registered with CUDA, or any host memory on a device that accesses pageable memory coherently.
const void* device_view(const void* p) {
    cudaPointerAttributes at;
    if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
        cudaGetLastError();
        return nullptr;
    }
    if (at.type == cudaMemoryTypeHost && at.devicePointer) return at.devicePointer;
    int dev = 0, pageable = 0;
    if (at.type == cudaMemoryTypeUnregistered && cudaGetDevice(&dev) == cudaSuccess &&
        cudaDeviceGetAttribute(&pageable, cudaDevAttrPageableMemoryAccessUsesHostPageTables, dev) == cudaSuccess &&
        pageable)
        return p;
    return nullptr;
}
}  // namespace

vfl_status bind_host_data(vfl_ctx* ctx, const void* xp, const void* xa, const int32_t* y, float* loss_out,
                          int64_t loss_cap, void* io_stream, int esz) {
    if (!ctx) return VFL_E_INVAL;
    if (ctx->broken) return VFL_E_CUDA;
    if (ctx->n_fwd != ctx->n_bwd || ctx->n_act != ctx->n_bwd)
        return ctx->fail(VFL_E_STATE, "vfl_bind_host_data with steps in flight");
    if (!xp) {
        TRY(sync_all(ctx));
        ctx->hio = false;
        ctx->h_copy = false;
        ctx->hc_xp = ctx->hc_xa = nullptr;
        ctx->hc_y = nullptr;
        ctx->h_xp = ctx->h_xa = nullptr;
        ctx->h_y = nullptr;
        ctx->hv_xp = ctx->hv_xa = nullptr;
        ctx->h_loss = nullptr;
        ctx->h_loss_cap = 0;
        ctx->io = nullptr;
        return VFL_OK;
    }
    if (!xa || !y || !io_stream) return ctx->fail(VFL_E_INVAL, "null host array or I/O stream");
    if (loss_out && loss_cap < 1) return ctx->fail(VFL_E_INVAL, "loss_cap must be >= 1");
    for (int w = 0; w < ctx->W; ++w)
        if (io_stream == ctx->ps[w] || io_stream == ctx->as[w])
            return ctx->fail(VFL_E_INVAL, "the I/O stream must not be a worker stream");
    const int n_cls = ctx->cfg.loss == VFL_LOSS_BCE ? 2 : ctx->T.back().out;
    for (long long i = 0; i < ctx->n_rows; ++i)
        if (y[i] < 0 || y[i] >= n_cls) return ctx->fail(VFL_E_INVAL, "label %d of row %lld outside [0, %d)", y[i], i, n_cls);
    const void* dxp = device_view(xp);
    const void* dxa = device_view(xa);
    const void* dy = device_view(y);
    const void* dl = loss_out ? device_view(loss_out) : nullptr;
    if (!dxp || !dxa || !dy || (loss_out && !dl))
        return ctx->fail(VFL_E_INVAL, "host arrays must be page-locked (cudaHostAlloc / cudaHostRegister)");
    TRY(sync_all(ctx));
    ctx->h_xp = static_cast<const float*>(dxp);
    ctx->h_xa = static_cast<const float*>(dxa);
    ctx->h_y = static_cast<const int32_t*>(dy);
    ctx->hv_xp = dxp;
    ctx->hv_xa = dxa;
    ctx->h_esz = esz;
    // the copy engines stage the rows when the host holds them page-locked in the slots' own layout
    auto pinned = [](const void* q) {
        cudaPointerAttributes at;
        const bool ok = cudaPointerGetAttributes(&at, q) == cudaSuccess && at.type == cudaMemoryTypeHost;
        cudaGetLastError();
        return ok;
    };
    const char* no_copy = std::getenv("VFL_DISABLE_COPY_STAGING");
    ctx->h_copy = esz == ctx->esz && ctx->ldxp == ctx->cfg.d_passive && ctx->ldxa == ctx->cfg.d_active &&
                  pinned(xp) && pinned(xa) && pinned(y) && !(no_copy && *no_copy && *no_copy != '0');
    ctx->hc_xp = static_cast<const char*>(xp);
    ctx->hc_xa = static_cast<const char*>(xa);
    ctx->hc_y = y;
    ctx->h_loss = static_cast<float*>(const_cast<void*>(dl));
    ctx->h_loss_cap = loss_out ? loss_cap : 0;
    ctx->io = static_cast<cudaStream_t>(io_stream);
    ctx->hio = true;
    return VFL_OK;
}

vfl_status vfl_bind_host_data(vfl_ctx* ctx, const float* xp, const float* xa, const int32_t* y, float* loss_out,
                              int64_t loss_cap, void* io_stream) {
    return bind_host_data(ctx, xp, xa, y, loss_out, loss_cap, io_stream, 4);
}

vfl_status vfl_bind_host_data_bf16(vfl_ctx* ctx, const uint16_t* xp, const uint16_t* xa, const int32_t* y,
                                   float* loss_out, int64_t loss_cap, void* io_stream) {
    if (!ctx) return VFL_E_INVAL;
    if (xp && !ctx->bf16) return ctx->fail(VFL_E_INVAL, "bf16 host data needs a bf16 context");
    return bind_host_data(ctx, xp, xa, y, loss_out, loss_cap, io_stream, 2);
}

vfl_status vfl_bind_host_data_bits(vfl_ctx* ctx, const uint32_t* xp_bits, const uint32_t* xa_bits, const int32_t* y,
                                   float* loss_out, int64_t loss_cap, void* io_stream) {
    return bind_host_data(ctx, xp_bits, xa_bits, y, loss_out, loss_cap, io_stream, 0);
}

vfl_status vfl_set_params(vfl_ctx* ctx, int32_t party, int32_t layer, const float* W, const float* b) {
    if (!ctx || !W || !b) return ctx ? ctx->fail(VFL_E_INVAL, "null parameter pointer") : VFL_E_INVAL;
    if (ctx->broken) return VFL_E_CUDA;
    if (ctx->started) return ctx->fail(VFL_E_STATE, "vfl_set_params after the first step");
    Layer* L = find_layer(ctx, party, layer);
    if (!L) return ctx->fail(VFL_E_INVAL, "no layer %d of party %d", layer, party);
    TRY(sync_all(ctx));
    const size_t nw = (size_t)L->out * L->in;
    // every replica (one unless in the parameter-server mode) starts from the same master
    for (int w = 0; w < (ctx->psmode ? ctx->W : 1); ++w) {
        CK(cudaMemcpy(L->Wr[w], W, nw * 4, cudaMemcpyHostToDevice));
        CK(cudaMemcpy(L->br[w], b, (size_t)L->out * 4, cudaMemcpyHostToDevice));
    }
    // every version slot gets the same compute copy (padding columns stay zero)
    for (int s = 0; s < ctx->S1; ++s) {
        CK(cudaMemset(L->cW[s], 0, (size_t)L->out * L->in_ld * ctx->esz));
        PLAUNCH(K_CAST, 0, 0, 0, launch_cast_rows(L->W, L->out, L->in, L->cW[s], L->in_ld, ctx->bf16, 0));
        CK(cudaMemcpy(L->cb[s], b, (size_t)L->out * 4, cudaMemcpyHostToDevice));
    }
    CK(cudaDeviceSynchronize());
    return VFL_OK;
}

vfl_status vfl_init_params(vfl_ctx* ctx, uint64_t seed) {
    if (!ctx) return VFL_E_INVAL;
    if (ctx->broken) return VFL_E_CUDA;
    if (ctx->started) return ctx->fail(VFL_E_STATE, "vfl_init_params after the first step");
    for (std::vector<Layer>* v : {&ctx->P, &ctx->A, &ctx->T})
        for (const Layer& L : *v) {
            const long long nw = (long long)L.out * L.in, n = nw + L.out;
            std::vector<float> vals((size_t)n);
            const uint32_t sub = ((uint32_t)L.party << 8) | (uint32_t)L.idx;
            const double scale = 1.0 / std::sqrt((double)L.in);
            for (long long blk = 0; blk * 4 < n; ++blk) {
                uint32_t w[4];
                philox4(seed, blk, sub, 0x49u, w);
                for (int j = 0; j < 4 && blk * 4 + j < n; ++j) {
                    const double u = (double)w[j] * (1.0 / 4294967296.0);
                    vals[(size_t)(blk * 4 + j)] = (float)((2.0 * u - 1.0) * scale);
                }
            }
            TRY(vfl_set_params(ctx, L.party, L.idx, vals.data(), vals.data() + nw));
        }
    return VFL_OK;
}

vfl_status vfl_get_params(vfl_ctx* ctx, int32_t party, int32_t layer, float* W, float* b) {
    if (!ctx || !W || !b) return ctx ? ctx->fail(VFL_E_INVAL, "null output pointer") : VFL_E_INVAL;
    if (ctx->broken) return VFL_E_CUDA;
    Layer* L = find_layer(ctx, party, layer);
    if (!L) return ctx->fail(VFL_E_INVAL, "no layer %d of party %d", layer, party);
    TRY(sync_all(ctx));
    CK(cudaMemcpy(W, L->W, (size_t)L->out * L->in * 4, cudaMemcpyDeviceToHost));
    CK(cudaMemcpy(b, L->b, (size_t)L->out * 4, cudaMemcpyDeviceToHost));
    return VFL_OK;
}

vfl_status vfl_get_grads(vfl_ctx* ctx, int32_t party, int32_t layer, int32_t worker, float* dW, float* db) {
    if (!ctx || !dW || !db) return ctx ? ctx->fail(VFL_E_INVAL, "null output pointer") : VFL_E_INVAL;
    if (ctx->broken) return VFL_E_CUDA;
    Layer* L = find_layer(ctx, party, layer);
    if (!L) return ctx->fail(VFL_E_INVAL, "no layer %d of party %d", layer, party);
    if (worker < 0 || worker >= ctx->W) return ctx->fail(VFL_E_INVAL, "worker %d out of range", worker);
    TRY(sync_all(ctx));
    const size_t nw = (size_t)L->out * L->in;
    std::vector<float> pw((size_t)L->nsplit * nw), pb((size_t)L->nsplit_b * L->out);
    CK(cudaMemcpy(pw.data(), L->pW[worker], pw.size() * 4, cudaMemcpyDeviceToHost));
    CK(cudaMemcpy(pb.data(), L->pb[worker], pb.size() * 4, cudaMemcpyDeviceToHost));
    for (size_t i = 0; i < nw; ++i) {
        float a = 0.f;
        for (int z = 0; z < L->nsplit; ++z) a += pw[z * nw + i];
        dW[i] = a;
    }
    for (int i = 0; i < L->out; ++i) {      // as the SGD kernel sums them: fp64, partials in order
        double a = 0.0;
        for (int z = 0; z < L->nsplit_b; ++z) a += pb[(size_t)z * L->out + i];
        db[i] = (float)a;
    }
    return VFL_OK;
}

vfl_status vfl_step_cursor(vfl_ctx* ctx, int64_t* k) {
    if (!ctx || !k) return VFL_E_INVAL;
    if (ctx->broken) return VFL_E_CUDA;
    if (ctx->n_fwd != ctx->n_bwd || ctx->n_act != ctx->n_bwd)
        return ctx->fail(VFL_E_STATE, "steps in flight: %lld published, %lld active, %lld finished", ctx->n_fwd,
                         ctx->n_act, ctx->n_bwd);
    *k = ctx->n_bwd;
    return VFL_OK;
}

vfl_status vfl_set_cursor(vfl_ctx* ctx, int64_t k) {
    if (!ctx) return VFL_E_INVAL;
    if (ctx->broken) return VFL_E_CUDA;
    if (k < 0) return ctx->fail(VFL_E_INVAL, "cursor %lld < 0", (long long)k);
    if (ctx->n_fwd != ctx->n_bwd || ctx->n_act != ctx->n_bwd)
        return ctx->fail(VFL_E_STATE, "vfl_set_cursor with steps in flight");
    TRY(sync_all(ctx));
    ctx->n_fwd = ctx->n_act = ctx->n_bwd = k;
    ctx->n_drops = 0;   // the batches trained so far are k unless vfl_set_drops says otherwise
    for (int i = 0; i < kInfoRing; ++i) ctx->step_id[i] = -1;
    ctx->ordered_floor = std::max<long long>(ctx->ordered_floor, k);
    for (int s = 0; s < kMaxSlots; ++s) ctx->slot_step_p[s] = ctx->grad_step[s] = -1;
    for (int w = 0; w < kMaxWorkers; ++w) ctx->last_act_step[w] = -1;
    ctx->started = true;
    return VFL_OK;
}

vfl_status vfl_get_version(vfl_ctx* ctx, int32_t party, int32_t layer, int64_t v, float* W, float* b) {
    if (!ctx || !W || !b) return ctx ? ctx->fail(VFL_E_INVAL, "null output pointer") : VFL_E_INVAL;
    if (ctx->broken) return VFL_E_CUDA;
    Layer* L = find_layer(ctx, party, layer);
    if (!L) return ctx->fail(VFL_E_INVAL, "no layer %d of party %d", layer, party);
    if (ctx->psmode) return ctx->fail(VFL_E_STATE, "the parameter-server mode stores replicas: use vfl_get_replica");
    int64_t k = 0;
    TRY(vfl_step_cursor(ctx, &k));
    if (v < std::max<int64_t>(0, k - ctx->cfg.staleness) || v > k)
        return ctx->fail(VFL_E_INVAL, "version %lld is not stored (cursor %lld, S=%d)", (long long)v, (long long)k,
                         ctx->cfg.staleness);
    TRY(sync_all(ctx));
    const int slot = (int)(v % ctx->S1);
    ++ctx->launches;
    CK(launch_to_f32(L->cW[slot], L->in_ld, L->out, L->in, ctx->bf16, ctx->scratch_f32, 0));
    CK(cudaMemcpy(W, ctx->scratch_f32, (size_t)L->out * L->in * 4, cudaMemcpyDeviceToHost));
    CK(cudaMemcpy(b, L->cb[slot], (size_t)L->out * 4, cudaMemcpyDeviceToHost));
    return VFL_OK;
}

vfl_status vfl_set_version(vfl_ctx* ctx, int32_t party, int32_t layer, int64_t v, const float* W, const float* b) {
    if (!ctx || !W || !b) return ctx ? ctx->fail(VFL_E_INVAL, "null parameter pointer") : VFL_E_INVAL;
    if (ctx->broken) return VFL_E_CUDA;
    Layer* L = find_layer(ctx, party, layer);
    if (!L) return ctx->fail(VFL_E_INVAL, "no layer %d of party %d", layer, party);
    if (ctx->psmode) return ctx->fail(VFL_E_STATE, "the parameter-server mode stores replicas: use vfl_set_replica");
    int64_t k = 0;
    TRY(vfl_step_cursor(ctx, &k));
    if (v < std::max<int64_t>(0, k - ctx->cfg.staleness) || v > k)
        return ctx->fail(VFL_E_INVAL, "version %lld cannot be stored (cursor %lld, S=%d)", (long long)v, (long long)k,
                         ctx->cfg.staleness);
    TRY(sync_all(ctx));
    const int slot = (int)(v % ctx->S1);
    const size_t nw = (size_t)L->out * L->in;
    // stage through the master's storage when v is not the current version
    float* tmp = ctx->scratch_f32;
    CK(cudaMemcpy(tmp, W, nw * 4, cudaMemcpyHostToDevice));
    CK(cudaMemset(L->cW[slot], 0, (size_t)L->out * L->in_ld * ctx->esz));
    ++ctx->launches;
    CK(launch_cast_rows(tmp, L->out, L->in, L->cW[slot], L->in_ld, ctx->bf16, 0));
    CK(cudaMemcpy(L->cb[slot], b, (size_t)L->out * 4, cudaMemcpyHostToDevice));
    if (v == k) {
        CK(cudaMemcpy(L->W, W, nw * 4, cudaMemcpyHostToDevice));
        CK(cudaMemcpy(L->b, b, (size_t)L->out * 4, cudaMemcpyHostToDevice));
    }
    CK(cudaDeviceSynchronize());
    return VFL_OK;
}

vfl_status vfl_get_replica(vfl_ctx* ctx, int32_t worker, int32_t party, int32_t layer, float* W, float* b) {
    if (!ctx || !W || !b) return ctx ? ctx->fail(VFL_E_INVAL, "null output pointer") : VFL_E_INVAL;
    if (ctx->broken) return VFL_E_CUDA;
    if (!ctx->psmode) return ctx->fail(VFL_E_STATE, "replicas exist only in the parameter-server mode");
    Layer* L = find_layer(ctx, party, layer);
    if (!L) return ctx->fail(VFL_E_INVAL, "no layer %d of party %d", layer, party);
    if (worker < 0 || worker >= ctx->W) return ctx->fail(VFL_E_INVAL, "worker %d out of range", worker);
    int64_t k = 0;
    TRY(vfl_step_cursor(ctx, &k));
    TRY(sync_all(ctx));
    CK(cudaMemcpy(W, L->Wr[worker], (size_t)L->out * L->in * 4, cudaMemcpyDeviceToHost));
    CK(cudaMemcpy(b, L->br[worker], (size_t)L->out * 4, cudaMemcpyDeviceToHost));
    return VFL_OK;
}

vfl_status vfl_set_replica(vfl_ctx* ctx, int32_t worker, int32_t party, int32_t layer, const float* W, const float* b) {
    if (!ctx || !W || !b) return ctx ? ctx->fail(VFL_E_INVAL, "null parameter pointer") : VFL_E_INVAL;
    if (ctx->broken) return VFL_E_CUDA;
    if (!ctx->psmode) return ctx->fail(VFL_E_STATE, "replicas exist only in the parameter-server mode");
    Layer* L = find_layer(ctx, party, layer);
    if (!L) return ctx->fail(VFL_E_INVAL, "no layer %d of party %d", layer, party);
    if (worker < 0 || worker >= ctx->W) return ctx->fail(VFL_E_INVAL, "worker %d out of range", worker);
    int64_t k = 0;
    TRY(vfl_step_cursor(ctx, &k));
    TRY(sync_all(ctx));
    const size_t nw = (size_t)L->out * L->in;
    CK(cudaMemcpy(L->Wr[worker], W, nw * 4, cudaMemcpyHostToDevice));
    CK(cudaMemcpy(L->br[worker], b, (size_t)L->out * 4, cudaMemcpyHostToDevice));
    // replica w's compute copy is version slot w, the cast of its master
    CK(cudaMemset(L->cW[worker], 0, (size_t)L->out * L->in_ld * ctx->esz));
    ++ctx->launches;
    CK(launch_cast_rows(L->Wr[worker], L->out, L->in, L->cW[worker], L->in_ld, ctx->bf16, 0));
    CK(cudaMemcpy(L->cb[worker], b, (size_t)L->out * 4, cudaMemcpyHostToDevice));
    CK(cudaDeviceSynchronize());
    return VFL_OK;
}

vfl_status vfl_ps_interval(int64_t t, int32_t dt0, int64_t* interval) {
    if (t < 1 || dt0 < 1 || !interval) return VFL_E_INVAL;
    *interval = ps_interval(t, dt0);
    return VFL_OK;
}

vfl_status vfl_gdp_sigma(double mu, int64_t batch, int64_t n_rows, int64_t queries, double* sigma) {
    if (!sigma || !(mu > 0.0) || batch < 1 || n_rows < 1 || queries < 1) return VFL_E_INVAL;
    *sigma = (double)batch * std::sqrt((double)queries) / (mu * (double)n_rows);
    return VFL_OK;
}


vfl_status vfl_make_drops(uint64_t seed, double rate, int64_t n_steps, uint8_t* drop) {
    if (!(rate >= 0.0 && rate <= 1.0) || n_steps < 0 || (n_steps > 0 && !drop)) {
        g_global_err = "vfl_make_drops: invalid argument";
        return VFL_E_INVAL;
    }
    const uint64_t thr = rate >= 1.0 ? (1ull << 32) : (uint64_t)std::floor(rate * 4294967296.0);
    for (int64_t k = 0; k < n_steps; ++k)
        drop[k] = thr >= (1ull << 32) || (uint64_t)philox_word0(seed, k, 2u, 0x4452u) < thr ? 1 : 0;
    return VFL_OK;
}

vfl_status vfl_make_schedule(uint64_t seed, int32_t S, int32_t kind, int64_t n_steps, int32_t* tau_p,
                             int32_t* tau_a) {
    if (S < 0 || n_steps < 0 || (n_steps > 0 && (!tau_p || !tau_a))) {
        g_global_err = "vfl_make_schedule: invalid argument";
        return VFL_E_INVAL;
    }
    if (kind != VFL_SCHED_SYNC && kind != VFL_SCHED_MAX && kind != VFL_SCHED_SEEDED) {
        g_global_err = "vfl_make_schedule: unknown kind";
        return VFL_E_INVAL;
    }
    for (int party = 0; party < 2; ++party) {
        int32_t* tau = party == 0 ? tau_p : tau_a;
        int32_t prev = 0;
        for (int64_t k = 0; k < n_steps; ++k) {
            int32_t t = 0;
            if (kind == VFL_SCHED_MAX) {
                t = (int32_t)std::min<int64_t>(k, S);
            } else if (kind == VFL_SCHED_SEEDED && k > 0) {
                // Philox4x32-10, counter (k lo, k hi, party, 0x5343), key (seed lo, seed hi); word 0
                const int64_t u = (int64_t)(philox_word0(seed, k, (uint32_t)party, 0x5343u) % (uint32_t)(S + 1));
                t = (int32_t)std::min<int64_t>(std::min<int64_t>(k, S), std::min<int64_t>(prev + 1, u));
            }
            tau[k] = t;
            prev = t;
        }
    }
    return VFL_OK;
}

vfl_status vfl_passive_forward(vfl_ctx* ctx, int64_t k, int32_t tau_p) {
    if (!ctx) return VFL_E_INVAL;
    if (ctx->broken) return VFL_E_CUDA;
    return do_passive_forward(ctx, k, tau_p);
}

vfl_status vfl_active_step(vfl_ctx* ctx, int64_t k, int32_t tau_a) {
    if (!ctx) return VFL_E_INVAL;
    if (ctx->broken) return VFL_E_CUDA;
    return do_active_step(ctx, k, tau_a);
}

vfl_status vfl_drop_step(vfl_ctx* ctx, int64_t k) {
    if (!ctx) return VFL_E_INVAL;
    if (ctx->broken) return VFL_E_CUDA;
    if (k != ctx->n_act) return ctx->fail(VFL_E_STATE, "drop_step(%lld): next active step is %lld", (long long)k, ctx->n_act);
    if (ctx->n_fwd > k + 1)
        return ctx->fail(VFL_E_STATE, "drop_step(%lld): step %lld is already published with the next batch",
                         (long long)k, ctx->n_fwd - 1);
    if (ctx->n_fwd == k) {   // the embedding never arrived: nothing was published for step k
        record_step(ctx, k, true);
        ctx->n_fwd = k + 1;
        ctx->started = true;
    } else if (!ctx->dropped(k)) {
        ctx->step_drop[k % kInfoRing] = 1;
        ++ctx->n_drops;
    }
    return do_drop_active(ctx, k);
}

vfl_status vfl_set_order(vfl_ctx* ctx, int32_t order) {
    if (!ctx) return VFL_E_INVAL;
    if (order != VFL_ORDER_OVERLAP && order != VFL_ORDER_UNIFORM) return ctx->fail(VFL_E_INVAL, "unknown order %d", order);
    if (ctx->n_fwd != ctx->n_bwd || ctx->n_act != ctx->n_bwd)
        return ctx->fail(VFL_E_STATE, "vfl_set_order with steps in flight");
    ctx->uniform = order == VFL_ORDER_UNIFORM;
    return VFL_OK;
}

vfl_status vfl_get_drops(vfl_ctx* ctx, int64_t* n) {
    if (!ctx || !n) return VFL_E_INVAL;
    *n = ctx->n_drops;
    return VFL_OK;
}

vfl_status vfl_set_drops(vfl_ctx* ctx, int64_t n) {
    if (!ctx) return VFL_E_INVAL;
    if (ctx->broken) return VFL_E_CUDA;
    if (ctx->n_fwd != ctx->n_bwd || ctx->n_act != ctx->n_bwd)
        return ctx->fail(VFL_E_STATE, "vfl_set_drops with steps in flight");
    if (n < 0 || n > ctx->n_fwd) return ctx->fail(VFL_E_INVAL, "drop count %lld outside [0, %lld]", (long long)n, ctx->n_fwd);
    ctx->n_drops = n;
    for (int i = 0; i < kInfoRing; ++i) ctx->step_id[i] = -1;
    return VFL_OK;
}

vfl_status vfl_passive_backward(vfl_ctx* ctx, int64_t k) {
    if (!ctx) return VFL_E_INVAL;
    if (ctx->broken) return VFL_E_CUDA;
    return do_passive_backward(ctx, k);
}

vfl_status vfl_train_steps(vfl_ctx* ctx, int64_t k0, int64_t n_steps, const int32_t* tau_p, const int32_t* tau_a,
                           const uint8_t* drop) {
    if (!ctx) return VFL_E_INVAL;
    if (ctx->broken) return VFL_E_CUDA;
    if (n_steps < 0 || (n_steps > 0 && (!tau_p || !tau_a))) return ctx->fail(VFL_E_INVAL, "invalid schedule arguments");
    if (k0 != ctx->n_fwd || k0 != ctx->n_act || k0 != ctx->n_bwd)
        return ctx->fail(VFL_E_STATE, "vfl_train_steps(%lld): steps before k0 are not all complete", (long long)k0);
    const long long end = k0 + n_steps;
    // Emit each phase as early as its inputs allow, so the publisher of step k+1
    // is queued ahead of the backward of step k whenever tau_p permits.
    while (ctx->n_bwd < end) {
        bool progressed = false;
        while (ctx->n_fwd < end && (ctx->psmode ? ps_need_bwd(ctx, ctx->n_fwd)
                                    : ctx->uniform ? ctx->n_fwd : ctx->n_fwd - tau_p[ctx->n_fwd]) <= ctx->n_bwd) {
            TRY(do_passive_forward(ctx, ctx->n_fwd, tau_p[ctx->n_fwd], drop && drop[ctx->n_fwd]));
            progressed = true;
        }
        while (ctx->n_act < ctx->n_fwd) {
            TRY(do_active_step(ctx, ctx->n_act, tau_a[ctx->n_act]));
            progressed = true;
        }
        if (ctx->n_bwd < ctx->n_act) {
            TRY(do_passive_backward(ctx, ctx->n_bwd));
            progressed = true;
        }
        if (!progressed) return ctx->fail(VFL_E_STATE, "schedule cannot make progress at step %lld", ctx->n_bwd);
    }
    return VFL_OK;
}

vfl_status vfl_train_epoch(vfl_ctx* ctx, int64_t epoch, const int32_t* tau_p, const int32_t* tau_a,
                           const uint8_t* drop, float* mean_loss_out) {
    if (!ctx) return VFL_E_INVAL;
    if (ctx->broken) return VFL_E_CUDA;
    if (epoch < 0) return ctx->fail(VFL_E_INVAL, "epoch %lld < 0", (long long)epoch);
    const long long k0 = epoch * ctx->nb;
    bool own_streams = true;
    for (int w = 0; w < ctx->W; ++w) own_streams = own_streams && ctx->ps[w] && ctx->as[w];
    if (ctx->uniform && !drop && own_streams && !ctx->prof_on) {
        // the epoch replays as a graph: the cached one of its shape updated in place, else a new capture
        vfl_graph*& g = ctx->epoch_graph[k0 % ctx->W];
        if (!g || g->n != ctx->nb || vfl_graph_update(ctx, g, k0, ctx->nb, tau_p, tau_a, nullptr) != VFL_OK) {
            if (ctx->broken) return VFL_E_CUDA;
            if (g) vfl_graph_destroy(g);
            g = nullptr;
            TRY(vfl_graph_capture(ctx, k0, ctx->nb, tau_p, tau_a, nullptr, &g));
        }
        TRY(vfl_graph_launch(ctx, g));
    } else {
        TRY(vfl_train_steps(ctx, k0, ctx->nb, tau_p, tau_a, drop));
    }
    if (!mean_loss_out) return VFL_OK;
    std::vector<float> loss((size_t)ctx->nb);
    TRY(vfl_read_losses(ctx, k0, ctx->nb, loss.data()));
    double tot = 0.0, rows = 0.0;
    for (long long i = 0; i < ctx->nb; ++i) {
        if (ctx->dropped(k0 + i)) continue;
        long long r0;
        const int n = ctx->batch_rows(k0 + i, &r0);
        tot += (double)loss[(size_t)i] * n;
        rows += n;
    }
    *mean_loss_out = rows > 0 ? (float)(tot / rows) : std::numeric_limits<float>::quiet_NaN();
    return VFL_OK;
}

namespace {

// Replace the plain edge from -> to by a programmatic one: `to` may launch once every CTA of `from`
// has signalled (griddepcontrol.launch_dependents) and runs its prologue, waiting in griddepcontrol.wait
// for `from` to complete before it reads from's output.  Left plain when the edge is not a direct one.
void make_programmatic(cudaGraph_t g, cudaGraphNode_t from, cudaGraphNode_t to) {
    if (cudaGraphRemoveDependencies(g, &from, &to, nullptr, 1) != cudaSuccess) {
        cudaGetLastError();
        return;
    }
    cudaGraphEdgeData ed;
    std::memset(&ed, 0, sizeof ed);
    ed.from_port = cudaGraphKernelNodePortProgrammatic;
    ed.type = cudaGraphDependencyTypeProgrammatic;
    if (cudaGraphAddDependencies(g, &from, &to, &ed, 1) != cudaSuccess) {
        cudaGetLastError();
        cudaGraphAddDependencies(g, &from, &to, nullptr, 1);
    }
}

// For each captured step: passive forward -> active step (the active step stages its weights and x^a
// and runs f_a before reading z^p), active step -> passive backward (weights and saved activations
// before dz^p), active step -> active update and passive backward -> passive update (launch latency
// hidden), and the passive update that produced the version a passive forward reads -> that forward
// (rows before the weights).
void programmatic_edges(vfl_ctx* ctx, cudaGraph_t g, long long k0, long long n, const int32_t* tau_p) {
    auto node = [&](int ph, long long k) -> cudaGraphNode_t {
        auto it = ctx->cap_nodes.find({ph, k});
        return it == ctx->cap_nodes.end() ? nullptr : it->second;
    };
    for (long long k = k0; k < k0 + n; ++k) {
        const std::pair<int, int> edges[4] = {
            {CAP_PFWD, CAP_ACTIVE}, {CAP_ACTIVE, CAP_PBWD}, {CAP_ACTIVE, CAP_AUPD}, {CAP_PBWD, CAP_PUPD}};
        for (const auto& ed : edges) {
            cudaGraphNode_t from = node(ed.first, k), to = node(ed.second, k);
            if (from && to) make_programmatic(g, from, to);
        }
        // the update that made the forward's weights: step v - 1 for version v = k - tau_p, the previous
        // step of the worker in the parameter-server mode (no edge when an averaging sits in between)
        // (in the uniform order the forward waits for the previous step's update, whatever it reads)
        const long long src = ctx->psmode ? k - ctx->W : ctx->uniform ? k - 1 : k - tau_p[k] - 1;
        cudaGraphNode_t from = node(CAP_PUPD, src), to = node(CAP_PFWD, k);
        if (from && to) make_programmatic(g, from, to);
    }
    // every other kernel starts by waiting for its producer (pdl_entry), so any remaining plain edge
    // between two kernel nodes whose target is not a fused kernel can be programmatic as well (the fused
    // path's few other kernels -- staging, averaging -- are off its critical chain: the per-edge queries
    // are skipped there, they cost the host more than they save)
    if (ctx->fused) return;
    size_t ne = 0;
    if (cudaGraphGetEdges(g, nullptr, nullptr, nullptr, &ne) != cudaSuccess || ne == 0) {
        cudaGetLastError();
        return;
    }
    std::vector<cudaGraphNode_t> from(ne), to(ne);
    std::vector<cudaGraphEdgeData> ed(ne);
    if (cudaGraphGetEdges(g, from.data(), to.data(), ed.data(), &ne) != cudaSuccess) {
        cudaGetLastError();
        return;
    }
    auto kernel_func = [](cudaGraphNode_t n) -> const void* {
        cudaGraphNodeType t;
        cudaKernelNodeParams kp;
        if (cudaGraphNodeGetType(n, &t) != cudaSuccess || t != cudaGraphNodeTypeKernel ||
            cudaGraphKernelNodeGetParams(n, &kp) != cudaSuccess) {
            cudaGetLastError();
            return nullptr;
        }
        return kp.func;
    };
    for (size_t i = 0; i < ne; ++i) {
        if (ed[i].type == cudaGraphDependencyTypeProgrammatic) continue;
        const void* ff = kernel_func(from[i]);
        const void* tf = kernel_func(to[i]);
        if (ff && tf && !is_fused_kernel(tf)) make_programmatic(g, from[i], to[i]);
    }
}

}  // namespace

}  // extern "C"

namespace {

// Record steps [k0, k0 + n) into a new cudaGraph (through vfl_train_steps on the context's streams in
// capture mode, the fused kernels' programmatic edges added) without running them.  The context's host
// state is left at k0; *after is the state once the captured steps have run.
vfl_status capture_window(vfl_ctx* ctx, vfl_graph* g, long long k0, long long n_steps, const int32_t* tau_p,
                          const int32_t* tau_a, const uint8_t* drop, cudaGraph_t* graph, HostState* after) {
    *graph = nullptr;
    const HostState before = save_state(ctx);
    cudaStream_t origin = ctx->ps[0];
    vfl_status st = VFL_OK;
    cudaStream_t ss[kMaxStreams];
    const int nss = ctx_streams(ctx, ss);
    cudaError_t e = cudaStreamBeginCapture(origin, cudaStreamCaptureModeThreadLocal);
    if (e == cudaSuccess) e = cudaEventRecord(g->fork, origin);
    for (int i = 0; i < nss && e == cudaSuccess; ++i)
        if (ss[i] != origin) e = cudaStreamWaitEvent(ss[i], g->fork, 0);
    const long long floor_before = ctx->ordered_floor;
    ctx->ordered_floor = std::max<long long>(ctx->ordered_floor, k0);
    ctx->cap_nodes.clear();
    ctx->capturing = true;
    if (e == cudaSuccess) st = vfl_train_steps(ctx, k0, n_steps, tau_p, tau_a, drop);
    ctx->capturing = false;
    ctx->ordered_floor = floor_before;
    // join every stream back into the origin, even after a failure, so that capture can end
    for (int i = 0; i < nss; ++i)
        if (ss[i] != origin && cudaEventRecord(g->join[i], ss[i]) == cudaSuccess)
            cudaStreamWaitEvent(origin, g->join[i], 0);
    cudaError_t e2 = cudaStreamEndCapture(origin, graph);
    if (e == cudaSuccess) e = e2;
    if (st == VFL_OK && e == cudaSuccess) programmatic_edges(ctx, *graph, k0, n_steps, tau_p);
    ctx->cap_nodes.clear();
    *after = save_state(ctx);
    after->launches -= before.launches;   // kernels per replay
    load_state(ctx, before);
    if (st != VFL_OK || e != cudaSuccess) {
        if (*graph) cudaGraphDestroy(*graph);
        *graph = nullptr;
        if (st != VFL_OK) return st;
        return ctx->cuda(e, "graph capture", __LINE__);
    }
    return VFL_OK;
}

vfl_status check_capture(vfl_ctx* ctx, long long k0) {
    for (int w = 0; w < ctx->W; ++w)
        if (!ctx->ps[w] || !ctx->as[w])
            return ctx->fail(VFL_E_STATE, "graph capture needs the caller's streams (vfl_set_streams)");
    if (k0 != ctx->n_fwd || k0 != ctx->n_act || k0 != ctx->n_bwd)
        return ctx->fail(VFL_E_STATE, "graph capture at %lld: steps before it are not all enqueued", k0);
    return VFL_OK;
}

}  // namespace

extern "C" {

vfl_status vfl_graph_capture(vfl_ctx* ctx, int64_t k0, int64_t n_steps, const int32_t* tau_p, const int32_t* tau_a,
                             const uint8_t* drop,
                             vfl_graph** out) {
    if (!ctx || !out) return VFL_E_INVAL;
    *out = nullptr;
    if (ctx->broken) return VFL_E_CUDA;
    TRY(check_capture(ctx, k0));
    // no synchronisation: earlier steps (a graph being replayed) may still run while the host captures the
    // next window; the capture records work without executing it and its replay is ordered after them
    vfl_graph* g = new vfl_graph();
    g->ctx = ctx;
    g->k0 = k0;
    g->n = n_steps;
    g->drops0 = ctx->n_drops;
    g->hio = ctx->hio;
    cudaError_t e = cudaEventCreateWithFlags(&g->fork, cudaEventDisableTiming);
    for (int i = 0; i < kMaxStreams && e == cudaSuccess; ++i) e = cudaEventCreateWithFlags(&g->join[i], cudaEventDisableTiming);
    if (e != cudaSuccess) {
        vfl_graph_destroy(g);
        return ctx->cuda(e, "cudaEventCreate", __LINE__);
    }
    cudaGraph_t graph = nullptr;
    HostState after;
    vfl_status st = capture_window(ctx, g, k0, n_steps, tau_p, tau_a, drop, &graph, &after);
    if (st != VFL_OK) {
        vfl_graph_destroy(g);
        return st;
    }
    e = cudaGraphInstantiate(&g->exec, graph, 0);
    // upload now (ordered on the origin stream, without waiting), so that the first replay does not pay for it
    if (e == cudaSuccess) e = cudaGraphUpload(g->exec, ctx->ps[0]);
    cudaGraphDestroy(graph);
    if (e != cudaSuccess) {
        vfl_graph_destroy(g);
        return ctx->cuda(e, "graph instantiate", __LINE__);
    }
    g->after = after;
    g->launches = after.launches;
    g->after.launches = 0;
    *out = g;
    return VFL_OK;
}

vfl_status vfl_graph_update(vfl_ctx* ctx, vfl_graph* g, int64_t k0, int64_t n_steps, const int32_t* tau_p,
                            const int32_t* tau_a, const uint8_t* drop) {
    if (!ctx || !g || g->ctx != ctx) return ctx ? ctx->fail(VFL_E_INVAL, "graph of another context") : VFL_E_INVAL;
    if (ctx->broken) return VFL_E_CUDA;
    TRY(check_capture(ctx, k0));
    cudaGraph_t graph = nullptr;
    HostState after;
    TRY(capture_window(ctx, g, k0, n_steps, tau_p, tau_a, drop, &graph, &after));
    cudaGraphExecUpdateResultInfo info;
    cudaError_t e = cudaGraphExecUpdate(g->exec, graph, &info);
    cudaGraphDestroy(graph);
    if (e == cudaErrorGraphExecUpdateFailure) {
        // not performed (another shape of graph): the executable graph still holds its old window
        cudaGetLastError();
        return ctx->fail(VFL_E_STATE, "steps [%lld, %lld) do not fit the graph's shape (update result %d)",
                         (long long)k0, (long long)(k0 + n_steps), (int)info.result);
    }
    if (e != cudaSuccess) return ctx->cuda(e, "cudaGraphExecUpdate", __LINE__);
    g->k0 = k0;
    g->n = n_steps;
    g->drops0 = ctx->n_drops;
    g->hio = ctx->hio;
    g->launches = after.launches;
    g->after = after;
    g->after.launches = 0;
    return VFL_OK;
}

vfl_status vfl_graph_launch(vfl_ctx* ctx, vfl_graph* g) {
    if (!ctx || !g || g->ctx != ctx) return ctx ? ctx->fail(VFL_E_INVAL, "graph of another context") : VFL_E_INVAL;
    if (ctx->broken) return VFL_E_CUDA;
    if (ctx->n_fwd != g->k0 || ctx->n_act != g->k0 || ctx->n_bwd != g->k0)
        return ctx->fail(VFL_E_STATE, "graph starts at step %lld but the context is at step %lld", g->k0, ctx->n_fwd);
    if (g->hio != ctx->hio) return ctx->fail(VFL_E_STATE, "graph captured with another host-data binding");
    if (g->drops0 != ctx->n_drops)
        return ctx->fail(VFL_E_STATE, "graph captured after %lld dropped steps, the context has %lld", g->drops0,
                         ctx->n_drops);
    cudaStream_t origin = ctx->ps[0];
    // order the replay after everything already enqueued on the context's streams, and theirs after it
    cudaStream_t ss[kMaxStreams];
    const int nss = ctx_streams(ctx, ss);
    for (int i = 0; i < nss; ++i) {
        if (ss[i] == origin) continue;
        CK(cudaEventRecord(g->join[i], ss[i]));
        CK(cudaStreamWaitEvent(origin, g->join[i], 0));
    }
    CK(cudaGraphLaunch(g->exec, origin));
    CK(cudaEventRecord(g->fork, origin));
    for (int i = 0; i < nss; ++i)
        if (ss[i] != origin) CK(cudaStreamWaitEvent(ss[i], g->fork, 0));
    const long long launched = ctx->launches + g->launches;
    load_state(ctx, g->after);
    ctx->launches = launched;
    ctx->ordered_floor = std::max<long long>(ctx->ordered_floor, g->k0 + g->n);
    return VFL_OK;
}

vfl_status vfl_graph_destroy(vfl_graph* g) {
    if (!g) return VFL_OK;
    if (g->exec) cudaGraphExecDestroy(g->exec);
    if (g->fork) cudaEventDestroy(g->fork);
    for (cudaEvent_t e : g->join)
        if (e) cudaEventDestroy(e);
    delete g;
    return VFL_OK;
}

vfl_status vfl_synchronize(vfl_ctx* ctx) {
    if (!ctx) return VFL_E_INVAL;
    if (ctx->broken) return VFL_E_CUDA;
    return sync_all(ctx);
}

vfl_status vfl_read_losses(vfl_ctx* ctx, int64_t k0, int64_t n, float* out) {
    if (!ctx || (n > 0 && !out)) return VFL_E_INVAL;
    if (ctx->broken) return VFL_E_CUDA;
    if (k0 < 0 || n < 0 || k0 + n > ctx->n_act || k0 < ctx->n_act - kLossCap)
        return ctx->fail(VFL_E_INVAL, "losses of steps [%lld, %lld) are not stored", (long long)k0, (long long)(k0 + n));
    TRY(sync_all(ctx));
    for (int64_t i = 0; i < n; ++i) {
        CK(cudaMemcpy(out + i, ctx->losses + ((k0 + i) % kLossCap), 4, cudaMemcpyDeviceToHost));
    }
    return VFL_OK;
}

vfl_status vfl_fetch_loss(vfl_ctx* ctx, int64_t k, float* host_out) {
    if (!ctx || !host_out) return VFL_E_INVAL;
    if (ctx->broken) return VFL_E_CUDA;
    if (k < 0 || k >= ctx->n_act || k < ctx->n_act - kLossCap)
        return ctx->fail(VFL_E_INVAL, "loss of step %lld is not stored", (long long)k);
    CK(cudaMemcpyAsync(host_out, ctx->losses + (k % kLossCap), 4, cudaMemcpyDeviceToHost, astream(ctx, k)));
    return VFL_OK;
}

vfl_status vfl_step_rows(vfl_ctx* ctx, int64_t k, int64_t* r0, int32_t* rows) {
    if (!ctx || !r0 || !rows) return VFL_E_INVAL;
    if (k < 0) return ctx->fail(VFL_E_INVAL, "step %lld < 0", (long long)k);
    long long r;
    *rows = ctx->batch_rows(k, &r);
    *r0 = r;
    return VFL_OK;
}

vfl_status vfl_tap(vfl_ctx* ctx, int64_t k, int32_t what, float* out, int64_t out_elems) {
    if (!ctx || !out) return VFL_E_INVAL;
    if (ctx->broken) return VFL_E_CUDA;
    TRY(sync_all(ctx));
    long long r0;
    const int rows = ctx->batch_rows(k, &r0);
    const int slot = (int)(k % ctx->S1);
    const int w = (int)(k % ctx->W);
    const void* src = nullptr;
    long long ld = 0;
    int cols = 0, bf = ctx->bf16;
    const int ep = ctx->P.back().out, ea = ctx->A.back().out;
    switch (what) {
        case VFL_TAP_EMB:
            if (ctx->slot_step_p[slot] != k) return ctx->fail(VFL_E_STATE, "embedding of step %lld is not stored", (long long)k);
            src = emb_dp(ctx) ? ctx->emb_pub[slot] : ctx->act_p[slot].back(); ld = ld8(ep); cols = ep;
            break;
        case VFL_TAP_GRAD:
            if (ctx->grad_step[slot] != k) return ctx->fail(VFL_E_STATE, "gradient of step %lld is not stored", (long long)k);
            src = ctx->grad[slot]; ld = ld8(ep); cols = ep;
            break;
        case VFL_TAP_LOGITS:
        case VFL_TAP_ZA:
        case VFL_TAP_DZA:
            if (ctx->last_act_step[w] != k) return ctx->fail(VFL_E_STATE, "active buffers of step %lld are not stored", (long long)k);
            if (what == VFL_TAP_LOGITS) { src = ctx->logits[w]; ld = ctx->T.back().out; cols = (int)ld; bf = 0; }
            else if (what == VFL_TAP_ZA) { src = ctx->act_a[w].back(); ld = ld8(ea); cols = ea; }
            else { src = ctx->dpre_a[w].back(); ld = ld8(ea); cols = ea; }
            break;
        default: {
            const int party = (what - 16) / 16, layer = (what - 16) % 16;
            if (what < 16 || party > 2) return ctx->fail(VFL_E_INVAL, "unknown tap %d", what);
            if (ctx->fused) return ctx->fail(VFL_E_STATE, "hidden activations are kept by the per-layer kernels only");
            if (party == 0) {
                if (layer >= (int)ctx->P.size()) return ctx->fail(VFL_E_INVAL, "no passive layer %d", layer);
                if (ctx->slot_step_p[slot] != k)
                    return ctx->fail(VFL_E_STATE, "passive activations of step %lld are not stored", (long long)k);
                src = ctx->act_p[slot][layer];
                cols = ctx->P[layer].out;
            } else {
                const std::vector<Layer>& v = party == 1 ? ctx->A : ctx->T;
                const int n = party == 1 ? (int)v.size() : (int)v.size() - 1;
                if (layer >= n) return ctx->fail(VFL_E_INVAL, "no stored layer %d of party %d", layer, party);
                if (ctx->last_act_step[w] != k)
                    return ctx->fail(VFL_E_STATE, "active buffers of step %lld are not stored", (long long)k);
                src = party == 1 ? ctx->act_a[w][layer] : ctx->act_t[w][layer];
                cols = v[layer].out;
            }
            ld = ld8(cols);
            break;
        }
    }
    if ((long long)rows * cols > out_elems)
        return ctx->fail(VFL_E_INVAL, "tap of step %lld needs %lld floats, the buffer holds %lld", (long long)k,
                         (long long)rows * cols, (long long)out_elems);
    ++ctx->launches;
    CK(launch_to_f32(src, ld, rows, cols, bf, ctx->scratch_f32, 0));
    CK(cudaMemcpy(out, ctx->scratch_f32, (size_t)rows * cols * 4, cudaMemcpyDeviceToHost));
    return VFL_OK;
}

vfl_status vfl_wait_channel(vfl_ctx* ctx, int32_t which, int64_t k, int64_t max_iters) {
    if (!ctx) return VFL_E_INVAL;
    if (ctx->broken) return VFL_E_CUDA;
    if ((which != 0 && which != 1) || k < 0 || max_iters < 1 || max_iters > (1ll << 24))
        return ctx->fail(VFL_E_INVAL, "invalid wait arguments");
    TRY(sync_all(ctx));
    const ChannelHeader* h = (which == 0 ? ctx->emb_hdr : ctx->grad_hdr) + (k % ctx->S1);
    PLAUNCH(K_HEADER, 0, 0, ctx->ps[0], launch_wait_header(h, k, max_iters, ctx->status, ctx->ps[0]));
    return sync_all(ctx);
}

vfl_status vfl_check_channel(vfl_ctx* ctx, int32_t which, int64_t k) {
    if (!ctx) return VFL_E_INVAL;
    if (ctx->broken) return VFL_E_CUDA;
    if ((which != 0 && which != 1) || k < 0) return ctx->fail(VFL_E_INVAL, "invalid check arguments");
    TRY(sync_all(ctx));
    const ChannelHeader* h = (which == 0 ? ctx->emb_hdr : ctx->grad_hdr) + (k % ctx->S1);
    PLAUNCH(K_HEADER, 0, 16, ctx->ps[0], launch_check_header(h, k, ctx->status, ctx->ps[0]));
    return sync_all(ctx);
}

int64_t vfl_kernel_launches(const vfl_ctx* ctx) { return ctx ? ctx->launches : 0; }

vfl_status vfl_exchange_bytes(const vfl_ctx* ctx, int64_t* emb, int64_t* grad) {
    if (!ctx || !emb || !grad) return VFL_E_INVAL;
    *emb = ctx->x_emb;
    *grad = ctx->x_grad;
    return VFL_OK;
}

vfl_status vfl_profile(vfl_ctx* ctx, int32_t enable) {
    if (!ctx) return VFL_E_INVAL;
    if (ctx->broken) return VFL_E_CUDA;
    if (enable) {
        for (ProfAgg& a : ctx->agg) a = ProfAgg();
        ctx->prof.clear();
        ctx->prof_on = true;
        return VFL_OK;
    }
    if (!ctx->prof_on) return VFL_OK;
    ctx->prof_on = false;
    TRY(sync_all(ctx));
    for (ProfRec& r : ctx->prof) {
        float ms = 0.f;
        const cudaError_t e = cudaEventElapsedTime(&ms, r.e0, r.e1);
        if (e != cudaSuccess) {
            // launches captured into a graph that has not run yet: nothing to fold
            cudaGetLastError();
            ctx->prof.clear();
            return ctx->fail(VFL_E_STATE, "timed launches have not run (a captured graph not launched?): %s",
                             cudaGetErrorString(e));
        }
        ProfAgg& a = ctx->agg[r.cls];
        a.n += 1;
        a.ms += ms;
        a.flops += r.flops;
        a.bytes += r.bytes;
        ctx->ev_spare.push_back(r.e0);
        ctx->ev_spare.push_back(r.e1);
    }
    ctx->prof.clear();
    return VFL_OK;
}

vfl_status vfl_profile_get(const vfl_ctx* ctx, int32_t cls, int64_t* launches, double* ms, double* flops,
                           double* bytes) {
    if (!ctx || cls < 0 || cls >= K_NCLASS || !launches || !ms || !flops || !bytes) return VFL_E_INVAL;
    const ProfAgg& a = ctx->agg[cls];
    *launches = a.n;
    *ms = a.ms;
    *flops = a.flops;
    *bytes = a.bytes;
    return VFL_OK;
}

const char* vfl_kernel_class_name(int32_t cls) { return cls >= 0 && cls < K_NCLASS ? kClassNames[cls] : nullptr; }

const char* vfl_last_error(const vfl_ctx* ctx) { return ctx ? ctx->err.c_str() : g_global_err.c_str(); }

}  // extern "C"
