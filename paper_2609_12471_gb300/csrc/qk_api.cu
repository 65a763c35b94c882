// libqk C ABI: configuration presets, packed weight layout, model loading,
// workspace layout and the host-side orchestration of the forward pass.
//
// Every entry point validates its arguments on the host before any launch,
// launches only on the caller's stream, never synchronises (except
// qk_check_status) and never allocates device memory.
#include <stdarg.h>
#include <stdio.h>
#include <string.h>

#include <atomic>
#include <new>

#include "qk_internal.cuh"

namespace qk {

static thread_local char g_err[512] = "";
static std::atomic<uint64_t> g_launches{0};

void note_launch(int n) { g_launches.fetch_add((uint64_t)n, std::memory_order_relaxed); }

bool prof_open(Model& m, int kind, cudaStream_t s) {
    if (!m.in_decode || m.prof_kind != kind || m.prof_used + 2 > (int)m.prof_ev.size()) return false;
    cudaEventRecord(m.prof_ev[m.prof_used++], s);
    return true;
}

void prof_close(Model& m, bool opened, cudaStream_t s) {
    if (opened) cudaEventRecord(m.prof_ev[m.prof_used++], s);
}

int set_error(int code, const char* fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_err, sizeof(g_err), fmt, ap);
    va_end(ap);
    return code;
}

int cuda_error(cudaError_t e, const char* what) {
    (void)cudaGetLastError();  // do not leave the error for the next call's launch check
    return set_error(QK_ECUDA, "%s: %s", what, cudaGetErrorString(e));
}

static size_t align256(size_t v) { return (v + 255) & ~(size_t)255; }

int validate_config(const qk_config& c) {
    if (c.dtype != QK_DTYPE_BF16 && c.dtype != QK_DTYPE_F32)
        return set_error(QK_EDTYPE, "dtype %d is neither QK_DTYPE_BF16 nor QK_DTYPE_F32", c.dtype);
    if (c.head_dim != 64 && c.head_dim != 128)
        return set_error(QK_EDTYPE, "head_dim %d unsupported (64 or 128)", c.head_dim);
    if (c.n_layers < 1 || c.n_q_heads < 1 || c.n_kv_heads < 1 || c.n_q_heads % c.n_kv_heads)
        return set_error(QK_ESHAPE, "bad layer / head counts (%d layers, %d q heads, %d kv heads)",
                         c.n_layers, c.n_q_heads, c.n_kv_heads);
    if (c.n_q_heads / c.n_kv_heads > 32)
        return set_error(QK_EDTYPE, "query heads per kv head > 32 unsupported");
    if (c.hidden < 64 || c.hidden % 64)
        return set_error(QK_ESHAPE, "hidden %d must be a positive multiple of 64", c.hidden);
    if (c.intermediate < 128 || c.intermediate % 128)
        return set_error(QK_ESHAPE, "intermediate %d must be a positive multiple of 128", c.intermediate);
    if (c.vocab < 4 || c.vocab % 4)
        return set_error(QK_ESHAPE, "vocab %d must be a positive multiple of 4", c.vocab);
    if (c.max_positions < 1 || c.reserved != 0)
        return set_error(QK_EINVAL, "max_positions must be >= 1 and reserved 0");
    if (!(c.rms_eps > 0.0) || !(c.rope_theta > 1.0))
        return set_error(QK_EINVAL, "rms_eps must be > 0 and rope_theta > 1");
    return QK_OK;
}

int packed_layout(const qk_config& c, PackedLayout* out) {
    QK_TRY(validate_config(c));
    size_t es = c.dtype == QK_DTYPE_BF16 ? 2 : 4;
    size_t H = c.hidden, d = c.head_dim, nq = c.n_q_heads, nkv = c.n_kv_heads, I = c.intermediate,
           V = c.vocab;
    size_t off = 0;
    auto take = [&](size_t bytes) {
        size_t o = off;
        off = align256(off + bytes);
        return o;
    };
    out->status = take(256);
    out->rope_cos = take((size_t)c.max_positions * (d / 2) * 4);
    out->rope_sin = take((size_t)c.max_positions * (d / 2) * 4);
    out->embed = take(V * H * es);
    out->layers.resize(c.n_layers);
    for (int l = 0; l < c.n_layers; ++l) {
        PackedLayout::L& L = out->layers[l];
        L.attn_norm = take(H * 4);
        L.q_norm = take(d * 4);
        L.k_norm = take(d * 4);
        L.mlp_norm = take(H * 4);
        L.w_qkv = take((nq + 2 * nkv) * d * H * es);
        L.w_o = take(H * nq * d * es);
        L.w_gu = take(2 * I * H * es);
        L.w_d = take(H * I * es);
    }
    out->final_norm = take(H * 4);
    out->lm_head = take(V * H * es);
    out->total = off;
    return QK_OK;
}

// ---------------------------------------------------------------- workspace layout
struct Workspace {
    float* x;       // [M, H] fp32 residual stream
    void* u;        // [M, H] normalised input of a linear layer
    void* qkv;      // [M, (nq + 2 nkv) d]
    void* o;        // [M, nq d] attention output
    void* h;        // [M, I] SwiGLU output
    void* gu;       // [M, 2 I] gate/up before SwiGLU (unfused path only)
    void* skv;      // scoring: K and V of one layer, [2][B, nkv, T, d]
    void* attn;     // decode: split-attention partials (bf16 models)
    float* part;    // decode: split-K partial products of the linear layers (bf16 models)
    bf16* xg;       // decode: bf16(x * g) for the next linear's input (fused path)
    float* ssq;     // decode: per-128-feature-tile sums of squares of x [H/128, M]
    int* tickets;   // decode: last-unit tickets of the fused linears
    float* logits;  // [logit_rows, V]
    int logit_rows;
    // scoring of bf16 models: per (row, 128-entry vocabulary tile) softmax statistics
    // formed in the lm_head epilogue instead of logits (null: logits + reduce)
    float2* lse_ms;  // [logit_rows, V / 128]
    int* lse_idx;    // [logit_rows, V / 128]
    float* lse_zt;   // [logit_rows]
    size_t total;
};

static const int kScoreLogitRows = 4096;

// The rollout keeps a cursor (step counter, per-row position / token / target,
// output slot) in 256-byte-aligned slots after the prefill/decode workspace.
static size_t rollout_cursor_bytes(int B) { return 5 * align256((size_t)(B > 1 ? B : 1) * 4); }

static const int kSplitMaxRows = 64;

// Decode steps of bf16 models with head_dim 128 and up to kSplitMaxRows rows run the
// fused path: tcgen05 linears whose k-block iterations are split evenly over the
// SMs; the last CTA of each tile sums its fp32 partials in k order and applies
// QK-norm + RoPE, the residual add (with the next norm's statistics) or SwiGLU.
static const int kTicketSlots = 4096;

static bool use_splitk(const Model& m, int M) {
    const qk_config& c = m.cfg;
    return c.dtype == QK_DTYPE_BF16 && M >= 1 && M <= kSplitMaxRows && c.head_dim == 128 &&
           c.hidden % 128 == 0 && c.intermediate % 128 == 0 && c.vocab % 128 == 0 &&
           c.vocab / 128 <= kTicketSlots && (2 * c.intermediate) / 128 <= kTicketSlots &&
           ((c.n_q_heads + 2 * c.n_kv_heads) * c.head_dim) / 128 <= kTicketSlots;
}

// Scoring of bf16 models forms the log-softmax statistics per vocabulary tile in the
// tcgen05 lm_head epilogue; the fp32 model (CUDA-core GEMM) materialises its logits.
static bool use_lse_head(const Model& m) {
    const qk_config& c = m.cfg;
    return c.dtype == QK_DTYPE_BF16 && c.vocab % 128 == 0 && c.hidden % 64 == 0;
}

static size_t splitk_part_floats(const Model& m, int M) {
    const qk_config& c = m.cfg;
    const int nqkv = (c.n_q_heads + 2 * c.n_kv_heads) * c.head_dim;
    const int widths[5] = {nqkv, c.hidden, 2 * c.intermediate, c.hidden, c.vocab};
    size_t f = 0;
    for (int n : widths) {
        const size_t g = gemm_fused_part_floats(M, n, m.num_sms);
        f = g > f ? g : f;
    }
    return f;
}

static int workspace_layout(const Model& m, int kind, int B, int T, int max_seq, Workspace* w,
                            char* base) {
    const qk_config& c = m.cfg;
    if (B < 1 || T < 1) return set_error(QK_ESHAPE, "batch %d and tokens %d must be >= 1", B, T);
    size_t es = m.es;
    size_t M = (size_t)B * (kind == QK_CALL_DECODE ? 1 : T);
    if (M > (size_t)1 << 24) return set_error(QK_ESHAPE, "too many tokens in one call (%zu)", M);
    size_t H = c.hidden, d = c.head_dim, nq = c.n_q_heads, nkv = c.n_kv_heads, I = c.intermediate;
    size_t off = 0;
    auto take = [&](size_t bytes) {
        char* p = base ? base + off : nullptr;
        off = align256(off + bytes);
        return (void*)p;
    };
    w->x = (float*)take(M * H * 4);
    w->u = take(M * H * es);
    w->qkv = take(M * (nq + 2 * nkv) * d * es);
    w->o = take(M * nq * d * es);
    w->h = take(M * I * es);
    w->gu = c.dtype == QK_DTYPE_F32 ? take(M * 2 * I * es) : nullptr;  // unfused SwiGLU path only
    w->skv = kind == QK_CALL_SCORE ? take(2 * (size_t)B * nkv * T * d * es) : nullptr;
    const bool fused = kind == QK_CALL_DECODE && use_splitk(m, B);
    w->part = fused ? (float*)take(splitk_part_floats(m, B) * 4) : nullptr;
    w->xg = fused ? (bf16*)take(M * H * 2) : nullptr;
    w->ssq = fused ? (float*)take((H / 128) * M * 4) : nullptr;
    w->tickets = fused ? (int*)take(kTicketSlots * 4) : nullptr;
    w->attn = nullptr;
    if (kind == QK_CALL_DECODE && c.dtype == QK_DTYPE_BF16 &&
        attn_decode_supported(c.head_dim, c.n_q_heads, c.n_kv_heads)) {
        if (max_seq < 1) return set_error(QK_ESHAPE, "max_seq must be >= 1");
        w->attn = take(attn_decode_scratch_bytes(B, c.n_q_heads, c.n_kv_heads, max_seq, m.num_sms));
    }
    size_t rows = kind == QK_CALL_SCORE ? (M < (size_t)kScoreLogitRows ? M : kScoreLogitRows) : B;
    w->logit_rows = (int)rows;
    w->lse_ms = nullptr;
    w->lse_idx = nullptr;
    w->lse_zt = nullptr;
    if (kind == QK_CALL_SCORE && use_lse_head(m)) {
        const size_t nvt = (size_t)c.vocab / 128;
        w->logits = nullptr;
        w->lse_ms = (float2*)take(rows * nvt * 8);
        w->lse_idx = (int*)take(rows * nvt * 4);
        w->lse_zt = (float*)take(rows * 4);
    } else {
        w->logits = (float*)take(rows * (size_t)c.vocab * 4);
    }
    w->total = off;
    return QK_OK;
}

// ---------------------------------------------------------------- forward pieces
struct KVView {
    char* base;        // layer 0's K
    size_t layer_bytes;  // bytes from one layer's K to the next layer's K (0: shared scratch)
    size_t half_bytes;   // bytes from a layer's K to its V
    KvPages kp;          // where a row's positions sit inside a layer's K (and V)
    void* k(int l) const { return base + (size_t)l * layer_bytes; }
    void* v(int l) const { return base + (size_t)l * layer_bytes + half_bytes; }
};

static KVView cache_view(const Model& m, void* kv, int max_batch, int max_seq) {
    const qk_config& c = m.cfg;
    size_t half = (size_t)max_batch * c.n_kv_heads * max_seq * c.head_dim * m.es;
    return KVView{(char*)kv, 2 * half, half, KvPages::dense(max_batch, max_seq)};
}

// A paged cache: per layer a K pool then a V pool of n_pages pages.
static KVView paged_view(const Model& m, void* kv, const qk_kv_pages& pg) {
    const qk_config& c = m.cfg;
    size_t half = (size_t)pg.n_pages * c.n_kv_heads * pg.page_size * c.head_dim * m.es;
    return KVView{(char*)kv, 2 * half, half, KvPages{pg.table, pg.per_row, pg.n_pages, pg.page_size}};
}

static void run_layer(Model& m, int l, const Workspace& w, int M, PosIndex pos,
                      const KVView& kv, cudaStream_t s) {
    const qk_config& c = m.cfg;
    const LayerW& L = m.layers[l];
    int H = c.hidden, d = c.head_dim, nq = c.n_q_heads, nkv = c.n_kv_heads, I = c.intermediate;
    int nqkv = (nq + 2 * nkv) * d;
    float eps = (float)c.rms_eps;
    bool pr;
    launch_rmsnorm(w.x, 1, 0, L.attn_norm, H, eps, w.u, c.dtype, M, s);
    pr = prof_open(m, QK_PROF_QKV, s);
    linear(m, w.u, H, L.w_qkv, w.qkv, nqkv, M, nqkv, H, EPI_STORE_ACT, w.gu, s);
    prof_close(m, pr, s);
    launch_qk_norm_rope(w.qkv, c.dtype, M, nq, nkv, d, L.q_norm, L.k_norm, eps, m.rope_cos,
                        m.rope_sin, c.max_positions, pos, kv.k(l), kv.v(l), kv.kp, m.status,
                        s);
    pr = prof_open(m, QK_PROF_ATTN, s);
    launch_attention(m, w.qkv, nqkv, kv.k(l), kv.v(l), M, kv.kp, pos, w.o,
                     w.attn, s);
    prof_close(m, pr, s);
    pr = prof_open(m, QK_PROF_O, s);
    linear(m, w.o, nq * d, L.w_o, w.x, H, M, H, nq * d, EPI_RESID_F32, w.gu, s);
    prof_close(m, pr, s);
    launch_rmsnorm(w.x, 1, 0, L.mlp_norm, H, eps, w.u, c.dtype, M, s);
    pr = prof_open(m, QK_PROF_GATE_UP, s);
    linear(m, w.u, H, L.w_gu, w.h, I, M, I, H, EPI_SWIGLU, w.gu, s);
    prof_close(m, pr, s);
    pr = prof_open(m, QK_PROF_DOWN, s);
    linear(m, w.h, I, L.w_d, w.x, H, M, H, I, EPI_RESID_F32, w.gu, s);
    prof_close(m, pr, s);
}

// One decoder layer of a fused decode step.  On entry w.x holds the residual,
// w.xg = bf16(x * g_attn) and w.ssq its tile sums of squares; on exit the same for
// the layer's output with gain g_next (the next layer's input norm or the final norm).
static void run_layer_fused(Model& m, int l, const Workspace& w, int M, PosIndex pos,
                            const KVView& kv, const float* g_next, cudaStream_t s) {
    const qk_config& c = m.cfg;
    const LayerW& L = m.layers[l];
    const int H = c.hidden, d = c.head_dim, nq = c.n_q_heads, nkv = c.n_kv_heads, I = c.intermediate;
    const int nqkv = (nq + 2 * nkv) * d;
    Fuse f{};
    f.tickets = w.tickets;
    f.part = w.part;
    f.ssq_in = w.ssq;
    f.n_ssq = H / 128;
    f.H = H;
    f.eps = (float)c.rms_eps;
    f.status = m.status;
    auto gemm = [&](const void* A, int lda, const void* W, int N, int K, const Fuse& fz) {
        int rc = launch_gemm_tc_fused((const bf16*)A, lda, (const bf16*)W, nullptr, M, N, K, fz,
                                      m.num_sms, m.status, s);
        if (rc != QK_OK && !m.deferred_error) m.deferred_error = rc;
    };
    bool pr;
    Fuse fq = f;
    fq.op = FUSE_QKV;
    fq.nq = nq;
    fq.nkv = nkv;
    fq.gq = L.q_norm;
    fq.gk = L.k_norm;
    fq.rope_cos = m.rope_cos;
    fq.rope_sin = m.rope_sin;
    fq.max_positions = c.max_positions;
    fq.pos = pos;
    fq.q_out = (bf16*)w.qkv;
    fq.q_ld = nqkv;
    fq.k_cache = (bf16*)kv.k(l);
    fq.v_cache = (bf16*)kv.v(l);
    fq.kv = kv.kp;
    pr = prof_open(m, QK_PROF_QKV, s);
    gemm(w.xg, H, L.w_qkv, nqkv, H, fq);
    prof_close(m, pr, s);
    pr = prof_open(m, QK_PROF_ATTN, s);
    launch_attention(m, w.qkv, nqkv, kv.k(l), kv.v(l), M, kv.kp, pos, w.o,
                     w.attn, s);
    prof_close(m, pr, s);
    Fuse fo = f;
    fo.op = FUSE_RESID;
    fo.x = w.x;
    fo.g_next = L.mlp_norm;
    fo.xg_out = w.xg;
    fo.ssq_out = w.ssq;
    pr = prof_open(m, QK_PROF_O, s);
    gemm(w.o, nq * d, L.w_o, H, nq * d, fo);
    prof_close(m, pr, s);
    Fuse fg = f;
    fg.op = FUSE_SWIGLU;
    fg.h_out = (bf16*)w.h;
    pr = prof_open(m, QK_PROF_GATE_UP, s);
    gemm(w.xg, H, L.w_gu, 2 * I, H, fg);
    prof_close(m, pr, s);
    Fuse fd = fo;
    fd.g_next = g_next;
    pr = prof_open(m, QK_PROF_DOWN, s);
    gemm(w.h, I, L.w_d, H, I, fd);
    prof_close(m, pr, s);
}

// Final norm of M_out selected rows (row r of the output reads residual row r * in_step + in_off),
// lm_head into `logits`, then log-prob / argmax per row.
static void run_head(Model& m, const Workspace& w, int M_out, int in_step, int in_off,
                     float* logits, OutIndex oi, float* lp, int32_t* am, cudaStream_t s,
                     bool normed = false, const int32_t* row_len = nullptr) {
    const qk_config& c = m.cfg;
    if (!normed)
        launch_rmsnorm(w.x, in_step, in_off, m.final_norm, c.hidden, (float)c.rms_eps, w.u,
                       c.dtype, M_out, s, row_len);
    bool pr = prof_open(m, QK_PROF_LM_HEAD, s);
    linear(m, w.u, c.hidden, m.lm_head, logits, c.vocab, M_out, c.vocab, c.hidden, EPI_STORE_F32,
           w.gu, s);
    prof_close(m, pr, s);
    if (lp || am)
        launch_logits_reduce(logits, M_out, c.vocab, oi, lp, am, m.status, s, nullptr,
                             m.sampling.out_tokens ? &m.sampling : nullptr);
}

// The split decode attention merges through tickets in its scratch that must be
// zero at the start of a step (each layer leaves them zero again).
static int clear_attn_tickets(const Model& m, const Workspace& w, int B, int max_seq, cudaStream_t s) {
    if (!w.attn) return QK_OK;
    const qk_config& c = m.cfg;
    int* t = attn_decode_tickets(w.attn, B, c.n_q_heads, c.n_kv_heads, max_seq, m.num_sms);
    QK_TRY_CUDA(cudaMemsetAsync(t, 0, (size_t)B * c.n_kv_heads * sizeof(int), s));
    return QK_OK;
}

int check_linear_operands(const Model& m, const void* A, int lda, const void* W, const void* C,
                          int out_es) {
    const int row_align = m.es == 2 ? 8 : 4;  // elements per 16 bytes
    if (((uintptr_t)A & 15) || ((uintptr_t)W & 15))
        return set_error(QK_EINVAL, "A and W must be 16-byte aligned (A %p, W %p)", A, W);
    if (lda % row_align)
        return set_error(QK_ESHAPE, "lda %d must be a multiple of %d elements (16 bytes)", lda,
                         row_align);
    if ((uintptr_t)C % (uintptr_t)out_es)
        return set_error(QK_EINVAL, "C must be aligned to its %d-byte elements", out_es);
    return QK_OK;
}

static int check_launch(const char* what) {
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_error(e, what);
    return QK_OK;
}

static int check_launch(Model& m, const char* what) {
    int rc = check_launch(what);
    if (rc == QK_OK && m.deferred_error) {
        rc = set_error(m.deferred_error, "%s: a tensor-map encode or kernel attribute call failed", what);
    }
    m.deferred_error = 0;
    return rc;
}

static int get_ws(const Model& m, int kind, int B, int T, int max_seq, void* ws, size_t ws_bytes,
                  Workspace* w) {
    QK_TRY(workspace_layout(m, kind, B, T, max_seq, w, nullptr));
    if (!ws) return set_error(QK_EINVAL, "workspace is NULL");
    if (((uintptr_t)ws & 255) != 0) return set_error(QK_EINVAL, "workspace must be 256-byte aligned");
    if (ws_bytes < w->total)
        return set_error(QK_ENOSPACE, "workspace has %zu bytes, needs %zu", ws_bytes, w->total);
    return workspace_layout(m, kind, B, T, max_seq, w, (char*)ws);
}

// A paged cache: the pool and table shapes (the table's contents are checked on the
// device: an entry outside [0, n_pages) sets QK_STATUS_BAD_PAGE).
static int check_pages(const Model& m, void* kv, const qk_kv_pages* pg, int B) {
    if (!kv || !pg || !pg->table) return set_error(QK_EINVAL, "kv cache, pages or page table is NULL");
    if (((uintptr_t)kv & 255) != 0) return set_error(QK_EINVAL, "kv cache must be 256-byte aligned");
    if (((uintptr_t)pg->table & 3) != 0) return set_error(QK_EINVAL, "page table must be 4-byte aligned");
    if (pg->n_pages < 1 || pg->per_row < 1 || pg->page_size < 128 || pg->page_size % 128)
        return set_error(QK_ESHAPE, "n_pages %d, per_row %d, page_size %d (>= 1, >= 1, a multiple of 128)",
                         pg->n_pages, pg->per_row, pg->page_size);
    const long long cap = (long long)pg->per_row * pg->page_size;
    if (cap > m.cfg.max_positions)
        return set_error(QK_ESHAPE, "per_row x page_size = %lld exceeds the RoPE table (%d positions)", cap,
                         m.cfg.max_positions);
    if (2 * (long long)pg->n_pages * m.cfg.n_kv_heads * pg->page_size >= (1ll << 31))
        return set_error(QK_ESHAPE, "a layer's pools exceed 2^31 rows of head_dim");
    if (B < 1) return set_error(QK_ESHAPE, "batch %d < 1", B);
    return QK_OK;
}

static int check_cache(const Model& m, void* kv, int max_batch, int max_seq, int B) {
    if (!kv) return set_error(QK_EINVAL, "kv cache is NULL");
    if (((uintptr_t)kv & 255) != 0) return set_error(QK_EINVAL, "kv cache must be 256-byte aligned");
    if (max_batch < 1 || max_seq < 1) return set_error(QK_ESHAPE, "max_batch / max_seq must be >= 1");
    if (B < 1 || B > max_batch) return set_error(QK_ESHAPE, "batch %d outside [1, %d]", B, max_batch);
    if (max_seq > m.cfg.max_positions)
        return set_error(QK_ESHAPE, "max_seq %d exceeds the RoPE table (%d positions)", max_seq,
                         m.cfg.max_positions);
    return QK_OK;
}

}  // namespace qk

using namespace qk;

// ================================================================ C ABI
extern "C" {

const char* qk_last_error(void) { return g_err; }

int qk_config_preset(const char* name, qk_config* out) {
    if (!name || !out) return set_error(QK_EINVAL, "null argument");
    qk_config c;
    memset(&c, 0, sizeof(c));
    c.rms_eps = 1e-6;
    c.rope_theta = 1e6;
    c.max_positions = 8192;
    if (!strcmp(name, "tiny_fp32")) {
        c.n_layers = 2; c.hidden = 256; c.n_q_heads = 4; c.n_kv_heads = 2; c.head_dim = 64;
        c.intermediate = 768; c.vocab = 4096; c.dtype = QK_DTYPE_F32;
    } else if (!strcmp(name, "q8b") || !strcmp(name, "q8b_layer")) {
        c.n_layers = strcmp(name, "q8b") ? 1 : 36; c.hidden = 4096; c.n_q_heads = 32;
        c.n_kv_heads = 8; c.head_dim = 128; c.intermediate = 12288; c.vocab = 151936;
        c.dtype = QK_DTYPE_BF16;
    } else {
        return set_error(QK_EINVAL, "unknown preset '%s'", name);
    }
    *out = c;
    return QK_OK;
}

int qk_weight_count(const qk_config* cfg, int* n) {
    if (!cfg || !n) return set_error(QK_EINVAL, "null argument");
    QK_TRY(validate_config(*cfg));
    *n = 3 + 11 * cfg->n_layers;
    return QK_OK;
}

int qk_model_packed_bytes(const qk_config* cfg, size_t* bytes) {
    if (!cfg || !bytes) return set_error(QK_EINVAL, "null argument");
    PackedLayout p;
    QK_TRY(packed_layout(*cfg, &p));
    *bytes = p.total;
    return QK_OK;
}

int qk_model_load(const qk_config* cfg, const void* const* tensors, int n_tensors, void* packed,
                  size_t packed_bytes, void* stream, qk_model** out) {
    if (!cfg || !tensors || !packed || !out) return set_error(QK_EINVAL, "null argument");
    *out = nullptr;
    PackedLayout p;
    QK_TRY(packed_layout(*cfg, &p));
    if (n_tensors != 3 + 11 * cfg->n_layers)
        return set_error(QK_EINVAL, "expected %d tensors, got %d", 3 + 11 * cfg->n_layers, n_tensors);
    for (int i = 0; i < n_tensors; ++i)
        if (!tensors[i]) return set_error(QK_EINVAL, "tensor %d is NULL", i);
    if (((uintptr_t)packed & 255) != 0) return set_error(QK_EINVAL, "packed buffer must be 256-byte aligned");
    if (packed_bytes < p.total)
        return set_error(QK_ENOSPACE, "packed buffer has %zu bytes, needs %zu", packed_bytes, p.total);
    cudaStream_t s = (cudaStream_t)stream;
    Model* m = new (std::nothrow) Model();
    if (!m) return set_error(QK_EINVAL, "host allocation failed");
    const qk_config& c = *cfg;
    m->cfg = c;
    m->es = c.dtype == QK_DTYPE_BF16 ? 2 : 4;
    m->packed = (char*)packed;
    m->packed_bytes = packed_bytes;
    auto fail = [&](int code) { delete m; return code; };
    cudaError_t e = cudaGetDevice(&m->device);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&m->num_sms, cudaDevAttrMultiProcessorCount, m->device);
    if (e != cudaSuccess) return fail(cuda_error(e, "device query"));
    char* B = (char*)packed;
    m->status = (uint32_t*)(B + p.status);
    m->rope_cos = (float*)(B + p.rope_cos);
    m->rope_sin = (float*)(B + p.rope_sin);
    m->embed = B + p.embed;
    m->final_norm = (float*)(B + p.final_norm);
    m->lm_head = B + p.lm_head;
    m->layers.resize(c.n_layers);
    size_t es = m->es, H = c.hidden, d = c.head_dim, nq = c.n_q_heads, nkv = c.n_kv_heads,
           I = c.intermediate, V = c.vocab;
    e = cudaMemsetAsync(m->status, 0, 256, s);
    if (e != cudaSuccess) return fail(cuda_error(e, "status clear"));
    launch_rope_table(m->rope_cos, m->rope_sin, c.max_positions, c.head_dim, c.rope_theta, s);
    int t = 0;
    auto copy = [&](void* dst, const void* src, size_t bytes) {
        return cudaMemcpyAsync(dst, src, bytes, cudaMemcpyDeviceToDevice, s);
    };
    if ((e = copy(m->embed, tensors[t++], V * H * es)) != cudaSuccess) return fail(cuda_error(e, "embed copy"));
    for (int l = 0; l < c.n_layers; ++l) {
        const PackedLayout::L& PL = p.layers[l];
        LayerW& L = m->layers[l];
        L.attn_norm = (float*)(B + PL.attn_norm);
        L.q_norm = (float*)(B + PL.q_norm);
        L.k_norm = (float*)(B + PL.k_norm);
        L.mlp_norm = (float*)(B + PL.mlp_norm);
        L.w_qkv = B + PL.w_qkv;
        L.w_o = B + PL.w_o;
        L.w_gu = B + PL.w_gu;
        L.w_d = B + PL.w_d;
        const void* const* T = tensors + t;
        t += 11;
        launch_widen_gain(T[0], c.dtype, L.attn_norm, (int)H, s);
        char* qkv = (char*)L.w_qkv;
        e = copy(qkv, T[1], nq * d * H * es);
        if (e == cudaSuccess) e = copy(qkv + nq * d * H * es, T[2], nkv * d * H * es);
        if (e == cudaSuccess) e = copy(qkv + (nq + nkv) * d * H * es, T[3], nkv * d * H * es);
        if (e != cudaSuccess) return fail(cuda_error(e, "qkv copy"));
        launch_widen_gain(T[4], c.dtype, L.q_norm, (int)d, s);
        launch_widen_gain(T[5], c.dtype, L.k_norm, (int)d, s);
        if ((e = copy(L.w_o, T[6], H * nq * d * es)) != cudaSuccess) return fail(cuda_error(e, "wo copy"));
        launch_widen_gain(T[7], c.dtype, L.mlp_norm, (int)H, s);
        // gate/up interleave: block i of 128 gate rows goes to rows [256 i, 256 i + 128),
        // the matching 128 up rows to [256 i + 128, 256 i + 256).
        size_t blk = 128 * H * es;
        e = cudaMemcpy2DAsync(L.w_gu, 2 * blk, T[8], blk, blk, I / 128, cudaMemcpyDeviceToDevice, s);
        if (e == cudaSuccess)
            e = cudaMemcpy2DAsync((char*)L.w_gu + blk, 2 * blk, T[9], blk, blk, I / 128,
                                  cudaMemcpyDeviceToDevice, s);
        if (e != cudaSuccess) return fail(cuda_error(e, "gate/up copy"));
        if ((e = copy(L.w_d, T[10], H * I * es)) != cudaSuccess) return fail(cuda_error(e, "wd copy"));
    }
    launch_widen_gain(tensors[t++], c.dtype, m->final_norm, (int)H, s);
    if ((e = copy(m->lm_head, tensors[t++], V * H * es)) != cudaSuccess) return fail(cuda_error(e, "lm_head copy"));
    int rc = check_launch("model load kernels");
    if (rc != QK_OK) return fail(rc);
    *out = (qk_model*)m;
    return QK_OK;
}

static void prof_release(Model& m) {
    for (cudaEvent_t e : m.prof_ev) cudaEventDestroy(e);
    m.prof_ev.clear();
    m.prof_used = 0;
    m.prof_kind = -1;
}

void qk_model_free(qk_model* m) {
    if (!m) return;
    prof_release(*(Model*)m);
    for (auto& g : ((Model*)m)->graphs) cudaGraphExecDestroy(g.exec);
    if (((Model*)m)->capture_stream) cudaStreamDestroy(((Model*)m)->capture_stream);
    delete (Model*)m;
}

int qk_profile_begin(qk_model* mh, int kind, int max_launches) {
    if (!mh) return set_error(QK_EINVAL, "null argument");
    Model& m = *(Model*)mh;
    if (kind < QK_PROF_QKV || kind > QK_PROF_LM_HEAD) return set_error(QK_EINVAL, "unknown kernel class %d", kind);
    if (max_launches < 1 || max_launches > (1 << 20)) return set_error(QK_EINVAL, "max_launches out of range");
    prof_release(m);
    m.prof_ev.resize(2 * (size_t)max_launches);
    for (size_t i = 0; i < m.prof_ev.size(); ++i) {
        cudaError_t e = cudaEventCreate(&m.prof_ev[i]);
        if (e != cudaSuccess) {
            m.prof_ev.resize(i);
            prof_release(m);
            return cuda_error(e, "cudaEventCreate");
        }
    }
    m.prof_kind = kind;
    return QK_OK;
}

int qk_profile_end(qk_model* mh, float* total_ms, int* launches) {
    if (!mh || !total_ms || !launches) return set_error(QK_EINVAL, "null argument");
    Model& m = *(Model*)mh;
    float tot = 0.f;
    int n = m.prof_used / 2;
    if (n > 0) {
        cudaError_t e = cudaEventSynchronize(m.prof_ev[2 * n - 1]);
        for (int i = 0; e == cudaSuccess && i < n; ++i) {
            float ms = 0.f;
            e = cudaEventElapsedTime(&ms, m.prof_ev[2 * i], m.prof_ev[2 * i + 1]);
            tot += ms;
        }
        if (e != cudaSuccess) {
            prof_release(m);
            return cuda_error(e, "profile events");
        }
    }
    prof_release(m);
    *total_ms = tot;
    *launches = n;
    return QK_OK;
}

uint64_t qk_launch_count(void) { return g_launches.load(); }

int qk_op_linear(qk_model* mh, const void* A, int lda, const void* W, void* C, int ldc, int M,
                 int N, int K, int epilogue, void* scratch, size_t scratch_bytes, void* stream) {
    if (!mh || !A || !W || !C) return set_error(QK_EINVAL, "null argument");
    Model& m = *(Model*)mh;
    if (M < 1 || N < 1 || K < 16 || K % 16 || lda < K || (epilogue == QK_EPI_SWIGLU && N % 128))
        return set_error(QK_ESHAPE, "bad linear shape M %d N %d K %d lda %d", M, N, K, lda);
    if (epilogue < QK_EPI_STORE || epilogue > QK_EPI_SWIGLU)
        return set_error(QK_EINVAL, "unknown epilogue %d", epilogue);
    if (ldc < N) return set_error(QK_ESHAPE, "ldc %d < N %d", ldc, N);
    const bool f32_out = epilogue == QK_EPI_STORE_F32 || epilogue == QK_EPI_RESID_F32;
    QK_TRY(check_linear_operands(m, A, lda, W, C, f32_out ? 4 : m.es));
    // Only the CUDA-core path (fp32 models) stages the gate/up product in scratch.
    size_t need = epilogue == QK_EPI_SWIGLU && m.cfg.dtype == QK_DTYPE_F32 ? (size_t)M * 2 * N * m.es : 0;
    if (need && (!scratch || scratch_bytes < need))
        return set_error(QK_ENOSPACE, "linear scratch has %zu bytes, needs %zu", scratch_bytes, need);
    linear(m, A, lda, W, C, ldc, M, N, K, epilogue, scratch, (cudaStream_t)stream);
    return check_launch(m, "linear");
}

int qk_debug_expire_next_wait(qk_model* mh, long long wait_cycles) {
    if (!mh) return set_error(QK_EINVAL, "null argument");
    if (wait_cycles < 1 || wait_cycles > (1ll << 31))
        return set_error(QK_EINVAL, "wait_cycles %lld outside [1, 2^31]", wait_cycles);
    ((Model*)mh)->test_wait_cycles = wait_cycles;
    return QK_OK;
}

int qk_kv_bytes(const qk_model* mh, int max_batch, int max_seq, size_t* bytes) {
    if (!mh || !bytes) return set_error(QK_EINVAL, "null argument");
    const Model& m = *(const Model*)mh;
    if (max_batch < 1 || max_seq < 1) return set_error(QK_ESHAPE, "max_batch / max_seq must be >= 1");
    *bytes = 2 * (size_t)m.cfg.n_layers * max_batch * m.cfg.n_kv_heads * max_seq * m.cfg.head_dim * m.es;
    return QK_OK;
}

int qk_kv_pages_bytes(const qk_model* mh, int n_pages, int page_size, size_t* bytes) {
    if (!mh || !bytes) return set_error(QK_EINVAL, "null argument");
    if (n_pages < 1 || page_size < 128 || page_size % 128)
        return set_error(QK_ESHAPE, "n_pages %d >= 1 and page_size %d a multiple of 128 are required", n_pages,
                         page_size);
    return qk_kv_bytes(mh, n_pages, page_size, bytes);  // the same bytes as n_pages rows of page_size
}

int qk_workspace_bytes(const qk_model* mh, int kind, int B, int T, int max_seq, size_t* bytes) {
    if (!mh || !bytes) return set_error(QK_EINVAL, "null argument");
    const Model& m = *(const Model*)mh;
    Workspace w;
    if (kind == QK_CALL_ROLLOUT) {
        Workspace w2;
        QK_TRY(workspace_layout(m, QK_CALL_PREFILL, B, T, max_seq, &w, nullptr));
        QK_TRY(workspace_layout(m, QK_CALL_DECODE, B, 1, max_seq, &w2, nullptr));
        *bytes = (w.total > w2.total ? w.total : w2.total) + rollout_cursor_bytes(B);
        return QK_OK;
    }
    if (kind == QK_CALL_BACKWARD) return backward_workspace_bytes(m, B, T, bytes);
    if (kind != QK_CALL_DECODE && kind != QK_CALL_PREFILL && kind != QK_CALL_SCORE)
        return set_error(QK_EINVAL, "unknown call kind %d", kind);
    QK_TRY(workspace_layout(m, kind, B, T, max_seq, &w, nullptr));
    *bytes = w.total;
    return QK_OK;
}

// start_dev (dev [B] or null): per-row first positions instead of start_pos; row_len
// (dev [B] or null): the head reads row b's token row_len[b] - 1 instead of T - 1.
static int prefill_impl(Model& m, const KVView& view, TokIndex tok, int B, int T,
                        int start_pos, float* last_logits, OutIndex oi, float* lp, int32_t* am,
                        void* ws, size_t ws_bytes, cudaStream_t s,
                        const int32_t* start_dev = nullptr, const int32_t* row_len = nullptr) {
    Workspace w;
    QK_TRY(get_ws(m, QK_CALL_PREFILL, B, T, view.kp.cap(), ws, ws_bytes, &w));
    int M = B * T;
    launch_embed(m.embed, m.cfg.dtype, m.cfg.vocab, m.cfg.hidden, tok, M, w.x, m.status, s);
    PosIndex pos{start_dev, start_pos, T};
    for (int l = 0; l < m.cfg.n_layers; ++l) run_layer(m, l, w, M, pos, view, s);
    if (last_logits || lp || am)
        run_head(m, w, B, T, T - 1, last_logits ? last_logits : w.logits, oi, lp, am, s, false,
                 row_len);
    return check_launch(m, "prefill");
}

int qk_prefill(qk_model* mh, void* kv, int max_batch, int max_seq, const int32_t* tokens, int B,
               int T, int start_pos, float* last_logits, const int32_t* targets, float* logprobs,
               int32_t* argmax, void* workspace, size_t ws_bytes, void* stream) {
    if (!mh || !tokens) return set_error(QK_EINVAL, "null argument");
    Model& m = *(Model*)mh;
    QK_TRY(check_cache(m, kv, max_batch, max_seq, B));
    if (T < 1 || start_pos < 0 || (long)start_pos + T > max_seq)
        return set_error(QK_ESHAPE, "positions [%d, %d) outside the cache of %d", start_pos,
                         start_pos + T, max_seq);
    if (logprobs && !targets) return set_error(QK_EINVAL, "logprobs requested without targets");
    OutIndex oi{1, 1, 1, 0, targets, 1, 0, 0};
    return prefill_impl(m, cache_view(m, kv, max_batch, max_seq), TokIndex{tokens, T, T, 0}, B, T,
                        start_pos, last_logits, oi, logprobs, argmax, workspace, ws_bytes,
                        (cudaStream_t)stream);
}

int qk_prefill_rows(qk_model* mh, void* kv, int max_batch, int max_seq, const int32_t* tokens, int B,
                    int T, const int32_t* start, const int32_t* len, float* last_logits,
                    void* workspace, size_t ws_bytes, void* stream) {
    if (!mh || !tokens || !start) return set_error(QK_EINVAL, "null argument");
    Model& m = *(Model*)mh;
    QK_TRY(check_cache(m, kv, max_batch, max_seq, B));
    if (T < 1 || T > max_seq) return set_error(QK_ESHAPE, "T %d outside 1 .. max_seq %d", T, max_seq);
    OutIndex oi{1, 1, 1, 0, nullptr, 1, 0, 0};
    return prefill_impl(m, cache_view(m, kv, max_batch, max_seq), TokIndex{tokens, T, T, 0}, B, T, 0,
                        last_logits, oi, nullptr, nullptr, workspace, ws_bytes, (cudaStream_t)stream,
                        start, len);
}

int qk_prefill_rows_paged(qk_model* mh, void* kv, const qk_kv_pages* pages, const int32_t* tokens,
                          int B, int T, const int32_t* start, const int32_t* len, float* last_logits,
                          void* workspace, size_t ws_bytes, void* stream) {
    if (!mh || !tokens || !start) return set_error(QK_EINVAL, "null argument");
    Model& m = *(Model*)mh;
    QK_TRY(check_pages(m, kv, pages, B));
    const int cap = pages->per_row * pages->page_size;
    if (T < 1 || T > cap) return set_error(QK_ESHAPE, "T %d outside 1 .. per_row x page_size %d", T, cap);
    OutIndex oi{1, 1, 1, 0, nullptr, 1, 0, 0};
    return prefill_impl(m, paged_view(m, kv, *pages), TokIndex{tokens, T, T, 0}, B, T, 0, last_logits, oi,
                        nullptr, nullptr, workspace, ws_bytes, (cudaStream_t)stream, start, len);
}

static int decode_impl(Model& m, const KVView& view, TokIndex tok, PosIndex pos,
                       int B, float* logits, OutIndex oi, float* lp, int32_t* am, void* ws,
                       size_t ws_bytes, cudaStream_t s) {
    Workspace w;
    QK_TRY(get_ws(m, QK_CALL_DECODE, B, 1, view.kp.cap(), ws, ws_bytes, &w));
    QK_TRY(clear_attn_tickets(m, w, B, view.kp.cap(), s));
    m.in_decode = true;
    if (w.part) {
        const qk_config& c = m.cfg;
        QK_TRY_CUDA(cudaMemsetAsync(w.tickets, 0, kTicketSlots * sizeof(int), s));
        launch_embed_gain(m.embed, c.vocab, tok, true, w.x, m.layers[0].attn_norm, w.xg, w.ssq, B,
                          c.hidden, m.status, s);
        for (int l = 0; l < c.n_layers; ++l)
            run_layer_fused(m, l, w, B, pos, view,
                            l + 1 < c.n_layers ? m.layers[l + 1].attn_norm : m.final_norm, s);
        if (logits || lp || am) {
            // logits = s_m * (W_lm (x g_final)), s_m the final RMSNorm scale of row m
            float* z = logits ? logits : w.logits;
            Fuse fl{};
            fl.op = FUSE_COLSCALE;
            fl.tickets = w.tickets;
            fl.part = w.part;
            fl.status = m.status;
            fl.ssq_in = w.ssq;
            fl.n_ssq = c.hidden / 128;
            fl.H = c.hidden;
            fl.eps = (float)c.rms_eps;
            bool pr = prof_open(m, QK_PROF_LM_HEAD, s);
            int rc = launch_gemm_tc_fused(w.xg, c.hidden, (const bf16*)m.lm_head, z, B, c.vocab,
                                          c.hidden, fl, m.num_sms, m.status, s);
            prof_close(m, pr, s);
            if (rc != QK_OK && !m.deferred_error) m.deferred_error = rc;
            if (lp || am)
                launch_logits_reduce(z, B, c.vocab, oi, lp, am, m.status, s, nullptr,
                                     m.sampling.out_tokens ? &m.sampling : nullptr);
        }
    } else {
        launch_embed(m.embed, m.cfg.dtype, m.cfg.vocab, m.cfg.hidden, tok, B, w.x, m.status, s);
        for (int l = 0; l < m.cfg.n_layers; ++l) run_layer(m, l, w, B, pos, view, s);
        if (logits || lp || am) run_head(m, w, B, 1, 0, logits ? logits : w.logits, oi, lp, am, s);
    }
    m.in_decode = false;
    return check_launch(m, "decode step");
}

int qk_decode_step(qk_model* mh, void* kv, int max_batch, int max_seq, const int32_t* tokens,
                   const int32_t* pos, int B, float* logits, const int32_t* targets,
                   float* logprobs, int32_t* argmax, void* workspace, size_t ws_bytes,
                   void* stream) {
    if (!mh || !tokens || !pos) return set_error(QK_EINVAL, "null argument");
    Model& m = *(Model*)mh;
    QK_TRY(check_cache(m, kv, max_batch, max_seq, B));
    if (logprobs && !targets) return set_error(QK_EINVAL, "logprobs requested without targets");
    OutIndex oi{1, 1, 1, 0, targets, 1, 0, 0};
    return decode_impl(m, cache_view(m, kv, max_batch, max_seq), TokIndex{tokens, 1, 1, 0},
                       PosIndex{pos, 0, 1}, B, logits, oi, logprobs, argmax, workspace, ws_bytes,
                       (cudaStream_t)stream);
}

int qk_decode_step_paged(qk_model* mh, void* kv, const qk_kv_pages* pages, const int32_t* tokens,
                         const int32_t* pos, int B, float* logits, const int32_t* targets,
                         float* logprobs, int32_t* argmax, void* workspace, size_t ws_bytes,
                         void* stream) {
    if (!mh || !tokens || !pos) return set_error(QK_EINVAL, "null argument");
    Model& m = *(Model*)mh;
    QK_TRY(check_pages(m, kv, pages, B));
    if (logprobs && !targets) return set_error(QK_EINVAL, "logprobs requested without targets");
    OutIndex oi{1, 1, 1, 0, targets, 1, 0, 0};
    return decode_impl(m, paged_view(m, kv, *pages), TokIndex{tokens, 1, 1, 0}, PosIndex{pos, 0, 1}, B,
                       logits, oi, logprobs, argmax, workspace, ws_bytes, (cudaStream_t)stream);
}

int qk_decode_layer(qk_model* mh, int layer, void* kv, int max_batch, int max_seq, float* x,
                    const int32_t* pos, int B, void* workspace, size_t ws_bytes, void* stream) {
    if (!mh || !x || !pos) return set_error(QK_EINVAL, "null argument");
    Model& m = *(Model*)mh;
    if (layer < 0 || layer >= m.cfg.n_layers)
        return set_error(QK_EINVAL, "layer %d outside [0, %d)", layer, m.cfg.n_layers);
    QK_TRY(check_cache(m, kv, max_batch, max_seq, B));
    Workspace w;
    QK_TRY(get_ws(m, QK_CALL_DECODE, B, 1, max_seq, workspace, ws_bytes, &w));
    w.x = x;
    cudaStream_t s = (cudaStream_t)stream;
    QK_TRY(clear_attn_tickets(m, w, B, max_seq, s));
    m.in_decode = true;
    if (w.part) {
        const LayerW& L = m.layers[layer];
        QK_TRY_CUDA(cudaMemsetAsync(w.tickets, 0, kTicketSlots * sizeof(int), s));
        launch_embed_gain(nullptr, m.cfg.vocab, TokIndex{}, false, w.x, L.attn_norm, w.xg, w.ssq, B,
                          m.cfg.hidden, m.status, s);
        run_layer_fused(m, layer, w, B, PosIndex{pos, 0, 1}, cache_view(m, kv, max_batch, max_seq),
                        L.attn_norm, s);
    } else {
        run_layer(m, layer, w, B, PosIndex{pos, 0, 1}, cache_view(m, kv, max_batch, max_seq), s);
    }
    m.in_decode = false;
    return check_launch(m, "decode layer");
}

static int score_impl(Model& m, const int32_t* tokens, int B, int T, float* logprobs,
                      int32_t* argmax, void* workspace, size_t ws_bytes, cudaStream_t s,
                      const GrpoArgs* grpo) {
    Workspace w;
    QK_TRY(get_ws(m, QK_CALL_SCORE, B, T, T, workspace, ws_bytes, &w));
    int M = B * T;
    // One layer's K and V live in scratch shaped like a cache of B rows x T positions;
    // every layer reuses it (layer stride 0).
    size_t half = (size_t)B * m.cfg.n_kv_heads * T * m.cfg.head_dim * m.es;
    KVView view{(char*)w.skv, 0, half, KvPages::dense(B, T)};
    launch_embed(m.embed, m.cfg.dtype, m.cfg.vocab, m.cfg.hidden, TokIndex{tokens, T, T, 0}, M, w.x,
                 m.status, s);
    PosIndex pos{nullptr, 0, T};
    for (int l = 0; l < m.cfg.n_layers; ++l) run_layer(m, l, w, M, pos, view, s);
    // lm_head over all rows in chunks; row r = b T + t scores tokens[b, t + 1] for t < T - 1.
    for (int r0 = 0; r0 < M; r0 += w.logit_rows) {
        int rows = M - r0 < w.logit_rows ? M - r0 : w.logit_rows;
        launch_rmsnorm(w.x + (size_t)r0 * m.cfg.hidden, 1, 0, m.final_norm, m.cfg.hidden,
                       (float)m.cfg.rms_eps, w.u, m.cfg.dtype, rows, s);
        OutIndex oi{T, T - 1, T - 1, 0, tokens, T, 1, r0};
        if (w.lse_ms) {
            // the softmax statistics per vocabulary tile come out of the lm_head epilogue
            Fuse lf{};
            lf.lse_ms = w.lse_ms;
            lf.lse_idx = w.lse_idx;
            lf.lse_zt = w.lse_zt;
            lf.lse_tok = tokens;
            lf.lse_T = T;
            lf.lse_row0 = r0;
            int rc = launch_gemm_tc((const bf16*)w.u, m.cfg.hidden, (const bf16*)m.lm_head, nullptr,
                                    m.cfg.vocab, rows, m.cfg.vocab, m.cfg.hidden, EPI_LSE, m.num_sms,
                                    m.status, s, 0, &lf);
            if (rc != QK_OK) return set_error(rc, "lm_head statistics launch");
            launch_lse_combine(w.lse_ms, w.lse_idx, w.lse_zt, m.cfg.vocab / 128, m.cfg.vocab, rows, oi,
                               logprobs, argmax, m.status, s, grpo);
        } else {
            linear(m, w.u, m.cfg.hidden, m.lm_head, w.logits, m.cfg.vocab, rows, m.cfg.vocab,
                   m.cfg.hidden, EPI_STORE_F32, w.gu, s);
            launch_logits_reduce(w.logits, rows, m.cfg.vocab, oi, logprobs, argmax, m.status, s, grpo);
        }
    }
    return QK_OK;
}

static int check_score_shape(const Model& m, int B, int T) {
    if (B < 1 || T < 2) return set_error(QK_ESHAPE, "scoring needs B >= 1 and T >= 2 (got %d, %d)", B, T);
    if (T > m.cfg.max_positions)
        return set_error(QK_ESHAPE, "T %d exceeds the RoPE table (%d)", T, m.cfg.max_positions);
    return QK_OK;
}

int qk_score_logprobs(qk_model* mh, const int32_t* tokens, int B, int T, float* logprobs,
                      int32_t* argmax, void* workspace, size_t ws_bytes, void* stream) {
    if (!mh || !tokens || !logprobs) return set_error(QK_EINVAL, "null argument");
    Model& m = *(Model*)mh;
    QK_TRY(check_score_shape(m, B, T));
    QK_TRY(score_impl(m, tokens, B, T, logprobs, argmax, workspace, ws_bytes, (cudaStream_t)stream,
                      nullptr));
    return check_launch(m, "score");
}

// ---------------------------------------------------------------- GRPO token loss
int qk_grpo_workspace_bytes(int B, size_t* bytes) {
    if (!bytes) return set_error(QK_EINVAL, "null argument");
    if (B < 1) return set_error(QK_ESHAPE, "batch %d must be >= 1", B);
    *bytes = grpo_scratch_bytes(B);
    return QK_OK;
}

static int grpo_args(const float* lp_old, const float* lp_ref, int B, int T, int ld,
                     const float* rewards, int group, const uint8_t* mask, float eps_low,
                     float eps_high, float beta, float* loss_tok, GrpoArgs* g) {
    if (!lp_old || !rewards || !loss_tok) return set_error(QK_EINVAL, "null argument");
    if (beta != 0.f && !lp_ref) return set_error(QK_EINVAL, "beta != 0 needs lp_ref");
    if (B < 1 || T < 1 || ld < T) return set_error(QK_ESHAPE, "need B >= 1, T >= 1, ld >= T");
    if (group < 1 || B % group) return set_error(QK_ESHAPE, "batch %d is not a multiple of group %d", B, group);
    if (!(eps_low >= 0.f && eps_low <= 1.f && eps_high >= 0.f))
        return set_error(QK_EINVAL, "clip band needs 0 <= eps_low <= 1 and eps_high >= 0");
    *g = GrpoArgs{lp_old, lp_ref, rewards, mask, loss_tok, group, ld, eps_low, eps_high, beta};
    return QK_OK;
}

int qk_grpo_token_loss(const float* lp, const float* lp_old, const float* lp_ref, int B, int T,
                       int ld, const float* rewards, int group, const uint8_t* mask,
                       float eps_low, float eps_high, float beta, float* loss_tok,
                       float* loss_mean, void* workspace, size_t ws_bytes, void* stream) {
    if (!lp) return set_error(QK_EINVAL, "null argument");
    GrpoArgs g;
    QK_TRY(grpo_args(lp_old, lp_ref, B, T, ld, rewards, group, mask, eps_low, eps_high, beta,
                     loss_tok, &g));
    if (!workspace || ws_bytes < grpo_scratch_bytes(B))
        return set_error(QK_ENOSPACE, "workspace has %zu bytes, needs %zu", ws_bytes,
                         grpo_scratch_bytes(B));
    launch_grpo_loss(lp, B, T, g, true, workspace, loss_mean, (cudaStream_t)stream);
    return check_launch("grpo token loss");
}

int qk_grpo_coef(const float* lp, const float* lp_old, const float* lp_ref, int B, int T, int ld,
                 const float* rewards, int group, const uint8_t* mask, float eps_low, float eps_high,
                 float beta, float* coef, float* loss_tok, float* loss_mean, void* workspace,
                 size_t ws_bytes, void* stream) {
    if (!lp || !coef) return set_error(QK_EINVAL, "null argument");
    GrpoArgs g;
    QK_TRY(grpo_args(lp_old, lp_ref, B, T, ld, rewards, group, mask, eps_low, eps_high, beta,
                     loss_tok, &g));
    if (!workspace || ws_bytes < grpo_scratch_bytes(B))
        return set_error(QK_ENOSPACE, "workspace has %zu bytes, needs %zu", ws_bytes,
                         grpo_scratch_bytes(B));
    cudaStream_t s = (cudaStream_t)stream;
    launch_grpo_loss(lp, B, T, g, true, workspace, loss_mean, s);
    launch_grpo_coef(lp, B, T, g, workspace, coef, s);
    return check_launch("grpo coefficients");
}

int qk_score_grpo(qk_model* mh, const int32_t* tokens, int B, int T, const float* lp_old,
                  const float* lp_ref, const float* rewards, int group, const uint8_t* mask,
                  float eps_low, float eps_high, float beta, float* logprobs, float* loss_tok,
                  float* loss_mean, void* workspace, size_t ws_bytes, void* stream) {
    if (!mh || !tokens || !logprobs) return set_error(QK_EINVAL, "null argument");
    Model& m = *(Model*)mh;
    QK_TRY(check_score_shape(m, B, T));
    GrpoArgs g;
    QK_TRY(grpo_args(lp_old, lp_ref, B, T - 1, T - 1, rewards, group, mask, eps_low, eps_high,
                     beta, loss_tok, &g));
    size_t score_bytes;
    QK_TRY(qk_workspace_bytes(mh, QK_CALL_SCORE, B, T, T, &score_bytes));
    score_bytes = align256(score_bytes);
    if (!workspace || ws_bytes < score_bytes + grpo_scratch_bytes(B))
        return set_error(QK_ENOSPACE, "workspace has %zu bytes, needs %zu", ws_bytes,
                         score_bytes + grpo_scratch_bytes(B));
    cudaStream_t s = (cudaStream_t)stream;
    QK_TRY(score_impl(m, tokens, B, T, logprobs, nullptr, workspace, score_bytes, s, &g));
    launch_grpo_loss(logprobs, B, T - 1, g, false, (char*)workspace + score_bytes, loss_mean, s);
    return check_launch(m, "score with GRPO loss");
}

// Rollout of B rows: prefill over the prompt, then N decode steps replayed from one
// captured graph.  Teacher forcing (sampled == nullptr): seq [B, P+N+1] supplies
// every input token and target.  Sampling: seq is the prompt [B, P]; the head of
// each step draws the next token into sampled [B, N+1] (m.sampling), and the next
// step reads it from there.
// The cache (dense or paged) was checked by the caller.
static int rollout_impl(Model& m, qk_model* mh, const KVView& view, const int32_t* seq, int B, int P,
                        int N, float* logprobs, int32_t* argmax, const SampleArgs* sampled,
                        void* workspace, size_t ws_bytes, cudaStream_t s) {
    const int max_seq = view.kp.cap();
    if (P < 1 || N < 0 || (long)P + N > max_seq)
        return set_error(QK_ESHAPE, "prompt %d + steps %d exceed the cache of %d", P, N, max_seq);
    size_t need;
    QK_TRY(qk_workspace_bytes(mh, QK_CALL_ROLLOUT, B, P, max_seq, &need));
    if (!workspace || ws_bytes < need)
        return set_error(QK_ENOSPACE, "workspace has %zu bytes, needs %zu", ws_bytes, need);
    struct SamplingScope {  // m.sampling is set only for the duration of this call
        Model& m;
        SamplingScope(Model& mm, const SampleArgs* a) : m(mm) { m.sampling = a ? *a : SampleArgs{}; }
        ~SamplingScope() { m.sampling = SampleArgs{}; }
    } scope(m, sampled);
    const int L = sampled ? P : P + N + 1;  // row length of seq
    OutIndex oi{1, 1, N + 1, 0, sampled ? nullptr : seq, L, P, 0};
    QK_TRY(prefill_impl(m, view, TokIndex{seq, P, L, 0}, B, P, 0, nullptr, oi, logprobs, argmax, workspace,
                        ws_bytes, s));
    if (N == 0) return QK_OK;
    // cursor slots
    const size_t slot = align256((size_t)B * 4);
    char* cur = (char*)workspace + (need - rollout_cursor_bytes(B));
    int32_t* step = (int32_t*)cur;
    int32_t* pos = (int32_t*)(cur + slot);
    int32_t* tok = (int32_t*)(cur + 2 * slot);
    int32_t* tgt = (int32_t*)(cur + 3 * slot);
    int32_t* off = (int32_t*)(cur + 4 * slot);
    QK_TRY_CUDA(cudaMemsetAsync(step, 0, sizeof(int32_t), s));
    OutIndex od{1, 1, N + 1, 0, sampled ? nullptr : tgt, 1, 0, 0, off};
    auto prepare = [&](cudaStream_t st) {
        if (sampled)
            launch_rollout_prepare_sampled(sampled->out_tokens, N + 1, P, B, step, pos, tok, off, st);
        else
            launch_rollout_prepare(seq, L, P, B, step, pos, tok, tgt, off, st);
    };
    auto one_step = [&]() -> int {
        prepare(s);
        return decode_impl(m, view, TokIndex{tok, 1, 1, 0}, PosIndex{pos, 0, 1}, B, nullptr, od, logprobs,
                           argmax, workspace, ws_bytes, s);
    };
    // Step 0 runs directly (it also performs any one-time kernel set-up).
    QK_TRY(one_step());
    if (N == 1) return QK_OK;
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    QK_TRY_CUDA(cudaStreamIsCapturing(s, &cs));
    if (cs != cudaStreamCaptureStatusNone) {  // already inside the caller's capture: no nesting
        for (int j = 1; j < N; ++j) QK_TRY(one_step());
        return QK_OK;
    }
    uint32_t inv_tau_bits = 0;
    if (sampled) memcpy(&inv_tau_bits, &sampled->inv_tau, 4);
    const uint64_t key[17] = {(uint64_t)(uintptr_t)view.base, (uint64_t)view.kp.n_pages,
                              (uint64_t)view.kp.page, (uint64_t)(uintptr_t)view.kp.table,
                              (uint64_t)view.kp.per_row, (uint64_t)(uintptr_t)seq, (uint64_t)B,
                              (uint64_t)P, (uint64_t)N, (uint64_t)(uintptr_t)logprobs,
                              (uint64_t)(uintptr_t)argmax, (uint64_t)(uintptr_t)workspace,
                              (uint64_t)ws_bytes, sampled ? 1ull : 0ull,
                              sampled ? (uint64_t)(uintptr_t)sampled->out_tokens : 0ull,
                              sampled ? (uint64_t)sampled->seed : 0ull, (uint64_t)inv_tau_bits};
    cudaGraphExec_t exec = nullptr;
    int kernels = 0;
    for (auto& g : m.graphs)
        if (!memcmp(g.key, key, sizeof(key))) {
            exec = g.exec;
            kernels = g.kernels;
        }
    if (!exec) {
        if (!m.capture_stream)
            QK_TRY_CUDA(cudaStreamCreateWithFlags(&m.capture_stream, cudaStreamNonBlocking));
        cudaStream_t cs_stream = m.capture_stream;
        QK_TRY_CUDA(cudaStreamBeginCapture(cs_stream, cudaStreamCaptureModeThreadLocal));
        const uint64_t before = g_launches.load();
        prepare(cs_stream);
        int rc = decode_impl(m, view, TokIndex{tok, 1, 1, 0}, PosIndex{pos, 0, 1}, B, nullptr, od, logprobs,
                             argmax, workspace, ws_bytes, cs_stream);
        kernels = (int)(g_launches.load() - before);
        g_launches.fetch_sub((uint64_t)kernels);  // counted again below, once per replay
        cudaGraph_t graph = nullptr;
        cudaError_t e = cudaStreamEndCapture(cs_stream, &graph);
        if (rc != QK_OK) {
            if (graph) cudaGraphDestroy(graph);
            return rc;
        }
        if (e != cudaSuccess) return cuda_error(e, "rollout step capture");
        e = cudaGraphInstantiate(&exec, graph, 0);
        cudaGraphDestroy(graph);
        if (e != cudaSuccess) return cuda_error(e, "rollout step graph instantiate");
        if (m.graphs.size() >= 8) {
            cudaGraphExecDestroy(m.graphs.front().exec);
            m.graphs.erase(m.graphs.begin());
        }
        Model::StepGraph g;
        memcpy(g.key, key, sizeof(key));
        g.exec = exec;
        g.kernels = kernels;
        m.graphs.push_back(g);
    }
    for (int j = 1; j < N; ++j) {
        QK_TRY_CUDA(cudaGraphLaunch(exec, s));
        note_launch(kernels);
    }
    return QK_OK;
}

int qk_rollout_teacher_forced(qk_model* mh, void* kv, int max_batch, int max_seq,
                              const int32_t* seq, int B, int P, int N, float* logprobs,
                              int32_t* argmax, void* workspace, size_t ws_bytes, void* stream) {
    if (!mh || !seq || !logprobs) return set_error(QK_EINVAL, "null argument");
    Model& m = *(Model*)mh;
    QK_TRY(check_cache(m, kv, max_batch, max_seq, B));
    return rollout_impl(m, mh, cache_view(m, kv, max_batch, max_seq), seq, B, P, N, logprobs, argmax,
                        nullptr, workspace, ws_bytes, (cudaStream_t)stream);
}

int qk_rollout_teacher_forced_paged(qk_model* mh, void* kv, const qk_kv_pages* pages, const int32_t* seq,
                                    int B, int P, int N, float* logprobs, int32_t* argmax, void* workspace,
                                    size_t ws_bytes, void* stream) {
    if (!mh || !seq || !logprobs) return set_error(QK_EINVAL, "null argument");
    Model& m = *(Model*)mh;
    QK_TRY(check_pages(m, kv, pages, B));
    return rollout_impl(m, mh, paged_view(m, kv, *pages), seq, B, P, N, logprobs, argmax, nullptr,
                        workspace, ws_bytes, (cudaStream_t)stream);
}

static int sampled_args(qk_model* mh, const int32_t* prompt, int B, int N, float tau, uint64_t seed,
                        int32_t* tokens, const float* logprobs, SampleArgs* sa) {
    if (!mh || !prompt || !tokens || !logprobs) return set_error(QK_EINVAL, "null argument");
    if (!(tau > 0.f) || !(1.f / tau < 3.0e38f)) return set_error(QK_EINVAL, "temperature must be > 0");
    if (B >= (1 << 24) || N + 1 >= (1 << 22) || ((Model*)mh)->cfg.vocab > (1 << 18))
        return set_error(QK_ESHAPE, "sampling counters need B < 2^24, N < 2^22, vocab <= 2^18");
    *sa = SampleArgs{(unsigned long long)seed, 1.f / tau, tokens};
    return QK_OK;
}

int qk_rollout_sampled(qk_model* mh, void* kv, int max_batch, int max_seq, const int32_t* prompt,
                       int B, int P, int N, float tau, uint64_t seed, int32_t* tokens,
                       float* logprobs, void* workspace, size_t ws_bytes, void* stream) {
    SampleArgs sa;
    QK_TRY(sampled_args(mh, prompt, B, N, tau, seed, tokens, logprobs, &sa));
    Model& m = *(Model*)mh;
    QK_TRY(check_cache(m, kv, max_batch, max_seq, B));
    return rollout_impl(m, mh, cache_view(m, kv, max_batch, max_seq), prompt, B, P, N, logprobs, nullptr,
                        &sa, workspace, ws_bytes, (cudaStream_t)stream);
}

int qk_rollout_sampled_paged(qk_model* mh, void* kv, const qk_kv_pages* pages, const int32_t* prompt, int B,
                             int P, int N, float tau, uint64_t seed, int32_t* tokens, float* logprobs,
                             void* workspace, size_t ws_bytes, void* stream) {
    SampleArgs sa;
    QK_TRY(sampled_args(mh, prompt, B, N, tau, seed, tokens, logprobs, &sa));
    Model& m = *(Model*)mh;
    QK_TRY(check_pages(m, kv, pages, B));
    return rollout_impl(m, mh, paged_view(m, kv, *pages), prompt, B, P, N, logprobs, nullptr, &sa,
                        workspace, ws_bytes, (cudaStream_t)stream);
}

int qk_check_status(qk_model* mh, void* stream, uint32_t* flags) {
    if (!mh) return set_error(QK_EINVAL, "null argument");
    Model& m = *(Model*)mh;
    cudaStream_t s = (cudaStream_t)stream;
    uint32_t v = 0;
    QK_TRY_CUDA(cudaStreamSynchronize(s));
    QK_TRY_CUDA(cudaMemcpy(&v, m.status, sizeof(v), cudaMemcpyDeviceToHost));
    QK_TRY_CUDA(cudaMemset(m.status, 0, sizeof(v)));
    if (flags) *flags = v;
    if (v & QK_STATUS_TIMEOUT)
        return set_error(QK_ETIMEOUT, "a bounded device wait expired (device status 0x%x)", v);
    if (v) return set_error(QK_EDEVICE, "device status 0x%x", v);
    return QK_OK;
}

}  // extern "C"
