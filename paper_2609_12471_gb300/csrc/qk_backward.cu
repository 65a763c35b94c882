// Backward pass of the decoder: the gradient, with respect to every weight tensor,
// of the token-weighted negative log-likelihood
//     loss = sum_{b, t < T-1} coef[b, t] * (-log p(tokens[b, t+1] | tokens[b, <= t])),
// which is the SFT objective of Eq. sft (Sec. "Task Serialization and SFT
// Objective") with coef = mask / (number of target tokens), and whose gradient is
// that of the GRPO objective of Eq. ppo (Sec. "GRPO Optimization") with
// coef = -d L / d lp (qk_grpo_coef).
//
// Schedule (one call, one stream):
//   1. forward over all layers, keeping each layer's activations (input residual x_l
//      and x_mid in fp32; norms, projections, rotated q / k, v, attention output and
//      log-sum-exp, SwiGLU inputs and output in the activation type);
//   2. head, in chunks of rows: lm_head logits -> per-row log-sum-exp (tile
//      statistics + combine), then dz = coef (softmax - onehot) in the activation
//      type from a second pass over the logits, dW_lm (+)= dz^T hn, d hn = dz W_lm;
//      final-norm backward;
//   3. per layer, last to first: the backward of the MLP and of W_o, then of the
//      attention (bf16, head_dim 128: one fused tcgen05 kernel that forms P and
//      dS = P (dP - D) on chip and accumulates dV, dK per key tile and dQ by TMA
//      reduce-add; otherwise P again from the stored log-sum-exp as [T, T] blocks
//      (causal tiles only), dS, dQ = dS K, dK and dV summed over each GQA group as
//      batched GEMMs), then QK-norm and RoPE, W_qkv and the input norm, adding into
//      the running residual gradient;
//   4. embedding gradient (scatter-add of the residual gradient).
// Every product is a bwd::Gemm (k_gemm_bwd.cu): tcgen05 for bf16 models, CUDA cores
// for fp32 models.  Gain gradients are reduced in a fixed order; the embedding
// gradient adds rows that share a token with fp32 atomics.
#include <math.h>

#include "bwd_common.cuh"

namespace qk {

using namespace bwd;

namespace {

constexpr int kHeadRows = 4096;  // lm_head rows per chunk (the dz buffer is [rows, V])

size_t align256(size_t v) { return (v + 255) & ~(size_t)255; }

// A buffer with one copy per layer.
struct PerLayer {
    char* base;
    size_t stride;
    void* at(int l) const { return base ? base + (size_t)l * stride : nullptr; }
};

struct BwdLayout {
    float* xs;  // (L + 1) x [M, H]: x_0 (embedding) .. x_L
    // kept from the forward pass, per layer
    PerLayer u1, qkv, qr, kvh, lse_a, O, x_mid, u2, gu, h;
    // one copy
    int* tgt;
    float* w;
    float* loss_rows;
    float* dx;
    void* dx_act;
    void* hn;
    float2* st_h;
    float* lse_h;
    float* zt;
    void* dz;
    float2* st_a;
    void* P;
    void* dgu;
    float* du;
    void* dO;
    float* Dv;
    void* dS;
    float* dqr;
    float* dkr;
    void* dqkv;
    float* part;
    size_t total;
};

bool fused_attn_bwd(const Model& m, int T) {
    const qk_config& c = m.cfg;
    return c.dtype == QK_DTYPE_BF16 && attn_bwd_supported(c.head_dim, c.n_q_heads, c.n_kv_heads, T);
}

int bwd_layout(const Model& m, int B, int T, char* base, BwdLayout* L) {
    const qk_config& c = m.cfg;
    const size_t es = m.es, M = (size_t)B * T, H = c.hidden, d = c.head_dim, nq = c.n_q_heads,
                 nkv = c.n_kv_heads, I = c.intermediate, V = c.vocab, nqkv = (nq + 2 * nkv) * d,
                 Z = (size_t)B * nq, nl = c.n_layers;
    const size_t Mc = M < (size_t)kHeadRows ? M : (size_t)kHeadRows;
    const size_t nct_v = cdiv(c.vocab, gemm_tile_n(m, c.vocab, 0));
    const size_t nct_a = cdiv(T, gemm_tile_n(m, T, 1));
    size_t off = 0;
    auto take = [&](size_t bytes) {
        void* p = base ? base + off : nullptr;
        off = align256(off + bytes);
        return p;
    };
    auto per_layer = [&](size_t bytes) {
        PerLayer q;
        q.stride = align256(bytes);
        q.base = (char*)take(q.stride * nl);
        return q;
    };
    L->xs = (float*)take((nl + 1) * M * H * 4);
    L->u1 = per_layer(M * H * es);
    L->qkv = per_layer(M * nqkv * es);
    L->qr = per_layer(M * nq * d * es);
    L->kvh = per_layer(2 * M * nkv * d * es);
    L->lse_a = per_layer(Z * T * 4);
    L->O = per_layer(M * nq * d * es);
    L->x_mid = per_layer(M * H * 4);
    L->u2 = per_layer(M * H * es);
    L->gu = per_layer(M * 2 * I * es);
    L->h = per_layer(M * I * es);
    L->tgt = (int*)take(M * 4);
    L->w = (float*)take(M * 4);
    L->loss_rows = (float*)take(M * 4);
    L->dx = (float*)take(M * H * 4);
    L->dx_act = take(M * H * es);
    L->hn = take(M * H * es);
    L->st_h = (float2*)take(Mc * nct_v * 8);
    L->lse_h = (float*)take(Mc * 4);
    L->zt = (float*)take(Mc * 4);
    L->dz = take(Mc * V * es);
    // the bf16 head_dim-128 path runs the fused attention backward: no [T, T] blocks
    const bool fused_attn = fused_attn_bwd(m, T);
    L->st_a = (float2*)take(Z * T * nct_a * 8);
    L->P = fused_attn ? nullptr : take(Z * T * T * es);
    L->dgu = take(M * 2 * I * es);
    L->du = (float*)take(M * H * 4);
    L->dO = take(M * nq * d * es);
    L->Dv = (float*)take(Z * T * 4);
    L->dS = fused_attn ? nullptr : take(Z * T * T * es);
    L->dqr = (float*)take(M * nq * d * 4);
    L->dkr = (float*)take(M * nkv * d * 4);
    L->dqkv = take(M * nqkv * es);
    const size_t nb = rms_part_rows((int)M);
    L->part = (float*)take(nb * (H > 2 * d ? H : 2 * d) * 4);
    L->total = off;
    return QK_OK;
}

// ------------------------------------------------------------------ GEMM builders
Op opk(const void* p, long long ld, int rows, int cols) {
    Op o{};
    o.ptr = p;
    o.ld = ld;
    o.rows = rows;
    o.cols = cols;
    o.zdiv = 1;
    o.zq = 1;
    o.pitch = 128;
    return o;
}
Op opm(const void* p, long long ld, int rows, int cols) {
    Op o = opk(p, ld, rows, cols);
    o.mn = 1;
    return o;
}
Out out2(void* C, long long ldc, int rows, int cols, const float* addend = nullptr) {
    Out o{};
    o.C = C;
    o.ldc = ldc;
    o.rows = rows;
    o.cols = cols;
    o.zq = 1;
    o.addend = addend;
    return o;
}
Sched sch(int Z, int M, int N, int K, int red = RED_FULL) {
    Sched s{};
    s.Z = Z;
    s.M = M;
    s.N = N;
    s.K = K;
    s.red = red;
    return s;
}
bwd::Epi epi_mode(int mode, int rows_per_z = 0) {
    bwd::Epi e{};
    e.mode = mode;
    e.scale = 1.f;
    e.rows_per_z = rows_per_z;
    return e;
}

struct Ctx {
    Model& m;
    const BwdLayout& L;
    int B, T, M;
    cudaStream_t s;
    char* act(void* p, size_t elems) const { return (char*)p + elems * m.es; }
};

// C[M, N] = X[M, K] W[N, K]^T (activation or fp32 store, fp32 with addend).
int lin_fwd(const Ctx& x, const void* X, int K, const void* W, int N, void* C, int mode,
            const float* addend = nullptr) {
    Gemm g{};
    g.A = opk(X, K, x.M, K);
    g.B = opk(W, K, N, K);
    g.out = out2(C, N, x.M, N, addend);
    g.epi = epi_mode(mode);
    g.sc = sch(1, x.M, N, K);
    return run_gemm(x.m, g, x.s);
}

// C[M, Kin] = dY[M, Nout] W[Nout, Kin] (rows of dY: stride ldy).
int lin_dx(const Ctx& x, const void* dY, long long ldy, const void* W, int Nout, int Kin, void* C,
           int mode, int M) {
    Gemm g{};
    g.A = opk(dY, ldy, M, Nout);
    g.B = opm(W, Kin, Nout, Kin);
    g.out = out2(C, Kin, M, Kin);
    g.epi = epi_mode(mode);
    g.sc = sch(1, M, Kin, Nout);
    return run_gemm(x.m, g, x.s);
}

// G[Mo, Kin] (+)= dY^T X over M token rows: output row i of G reads column
// xb + (i / 128) pitch + i % 128 of dY (row stride ldy, cols_dy columns).
int lin_dw(const Ctx& x, const void* dY, long long ldy, int cols_dy, int xb, int pitch, int Mo,
           const void* X, long long ldx, int Kin, float* G, bool add, int M) {
    Gemm g{};
    g.A = opm(dY, ldy, M, cols_dy);
    g.A.xb = xb;
    g.A.pitch = pitch;
    g.B = opm(X, ldx, M, Kin);
    g.out = out2(G, Kin, Mo, Kin, add ? G : nullptr);
    g.epi = epi_mode(E_F32);
    g.sc = sch(1, Mo, Kin, M);
    return run_gemm(x.m, g, x.s);
}

// Attention operands.  Token-major buffers [M, heads * d]: batch entry z = b nq + h (or
// b nkv + g) selects rows b T .. and the head's d columns.  Head-major K / V ([2][B][nkv][T][d],
// K then V): the kv head of query head z is plane z / (nq / nkv).
Op head_op(const void* p, int ld, int M, int heads, int d, int T, bool mn) {
    Op o = mn ? opm(p, ld, M, ld) : opk(p, ld, M, ld);
    o.zq = heads;
    o.zx = d;
    o.zy = T;
    return o;
}
Op kv_op(const void* kvh, int M, int nkv, int d, int T, int grp, bool mn, bool v) {
    const int rows = M * nkv;
    Op o = mn ? opm(kvh, d, 2 * rows, d) : opk(kvh, d, 2 * rows, d);
    o.yb = v ? rows : 0;
    o.zdiv = grp;
    o.zy = T;
    return o;
}

// S = q k^T / sqrt(d) over the causal tiles of every (row, query head), epilogue e.
Gemm scores_gemm(const Ctx& x, int l, const bwd::Epi& e) {
    const qk_config& c = x.m.cfg;
    const int d = c.head_dim, nq = c.n_q_heads, nkv = c.n_kv_heads, T = x.T, M = x.M;
    Gemm g{};
    g.A = head_op(x.L.qr.at(l), nq * d, M, nq, d, T, false);
    g.B = kv_op(x.L.kvh.at(l), M, nkv, d, T, nq / nkv, false, false);
    g.sc = sch(x.B * nq, T, T, d);
    g.sc.tri = 1;
    g.epi = e;
    g.epi.scale = 1.f / sqrtf((float)d);
    g.epi.causal = 1;
    g.epi.rows_per_z = T;
    g.out = out2(x.L.P, T, x.B * nq * T, T);
    g.out.zrow = T;
    return g;
}

// P = softmax of the causal scores of layer l from its stored log-sum-exp.
int probs(const Ctx& x, int l) {
    bwd::Epi e = epi_mode(E_SOFTMAX);
    e.lse = (const float*)x.L.lse_a.at(l);
    return run_gemm(x.m, scores_gemm(x, l, e), x.s);
}

// Causal attention of layer l: O and the per-row log-sum-exp.  bf16 models with
// head_dim 128: the tcgen05 flash kernel (k_attn_prefill.cu); otherwise scores ->
// statistics -> P -> P V through the batched GEMM.
int attn_fwd(const Ctx& x, int l) {
    Model& m = x.m;
    const qk_config& c = m.cfg;
    const int d = c.head_dim, nq = c.n_q_heads, nkv = c.n_kv_heads, T = x.T, M = x.M, Z = x.B * nq;
    const BwdLayout& L = x.L;
    float* lse = (float*)L.lse_a.at(l);
    if (c.dtype == QK_DTYPE_BF16 && attn_prefill_supported(d, nq, nkv))
        return launch_attn_prefill((const bf16*)L.qr.at(l), nq * d, L.kvh.at(l), nq, nkv, KvPages::dense(x.B, T),
                                   x.B, T, 0, nullptr, (bf16*)L.O.at(l), m.num_sms, m.status, x.s, lse);
    const int tn = gemm_tile_n(m, T, 1);
    bwd::Epi e = epi_mode(E_STATS);
    e.stats = L.st_a;
    e.n_ct = cdiv(T, tn);
    Gemm g = scores_gemm(x, l, e);
    g.out = out2(nullptr, T, Z * T, T);
    QK_TRY(run_gemm(m, g, x.s));
    launch_stats_combine(L.st_a, cdiv(T, tn), tn, 1, Z * T, T, lse, nullptr, nullptr, nullptr, x.s);
    QK_TRY(probs(x, l));
    Gemm pv{};
    pv.A = opk(L.P, T, Z * T, T);
    pv.A.zy = T;
    pv.B = kv_op(L.kvh.at(l), M, nkv, d, T, nq / nkv, true, true);
    pv.sc = sch(Z, T, d, T, RED_PREFIX);
    pv.sc.desc_m = 1;
    pv.epi = epi_mode(E_ACT, T);
    pv.out = out2(L.O.at(l), nq * d, M, nq * d);
    pv.out.zq = nq;
    pv.out.zrow = T;
    pv.out.zcol = d;
    return run_gemm(m, pv, x.s);
}

// ------------------------------------------------------------------ layer forward
// x_out = layer l (x_in); keeps the layer's activations (u1, qkv, qr, kvh, lse, O, x_mid,
// u2, gu, h) for its backward.
int layer_fwd(const Ctx& x, int l, const float* x_in, float* x_out) {
    Model& m = x.m;
    const qk_config& c = m.cfg;
    const LayerW& W = m.layers[l];
    const BwdLayout& L = x.L;
    const int H = c.hidden, d = c.head_dim, nq = c.n_q_heads, nkv = c.n_kv_heads, I = c.intermediate;
    const int nqkv = (nq + 2 * nkv) * d, T = x.T, M = x.M;
    const float eps = (float)c.rms_eps;
    launch_rmsnorm(x_in, 1, 0, W.attn_norm, H, eps, L.u1.at(l), c.dtype, M, x.s);
    QK_TRY(lin_fwd(x, L.u1.at(l), H, W.w_qkv, nqkv, L.qkv.at(l), E_ACT));
    launch_qk_fwd(L.qkv.at(l), nqkv, M, T, nq, nkv, d, W.q_norm, W.k_norm, eps, m.rope_cos, m.rope_sin,
                  L.qr.at(l), L.kvh.at(l), c.dtype, x.s);
    QK_TRY(attn_fwd(x, l));
    float* x_mid = (float*)L.x_mid.at(l);
    QK_TRY(lin_fwd(x, L.O.at(l), nq * d, W.w_o, H, x_mid, E_F32, x_in));
    launch_rmsnorm(x_mid, 1, 0, W.mlp_norm, H, eps, L.u2.at(l), c.dtype, M, x.s);
    QK_TRY(lin_fwd(x, L.u2.at(l), H, W.w_gu, 2 * I, L.gu.at(l), E_ACT));
    launch_swiglu_fwd(L.gu.at(l), M, I, L.h.at(l), c.dtype, x.s);
    return lin_fwd(x, L.h.at(l), I, W.w_d, H, x_out, E_F32, x_mid);
}

// ------------------------------------------------------------------ layer backward
// Given dx = d loss / d x_{l+1} (fp32 and its activation copy), leaves d loss / d x_l
// there and writes the layer's weight gradients G[0..10] (canonical order).
int layer_bwd(const Ctx& x, int l, float* const* G, bool acc) {
    Model& m = x.m;
    const qk_config& c = m.cfg;
    const LayerW& W = m.layers[l];
    const BwdLayout& L = x.L;
    const int H = c.hidden, d = c.head_dim, nq = c.n_q_heads, nkv = c.n_kv_heads, I = c.intermediate;
    const int nqkv = (nq + 2 * nkv) * d, T = x.T, M = x.M, Z = x.B * nq, Zk = x.B * nkv, grp = nq / nkv;
    const float eps = (float)c.rms_eps;
    const float* x_in = L.xs + (size_t)l * M * H;
    const int nb = rms_part_rows(M);
    void* u1 = L.u1.at(l);
    void* qkv = L.qkv.at(l);
    void* qr = L.qr.at(l);
    void* kvh = L.kvh.at(l);
    void* O = L.O.at(l);
    void* u2 = L.u2.at(l);
    void* gu = L.gu.at(l);
    // ---- MLP: x_out = x_mid + W_d h, h = silu(W_g u2) * (W_u u2)
    QK_TRY(lin_dw(x, L.dx_act, H, H, 0, 128, H, L.h.at(l), I, I, G[10], acc, M));
    {  // dh = dx W_d with the SwiGLU backward in the epilogue: dgu = (dg, du) from gu
        Gemm g{};
        g.A = opk(L.dx_act, H, M, H);
        g.B = opm(W.w_d, I, H, I);
        g.out = out2(L.dgu, 2 * I, M, 2 * I);
        g.epi = epi_mode(E_SWIGLU_BWD);
        g.epi.P = gu;
        g.sc = sch(1, M, I, H);
        QK_TRY(run_gemm(m, g, x.s));
    }
    QK_TRY(lin_dw(x, L.dgu, 2 * I, 2 * I, 0, 256, I, u2, H, H, G[8], acc, M));
    QK_TRY(lin_dw(x, L.dgu, 2 * I, 2 * I, 128, 256, I, u2, H, H, G[9], acc, M));
    QK_TRY(lin_dx(x, L.dgu, 2 * I, W.w_gu, 2 * I, H, L.du, E_F32, M));
    launch_rms_bwd((const float*)L.x_mid.at(l), W.mlp_norm, L.du, M, H, eps, 0, L.dx, L.dx_act, L.part,
                   c.dtype, x.s);
    launch_gain_reduce(L.part, nb, H, H, G[7], acc, x.s);
    // ---- attention output: x_mid = x_in + W_o o
    QK_TRY(lin_dw(x, L.dx_act, H, H, 0, 128, H, O, nq * d, nq * d, G[6], acc, M));
    QK_TRY(lin_dx(x, L.dx_act, H, W.w_o, H, nq * d, L.dO, E_ACT, M));
    launch_attn_d(L.dO, O, M, T, nq, d, L.Dv, c.dtype, x.s);
    if (fused_attn_bwd(m, T)) {  // P and dS stay on chip (k_attn_bwd.cu)
        QK_TRY_CUDA(cudaMemsetAsync(L.dqr, 0, (size_t)M * nq * d * 4, x.s));
        const int rc = launch_attn_bwd((const bf16*)qr, (const bf16*)L.dO, (const bf16*)kvh,
                                       (const float*)L.lse_a.at(l), L.Dv, L.dqr, L.dkr, (bf16*)L.dqkv, nqkv,
                                       (nq + nkv) * d, x.B, T, nq, nkv, m.num_sms, m.status, x.s);
        if (rc != QK_OK) return set_error(rc, "fused attention backward launch");
    } else {
    // P again from the stored log-sum-exp, then dS = P (dO V^T - D) / sqrt(d)
    QK_TRY(probs(x, l));
    Gemm g{};
    g.A = head_op(L.dO, nq * d, M, nq, d, T, false);
    g.B = kv_op(kvh, M, nkv, d, T, grp, false, true);
    g.sc = sch(Z, T, T, d);
    g.sc.tri = 1;
    g.epi = epi_mode(E_DS, T);
    g.epi.scale = 1.f / sqrtf((float)d);
    g.epi.P = L.P;
    g.epi.D = L.Dv;
    g.out = out2(L.dS, T, Z * T, T);
    g.out.zrow = T;
    QK_TRY(run_gemm(m, g, x.s));
    // dq_rot = dS k (keys up to the tile's last query)
    Gemm gq{};
    gq.A = opk(L.dS, T, Z * T, T);
    gq.A.zy = T;
    gq.B = kv_op(kvh, M, nkv, d, T, grp, true, false);
    gq.sc = sch(Z, T, d, T, RED_PREFIX);
    gq.sc.desc_m = 1;
    gq.epi = epi_mode(E_F32, T);
    gq.out = out2(L.dqr, nq * d, M, nq * d);
    gq.out.zq = nq;
    gq.out.zrow = T;
    gq.out.zcol = d;
    QK_TRY(run_gemm(m, gq, x.s));
    // dk_rot = sum over the group's heads of dS^T q; dv = sum of P^T dO (queries from the key tile on)
    Gemm gk{};
    gk.A = opm(L.dS, T, Z * T, T);
    gk.A.zy = grp * T;
    gk.A.kwrap = T;
    gk.A.kwy = T;
    gk.B = opm(qr, nq * d, M, nq * d);
    gk.B.zq = nkv;
    gk.B.zx = grp * d;
    gk.B.zy = T;
    gk.B.kwrap = T;
    gk.B.kwx = d;
    gk.sc = sch(Zk, T, d, grp * T, RED_SUFFIX);
    gk.sc.seg = T;
    gk.epi = epi_mode(E_F32, T);
    gk.out = out2(L.dkr, nkv * d, M, nkv * d);
    gk.out.zq = nkv;
    gk.out.zrow = T;
    gk.out.zcol = d;
    QK_TRY(run_gemm(m, gk, x.s));
    Gemm gv = gk;
    gv.A.ptr = L.P;
    gv.B.ptr = L.dO;
    gv.epi = epi_mode(E_ACT, T);
    gv.out = out2(x.act(L.dqkv, (size_t)(nq + nkv) * d), nqkv, M, nkv * d);
    gv.out.zq = nkv;
    gv.out.zrow = T;
    gv.out.zcol = d;
    QK_TRY(run_gemm(m, gv, x.s));
    }
    // ---- QK-norm + RoPE, then the projections
    launch_qk_bwd(L.dqr, L.dkr, qkv, nqkv, M, T, nq, nkv, d, W.q_norm, W.k_norm, eps, m.rope_cos,
                  m.rope_sin, L.dqkv, L.part, c.dtype, x.s);
    launch_gain_reduce(L.part, nb, d, 2 * d, G[4], acc, x.s);
    launch_gain_reduce(L.part + d, nb, d, 2 * d, G[5], acc, x.s);
    QK_TRY(lin_dw(x, L.dqkv, nqkv, nqkv, 0, 128, nq * d, u1, H, H, G[1], acc, M));
    QK_TRY(lin_dw(x, L.dqkv, nqkv, nqkv, nq * d, 128, nkv * d, u1, H, H, G[2], acc, M));
    QK_TRY(lin_dw(x, L.dqkv, nqkv, nqkv, (nq + nkv) * d, 128, nkv * d, u1, H, H, G[3], acc, M));
    QK_TRY(lin_dx(x, L.dqkv, nqkv, W.w_qkv, nqkv, H, L.du, E_F32, M));
    launch_rms_bwd(x_in, W.attn_norm, L.du, M, H, eps, 0, L.dx, L.dx_act, L.part, c.dtype, x.s);
    launch_gain_reduce(L.part, nb, H, H, G[0], acc, x.s);
    return QK_OK;
}

int backward_impl(Model& m, const int32_t* tokens, int B, int T, const float* coef, float* const* grads,
                  bool acc, float* loss, void* ws, cudaStream_t s) {
    const qk_config& c = m.cfg;
    BwdLayout L;
    QK_TRY(bwd_layout(m, B, T, (char*)ws, &L));
    const int M = B * T, H = c.hidden, V = c.vocab, nl = c.n_layers;
    Ctx x{m, L, B, T, M, s};
    const float eps = (float)c.rms_eps;
    launch_rows_prep(tokens, B, T, coef, V, L.tgt, L.w, m.status, s);
    launch_embed(m.embed, c.dtype, V, H, TokIndex{tokens, T, T, 0}, M, L.xs, m.status, s);
    for (int l = 0; l < nl; ++l)
        QK_TRY(layer_fwd(x, l, L.xs + (size_t)l * M * H, L.xs + (size_t)(l + 1) * M * H));
    // ---- head
    const float* xL = L.xs + (size_t)nl * M * H;
    float* g_lm = grads[2 + 11 * nl];
    launch_rmsnorm(xL, 1, 0, m.final_norm, H, eps, L.hn, c.dtype, M, s);
    const int tn = gemm_tile_n(m, V, 0), nct = cdiv(V, tn);
    for (int r0 = 0; r0 < M; r0 += kHeadRows) {
        const int rows = M - r0 < kHeadRows ? M - r0 : kHeadRows;
        const void* hn = x.act(L.hn, (size_t)r0 * H);
        Gemm g{};
        g.A = opk(hn, H, rows, H);
        g.B = opk(m.lm_head, H, V, H);
        g.sc = sch(1, rows, V, H);
        g.epi = epi_mode(E_STATS, rows);
        g.epi.tgt = L.tgt + r0;
        g.epi.zt = L.zt;
        g.epi.stats = L.st_h;
        g.epi.n_ct = nct;
        g.out = out2(nullptr, V, rows, V);
        QK_TRY(run_gemm(m, g, s));
        launch_stats_combine(L.st_h, nct, tn, 0, rows, rows, L.lse_h, L.w + r0, L.zt, L.loss_rows + r0, s);
        g.epi.mode = E_SOFTMAX;
        g.epi.lse = L.lse_h;
        g.epi.w = L.w + r0;
        g.out = out2(L.dz, V, rows, V);
        QK_TRY(run_gemm(m, g, s));
        QK_TRY(lin_dw(x, L.dz, V, V, 0, 128, V, hn, H, H, g_lm, acc || r0 > 0, rows));
        QK_TRY(lin_dx(x, L.dz, V, m.lm_head, V, H, L.du + (size_t)r0 * H, E_F32, rows));
    }
    const int nb = rms_part_rows(M);
    launch_rms_bwd(xL, m.final_norm, L.du, M, H, eps, 1, L.dx, L.dx_act, L.part, c.dtype, s);
    launch_gain_reduce(L.part, nb, H, H, grads[1 + 11 * nl], acc, s);
    if (loss) launch_sum(L.loss_rows, M, loss, s);
    // ---- layers, last to first
    for (int l = nl - 1; l >= 0; --l) QK_TRY(layer_bwd(x, l, grads + 1 + 11 * l, acc));
    // ---- embedding
    if (!acc) QK_TRY_CUDA(cudaMemsetAsync(grads[0], 0, (size_t)V * H * 4, s));
    launch_embed_bwd(tokens, L.dx, M, H, V, grads[0], s);
    return QK_OK;
}

}  // namespace

// Rows of a bf16 call are padded to a multiple of 128 positions (the tensor-core tiles'
// granularity): the padding follows every real position, so under causal attention no
// real position sees it, and its coefficients are zero, so it adds nothing to the loss
// and receives no gradient.
static int padded_len(const Model& m, int T) {
    return m.cfg.dtype == QK_DTYPE_BF16 && T % 128 ? (T + 127) / 128 * 128 : T;
}

// Workspace: the layout for the padded length, then (when padding) the padded tokens
// [B, Tp] and coefficients [B, Tp - 1].
static size_t pad_bytes(int B, int T, int Tp) {
    if (Tp == T) return 0;
    return align256((size_t)B * Tp * 4) + align256((size_t)B * (Tp - 1) * 4);
}

int backward_workspace_bytes(const Model& m, int B, int T, size_t* bytes) {
    if (B < 1 || T < 2) return set_error(QK_ESHAPE, "backward needs B >= 1 and T >= 2");
    const int Tp = padded_len(m, T);
    if ((size_t)B * Tp > ((size_t)1 << 24)) return set_error(QK_ESHAPE, "too many tokens in one call");
    BwdLayout L;
    QK_TRY(bwd_layout(m, B, Tp, nullptr, &L));
    *bytes = L.total + pad_bytes(B, T, Tp);
    return QK_OK;
}

}  // namespace qk

using namespace qk;

extern "C" int qk_backward_logprob(qk_model* mh, const int32_t* tokens, int B, int T, const float* coef,
                                   float* const* grads, int n_grads, int accumulate, float* loss,
                                   void* workspace, size_t ws_bytes, void* stream) {
    if (!mh || !tokens || !coef || !grads) return set_error(QK_EINVAL, "null argument");
    Model& m = *(Model*)mh;
    const qk_config& c = m.cfg;
    const int want = 3 + 11 * c.n_layers;
    if (n_grads != want) return set_error(QK_EINVAL, "n_grads %d, the model has %d tensors", n_grads, want);
    for (int i = 0; i < want; ++i)
        if (!grads[i] || ((uintptr_t)grads[i] & 15))
            return set_error(QK_EINVAL, "gradient buffer %d is NULL or not 16-byte aligned", i);
    size_t need = 0;
    QK_TRY(backward_workspace_bytes(m, B, T, &need));
    const int Tp = padded_len(m, T);
    if (Tp > c.max_positions)
        return set_error(QK_ESHAPE, "T %d (%d padded) exceeds max_positions %d", T, Tp, c.max_positions);
    if (c.dtype == QK_DTYPE_BF16 &&
        (c.head_dim != 128 || c.vocab % 64 || c.hidden % 64 || ((uintptr_t)tokens & 3) || ((uintptr_t)coef & 3)))
        return set_error(QK_ESHAPE, "bf16 backward needs head_dim 128 and vocab, hidden %% 64 == 0");
    if (!workspace || ((uintptr_t)workspace & 255)) return set_error(QK_EINVAL, "workspace NULL or not 256-byte aligned");
    if (ws_bytes < need) return set_error(QK_ENOSPACE, "workspace has %zu bytes, needs %zu", ws_bytes, need);
    cudaGetLastError();
    cudaStream_t s = (cudaStream_t)stream;
    if (Tp != T) {  // padded copies of the rows after the layout's buffers
        BwdLayout L;
        QK_TRY(bwd_layout(m, B, Tp, nullptr, &L));
        int32_t* tok_p = (int32_t*)((char*)workspace + L.total);
        float* coef_p = (float*)((char*)tok_p + align256((size_t)B * Tp * 4));
        launch_pad_rows(tokens, coef, B, T, Tp, tok_p, coef_p, s);
        tokens = tok_p;
        coef = coef_p;
    }
    int rc = backward_impl(m, tokens, B, Tp, coef, grads, accumulate != 0, loss, workspace, s);
    if (rc != QK_OK) return rc;
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_error(e, "backward launches");
    return QK_OK;
}
