// Kernel selection for the linear layers and attention of one forward call.
#include "bwd_common.cuh"

namespace qk {

// bf16: up to kGemvMaxRows token rows stream the weights through the CUDA-core
// GEMV (bound by reading W); 256 or more rows whose shape fills the SMs with 256 x 256
// tiles go to the batched tcgen05 GEMM of k_gemm_bwd.cu; other row counts to the
// swap-AB tcgen05 GEMM of k_gemm_tc.cu.  fp32: CUDA-core GEMM (no TF32).
void linear(Model& m, const void* A, int lda, const void* W, void* C, int ldc, int M, int N,
            int K, int epi, void* gu, cudaStream_t s) {
    const int dt = m.cfg.dtype;
    if (dt == QK_DTYPE_BF16 && M <= kGemvMaxRows) {
        launch_gemv_bf16((const bf16*)A, lda, (const bf16*)W, C, ldc, M, N, K, epi, s);
        return;
    }
    // 256 or more rows (prefill / scoring): 256 x 256 tensor-core tiles when they fit
    if (dt == QK_DTYPE_BF16 && m.test_wait_cycles == 0 && bwd::linear_large(m, A, lda, W, C, ldc, M, N, K, epi, s))
        return;
    if (dt == QK_DTYPE_BF16 && gemm_tc_supported(A, lda, N, K)) {
        const long long test_wait = m.test_wait_cycles;  // one launch only
        m.test_wait_cycles = 0;
        int rc = launch_gemm_tc((const bf16*)A, lda, (const bf16*)W, C, ldc, M, N, K, epi,
                                m.num_sms, m.status, s, test_wait);
        if (rc != QK_OK && !m.deferred_error) m.deferred_error = rc;
        return;
    }
    if (epi == EPI_SWIGLU) {
        launch_gemm_simt(A, lda, W, gu, 2 * N, M, 2 * N, K, dt, EPI_STORE_ACT, s);
        launch_swiglu(gu, C, dt, M, N, s);
        return;
    }
    launch_gemm_simt(A, lda, W, C, ldc, M, N, K, dt, epi, s);
}

void launch_attention(Model& m, const void* q, int q_ld, const void* k_cache, const void* v_cache,
                      int M, const KvPages& kp, PosIndex pos, void* o, void* scratch,
                      cudaStream_t s) {
    const qk_config& c = m.cfg;
    // the tensor-core kernels address V as the rows after K's pool
    const bool v_follows = (const char*)v_cache == (const char*)k_cache + (size_t)kp.n_pages * c.n_kv_heads *
                                                                         kp.page * c.head_dim * 2;
    if (c.dtype == QK_DTYPE_BF16 && pos.T == 1 && scratch &&
        attn_decode_supported(c.head_dim, c.n_q_heads, c.n_kv_heads) && v_follows) {
        int rc = launch_attn_decode((const bf16*)q, q_ld, k_cache, c.n_q_heads, c.n_kv_heads,
                                    kp, M, pos, scratch, (bf16*)o, m.num_sms, m.status, s);
        if (rc != QK_OK && !m.deferred_error) m.deferred_error = rc;
        return;
    }
    if (c.dtype == QK_DTYPE_BF16 && pos.T > 1 &&
        attn_prefill_supported(c.head_dim, c.n_q_heads, c.n_kv_heads) && v_follows) {
        int rc = launch_attn_prefill((const bf16*)q, q_ld, k_cache, c.n_q_heads, c.n_kv_heads,
                                     kp, M / pos.T, pos.T, pos.start, pos.pos_dev,
                                     (bf16*)o, m.num_sms, m.status, s);
        if (rc != QK_OK && !m.deferred_error) m.deferred_error = rc;
        return;
    }
    launch_attention_simt(q, q_ld, k_cache, v_cache, c.dtype, M, c.n_q_heads, c.n_kv_heads,
                          c.head_dim, kp, pos, o, m.status, s);
}

}  // namespace qk
