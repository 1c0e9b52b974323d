/*
 * FLARE block-denoising attention step: plain fp64 CPU oracle.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing on the product path may call, link or
 * load this file; only the tests, the smoke check and the CPU-baseline leg of
 * the benchmark do.  It shares no code, header, constant or helper with the
 * CUDA library: the two meet only through the seeded inputs.
 *
 * Every routine is the paper's definition written out, slowly and in double
 * precision, in the paper's order and notation:
 *
 *   gated delta rule, per step (Appendix "Single-stream chunkwise training",
 *   Eq. per-step-fwd):
 *       S_pre_t = exp(g_t) S_{t-1}
 *       u_t     = v_t - S_pre_t^T k_t
 *       delta_t = beta_t u_t
 *       S_t     = S_pre_t + k_t delta_t^T
 *       o_t     = s S_t^T q_t                       (token-causal readout)
 *   noisy block forward (Eq. noisy-block-fwd): the block starts from the
 *   committed state and every block position reads the block-end state,
 *       o~_l = s S_B^T q~_l   for all l in the block.
 *   commit at accepted length r (serving appendix, "Recovering the recurrent
 *   state at the accept boundary"): the pool slot becomes S^(r) = S_r, and
 *   r = 0 leaves it unchanged.
 *   AR-Trust verify round (decoding appendix, block layout; serving appendix,
 *   cache-and-scatter): anchor and verify rows read S_{t+1} token-causally,
 *   draft rows read S_L, the states after the anchor and each verify token
 *   are cached, and the commit copies the cached state at the accepted
 *   offset into the pool.
 *   two-stream training forward (Eq. noisy-block-fwd): each noisy block is
 *   seeded with the clean state before it, runs its own tokens and reads its
 *   block-end state; the clean state advances block by block (Eq. f-blk).
 *   two-stream causal ShortConv (Eq. short-conv-noisy): lags inside the block
 *   read the block, earlier lags the committed W-1-token clean state; the
 *   state is committed as the last W-1 tokens of (state ++ accepted rows).
 *   chunkwise form (Eq. chunk-state / Eq. f-blk with WY-corrected values):
 *   an independent second implementation used only to pin the first.
 *   softmax retrieval over a visible set (Eq. softmax-retrieval) with the
 *   Diffusion-Trust block mask: every block row sees the whole paged prefix
 *   and (bidirectional mode) every block token, or (token-causal mode) the
 *   block tokens up to and including itself.
 *
 * Element types of the inputs: 0 = bf16 (raw 16-bit patterns), 1 = fp32,
 * 2 = fp64.  Converting a bf16 or fp32 value to double is exact, so the
 * oracle computes on exactly the values the GPU sees.
 */
#include <math.h>
#include <stddef.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

enum { ORC_BF16 = 0, ORC_F32 = 1, ORC_F64 = 2 };

static double ld(const void* p, int dt, size_t i) {
  if (dt == ORC_F64) return ((const double*)p)[i];
  if (dt == ORC_F32) return (double)((const float*)p)[i];
  uint32_t bits = ((uint32_t)((const uint16_t*)p)[i]) << 16;
  float f;
  memcpy(&f, &bits, sizeof f);
  return (double)f;
}

static void set_threads(int nthreads) {
#ifdef _OPENMP
  if (nthreads > 0) omp_set_num_threads(nthreads);
#else
  (void)nthreads;
#endif
}

int oracle_max_threads(void) {
#ifdef _OPENMP
  return omp_get_max_threads();
#else
  return 1;
#endif
}

/*
 * Gated delta rule over one block for every (request r, value head j),
 * following Eq. per-step-fwd token by token.
 *
 * Shapes (row-major):
 *   q, k        [R, B, Hk, dk]       (q may be NULL when no readout is asked)
 *   v           [R, B, Hv, dv]
 *   log_decay   [R, B, Hv]   g_t, the log-gate; alpha_t = exp(g_t)
 *   beta        [R, B, Hv]
 *   state_pool  [num_slots, Hv, dk, dv], S[i][j] at i*dv + j, so o = S^T q
 *   state_slot  [R]          pool slot holding request r's committed state
 *   accept_len  [R] or NULL  length r at which to take the committed state
 *                            (NULL means the full block, r = B)
 * Outputs (each may be NULL):
 *   out_blockend [R, B, Hv, dv]  o~_l = s S_B^T q_l   (Eq. noisy-block-fwd)
 *   out_causal   [R, B, Hv, dv]  o_t  = s S_t^T q_t   (Eq. per-step-fwd)
 *   state_out    [R, Hv, dk, dv] S_{accept_len[r]}
 * Value head j reads q/k head floor(j * Hk / Hv).
 * Returns 0, or -1 for an invalid slot or accepted length.
 */
int oracle_gdr_per_token(int R, int B, int Hk, int Hv, int dk, int dv, double s,
                         int act_dt, const void* q, const void* k, const void* v,
                         int gate_dt, const void* log_decay, const void* beta,
                         int state_dt, const void* state_pool, int num_slots,
                         const int32_t* state_slot, const int32_t* accept_len,
                         double* out_blockend, double* out_causal, double* state_out,
                         int nthreads) {
  for (int r = 0; r < R; ++r) {
    if (state_slot[r] < 0 || state_slot[r] >= num_slots) return -1;
    if (accept_len && (accept_len[r] < 0 || accept_len[r] > B)) return -1;
  }
  set_threads(nthreads);
#pragma omp parallel for schedule(dynamic, 1)
  for (long item = 0; item < (long)R * Hv; ++item) {
    const int r = (int)(item / Hv), j = (int)(item % Hv);
    const int h = (int)(((long)j * Hk) / Hv);
    const int r_acc = accept_len ? accept_len[r] : B;
    double* S = (double*)malloc(sizeof(double) * dk * dv);
    double* u = (double*)malloc(sizeof(double) * dv);
    double* kt = (double*)malloc(sizeof(double) * dk);
    double* qt = (double*)malloc(sizeof(double) * dk);
    const size_t s0 = ((size_t)state_slot[r] * Hv + j) * dk * dv;
    for (int e = 0; e < dk * dv; ++e) S[e] = ld(state_pool, state_dt, s0 + e);
    if (state_out && r_acc == 0)
      for (int e = 0; e < dk * dv; ++e) state_out[(size_t)item * dk * dv + e] = S[e];
    for (int t = 0; t < B; ++t) {
      const size_t kq = (((size_t)r * B + t) * Hk + h) * dk;
      const size_t vo = (((size_t)r * B + t) * Hv + j) * dv;
      const size_t gb = ((size_t)r * B + t) * Hv + j;
      const double alpha = exp(ld(log_decay, gate_dt, gb));
      const double bt = ld(beta, gate_dt, gb);
      for (int i = 0; i < dk; ++i) kt[i] = ld(k, act_dt, kq + i);
      /* gating decay: S_pre = exp(g_t) S_{t-1} */
      for (int e = 0; e < dk * dv; ++e) S[e] *= alpha;
      /* prediction error u_t = v_t - S_pre^T k_t, delta update delta_t = beta_t u_t */
      for (int c = 0; c < dv; ++c) u[c] = 0.0;
      for (int i = 0; i < dk; ++i)
        for (int c = 0; c < dv; ++c) u[c] += S[i * dv + c] * kt[i];
      for (int c = 0; c < dv; ++c) u[c] = bt * (ld(v, act_dt, vo + c) - u[c]);
      /* outer-product write S_t = S_pre + k_t delta_t^T */
      for (int i = 0; i < dk; ++i)
        for (int c = 0; c < dv; ++c) S[i * dv + c] += kt[i] * u[c];
      /* token-causal output o_t = s S_t^T q_t */
      if (out_causal) {
        for (int i = 0; i < dk; ++i) qt[i] = ld(q, act_dt, kq + i);
        for (int c = 0; c < dv; ++c) {
          double acc = 0.0;
          for (int i = 0; i < dk; ++i) acc += S[i * dv + c] * qt[i];
          out_causal[vo + c] = s * acc;
        }
      }
      if (state_out && t + 1 == r_acc)
        for (int e = 0; e < dk * dv; ++e) state_out[(size_t)item * dk * dv + e] = S[e];
    }
    /* block-end readout: every block row reads S_B (Eq. noisy-block-fwd) */
    if (out_blockend)
      for (int l = 0; l < B; ++l) {
        const size_t ql = (((size_t)r * B + l) * Hk + h) * dk;
        const size_t ol = (((size_t)r * B + l) * Hv + j) * dv;
        for (int i = 0; i < dk; ++i) qt[i] = ld(q, act_dt, ql + i);
        for (int c = 0; c < dv; ++c) {
          double acc = 0.0;
          for (int i = 0; i < dk; ++i) acc += S[i * dv + c] * qt[i];
          out_blockend[ol + c] = s * acc;
        }
      }
    free(qt);
    free(kt);
    free(u);
    free(S);
  }
  return 0;
}

/*
 * AR-Trust verify round, gated-delta-rule part (decoding appendix, "AR-Trust
 * sampling": the block is [anchor, d_0 .. d_{K-1}, MASK ...]; serving
 * appendix, "Recovering the recurrent state at the accept boundary", path (b),
 * cache-and-scatter).  For request r with K = verify_len[r] the block's rows
 * 0..K (anchor and verify rows) are token-causal and rows K+1..L-1 (padding and
 * draft rows) read the whole block.  From S0 = state_pool[state_slot[r]][j]
 * the gated delta rule (Eq. per-step-fwd) runs over all L block tokens; with
 * S_n the state after tokens 0..n-1:
 *   out[r][t][j]        = s S_{t+1}^T q_t   for t <= K   (token-causal rows)
 *   out[r][t][j]        = s S_L^T q_t       for t >  K   (bidirectional rows)
 *   records[r][t][j]    = S_{t+1}           for t <  K   (S^(t): the anchor and
 *                                                          t accepted drafts)
 *   state_out[r][j]     = S_{K+1}                        (S^(K): every draft accepted)
 * Shapes: q, k [R,L,Hk,dk]; v [R,L,Hv,dv]; log_decay, beta [R,L,Hv];
 * state_pool [num_slots,Hv,dk,dv]; state_slot, verify_len [R];
 * out [R,L,Hv,dv]; records [R,max_verify,Hv,dk,dv] (entries t >= K untouched);
 * state_out [R,Hv,dk,dv].  Returns -1 for an invalid slot or verify length
 * (verify_len[r] outside [0, min(max_verify, L-1)]).
 */
int oracle_gdr_verify(int R, int L, int Hk, int Hv, int dk, int dv, double s, int max_verify,
                      int act_dt, const void* q, const void* k, const void* v,
                      int gate_dt, const void* log_decay, const void* beta,
                      int state_dt, const void* state_pool, int num_slots,
                      const int32_t* state_slot, const int32_t* verify_len,
                      double* out, double* records, double* state_out, int nthreads) {
  for (int r = 0; r < R; ++r) {
    if (state_slot[r] < 0 || state_slot[r] >= num_slots) return -1;
    if (verify_len[r] < 0 || verify_len[r] > max_verify || verify_len[r] > L - 1) return -1;
  }
  set_threads(nthreads);
  const size_t nst = (size_t)dk * dv;
#pragma omp parallel for schedule(dynamic, 1)
  for (long item = 0; item < (long)R * Hv; ++item) {
    const int r = (int)(item / Hv), j = (int)(item % Hv);
    const int h = (int)(((long)j * Hk) / Hv);
    const int K = verify_len[r];
    double* S = (double*)malloc(sizeof(double) * nst);
    double* u = (double*)malloc(sizeof(double) * dv);
    double* kt = (double*)malloc(sizeof(double) * dk);
    double* qt = (double*)malloc(sizeof(double) * dk);
    const size_t s0 = ((size_t)state_slot[r] * Hv + j) * nst;
    for (size_t e = 0; e < nst; ++e) S[e] = ld(state_pool, state_dt, s0 + e);
    for (int t = 0; t < L; ++t) {
      const size_t kq = (((size_t)r * L + t) * Hk + h) * dk;
      const size_t vo = (((size_t)r * L + t) * Hv + j) * dv;
      const size_t gb = ((size_t)r * L + t) * Hv + j;
      const double alpha = exp(ld(log_decay, gate_dt, gb));
      const double bt = ld(beta, gate_dt, gb);
      for (int i = 0; i < dk; ++i) kt[i] = ld(k, act_dt, kq + i);
      /* S_pre = exp(g_t) S;  u_t = v_t - S_pre^T k_t;  S = S_pre + k_t (beta_t u_t)^T */
      for (size_t e = 0; e < nst; ++e) S[e] *= alpha;
      for (int c = 0; c < dv; ++c) u[c] = 0.0;
      for (int i = 0; i < dk; ++i)
        for (int c = 0; c < dv; ++c) u[c] += S[i * dv + c] * kt[i];
      for (int c = 0; c < dv; ++c) u[c] = bt * (ld(v, act_dt, vo + c) - u[c]);
      for (int i = 0; i < dk; ++i)
        for (int c = 0; c < dv; ++c) S[i * dv + c] += kt[i] * u[c];
      /* anchor and verify rows read the state right after their own token */
      if (t <= K) {
        for (int i = 0; i < dk; ++i) qt[i] = ld(q, act_dt, kq + i);
        for (int c = 0; c < dv; ++c) {
          double acc = 0.0;
          for (int i = 0; i < dk; ++i) acc += S[i * dv + c] * qt[i];
          out[vo + c] = s * acc;
        }
      }
      /* cache S^(t) for the verify positions, the live state after the last one */
      if (t < K)
        memcpy(records + (((size_t)r * max_verify + t) * Hv + j) * nst, S, sizeof(double) * nst);
      if (t == K) memcpy(state_out + (size_t)item * nst, S, sizeof(double) * nst);
    }
    /* padding and draft rows read the block-end state S_L */
    for (int t = K + 1; t < L; ++t) {
      const size_t ql = (((size_t)r * L + t) * Hk + h) * dk;
      const size_t ol = (((size_t)r * L + t) * Hv + j) * dv;
      for (int i = 0; i < dk; ++i) qt[i] = ld(q, act_dt, ql + i);
      for (int c = 0; c < dv; ++c) {
        double acc = 0.0;
        for (int i = 0; i < dk; ++i) acc += S[i * dv + c] * qt[i];
        out[ol + c] = s * acc;
      }
    }
    free(qt);
    free(kt);
    free(u);
    free(S);
  }
  return 0;
}

/*
 * The same quantities computed a second, independent way: the chunkwise
 * (WY / UT) form of the appendix, "Chunkwise-parallel form",
 * "Chunk-corrected values" and Eq. chunk-state, applied to one block.
 *
 *   gamma_t = sum_{i<=t} g_i                          (cumulative log-gate G_t)
 *   A[t][i] = beta_t exp(gamma_t - gamma_i) (k_t . k_i)        for i < t
 *   (I + A) delta = diag(beta) (V - diag(exp(gamma)) K S0)     (forward substitution)
 *   S_r = exp(gamma_r) S0 + sum_{i<=r} exp(gamma_r - gamma_i) k_i delta_i^T
 *   o~_l = s (exp(gamma_B) S0^T q_l + sum_{i<=B} exp(gamma_B - gamma_i) (q_l . k_i) delta_i)
 *
 * delta here is the per-step delta update (the WY-corrected value scaled by
 * beta); Eq. chunk-state with r = B is Eq. f-blk.  Same arguments and outputs
 * as oracle_gdr_per_token except that token-causal outputs are not formed.
 */
int oracle_gdr_chunked(int R, int B, int Hk, int Hv, int dk, int dv, double s,
                       int act_dt, const void* q, const void* k, const void* v,
                       int gate_dt, const void* log_decay, const void* beta,
                       int state_dt, const void* state_pool, int num_slots,
                       const int32_t* state_slot, const int32_t* accept_len,
                       double* out_blockend, double* state_out, int nthreads) {
  for (int r = 0; r < R; ++r) {
    if (state_slot[r] < 0 || state_slot[r] >= num_slots) return -1;
    if (accept_len && (accept_len[r] < 0 || accept_len[r] > B)) return -1;
  }
  set_threads(nthreads);
#pragma omp parallel for schedule(dynamic, 1)
  for (long item = 0; item < (long)R * Hv; ++item) {
    const int r = (int)(item / Hv), j = (int)(item % Hv);
    const int h = (int)(((long)j * Hk) / Hv);
    const int r_acc = accept_len ? accept_len[r] : B;
    double* S0 = (double*)malloc(sizeof(double) * dk * dv);
    double* gam = (double*)malloc(sizeof(double) * (B + 1));
    double* A = (double*)calloc((size_t)B * B, sizeof(double));
    double* delta = (double*)malloc(sizeof(double) * B * dv);
    const size_t s0 = ((size_t)state_slot[r] * Hv + j) * dk * dv;
    for (int e = 0; e < dk * dv; ++e) S0[e] = ld(state_pool, state_dt, s0 + e);
#define KEL(t, i) ld(k, act_dt, (((size_t)r * B + (t)) * Hk + h) * dk + (i))
#define QEL(t, i) ld(q, act_dt, (((size_t)r * B + (t)) * Hk + h) * dk + (i))
#define VEL(t, c) ld(v, act_dt, (((size_t)r * B + (t)) * Hv + j) * dv + (c))
#define GB(t) (((size_t)r * B + (t)) * Hv + j)
    /* gam[t+1] = gamma after token t (1-based cumulative), gam[0] = 0 */
    gam[0] = 0.0;
    for (int t = 0; t < B; ++t) gam[t + 1] = gam[t] + ld(log_decay, gate_dt, GB(t));
    for (int t = 0; t < B; ++t)
      for (int i = 0; i < t; ++i) {
        double kk = 0.0;
        for (int e = 0; e < dk; ++e) kk += KEL(t, e) * KEL(i, e);
        A[t * B + i] = ld(beta, gate_dt, GB(t)) * exp(gam[t + 1] - gam[i + 1]) * kk;
      }
    /* right-hand side, then forward substitution through the unit lower-triangular I + A */
    for (int t = 0; t < B; ++t) {
      const double bt = ld(beta, gate_dt, GB(t));
      const double G = exp(gam[t + 1]);
      for (int c = 0; c < dv; ++c) {
        double ks = 0.0;
        for (int i = 0; i < dk; ++i) ks += KEL(t, i) * S0[i * dv + c];
        double x = bt * (VEL(t, c) - G * ks);
        for (int i = 0; i < t; ++i) x -= A[t * B + i] * delta[i * dv + c];
        delta[t * dv + c] = x;
      }
    }
    if (state_out) {
      double* So = state_out + (size_t)item * dk * dv;
      const double Gr = exp(gam[r_acc]);
      for (int i = 0; i < dk; ++i)
        for (int c = 0; c < dv; ++c) {
          double acc = Gr * S0[i * dv + c];
          for (int t = 0; t < r_acc; ++t)
            acc += exp(gam[r_acc] - gam[t + 1]) * KEL(t, i) * delta[t * dv + c];
          So[i * dv + c] = acc;
        }
    }
    if (out_blockend) {
      const double GB_ = exp(gam[B]);
      for (int l = 0; l < B; ++l)
        for (int c = 0; c < dv; ++c) {
          double acc = 0.0;
          for (int i = 0; i < dk; ++i) acc += QEL(l, i) * S0[i * dv + c];
          acc *= GB_;
          for (int t = 0; t < B; ++t) {
            double qk = 0.0;
            for (int e = 0; e < dk; ++e) qk += QEL(l, e) * KEL(t, e);
            acc += exp(gam[B] - gam[t + 1]) * qk * delta[t * dv + c];
          }
          out_blockend[(((size_t)r * B + l) * Hv + j) * dv + c] = s * acc;
        }
    }
#undef KEL
#undef QEL
#undef VEL
#undef GB
    free(delta);
    free(A);
    free(gam);
    free(S0);
  }
  return 0;
}

/*
 * Two-stream training forward of a gated-delta-rule layer, noisy stream
 * (appendix "Two-stream recurrence and block-level chain rule",
 * Eq. noisy-block-fwd; Route II computes exactly this, "Fused forward
 * kernel").  For sequence n and value head j the clean recurrence
 * (Eq. per-step-fwd on the clean tokens) starts from S_init[n][j]; block b
 * covers positions bB .. bB+B-1 (0-based).  The noisy recurrence of block b
 * starts from the clean state before the block, S_{bB}, runs the block's B
 * noisy tokens through Eq. per-step-fwd, and every noisy position of the
 * block reads the noisy block-end state:
 *     out[n][l][j] = s S~_{bB+B}^T q~_l      for every l in block b.
 * The clean state then advances over the block's clean tokens (which is
 * f_blk of Eq. f-blk).  Between blocks the noisy state is discarded.
 * chunk_states_out[n][j][c] (nullable) records the clean state at each chunk
 * start (positions cC); with chunk_states_in (nullable) the clean state is
 * instead reset to chunk_states_in[n][j][c] at each chunk start, so that the
 * computation starts from the same (rounded) chunk states a kernel is given.
 * Shapes: clean k [N,L,Hk,dk], v [N,L,Hv,dv], g, beta [N,L,Hv]; noisy q, k
 * [N,L,Hk,dk], v [N,L,Hv,dv], g, beta [N,L,Hv]; S_init [N,Hv,dk,dv]; out
 * [N,L,Hv,dv]; chunk states [N,Hv,L/C,dk,dv].  Requires B | C and C | L.
 */
int oracle_two_stream_fwd(int N, int L, int Hk, int Hv, int dk, int dv, int B, int C, double s,
                          int act_dt, const void* k, const void* v, int gate_dt, const void* g,
                          const void* beta, const void* qn, const void* kn, const void* vn,
                          const void* gn, const void* betan, int state_dt, const void* S_init,
                          const void* chunk_states_in, double* out, double* chunk_states_out,
                          int nthreads) {
  if (B < 1 || C < B || C % B != 0 || L % C != 0) return -1;
  const int n_chunks = L / C;
  const size_t nst = (size_t)dk * dv;
  set_threads(nthreads);
#pragma omp parallel for schedule(dynamic, 1)
  for (long item = 0; item < (long)N * Hv; ++item) {
    const int n = (int)(item / Hv), j = (int)(item % Hv);
    const int h = (int)(((long)j * Hk) / Hv);
    double* S = (double*)malloc(sizeof(double) * nst);
    double* Sn = (double*)malloc(sizeof(double) * nst);
    double* u = (double*)malloc(sizeof(double) * dv);
    double* kt = (double*)malloc(sizeof(double) * dk);
    for (size_t e = 0; e < nst; ++e) S[e] = ld(S_init, state_dt, (size_t)item * nst + e);
    /* one gated-delta-rule step (Eq. per-step-fwd) of state X on token t of a stream */
#define GDR_STEP(X, KK, VV, GG, BB, t)                                                    \
  do {                                                                                    \
    const size_t kq_ = (((size_t)n * L + (t)) * Hk + h) * dk;                             \
    const size_t vo_ = (((size_t)n * L + (t)) * Hv + j) * dv;                             \
    const size_t gb_ = ((size_t)n * L + (t)) * Hv + j;                                    \
    const double alpha_ = exp(ld(GG, gate_dt, gb_)), bt_ = ld(BB, gate_dt, gb_);          \
    for (int i = 0; i < dk; ++i) kt[i] = ld(KK, act_dt, kq_ + i);                         \
    for (size_t e = 0; e < nst; ++e) (X)[e] *= alpha_;                                    \
    for (int c = 0; c < dv; ++c) u[c] = 0.0;                                              \
    for (int i = 0; i < dk; ++i)                                                          \
      for (int c = 0; c < dv; ++c) u[c] += (X)[i * dv + c] * kt[i];                       \
    for (int c = 0; c < dv; ++c) u[c] = bt_ * (ld(VV, act_dt, vo_ + c) - u[c]);           \
    for (int i = 0; i < dk; ++i)                                                          \
      for (int c = 0; c < dv; ++c) (X)[i * dv + c] += kt[i] * u[c];                      \
  } while (0)
    for (int b = 0; b < L / B; ++b) {
      const int t0 = b * B;
      if (t0 % C == 0) {
        const size_t co = ((size_t)item * n_chunks + t0 / C) * nst;
        if (chunk_states_in)
          for (size_t e = 0; e < nst; ++e) S[e] = ld(chunk_states_in, state_dt, co + e);
        if (chunk_states_out) memcpy(chunk_states_out + co, S, sizeof(double) * nst);
      }
      /* noisy block: seeded with the clean state before the block */
      memcpy(Sn, S, sizeof(double) * nst);
      for (int t = t0; t < t0 + B; ++t) GDR_STEP(Sn, kn, vn, gn, betan, t);
      for (int l = t0; l < t0 + B; ++l) {
        const size_t ql = (((size_t)n * L + l) * Hk + h) * dk;
        const size_t ol = (((size_t)n * L + l) * Hv + j) * dv;
        for (int i = 0; i < dk; ++i) kt[i] = ld(qn, act_dt, ql + i);
        for (int c = 0; c < dv; ++c) {
          double acc = 0.0;
          for (int i = 0; i < dk; ++i) acc += Sn[i * dv + c] * kt[i];
          out[ol + c] = s * acc;
        }
      }
      /* clean stream advances over the block (f_blk) */
      for (int t = t0; t < t0 + B; ++t) GDR_STEP(S, k, v, g, beta, t);
    }
#undef GDR_STEP
    free(kt);
    free(u);
    free(Sn);
    free(S);
  }
  return 0;
}

/*
 * Two-stream causal ShortConv of a block (appendix "1D Causal ShortConv:
 * implementation routes", Eq. short-conv-clean / Eq. short-conv-noisy), in
 * its serving form.  A depthwise causal convolution of width W over C
 * channels; for request r and block row l (0-based inside the block) the lag-i
 * input is the block's own row l - i when it lies inside the block, and
 * otherwise the committed conv state, i.e. the last W - 1 clean tokens before
 * the block (the state "is a raw tensor slice" of the clean stream):
 *     z_{l,i} = x[r][l-i]                      if l - i >= 0
 *             = conv_state[slot][W-1 + l-i]    otherwise (oldest row first)
 *     y[r][l][c] = act(bias[c] + sum_{i<W} w[c][i] z_{l,i}[c])
 * act is the identity (act = 0) or SiLU u / (1 + exp(-u)) (act = 1); bias may
 * be NULL.  With accept_len non-NULL the state is then committed at length
 * n = accept_len[r]: state_out[r] = the last W - 1 rows of
 * (conv_state[slot] ++ x[r][0..n-1]); n = 0 keeps the old state.
 * Shapes: x [R,B,C]; conv_state [num_slots, W-1, C]; weight [C, W] (w[c][i]
 * multiplies lag i); bias [C]; out [R,B,C]; state_out [R, W-1, C].
 * Returns -1 for an invalid slot, width or accepted length.
 */
int oracle_short_conv(int R, int B, int C, int W, int act, int act_dt, const void* x,
                      const void* conv_state, int num_slots, const int32_t* state_slot,
                      int w_dt, const void* weight, const void* bias,
                      const int32_t* accept_len, double* out, double* state_out) {
  if (W < 1 || (act != 0 && act != 1)) return -1;
  for (int r = 0; r < R; ++r) {
    if (state_slot[r] < 0 || state_slot[r] >= num_slots) return -1;
    if (accept_len && (accept_len[r] < 0 || accept_len[r] > B)) return -1;
  }
  const int Wm = W - 1;
  for (int r = 0; r < R; ++r) {
    const size_t st = (size_t)state_slot[r] * Wm * C;
    for (int l = 0; l < B; ++l)
      for (int c = 0; c < C; ++c) {
        double acc = bias ? ld(bias, w_dt, c) : 0.0;
        for (int i = 0; i < W; ++i) {
          const int pos = l - i;
          const double z = pos >= 0 ? ld(x, act_dt, ((size_t)r * B + pos) * C + c)
                                     : ld(conv_state, act_dt, st + (size_t)(Wm + pos) * C + c);
          acc += ld(weight, w_dt, (size_t)c * W + i) * z;
        }
        out[((size_t)r * B + l) * C + c] = act ? acc / (1.0 + exp(-acc)) : acc;
      }
    if (accept_len && state_out) {
      const int n = accept_len[r];
      /* sequence (old state ++ accepted rows); keep its last W - 1 rows */
      for (int j = 0; j < Wm; ++j) {
        const int pos = n - Wm + j; /* position in the block, negative = old state */
        for (int c = 0; c < C; ++c)
          state_out[((size_t)r * Wm + j) * C + c] =
              pos >= 0 ? ld(x, act_dt, ((size_t)r * B + pos) * C + c)
                       : ld(conv_state, act_dt, st + (size_t)(Wm + pos) * C + c);
      }
    }
  }
  return 0;
}

/*
 * Dense copy of request r's paged prefix for one pool (K or V):
 * token j < prefix_len[r] lives in page page_table[r * max_pages + j / page_size],
 * row j % page_size, of the pool laid out [num_pages, Hkv, page_size, D].
 * out is [prefix_len[r], Hkv, D] in fp64.  Returns -1 on an invalid page id or
 * a prefix longer than max_pages * page_size.
 */
int oracle_gather_prefix(int r, int Hkv, int D, int page_size, int num_pages, int max_pages,
                         int act_dt, const void* pool, const int32_t* page_table,
                         const int32_t* prefix_len, double* out) {
  const int P = prefix_len[r];
  if (P < 0 || P > max_pages * page_size) return -1;
  for (int jt = 0; jt < P; ++jt) {
    const int page = page_table[(size_t)r * max_pages + jt / page_size];
    if (page < 0 || page >= num_pages) return -1;
    for (int hk = 0; hk < Hkv; ++hk)
      for (int d = 0; d < D; ++d)
        out[((size_t)jt * Hkv + hk) * D + d] =
            ld(pool, act_dt, (((size_t)page * Hkv + hk) * page_size + jt % page_size) * D + d);
  }
  return 0;
}

/*
 * Block-query softmax attention (Eq. softmax-retrieval) with the
 * Diffusion-Trust block mask.  For request r, query head h (kv head
 * h / (Hq / Hkv)) and block row t the visible set is every prefix token
 * j < prefix_len[r] (read through the page table) plus the block tokens i
 * with i < B (mask_mode 0, bidirectional denoise pass) or i <= t
 * (mask_mode 1, token-causal state-update pass).  Mask modes 2 and 3 are the
 * compact per-row encoding of the serving appendix's dLLM mask modes (AR-Trust
 * block: anchor and verify rows token-causal, draft rows bidirectional over
 * the block): row t is token-causal when row_type[t] == 0 and bidirectional
 * when it is 1, with row_type [B] shared by every request (mode 2) or
 * [R, B] per request (mode 3).  Every row sees the whole prefix in every mode
 * (the prefix-tile visibility invariant).  Two passes in fp64:
 *   z_i = scale (q . k_i),  m = max_i z_i,  w_i = exp(z_i - m),
 *   o = sum_i w_i v_i / sum_i w_i,  lse = m + log(sum_i w_i).
 * Shapes: q [R,B,Hq,D]; k_blk, v_blk [R,B,Hkv,D]; pools
 * [num_pages,Hkv,page_size,D]; page_table [R,max_pages]; prefix_len [R];
 * out [R,B,Hq,D]; lse [R,B,Hq] (may be NULL); row_type (modes 2 and 3 only)
 * uint8 [B] or [R,B], each entry 0 or 1.
 */
int oracle_block_softmax(int R, int B, int Hq, int Hkv, int D, int page_size, int num_pages,
                         int max_pages, double scale, int mask_mode, int act_dt,
                         const void* q, const void* k_blk, const void* v_blk,
                         const void* k_pool, const void* v_pool,
                         const int32_t* page_table, const int32_t* prefix_len,
                         const uint8_t* row_type, double* out, double* lse, int nthreads) {
  if (Hkv <= 0 || Hq % Hkv != 0) return -1;
  if (mask_mode < 0 || mask_mode > 3) return -1;
  if (mask_mode >= 2) {
    if (!row_type) return -1;
    const long n_types = mask_mode == 2 ? B : (long)R * B;
    for (long i = 0; i < n_types; ++i)
      if (row_type[i] > 1) return -1;
  }
  for (int r = 0; r < R; ++r) {
    const int P = prefix_len[r];
    if (P < 0 || P > max_pages * page_size) return -1;
    for (int pg = 0; pg < (P + page_size - 1) / page_size; ++pg) {
      const int page = page_table[(size_t)r * max_pages + pg];
      if (page < 0 || page >= num_pages) return -1;
    }
  }
  const int G = Hq / Hkv;
  set_threads(nthreads);
#pragma omp parallel for schedule(dynamic, 1)
  for (long item = 0; item < (long)R * Hq * B; ++item) {
    const int r = (int)(item / ((long)Hq * B));
    const int h = (int)((item / B) % Hq);
    const int t = (int)(item % B);
    const int kvh = h / G;
    const int P = prefix_len[r];
    int causal_row = mask_mode == 1;
    if (mask_mode == 2) causal_row = row_type[t] == 0;
    if (mask_mode == 3) causal_row = row_type[(size_t)r * B + t] == 0;
    const int nblk = causal_row ? t + 1 : B;
    const int n = P + nblk;
    double* z = (double*)malloc(sizeof(double) * (n > 0 ? n : 1));
    double* qv = (double*)malloc(sizeof(double) * D);
    const size_t qo = (((size_t)r * B + t) * Hq + h) * D;
    for (int d = 0; d < D; ++d) qv[d] = ld(q, act_dt, qo + d);
    /* visible keys: prefix first, then the block */
    for (int jt = 0; jt < n; ++jt) {
      double acc = 0.0;
      if (jt < P) {
        const int page = page_table[(size_t)r * max_pages + jt / page_size];
        const size_t ko = (((size_t)page * Hkv + kvh) * page_size + jt % page_size) * D;
        for (int d = 0; d < D; ++d) acc += qv[d] * ld(k_pool, act_dt, ko + d);
      } else {
        const size_t ko = (((size_t)r * B + (jt - P)) * Hkv + kvh) * D;
        for (int d = 0; d < D; ++d) acc += qv[d] * ld(k_blk, act_dt, ko + d);
      }
      z[jt] = scale * acc;
    }
    double m = -INFINITY;
    for (int jt = 0; jt < n; ++jt) m = z[jt] > m ? z[jt] : m;
    double Z = 0.0;
    for (int jt = 0; jt < n; ++jt) {
      z[jt] = exp(z[jt] - m);
      Z += z[jt];
    }
    for (int d = 0; d < D; ++d) {
      double acc = 0.0;
      for (int jt = 0; jt < n; ++jt) {
        double vv;
        if (jt < P) {
          const int page = page_table[(size_t)r * max_pages + jt / page_size];
          vv = ld(v_pool, act_dt, (((size_t)page * Hkv + kvh) * page_size + jt % page_size) * D + d);
        } else {
          vv = ld(v_blk, act_dt, (((size_t)r * B + (jt - P)) * Hkv + kvh) * D + d);
        }
        acc += z[jt] * vv;
      }
      out[qo + d] = acc / Z;
    }
    if (lse) lse[((size_t)r * B + t) * Hq + h] = m + log(Z);
    free(qv);
    free(z);
  }
  return 0;
}

/*
 * KV append of the state-update pass (serving appendix: after the last denoise
 * step the token-causal pass appends the block's keys and values to the cache):
 * for request r the first n = append_len[r] block tokens (all B when
 * append_len is NULL) go to prefix positions prefix_len[r] + t, i.e. page
 * page_table[r][(P + t) / page_size], row (P + t) % page_size, of both pools
 * ([num_pages, Hkv, page_size, D]).  Elements are copied bit for bit; nothing
 * else in the pools changes and prefix_len is not updated (that is the
 * caller's bookkeeping).  elem_bytes is the size of one element.
 * Returns -1 (and writes nothing) if any request's range or page is invalid.
 */
int oracle_append_kv(int R, int B, int Hkv, int D, int page_size, int num_pages, int max_pages,
                     int elem_bytes, const void* k_blk, const void* v_blk, void* k_pool,
                     void* v_pool, const int32_t* page_table, const int32_t* prefix_len,
                     const int32_t* append_len) {
  for (int r = 0; r < R; ++r) {
    const int P = prefix_len[r];
    const int n = append_len ? append_len[r] : B;
    if (n < 0 || n > B || P < 0 || P + n > max_pages * page_size) return -1;
    for (int t = 0; t < n; ++t) {
      const int page = page_table[(size_t)r * max_pages + (P + t) / page_size];
      if (page < 0 || page >= num_pages) return -1;
    }
  }
  const size_t row = (size_t)D * elem_bytes;
  for (int r = 0; r < R; ++r) {
    const int P = prefix_len[r];
    const int n = append_len ? append_len[r] : B;
    for (int t = 0; t < n; ++t) {
      const int pos = P + t;
      const int page = page_table[(size_t)r * max_pages + pos / page_size];
      for (int hk = 0; hk < Hkv; ++hk) {
        const size_t dst = (((size_t)page * Hkv + hk) * page_size + pos % page_size) * row;
        const size_t src = (((size_t)r * B + t) * Hkv + hk) * row;
        memcpy((char*)k_pool + dst, (const char*)k_blk + src, row);
        memcpy((char*)v_pool + dst, (const char*)v_blk + src, row);
      }
    }
  }
  return 0;
}
