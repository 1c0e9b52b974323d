/*
 * flare.h -- C ABI of the FLARE block-denoising attention step on GB300 (sm_103a).
 *
 * FLARE serves a hybrid backbone (gated-delta-rule linear attention layers
 * interleaved with softmax attention layers) by denoising a block of B tokens
 * per request.  Each block is processed by two kinds of forward pass (serving
 * appendix, "Differences between the denoise pass and the state-update pass"):
 *   - denoise passes read the committed recurrent state and the paged KV
 *     prefix but write neither;
 *   - one state-update pass writes the recurrent state at the accepted length.
 * This library exposes exactly the per-layer attention work of those passes:
 *
 *   flare_block_linear_attn   gated-delta-rule block pass, block-end readout
 *   flare_commit_state        write S^(r) into the state pool
 *   flare_block_softmax_attn  block queries over paged prefix + block
 *   flare_append_kv           append the finalized block to the paged cache
 *   flare_short_conv          two-stream causal ShortConv of the block, conv-state commit
 *
 * and the attention work of an AR-Trust verify round (decoding appendix):
 *
 *   flare_verify_linear_attn  token-causal anchor/verify rows, bidirectional
 *                             draft rows, verify states cached
 *   flare_verify_commit       restore the state at the accepted offset
 *   flare_block_softmax_attn  with the per-row ROW_TYPE mask modes
 *
 * and, for training, the fused two-stream forward of a GDN layer:
 *
 *   flare_two_stream_fwd      noisy blocks seeded from the on-chip clean state
 *
 * Conventions shared by every call
 * --------------------------------
 *  - All tensor arguments are DEVICE pointers to contiguous row-major arrays
 *    in the shapes stated per call.  Integer arrays are int32.  Activation,
 *    state, pool, filter and output arrays must start on a 16-byte boundary
 *    (they are moved in 16-byte pieces); a misaligned one is rejected with
 *    FLARE_ERR_INVALID_ARGUMENT.
 *  - Ownership: the caller allocates and frees every buffer (inputs, outputs,
 *    pools, workspace, status word).  The library allocates no device memory,
 *    frees nothing and never synchronizes inside a compute call.  Work is
 *    enqueued on `stream` (a cudaStream_t passed as void*, NULL = legacy
 *    default stream); a call returns once its kernels are enqueued.
 *  - Errors a host can see (null pointer, unsupported size, bad dtype, too
 *    small workspace) are returned immediately and nothing is launched.
 *  - Errors only the device can see (a page id, state slot, prefix length or
 *    accepted length out of range) set bits in *dev_status with an atomic OR
 *    (FLARE_DEV_* below); the offending (request, head) item is skipped and its
 *    outputs are left untouched.  Nothing traps.  The caller clears
 *    *dev_status (4 bytes, device memory) and reads it back, e.g. with
 *    flare_read_status.
 *  - Kernels are launched on the current CUDA device; all pointers must live
 *    on that device.
 */
#ifndef FLARE_H_
#define FLARE_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum flare_status {
  FLARE_OK = 0,
  FLARE_ERR_INVALID_ARGUMENT = 1, /* null pointer, inconsistent sizes */
  FLARE_ERR_UNSUPPORTED = 2,      /* sizes or dtypes the library does not implement */
  FLARE_ERR_CUDA = 3,             /* a CUDA runtime call failed (launch, attribute) */
  FLARE_ERR_DEVICE_STATUS = 4     /* flare_read_status found device error bits */
} flare_status;

typedef enum flare_dtype { FLARE_DT_BF16 = 0, FLARE_DT_F32 = 1 } flare_dtype;

/* Softmax block mask (decoding appendix, attention patterns): every block row
 * sees the whole prefix; in the denoise pass (BIDIR) it also sees every block
 * token, in the state-update pass (CAUSAL) the block tokens up to itself.
 * The two ROW_TYPE modes are the compact (B, row_type_1..B) encoding of the
 * serving appendix's native dLLM mask modes, used by the AR-Trust verify
 * round (anchor and verify rows token-causal, draft rows bidirectional over
 * the block): desc->row_type gives one type per block row, shared by the
 * batch (UNIFORM, [B]) or per request (PER_REQUEST, [R, B]).  Prefix tiles are
 * unmasked for every row type. */
typedef enum flare_mask_mode {
  FLARE_MASK_BLOCK_BIDIR = 0,
  FLARE_MASK_BLOCK_CAUSAL = 1,
  FLARE_MASK_ROW_TYPE_UNIFORM = 2,
  FLARE_MASK_ROW_TYPE_PER_REQUEST = 3
} flare_mask_mode;

/* Row types (uint8) of the ROW_TYPE mask modes.  A value other than these two
 * reads as FLARE_ROW_BIDIR. */
#define FLARE_ROW_CAUSAL 0 /* anchor / verify row: block tokens 0..t */
#define FLARE_ROW_BIDIR 1  /* draft / MASK row: every block token */

/* Device status bits (OR-ed into *dev_status). */
#define FLARE_DEV_BAD_SLOT 0x1       /* state_slot[r] outside [0, num_state_slots) */
#define FLARE_DEV_BAD_PAGE 0x2       /* page id outside [0, num_pages) */
#define FLARE_DEV_BAD_PREFIX_LEN 0x4 /* prefix_len[r] < 0 or > max_pages_per_req * page_size */
#define FLARE_DEV_BAD_ACCEPT_LEN 0x8 /* accept_len[r] outside [0, block_len] */
#define FLARE_DEV_WAIT_TIMEOUT 0x10  /* an in-kernel pipeline wait gave up (bounded spin) */
#define FLARE_DEV_BAD_VERIFY_LEN 0x20 /* verify_len[r] outside [0, min(max_verify, block_len-1)],
                                         or an accepted offset outside [0, verify_len[r]] */

/* Activation applied after the ShortConv. */
typedef enum flare_activation { FLARE_ACT_NONE = 0, FLARE_ACT_SILU = 1 } flare_activation;

/* Gated-delta-rule layer shape.
 *   num_requests R, block_len B (1..64), num_qk_heads Hk, num_v_heads Hv
 *   (Hv a multiple of Hk; value head j reads q/k head j / (Hv / Hk)),
 *   head_dim_k dk and head_dim_v dv (each 64 or 128), num_state_slots in the
 *   pool, act_dtype of q/k/v/out, scale s of the readout (the paper's
 *   s = 1/sqrt(dk); pass it explicitly). */
typedef struct flare_linear_desc {
  int32_t num_requests;
  int32_t block_len;
  int32_t num_qk_heads;
  int32_t num_v_heads;
  int32_t head_dim_k;
  int32_t head_dim_v;
  int32_t num_state_slots;
  flare_dtype act_dtype;
  float scale;
} flare_linear_desc;

/* Softmax layer shape.
 *   num_requests R, block_len B (1..64), num_q_heads Hq, num_kv_heads Hkv
 *   (Hq a multiple of Hkv; q head h reads kv head h / (Hq / Hkv)), head_dim D
 *   (64, 128 or 256), page_size p (16 or 64 tokens), num_pages in each pool,
 *   max_pages_per_req (columns of the page table), act_dtype of every
 *   activation and pool, scale of the logits (the paper's 1/sqrt(D)),
 *   mask_mode as above; row_type is a DEVICE pointer to uint8 row types
 *   ([B] or [R, B]) for the ROW_TYPE modes and is ignored (may be NULL) in
 *   the others. */
typedef struct flare_softmax_desc {
  int32_t num_requests;
  int32_t block_len;
  int32_t num_q_heads;
  int32_t num_kv_heads;
  int32_t head_dim;
  int32_t page_size;
  int32_t num_pages;
  int32_t max_pages_per_req;
  flare_dtype act_dtype;
  float scale;
  flare_mask_mode mask_mode;
  const uint8_t* row_type;
} flare_softmax_desc;

/* ShortConv shape (the depthwise causal convolution in front of a GDN layer's
 * q/k/v projections).
 *   num_requests R, block_len B (>= 1), channels C (a multiple of 8), width W
 *   (1..4), num_state_slots in the conv-state pool, act_dtype of x, the conv
 *   state and out, activation after the bias. */
typedef struct flare_conv_desc {
  int32_t num_requests;
  int32_t block_len;
  int32_t channels;
  int32_t width;
  int32_t num_state_slots;
  flare_dtype act_dtype;
  flare_activation activation;
} flare_conv_desc;

/* Two-stream training layer shape (the noisy stream of a GDN layer).
 *   num_seqs N, seq_len L (a multiple of chunk_len), chunk_len C (64, the
 *   chunk of the clean chunkwise pass), block_len B (1, 2, 4, 8 or 16; the
 *   diffusion block), num_qk_heads Hk, num_v_heads Hv (a multiple of Hk),
 *   head_dim_k = head_dim_v = 128, act_dtype of the activations and the
 *   output, scale s of the readout. */
typedef struct flare_two_stream_desc {
  int32_t num_seqs;
  int32_t seq_len;
  int32_t chunk_len;
  int32_t block_len;
  int32_t num_qk_heads;
  int32_t num_v_heads;
  int32_t head_dim_k;
  int32_t head_dim_v;
  flare_dtype act_dtype;
  float scale;
} flare_two_stream_desc;

/*
 * Denoise pass of a gated-delta-rule layer (Eq. flare-gdn-schedule, noisy
 * branch; Eq. noisy-block-fwd).  For each request r and value head j the block
 * recurrence starts from S0 = state_pool[state_slot[r]][j] and runs the B
 * block tokens through the gated delta rule (Eq. per-step-fwd); every block
 * position then reads the block-end state:
 *     out[r][l][j] = scale * S_B^T q[r][l][h],   h = j / (Hv / Hk),  all l.
 * The state pool is read and NEVER written.
 *   q, k        [R, B, Hk, dk]   act_dtype
 *   v           [R, B, Hv, dv]   act_dtype
 *   log_decay   [R, B, Hv]       fp32, g_t (the gate is exp(g_t))
 *   beta        [R, B, Hv]       fp32
 *   state_pool  [num_state_slots, Hv, dk, dv] fp32, S[i][c] at i*dv + c
 *   state_slot  [R]              int32
 *   out         [R, B, Hv, dv]   act_dtype
 *   dev_status  int32 (device)   FLARE_DEV_BAD_SLOT
 */
flare_status flare_block_linear_attn(const flare_linear_desc* desc, const void* q,
                                     const void* k, const void* v, const float* log_decay,
                                     const float* beta, const float* state_pool,
                                     const int32_t* state_slot, void* out, int32_t* dev_status,
                                     void* stream);

/*
 * State commit at the accepted length (serving appendix, "Recovering the
 * recurrent state at the accept boundary"; Eq. chunk-state / Eq. f-blk for a
 * full block).  With the state-update pass's own block inputs, for each
 * request r with n = accept_len[r] in [0, B]:
 *     state_pool[state_slot[r]][j] <- S_n,
 * the state after the first n block tokens of the gated delta rule started
 * from the committed state.  n = 0 leaves the slot untouched (bit-identical);
 * n = B applies the full clean-transition map.  Written in place.
 * If causal_out is non-NULL the token-causal outputs of the state-update pass
 * are written for every block position t (Eq. per-step-fwd, o_t line):
 *     causal_out[r][t][j] = scale * S_t^T q[r][t][h]   (q must then be non-NULL).
 * Precondition: the state_slot entries are distinct within one call.
 *   q (nullable), k, v, log_decay, beta, state_pool, state_slot: as above
 *   accept_len  [R]             int32
 *   causal_out  [R, B, Hv, dv]  act_dtype, nullable
 *   dev_status  FLARE_DEV_BAD_SLOT | FLARE_DEV_BAD_ACCEPT_LEN
 */
flare_status flare_commit_state(const flare_linear_desc* desc, const void* q, const void* k,
                                const void* v, const float* log_decay, const float* beta,
                                float* state_pool, const int32_t* state_slot,
                                const int32_t* accept_len, void* causal_out,
                                int32_t* dev_status, void* stream);

/*
 * AR-Trust verify round of a gated-delta-rule layer (decoding appendix,
 * "AR-Trust sampling", block layout; serving appendix, "Recovering the
 * recurrent state at the accept boundary", path (b) cache-and-scatter).
 * The block of L = desc->block_len tokens is [anchor, d_0 .. d_{K-1},
 * MASK ...] with K = verify_len[r] held drafts (0 on a cold start).  For each
 * request r and value head j the gated delta rule (Eq. per-step-fwd) runs
 * from S0 = state_pool[state_slot[r]][j] over all L tokens; with S_n the state
 * after block tokens 0..n-1:
 *     out[r][t][j]   = scale * S_{t+1}^T q[r][t][h]   t <= K (anchor, verify rows:
 *                                                     token-causal)
 *     out[r][t][j]   = scale * S_L^T q[r][t][h]       t >  K (draft rows: the
 *                                                     whole block)
 *     verify_states[r][t][j] = S_{t+1}                t <  K (S^(t): the anchor
 *                                                     and t accepted drafts)
 *     state_pool[state_slot[r]][j] <- S_{K+1}         (S^(K), written in place)
 * so the live pool holds the state after every verify token, and
 * flare_verify_commit restores S^(a) when only a < K drafts are accepted.
 * Entries t >= K of verify_states are not written.
 * Precondition: the state_slot entries are distinct within one call.
 *   q, k           [R, L, Hk, dk]           act_dtype
 *   v              [R, L, Hv, dv]           act_dtype
 *   log_decay,beta [R, L, Hv]               fp32
 *   state_pool     [num_state_slots, Hv, dk, dv] fp32, read and written
 *   state_slot     [R]                      int32
 *   verify_len     [R]                      int32 in [0, min(max_verify, L - 1)]
 *   out            [R, L, Hv, dv]           act_dtype
 *   verify_states  [R, max_verify, Hv, dk, dv] fp32 (may be NULL if max_verify = 0)
 *   dev_status     FLARE_DEV_BAD_SLOT | FLARE_DEV_BAD_VERIFY_LEN (the request is
 *                  skipped: nothing of it is written)
 */
flare_status flare_verify_linear_attn(const flare_linear_desc* desc, int32_t max_verify,
                                      const void* q, const void* k, const void* v,
                                      const float* log_decay, const float* beta,
                                      float* state_pool, const int32_t* state_slot,
                                      const int32_t* verify_len, void* out, float* verify_states,
                                      int32_t* dev_status, void* stream);

/*
 * Gather-scatter commit of an AR-Trust verify round across layers (serving
 * appendix, path (b)): once the verify decision is known, for every layer l
 * and request r with accepted offset a = accept[r] (drafts accepted, in
 * [0, verify_len[r]]):
 *     a <  verify_len[r]:  state_pools[l][state_slot[r]] <- verify_states[l][r][a]
 *     a == verify_len[r]:  nothing (the pool already holds S^(K))
 * A bit-for-bit copy, one launch for all layers.
 *   desc           only num_requests, num_v_heads, head_dim_k, head_dim_v and
 *                  num_state_slots are used
 *   num_layers     1 .. 64
 *   verify_states  HOST array of num_layers DEVICE pointers, each
 *                  [R, max_verify, Hv, dk, dv] fp32 as written by
 *                  flare_verify_linear_attn
 *   state_pools    HOST array of num_layers DEVICE pointers, each
 *                  [num_state_slots, Hv, dk, dv] fp32
 *   state_slot, accept, verify_len  [R] int32 (device)
 *   dev_status     FLARE_DEV_BAD_SLOT | FLARE_DEV_BAD_VERIFY_LEN (the request is
 *                  skipped)
 */
flare_status flare_verify_commit(const flare_linear_desc* desc, int32_t max_verify,
                                 int32_t num_layers, const float* const* verify_states,
                                 float* const* state_pools, const int32_t* state_slot,
                                 const int32_t* accept, const int32_t* verify_len,
                                 int32_t* dev_status, void* stream);

/*
 * Two-stream causal ShortConv of a block (appendix "1D Causal ShortConv:
 * implementation routes", Eq. short-conv-noisy, serving form) and, optionally,
 * the commit of its conv state.  For request r and block row l the lag-i input
 * (i < W) is the block's own row l - i when l - i >= 0, and otherwise row
 * W - 1 + (l - i) of the committed conv state, which holds the last W - 1
 * clean tokens before the block, oldest first:
 *     out[r][l][c] = act(bias[c] + sum_i weight[c][i] * z_{l,i}[c])
 * (act: identity or SiLU u / (1 + e^-u); fp32 arithmetic, one rounding to
 * act_dtype).  The denoise passes call it with the noisy block and no commit;
 * the state-update pass (and an AR-Trust round with the anchor plus the
 * accepted drafts) passes accept_len: after the outputs, each request's slot
 * becomes the last W - 1 rows of (old state ++ block rows 0..n-1),
 * n = accept_len[r] in [0, B], a bit copy; n = 0 leaves it unchanged.
 * Precondition: the state_slot entries are distinct within a committing call.
 *   x           [R, B, C]                 act_dtype
 *   conv_state  [num_state_slots, W-1, C] act_dtype (read; written only with accept_len)
 *   state_slot  [R]                       int32
 *   weight      [C, W]                    fp32, weight[c][i] multiplies lag i
 *   bias        [C]                       fp32, nullable
 *   accept_len  [R]                       int32, nullable (no commit)
 *   out         [R, B, C]                 act_dtype
 *   dev_status  FLARE_DEV_BAD_SLOT | FLARE_DEV_BAD_ACCEPT_LEN (the request is skipped)
 */
flare_status flare_short_conv(const flare_conv_desc* desc, const void* x, void* conv_state,
                              const int32_t* state_slot, const float* weight, const float* bias,
                              const int32_t* accept_len, void* out, int32_t* dev_status,
                              void* stream);

/*
 * Two-stream training forward of a gated-delta-rule layer, noisy stream: the
 * Route II fused forward (appendix "Two-stream recurrence and block-level
 * chain rule", Eq. noisy-block-fwd and Eq. f-blk; "Route II: fused
 * two-stream").  Sequence n is L clean tokens and L noisy tokens over the
 * same positions, cut into blocks of B.  The noisy recurrence of block b
 * starts from the clean state before the block, S_{bB}, runs the block's
 * noisy tokens through the gated delta rule (Eq. per-step-fwd), and every
 * noisy position of the block reads the noisy block-end state:
 *     out[n][l][j] = scale * S~_{bB+B}^T q~[n][l][h]     (l in block b)
 * The clean state S_{bB} comes from chunk_states (the clean state at the
 * start of each C-token chunk, as the clean chunkwise pass produces it)
 * advanced over the clean tokens of the chunk's earlier blocks (f_blk), on
 * chip; no block-boundary state is written.  The clean outputs are the clean
 * chunkwise pass's and are not formed here.  Value head j reads q/k head
 * j / (Hv / Hk).  Arithmetic: bf16 activations run the state's products and
 * updates as tf32 tensor-core products with fp32 accumulation (the state
 * itself stays fp32); fp32 activations run exact fp32.
 *   chunk_states  [N, Hv, L/C, dk, dv]   fp32
 *   k, v          [N, L, Hk, dk], [N, L, Hv, dv]   clean, act_dtype
 *   log_decay, beta [N, L, Hv]           clean, fp32
 *   q_noisy, k_noisy [N, L, Hk, dk], v_noisy [N, L, Hv, dv]   act_dtype
 *   log_decay_noisy, beta_noisy [N, L, Hv] fp32
 *   out_noisy     [N, L, Hv, dv]         act_dtype
 *   dev_status    int32 status word (bits OR-ed in, never cleared)
 * Every index is derived from the shape, so the only device-detected error is
 * FLARE_DEV_WAIT_TIMEOUT (a tensor-core pipeline wait that gave up; the
 * outputs of the affected chunk are then incomplete).
 */
flare_status flare_two_stream_fwd(const flare_two_stream_desc* desc, const float* chunk_states,
                                  const void* k, const void* v, const float* log_decay,
                                  const float* beta, const void* q_noisy, const void* k_noisy,
                                  const void* v_noisy, const float* log_decay_noisy,
                                  const float* beta_noisy, void* out_noisy, int32_t* dev_status,
                                  void* stream);

/*
 * Bytes of device workspace flare_block_softmax_attn needs for `desc`
 * (the longest-first order of the work units and the partial outputs of split
 * prefixes).  May be 0.  Host-only, no GPU work.
 */
flare_status flare_softmax_workspace_size(const flare_softmax_desc* desc, size_t* bytes);

/*
 * Block-query softmax attention over a paged KV prefix (Eq. softmax-retrieval
 * with the Diffusion-Trust block mask; native dLLM mask modes of the serving
 * appendix).  For request r, query head h (kv head h / (Hq / Hkv)) and block
 * row t the visible keys are the prefix tokens j < prefix_len[r], read from
 * page page_table[r][j / p], row j % p of the pools, followed by the block's
 * own keys (all B of them in BIDIR mode and for FLARE_ROW_BIDIR rows, 0..t in
 * CAUSAL mode and for FLARE_ROW_CAUSAL rows):
 *     out[r][t][h] = sum_i softmax_i(scale * q . k_i) v_i
 *     lse[r][t][h] = log sum_i exp(scale * q . k_i)          (natural log)
 * The block's keys/values are not in the pools (they are appended only by the
 * state-update pass).  Pool rows past a request's prefix end are never used,
 * whatever they hold.
 *   q              [R, B, Hq, D]                 act_dtype
 *   k_blk, v_blk   [R, B, Hkv, D]                act_dtype
 *   k_pool, v_pool [num_pages, Hkv, p, D]        act_dtype
 *   page_table     [R, max_pages_per_req]        int32
 *   prefix_len     [R]                           int32
 *   out            [R, B, Hq, D]                 act_dtype
 *   lse            [R, B, Hq]                    fp32, nullable
 *   workspace      >= flare_softmax_workspace_size bytes, 256-byte aligned
 *                  (may be NULL when that size is 0)
 *   dev_status     FLARE_DEV_BAD_PAGE | FLARE_DEV_BAD_PREFIX_LEN | FLARE_DEV_WAIT_TIMEOUT
 */
flare_status flare_block_softmax_attn(const flare_softmax_desc* desc, const void* q,
                                      const void* k_blk, const void* v_blk, const void* k_pool,
                                      const void* v_pool, const int32_t* page_table,
                                      const int32_t* prefix_len, void* out, float* lse,
                                      void* workspace, size_t workspace_bytes,
                                      int32_t* dev_status, void* stream);

/*
 * KV append of the state-update pass (serving appendix, Diffusion-Trust
 * serving loop: after the last denoise step the token-causal pass writes the
 * recurrent state back and appends the block's keys and values to the cache).
 * For request r the first n = append_len[r] block tokens (all B when
 * append_len is NULL) are copied bit for bit to prefix positions
 * prefix_len[r] + t, t < n, i.e. page page_table[r][(P + t) / p], row
 * (P + t) % p of both pools.  Page allocation is the caller's: the table
 * entries for those positions must already name pages.  prefix_len is not
 * updated (advance it by n afterwards).  Nothing else in the pools changes.
 *   k_blk, v_blk   [R, B, Hkv, D]             act_dtype (desc->act_dtype)
 *   k_pool, v_pool [num_pages, Hkv, p, D]     act_dtype, written in place
 *   page_table     [R, max_pages_per_req]     int32
 *   prefix_len     [R]                        int32
 *   append_len     [R]                        int32 in [0, B], nullable
 *   dev_status     FLARE_DEV_BAD_ACCEPT_LEN (n out of range),
 *                  FLARE_DEV_BAD_PREFIX_LEN (P + n beyond the table),
 *                  FLARE_DEV_BAD_PAGE; the request is skipped.
 * Only the shape fields, page_size, num_pages, max_pages_per_req and
 * act_dtype of desc are used.
 */
flare_status flare_append_kv(const flare_softmax_desc* desc, const void* k_blk, const void* v_blk,
                             void* k_pool, void* v_pool, const int32_t* page_table,
                             const int32_t* prefix_len, const int32_t* append_len,
                             int32_t* dev_status, void* stream);

/* Size of the library-owned scratch array used by flare_block_softmax_attn_noalloc. */
#define FLARE_NOALLOC_SCRATCH_BYTES (64u * 1024u * 1024u)

/*
 * flare_block_softmax_attn for callers that cannot allocate device memory.
 * The paper has no counterpart; this is a deployment convenience.
 * Some callers cannot supply a workspace: a serving engine whose memory
 * manager owns all device memory and forbids cudaMalloc/cudaFree while
 * requests are in flight (they synchronize the device and can fail under
 * memory pressure), or a plugin host that passes only the request's own
 * tensors.  Same arguments, layouts, outputs and status bits as
 * flare_block_softmax_attn, minus the workspace: the workspace (work order and split partials) lives in a
 * file-scope device array of FLARE_NOALLOC_SCRATCH_BYTES that the library
 * holds on every GPU that loads it, until the process exits.
 *  - This call allocates nothing (no cudaMalloc, cudaFree or allocating
 *    library routine).
 *  - The first call on each device looks up the array's device address
 *    (cudaGetSymbolAddress, current device) and caches it.  With CUDA's
 *    default lazy module loading that lookup is also when the array's memory
 *    is committed on the device, so make the first call (a warm-up call will
 *    do) at start-up: before the engine reserves its memory pool, and before
 *    any stream capture.  CUDA_MODULE_LOADING=EAGER commits it when the
 *    library is loaded instead.
 *  - The cached address belongs to the device's current context: after
 *    cudaDeviceReset (or anything else that destroys the primary context)
 *    this entry point must not be called again in the process.
 *  - If the shape needs more scratch than FLARE_NOALLOC_SCRATCH_BYTES
 *    (flare_softmax_workspace_size reports the need), the call returns
 *    FLARE_ERR_UNSUPPORTED and launches nothing.
 *  - Every call shares the one array: calls that overlap on the GPU (other
 *    streams, other host threads) race on it and must be serialized by the
 *    caller.  No part of it needs to start at zero.
 */
flare_status flare_block_softmax_attn_noalloc(const flare_softmax_desc* desc, const void* q,
                                              const void* k_blk, const void* v_blk,
                                              const void* k_pool, const void* v_pool,
                                              const int32_t* page_table,
                                              const int32_t* prefix_len, void* out, float* lse,
                                              int32_t* dev_status, void* stream);

/*
 * Test/debug helper: dense copy of request `request`'s paged prefix,
 * k_out/v_out [prefix_len[request], Hkv, D] act_dtype (the caller sizes them
 * from the prefix length it wrote).  Same page arithmetic as the attention
 * kernels; bit-exact copy.  dev_status: FLARE_DEV_BAD_PAGE | FLARE_DEV_BAD_PREFIX_LEN.
 */
flare_status flare_debug_gather_prefix(const flare_softmax_desc* desc, const void* k_pool,
                                       const void* v_pool, const int32_t* page_table,
                                       const int32_t* prefix_len, int32_t request, void* k_out,
                                       void* v_out, int32_t* dev_status, void* stream);

/*
 * Test helper for failure detection: one CTA waits on a pipeline barrier that
 * nothing ever completes, through the bounded wait every pipelined kernel
 * uses, gives up after limit_ns nanoseconds (1 us .. 1 s; else
 * FLARE_ERR_INVALID_ARGUMENT) and sets FLARE_DEV_WAIT_TIMEOUT in dev_status.
 * The context stays usable afterwards.
 */
flare_status flare_debug_wait_timeout(int32_t* dev_status, uint64_t limit_ns, void* stream);

/*
 * Waits for `stream`, copies the status word to *bits_out (nullable) and
 * returns FLARE_ERR_DEVICE_STATUS if any bit is set, FLARE_ERR_CUDA if the
 * stream reported an error, else FLARE_OK.  This is the one call that
 * synchronizes.
 */
flare_status flare_read_status(const int32_t* dev_status, void* stream, int32_t* bits_out);

/* Static string naming a status code. */
const char* flare_status_string(flare_status status);

/* Number of kernels this library has enqueued since it was loaded, over all
 * devices and threads (diagnostic; a relaxed atomic counter). */
uint64_t flare_launch_count(void);

#ifdef __cplusplus
}
#endif

#endif /* FLARE_H_ */
