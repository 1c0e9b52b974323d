// C ABI of the FLARE attention step: argument checks, work planning, launch.
// The declarations and the contract of every entry point are in flare.h.
#include <cuda_runtime.h>
#include <stdint.h>
#include <string.h>

#include <atomic>

#include "flare.h"
#include "kernels.h"

using namespace flare;

namespace {

bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

bool valid_dtype(flare_dtype d) { return d == FLARE_DT_BF16 || d == FLARE_DT_F32; }

flare_status check_linear(const flare_linear_desc* d) {
  if (!d) return FLARE_ERR_INVALID_ARGUMENT;
  if (d->num_requests < 0 || d->block_len < 1 || d->num_qk_heads < 1 || d->num_v_heads < 1 ||
      d->num_state_slots < 1 || !valid_dtype(d->act_dtype))
    return FLARE_ERR_INVALID_ARGUMENT;
  if (d->num_v_heads % d->num_qk_heads != 0) return FLARE_ERR_INVALID_ARGUMENT;
  if (d->block_len > 64) return FLARE_ERR_UNSUPPORTED;
  if ((d->head_dim_k != 64 && d->head_dim_k != 128) ||
      (d->head_dim_v != 64 && d->head_dim_v != 128))
    return FLARE_ERR_UNSUPPORTED;
  return FLARE_OK;
}

flare_status check_softmax(const flare_softmax_desc* d) {
  if (!d) return FLARE_ERR_INVALID_ARGUMENT;
  if (d->num_requests < 0 || d->block_len < 1 || d->num_q_heads < 1 || d->num_kv_heads < 1 ||
      d->page_size < 1 || d->num_pages < 0 || d->max_pages_per_req < 0 ||
      !valid_dtype(d->act_dtype))
    return FLARE_ERR_INVALID_ARGUMENT;
  if (d->mask_mode != FLARE_MASK_BLOCK_BIDIR && d->mask_mode != FLARE_MASK_BLOCK_CAUSAL &&
      d->mask_mode != FLARE_MASK_ROW_TYPE_UNIFORM &&
      d->mask_mode != FLARE_MASK_ROW_TYPE_PER_REQUEST)
    return FLARE_ERR_INVALID_ARGUMENT;
  if ((d->mask_mode == FLARE_MASK_ROW_TYPE_UNIFORM ||
       d->mask_mode == FLARE_MASK_ROW_TYPE_PER_REQUEST) && !d->row_type)
    return FLARE_ERR_INVALID_ARGUMENT;
  if (!(d->scale >= 0.f) || !(d->scale < 3.0e38f)) return FLARE_ERR_INVALID_ARGUMENT;
  if (d->num_q_heads % d->num_kv_heads != 0) return FLARE_ERR_INVALID_ARGUMENT;
  if (d->block_len > 64) return FLARE_ERR_UNSUPPORTED;
  if (d->head_dim != 64 && d->head_dim != 128 && d->head_dim != 256) return FLARE_ERR_UNSUPPORTED;
  if (d->page_size != 16 && d->page_size != 32 && d->page_size != 64 && d->page_size != 128)
    return FLARE_ERR_UNSUPPORTED;
  if ((int64_t)d->max_pages_per_req * d->page_size > (1 << 24)) return FLARE_ERR_UNSUPPORTED;
  return FLARE_OK;
}

int device_sms() {
  int dev = 0, n = kNumSMs;
  if (cudaGetDevice(&dev) == cudaSuccess)
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
  return n > 0 ? n : kNumSMs;
}

SoftmaxParams softmax_params(const flare_softmax_desc* d) {
  SoftmaxParams p;
  memset(&p, 0, sizeof p);
  p.R = d->num_requests;
  p.B = d->block_len;
  p.Hq = d->num_q_heads;
  p.Hkv = d->num_kv_heads;
  p.G = d->num_q_heads / d->num_kv_heads;
  p.D = d->head_dim;
  p.page_size = d->page_size;
  p.num_pages = d->num_pages;
  p.max_pages = d->max_pages_per_req;
  p.scale_log2 = d->scale * 1.4426950408889634f;
  p.causal = d->mask_mode == FLARE_MASK_BLOCK_CAUSAL;
  if (d->mask_mode == FLARE_MASK_ROW_TYPE_UNIFORM || d->mask_mode == FLARE_MASK_ROW_TYPE_PER_REQUEST) {
    p.row_type = d->row_type;
    p.row_type_stride = d->mask_mode == FLARE_MASK_ROW_TYPE_PER_REQUEST ? d->block_len : 0;
  }
  return p;
}

SoftmaxPlan plan_for(const flare_softmax_desc* d) {
  return plan_softmax(d->num_requests, d->block_len, d->num_q_heads, d->num_kv_heads,
                      d->head_dim, d->page_size, d->max_pages_per_req,
                      d->act_dtype == FLARE_DT_BF16, device_sms());
}

}  // namespace

namespace flare {

static std::atomic<uint64_t> g_launches{0};
void note_launches(int n) { g_launches.fetch_add((uint64_t)n, std::memory_order_relaxed); }

SoftmaxPlan plan_softmax(int R, int B, int Hq, int Hkv, int D, int page_size, int max_pages,
                         bool bf16, int num_sms) {
  SoftmaxPlan pl;
  memset(&pl, 0, sizeof pl);
  const int G = Hq / Hkv, M = B * G;
  const long prefix_max = (long)max_pages * page_size;
  if (bf16 && softmax_tc_supported(B, Hq, Hkv, D, page_size)) {
    // tensor-core kernel: 128 query rows per CTA, one CTA per SM, work units
    // started longest first.  Split the prefix only when the batch has fewer
    // work items than SMs (then aim at two CTAs per SM), and keep at least 16
    // tiles (1024 keys) per split so partials stay small.
    pl.kernel = 1;
    pl.rows_per_cta = 128;
    const long items = (long)R * Hkv * ((M + 127) / 128);
    const long tiles = (prefix_max + 63) / 64;
    long ns = 1;
    if (items > 0 && items < num_sms) ns = (2L * num_sms + items - 1) / items;
    const long cap = tiles / 16 > 1 ? tiles / 16 : 1;
    if (ns > cap) ns = cap;
    if (ns > 64) ns = 64;  // the merge keeps 128 x n_split weights in shared memory
    const long tps = ns > 0 ? (tiles + ns - 1) / ns : 1;
    pl.split_len = (int)((tps > 0 ? tps : 1) * 64);
    pl.n_split = tiles > 0 ? (int)((tiles + tps - 1) / tps) : 1;
    if (pl.n_split < 1) pl.n_split = 1;
  } else {
    pl.kernel = 0;
    pl.rows_per_cta = 16;
    const long total_max = prefix_max + B;
    const long base = (long)R * Hkv * ((M + pl.rows_per_cta - 1) / pl.rows_per_cta);
    const long target = 4L * num_sms;
    long ns = base > 0 ? (target + base - 1) / base : 1;
    const long max_split = (total_max + 255) / 256;
    if (ns > max_split) ns = max_split;
    if (ns < 1) ns = 1;
    long len = (total_max + ns - 1) / ns;
    len = (len + 63) / 64 * 64;
    ns = (total_max + len - 1) / len;
    pl.n_split = (int)ns;
    pl.split_len = (int)len;
  }
  if (pl.n_split > 1) {
    const size_t rows = (size_t)R * Hkv * pl.n_split * M;
    pl.ws_o_bytes = (rows * D * sizeof(float) + 255) / 256 * 256;
    pl.ws_lse_bytes = (rows * sizeof(float) + 255) / 256 * 256;
  }
  // tensor-core kernel: the work units in longest-first order, and per row
  // tile a count of finished splits (the last one merges the partials)
  if (pl.kernel == 1) {
    // order [R*n_split], n_valid [1], bad-request mask [ceil(R/32)]
    pl.ws_order_bytes =
        (((size_t)R * pl.n_split + 1 + (size_t)(R + 31) / 32) * sizeof(int32_t) + 255) / 256 * 256;
    // one CTA per work item when the prefix is split, else one per SM (at most
    // one per work item) walking the items
    const long n_items = (long)((M + 127) / 128) * Hkv * R * pl.n_split;
    pl.num_ctas = (int)(pl.n_split > 1 ? n_items : (n_items < num_sms ? n_items : num_sms));
    if (pl.n_split > 1)
      pl.ws_count_bytes =
          ((size_t)R * Hkv * ((M + 127) / 128) * sizeof(int32_t) + 255) / 256 * 256;
  }
  pl.workspace_bytes = pl.ws_o_bytes + pl.ws_lse_bytes + pl.ws_order_bytes + pl.ws_count_bytes;
  return pl;
}

cudaError_t launch_softmax(const SoftmaxParams& p, const SoftmaxPlan& plan, bool bf16,
                           cudaStream_t stream) {
  if (plan.kernel == 1) return launch_softmax_tc(p, plan, stream);
  return launch_softmax_simt(p, plan, bf16, stream);
}

}  // namespace flare

extern "C" {

const char* flare_status_string(flare_status s) {
  switch (s) {
    case FLARE_OK: return "FLARE_OK";
    case FLARE_ERR_INVALID_ARGUMENT: return "FLARE_ERR_INVALID_ARGUMENT";
    case FLARE_ERR_UNSUPPORTED: return "FLARE_ERR_UNSUPPORTED";
    case FLARE_ERR_CUDA: return "FLARE_ERR_CUDA";
    case FLARE_ERR_DEVICE_STATUS: return "FLARE_ERR_DEVICE_STATUS";
  }
  return "FLARE_ERR_UNKNOWN";
}

flare_status flare_block_linear_attn(const flare_linear_desc* d, const void* q, const void* k,
                                     const void* v, const float* log_decay, const float* beta,
                                     const float* state_pool, const int32_t* state_slot,
                                     void* out, int32_t* dev_status, void* stream) {
  flare_status st = check_linear(d);
  if (st != FLARE_OK) return st;
  if (!q || !k || !v || !log_decay || !beta || !state_pool || !state_slot || !out || !dev_status)
    return FLARE_ERR_INVALID_ARGUMENT;
  if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(state_pool) ||
      !aligned16(out))
    return FLARE_ERR_INVALID_ARGUMENT;
  if (d->num_requests == 0) return FLARE_OK;
  GdrParams p;
  memset(&p, 0, sizeof p);
  p.R = d->num_requests;
  p.B = d->block_len;
  p.Hk = d->num_qk_heads;
  p.Hv = d->num_v_heads;
  p.dk = d->head_dim_k;
  p.dv = d->head_dim_v;
  p.nslots = d->num_state_slots;
  p.scale = d->scale;
  p.q = q;
  p.k = k;
  p.v = v;
  p.log_decay = log_decay;
  p.beta = beta;
  p.state_pool = const_cast<float*>(state_pool);  // read only: write_state = 0
  p.state_slot = state_slot;
  p.out_blockend = out;
  p.write_state = 0;
  p.dev_status = dev_status;
  const bool bf16 = d->act_dtype == FLARE_DT_BF16;
  // bf16: the persistent tensor-core kernels for 128 x 128 states (B <= 32,
  // and 33..64 as one chunk), the one-CTA-per-item tensor-core kernel for the
  // other shapes; fp32 the CUDA-core recurrence
  cudaError_t e;
  if (bf16 && gdr_denoise_persist_supported(p.B, p.dk, p.dv))
    e = launch_gdr_denoise_persist(p, static_cast<cudaStream_t>(stream));
  else if (bf16 && gdr_denoise_chunk64_supported(p.B, p.dk, p.dv))
    e = launch_gdr_denoise_chunk64(p, static_cast<cudaStream_t>(stream));
  else if (bf16 && gdr_denoise_tc_supported(p.B, p.dk, p.dv))
    e = launch_gdr_denoise_tc(p, static_cast<cudaStream_t>(stream));
  else
    e = launch_gdr_recurrent(p, bf16, static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? FLARE_OK : FLARE_ERR_CUDA;
}

flare_status flare_commit_state(const flare_linear_desc* d, const void* q, const void* k,
                                const void* v, const float* log_decay, const float* beta,
                                float* state_pool, const int32_t* state_slot,
                                const int32_t* accept_len, void* causal_out,
                                int32_t* dev_status, void* stream) {
  flare_status st = check_linear(d);
  if (st != FLARE_OK) return st;
  if (!k || !v || !log_decay || !beta || !state_pool || !state_slot || !accept_len ||
      !dev_status || (causal_out && !q))
    return FLARE_ERR_INVALID_ARGUMENT;
  if ((q && !aligned16(q)) || !aligned16(k) || !aligned16(v) || !aligned16(state_pool) ||
      (causal_out && !aligned16(causal_out)))
    return FLARE_ERR_INVALID_ARGUMENT;
  if (d->num_requests == 0) return FLARE_OK;
  GdrParams p;
  memset(&p, 0, sizeof p);
  p.R = d->num_requests;
  p.B = d->block_len;
  p.Hk = d->num_qk_heads;
  p.Hv = d->num_v_heads;
  p.dk = d->head_dim_k;
  p.dv = d->head_dim_v;
  p.nslots = d->num_state_slots;
  p.scale = d->scale;
  p.q = causal_out ? q : nullptr;
  p.k = k;
  p.v = v;
  p.log_decay = log_decay;
  p.beta = beta;
  p.state_pool = state_pool;
  p.state_slot = state_slot;
  p.accept_len = accept_len;
  p.out_causal = causal_out;
  p.write_state = 1;
  p.dev_status = dev_status;
  const bool bf16 = d->act_dtype == FLARE_DT_BF16;
  // bf16 blocks of the 128 x 128 state without token-causal outputs take the
  // tensor-core chunkwise commit, the rest the register recurrence
  const cudaError_t e =
      (bf16 && !causal_out && gdr_commit_tc_supported(p.B, p.dk, p.dv))
          ? launch_gdr_commit_tc(p, static_cast<cudaStream_t>(stream))
          : launch_gdr_commit(p, bf16, static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? FLARE_OK : FLARE_ERR_CUDA;
}

flare_status flare_verify_linear_attn(const flare_linear_desc* d, int32_t max_verify,
                                      const void* q, const void* k, const void* v,
                                      const float* log_decay, const float* beta,
                                      float* state_pool, const int32_t* state_slot,
                                      const int32_t* verify_len, void* out, float* verify_states,
                                      int32_t* dev_status, void* stream) {
  flare_status st = check_linear(d);
  if (st != FLARE_OK) return st;
  if (max_verify < 0) return FLARE_ERR_INVALID_ARGUMENT;
  if (!q || !k || !v || !log_decay || !beta || !state_pool || !state_slot || !verify_len ||
      !out || !dev_status || (max_verify > 0 && !verify_states))
    return FLARE_ERR_INVALID_ARGUMENT;
  if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(state_pool) ||
      !aligned16(out) || !aligned16(verify_states))
    return FLARE_ERR_INVALID_ARGUMENT;
  if (d->num_requests == 0) return FLARE_OK;
  GdrParams p;
  memset(&p, 0, sizeof p);
  p.R = d->num_requests;
  p.B = d->block_len;
  p.Hk = d->num_qk_heads;
  p.Hv = d->num_v_heads;
  p.dk = d->head_dim_k;
  p.dv = d->head_dim_v;
  p.nslots = d->num_state_slots;
  p.scale = d->scale;
  p.q = q;
  p.k = k;
  p.v = v;
  p.log_decay = log_decay;
  p.beta = beta;
  p.state_pool = state_pool;
  p.state_slot = state_slot;
  p.out_causal = out;
  p.write_state = 1;
  p.verify_len = verify_len;
  p.max_verify = max_verify;
  p.verify_states = verify_states;
  p.dev_status = dev_status;
  const cudaError_t e = launch_gdr_verify(p, d->act_dtype == FLARE_DT_BF16,
                                          static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? FLARE_OK : FLARE_ERR_CUDA;
}

flare_status flare_verify_commit(const flare_linear_desc* d, int32_t max_verify,
                                 int32_t num_layers, const float* const* verify_states,
                                 float* const* state_pools, const int32_t* state_slot,
                                 const int32_t* accept, const int32_t* verify_len,
                                 int32_t* dev_status, void* stream) {
  flare_status st = check_linear(d);
  if (st != FLARE_OK) return st;
  if (max_verify < 0 || num_layers < 1) return FLARE_ERR_INVALID_ARGUMENT;
  if (num_layers > kMaxVerifyLayers) return FLARE_ERR_UNSUPPORTED;
  if (!verify_states || !state_pools || !state_slot || !accept || !verify_len || !dev_status)
    return FLARE_ERR_INVALID_ARGUMENT;
  VerifyCommitParams p;
  memset(&p, 0, sizeof p);
  for (int l = 0; l < num_layers; ++l) {
    if (!state_pools[l] || (max_verify > 0 && !verify_states[l]))
      return FLARE_ERR_INVALID_ARGUMENT;
    if (!aligned16(state_pools[l]) || !aligned16(verify_states[l]))
      return FLARE_ERR_INVALID_ARGUMENT;
    p.records[l] = verify_states[l];
    p.pools[l] = state_pools[l];
  }
  if (d->num_requests == 0 || max_verify == 0) return FLARE_OK;
  p.R = d->num_requests;
  p.max_verify = max_verify;
  p.nslots = d->num_state_slots;
  p.n_layers = num_layers;
  p.state_elems = (size_t)d->num_v_heads * d->head_dim_k * d->head_dim_v;
  p.state_slot = state_slot;
  p.accept = accept;
  p.verify_len = verify_len;
  p.dev_status = dev_status;
  const cudaError_t e = launch_verify_commit(p, static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? FLARE_OK : FLARE_ERR_CUDA;
}

flare_status flare_short_conv(const flare_conv_desc* d, const void* x, void* conv_state,
                              const int32_t* state_slot, const float* weight, const float* bias,
                              const int32_t* accept_len, void* out, int32_t* dev_status,
                              void* stream) {
  if (!d) return FLARE_ERR_INVALID_ARGUMENT;
  if (d->num_requests < 0 || d->block_len < 1 || d->channels < 1 || d->num_state_slots < 1 ||
      d->width < 1 || !valid_dtype(d->act_dtype) ||
      (d->activation != FLARE_ACT_NONE && d->activation != FLARE_ACT_SILU))
    return FLARE_ERR_INVALID_ARGUMENT;
  if (d->width > 4 || d->channels % 8 != 0) return FLARE_ERR_UNSUPPORTED;
  if (!x || !state_slot || !weight || !out || !dev_status || (d->width > 1 && !conv_state))
    return FLARE_ERR_INVALID_ARGUMENT;
  if (!aligned16(x) || !aligned16(conv_state) || !aligned16(weight) || !aligned16(bias) ||
      !aligned16(out))
    return FLARE_ERR_INVALID_ARGUMENT;
  if (d->num_requests == 0) return FLARE_OK;
  ConvParams p;
  memset(&p, 0, sizeof p);
  p.R = d->num_requests;
  p.B = d->block_len;
  p.C = d->channels;
  p.W = d->width;
  p.nslots = d->num_state_slots;
  p.silu = d->activation == FLARE_ACT_SILU;
  p.x = x;
  p.conv_state = conv_state;
  p.state_slot = state_slot;
  p.weight = weight;
  p.bias = bias;
  p.accept_len = accept_len;
  p.out = out;
  p.dev_status = dev_status;
  const cudaError_t e = launch_short_conv(p, d->act_dtype == FLARE_DT_BF16,
                                          static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? FLARE_OK : FLARE_ERR_CUDA;
}

flare_status flare_two_stream_fwd(const flare_two_stream_desc* d, const float* chunk_states,
                                  const void* k, const void* v, const float* log_decay,
                                  const float* beta, const void* q_noisy, const void* k_noisy,
                                  const void* v_noisy, const float* log_decay_noisy,
                                  const float* beta_noisy, void* out_noisy, int32_t* dev_status,
                                  void* stream) {
  if (!d) return FLARE_ERR_INVALID_ARGUMENT;
  if (d->num_seqs < 0 || d->seq_len < 0 || d->chunk_len < 1 || d->block_len < 1 ||
      d->num_qk_heads < 1 || d->num_v_heads < 1 || d->num_v_heads % d->num_qk_heads != 0 ||
      !valid_dtype(d->act_dtype))
    return FLARE_ERR_INVALID_ARGUMENT;
  if (d->chunk_len != two_stream_chunk_len() || d->seq_len % d->chunk_len != 0)
    return FLARE_ERR_UNSUPPORTED;
  const int B = d->block_len;
  if (B != 1 && B != 2 && B != 4 && B != 8 && B != 16) return FLARE_ERR_UNSUPPORTED;
  if (d->head_dim_k != 128 || d->head_dim_v != 128) return FLARE_ERR_UNSUPPORTED;
  if (!chunk_states || !k || !v || !log_decay || !beta || !q_noisy || !k_noisy || !v_noisy ||
      !log_decay_noisy || !beta_noisy || !out_noisy || !dev_status)
    return FLARE_ERR_INVALID_ARGUMENT;
  if (!aligned16(chunk_states) || !aligned16(k) || !aligned16(v) || !aligned16(q_noisy) ||
      !aligned16(k_noisy) || !aligned16(v_noisy) || !aligned16(out_noisy))
    return FLARE_ERR_INVALID_ARGUMENT;
  if (d->num_seqs == 0 || d->seq_len == 0) return FLARE_OK;
  TwoStreamParams p;
  memset(&p, 0, sizeof p);
  p.N = d->num_seqs;
  p.L = d->seq_len;
  p.B = B;
  p.Hk = d->num_qk_heads;
  p.Hv = d->num_v_heads;
  p.dk = d->head_dim_k;
  p.dv = d->head_dim_v;
  p.scale = d->scale;
  p.chunk_states = chunk_states;
  p.k = k;
  p.v = v;
  p.g = log_decay;
  p.beta = beta;
  p.qn = q_noisy;
  p.kn = k_noisy;
  p.vn = v_noisy;
  p.gn = log_decay_noisy;
  p.betan = beta_noisy;
  p.out = out_noisy;
  p.dev_status = dev_status;
  const cudaError_t e = launch_two_stream_fwd(p, d->act_dtype == FLARE_DT_BF16,
                                              static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? FLARE_OK : FLARE_ERR_CUDA;
}

flare_status flare_softmax_workspace_size(const flare_softmax_desc* d, size_t* bytes) {
  flare_status st = check_softmax(d);
  if (st != FLARE_OK) return st;
  if (!bytes) return FLARE_ERR_INVALID_ARGUMENT;
  *bytes = d->num_requests == 0 ? 0 : plan_for(d).workspace_bytes;
  return FLARE_OK;
}

flare_status flare_block_softmax_attn(const flare_softmax_desc* d, const void* q,
                                      const void* k_blk, const void* v_blk, const void* k_pool,
                                      const void* v_pool, const int32_t* page_table,
                                      const int32_t* prefix_len, void* out, float* lse,
                                      void* workspace, size_t workspace_bytes,
                                      int32_t* dev_status, void* stream) {
  flare_status st = check_softmax(d);
  if (st != FLARE_OK) return st;
  if (!q || !k_blk || !v_blk || !prefix_len || !out || !dev_status)
    return FLARE_ERR_INVALID_ARGUMENT;
  if (d->max_pages_per_req > 0 && (!k_pool || !v_pool || !page_table))
    return FLARE_ERR_INVALID_ARGUMENT;
  if (!aligned16(q) || !aligned16(k_blk) || !aligned16(v_blk) || !aligned16(k_pool) ||
      !aligned16(v_pool) || !aligned16(out))
    return FLARE_ERR_INVALID_ARGUMENT;
  if (d->num_requests == 0) return FLARE_OK;
  const SoftmaxPlan plan = plan_for(d);
  if (workspace_bytes < plan.workspace_bytes) return FLARE_ERR_INVALID_ARGUMENT;
  if (plan.workspace_bytes && (!workspace || ((uintptr_t)workspace & 255u)))
    return FLARE_ERR_INVALID_ARGUMENT;
  SoftmaxParams p = softmax_params(d);
  p.q = q;
  p.k_blk = k_blk;
  p.v_blk = v_blk;
  p.k_pool = k_pool;
  p.v_pool = v_pool;
  p.page_table = page_table;
  p.prefix_len = prefix_len;
  p.out = out;
  p.lse = lse;
  p.n_split = plan.n_split;
  p.split_len = plan.split_len;
  if (plan.workspace_bytes) {
    char* ws = static_cast<char*>(workspace);
    if (plan.ws_o_bytes) {
      p.ws_o = reinterpret_cast<float*>(ws);
      p.ws_lse = reinterpret_cast<float*>(ws + plan.ws_o_bytes);
    }
    if (plan.ws_order_bytes) {
      p.order = reinterpret_cast<int32_t*>(ws + plan.ws_o_bytes + plan.ws_lse_bytes);
      p.n_valid = p.order + (size_t)p.R * plan.n_split;
      p.bad_mask = reinterpret_cast<uint32_t*>(p.n_valid + 1);
    }
    if (plan.ws_count_bytes)
      p.counters = reinterpret_cast<int32_t*>(ws + plan.ws_o_bytes + plan.ws_lse_bytes +
                                              plan.ws_order_bytes);
  }
  p.dev_status = dev_status;
  const cudaError_t e = launch_softmax(p, plan, d->act_dtype == FLARE_DT_BF16,
                                       static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? FLARE_OK : FLARE_ERR_CUDA;
}

flare_status flare_append_kv(const flare_softmax_desc* d, const void* k_blk, const void* v_blk,
                             void* k_pool, void* v_pool, const int32_t* page_table,
                             const int32_t* prefix_len, const int32_t* append_len,
                             int32_t* dev_status, void* stream) {
  flare_status st = check_softmax(d);
  if (st != FLARE_OK) return st;
  if (!k_blk || !v_blk || !k_pool || !v_pool || !page_table || !prefix_len || !dev_status)
    return FLARE_ERR_INVALID_ARGUMENT;
  if (!aligned16(k_blk) || !aligned16(v_blk) || !aligned16(k_pool) || !aligned16(v_pool))
    return FLARE_ERR_INVALID_ARGUMENT;
  if (d->num_requests == 0) return FLARE_OK;
  SoftmaxParams p = softmax_params(d);
  p.k_blk = k_blk;
  p.v_blk = v_blk;
  p.page_table = page_table;
  p.prefix_len = prefix_len;
  p.dev_status = dev_status;
  const int elem = d->act_dtype == FLARE_DT_BF16 ? 2 : 4;
  const cudaError_t e = launch_append_kv(p, append_len, k_pool, v_pool, elem,
                                         static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? FLARE_OK : FLARE_ERR_CUDA;
}

flare_status flare_debug_gather_prefix(const flare_softmax_desc* d, const void* k_pool,
                                       const void* v_pool, const int32_t* page_table,
                                       const int32_t* prefix_len, int32_t request, void* k_out,
                                       void* v_out, int32_t* dev_status, void* stream) {
  flare_status st = check_softmax(d);
  if (st != FLARE_OK) return st;
  if (!k_pool || !v_pool || !page_table || !prefix_len || !k_out || !v_out || !dev_status)
    return FLARE_ERR_INVALID_ARGUMENT;
  if (request < 0 || request >= d->num_requests) return FLARE_ERR_INVALID_ARGUMENT;
  SoftmaxParams p = softmax_params(d);
  p.k_pool = k_pool;
  p.v_pool = v_pool;
  p.page_table = page_table;
  p.prefix_len = prefix_len;
  p.dev_status = dev_status;
  const cudaError_t e = launch_gather_prefix(p, request, k_out, v_out,
                                             d->act_dtype == FLARE_DT_BF16,
                                             static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? FLARE_OK : FLARE_ERR_CUDA;
}

flare_status flare_debug_wait_timeout(int32_t* dev_status, uint64_t limit_ns, void* stream) {
  if (!dev_status || limit_ns < 1000ull || limit_ns > 1000000000ull)
    return FLARE_ERR_INVALID_ARGUMENT;
  const cudaError_t e =
      launch_debug_wait_timeout(dev_status, limit_ns, static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? FLARE_OK : FLARE_ERR_CUDA;
}

uint64_t flare_launch_count(void) { return g_launches.load(std::memory_order_relaxed); }

flare_status flare_read_status(const int32_t* dev_status, void* stream, int32_t* bits_out) {
  if (!dev_status) return FLARE_ERR_INVALID_ARGUMENT;
  int32_t bits = 0;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (cudaMemcpyAsync(&bits, dev_status, sizeof bits, cudaMemcpyDeviceToHost, s) != cudaSuccess)
    return FLARE_ERR_CUDA;
  if (cudaStreamSynchronize(s) != cudaSuccess) return FLARE_ERR_CUDA;
  if (bits_out) *bits_out = bits;
  return bits ? FLARE_ERR_DEVICE_STATUS : FLARE_OK;
}

}  // extern "C"
