// Internal launch interface between the C ABI layer and the kernels.
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

namespace flare {

constexpr int kNumSMs = 152;  // GB300: 2 dies x 76 SMs (re-read at run time)

// Counts kernel launches for flare_launch_count().
void note_launches(int n);

struct GdrParams {
  int R, B, Hk, Hv, dk, dv, nslots;
  float scale;
  const void* q;  // [R,B,Hk,dk], nullable when no readout is asked
  const void* k;  // [R,B,Hk,dk]
  const void* v;  // [R,B,Hv,dv]
  const float* log_decay;  // [R,B,Hv]
  const float* beta;       // [R,B,Hv]
  float* state_pool;       // [nslots,Hv,dk,dv]; written only when write_state
  const int32_t* state_slot;  // [R]
  const int32_t* accept_len;  // [R] or nullptr (= B)
  void* out_blockend;         // [R,B,Hv,dv] or nullptr
  void* out_causal;           // [R,B,Hv,dv] or nullptr
  int write_state;
  // AR-Trust verify round
  const int32_t* verify_len;  // [R] or nullptr
  int max_verify;
  float* verify_states;       // [R,max_verify,Hv,dk,dv]
  int32_t* dev_status;
};

struct SoftmaxParams {
  int R, B, Hq, Hkv, G, D, page_size, num_pages, max_pages;
  float scale_log2;  // logit scale * log2(e)
  int causal;
  const uint8_t* row_type;  // per-row types (0 = token-causal) or nullptr
  int row_type_stride;      // 0 (one layout for the batch) or B (per request)
  const void* q;      // [R,B,Hq,D]
  const void* k_blk;  // [R,B,Hkv,D]
  const void* v_blk;
  const void* k_pool;  // [num_pages,Hkv,page_size,D]
  const void* v_pool;
  const int32_t* page_table;  // [R,max_pages]
  const int32_t* prefix_len;  // [R]
  void* out;                  // [R,B,Hq,D]
  float* lse;                 // [R,B,Hq] or nullptr
  float* ws_o;                // split partial outputs [R*Hkv][n_split][B*G][D]
  float* ws_lse;              // split partial lse     [R*Hkv][n_split][B*G]
  int n_split, split_len;
  int32_t* order;             // [R*n_split] valid work units (r, split), longest first
  int32_t* n_valid;           // number of valid work units in `order`
  uint32_t* bad_mask;         // [ceil(R/32)] requests with a bad prefix length or page id
  int32_t* counters;          // [R*Hkv*ceil(B*G/128)] finished splits per row tile (n_split > 1)
  int32_t* dev_status;
};

// Work decomposition of the softmax call; identical for the workspace query
// and the launch.
struct SoftmaxPlan {
  int kernel;  // 0 = CUDA-core kernel, 1 = tensor-core kernel
  int rows_per_cta;
  int n_split;
  int split_len;
  int num_ctas;  // tensor-core kernel: CTAs launched
  size_t ws_o_bytes, ws_lse_bytes, ws_order_bytes, ws_count_bytes;
  size_t workspace_bytes;
};

size_t gdr_recurrent_smem_bytes(int dk, int dv, int threads);
bool gdr_denoise_tc_supported(int B, int dk, int dv);
bool gdr_denoise_persist_supported(int B, int dk, int dv);
cudaError_t launch_gdr_denoise_persist(const GdrParams& p, cudaStream_t stream);
bool gdr_denoise_chunk64_supported(int B, int dk, int dv);
cudaError_t launch_gdr_denoise_chunk64(const GdrParams& p, cudaStream_t stream);
cudaError_t launch_gdr_commit(const GdrParams& p, bool bf16, cudaStream_t stream);
bool gdr_commit_tc_supported(int B, int dk, int dv);
cudaError_t launch_gdr_commit_tc(const GdrParams& p, cudaStream_t stream);
cudaError_t launch_gdr_verify(const GdrParams& p, bool bf16, cudaStream_t stream);

constexpr int kMaxVerifyLayers = 64;
struct VerifyCommitParams {
  int R, max_verify, nslots, n_layers;
  size_t state_elems;  // Hv * dk * dv
  const float* records[kMaxVerifyLayers];
  float* pools[kMaxVerifyLayers];
  const int32_t* state_slot;
  const int32_t* accept;
  const int32_t* verify_len;
  int32_t* dev_status;
};
cudaError_t launch_verify_commit(const VerifyCommitParams& p, cudaStream_t stream);

struct ConvParams {
  int R, B, C, W, nslots, silu;
  const void* x;              // [R,B,C]
  void* conv_state;           // [nslots,W-1,C]
  const int32_t* state_slot;  // [R]
  const float* weight;        // [C,W]
  const float* bias;          // [C] or nullptr
  const int32_t* accept_len;  // [R] or nullptr (no commit)
  void* out;                  // [R,B,C]
  int32_t* dev_status;
};
cudaError_t launch_short_conv(const ConvParams& p, bool bf16, cudaStream_t stream);

struct TwoStreamParams {
  int N, L, B, Hk, Hv, dk, dv;
  float scale;
  const float* chunk_states;  // [N,Hv,L/64,dk,dv]
  const void* k;              // clean [N,L,Hk,dk]
  const void* v;              // clean [N,L,Hv,dv]
  const float* g;             // clean log-gates [N,L,Hv]
  const float* beta;
  const void* qn;             // noisy [N,L,Hk,dk]
  const void* kn;
  const void* vn;             // noisy [N,L,Hv,dv]
  const float* gn;
  const float* betan;
  void* out;                  // [N,L,Hv,dv]
  int32_t* dev_status;
};
int two_stream_chunk_len();
cudaError_t launch_two_stream_fwd(const TwoStreamParams& p, bool bf16, cudaStream_t stream);
bool two_stream_chunk_supported(int B, int dk, int dv);
cudaError_t launch_two_stream_chunk(const TwoStreamParams& p, cudaStream_t stream);
cudaError_t launch_gdr_denoise_tc(const GdrParams& p, cudaStream_t stream);
cudaError_t launch_gdr_recurrent(const GdrParams& p, bool bf16, cudaStream_t stream);

SoftmaxPlan plan_softmax(int R, int B, int Hq, int Hkv, int D, int page_size, int max_pages,
                         bool bf16, int num_sms);
cudaError_t launch_softmax(const SoftmaxParams& p, const SoftmaxPlan& plan, bool bf16,
                           cudaStream_t stream);
cudaError_t launch_softmax_simt(const SoftmaxParams& p, const SoftmaxPlan& plan, bool bf16,
                                cudaStream_t stream);
cudaError_t launch_softmax_tc(const SoftmaxParams& p, const SoftmaxPlan& plan,
                              cudaStream_t stream);
cudaError_t launch_softmax_combine(const SoftmaxParams& p, bool bf16, cudaStream_t stream);
bool softmax_tc_supported(int B, int Hq, int Hkv, int D, int page_size);
cudaError_t launch_append_kv(const SoftmaxParams& p, const int32_t* append_len, void* k_pool,
                             void* v_pool, int elem_bytes, cudaStream_t stream);
cudaError_t launch_debug_wait_timeout(int32_t* status, uint64_t limit_ns, cudaStream_t stream);
cudaError_t launch_gather_prefix(const SoftmaxParams& p, int request, void* k_out, void* v_out,
                                 bool bf16, cudaStream_t stream);

}  // namespace flare
