// Internal definitions shared by the kvq CUDA translation units.
#pragma once

#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/kvq.h"

namespace kvq {

constexpr int kHeadDim = 128;
constexpr int kGroup = 32;
constexpr int kMaxGq = 8;        // largest n_q_heads / n_kv_heads supported
constexpr int kMaxSplits = 256;    // splits per (sequence, kv-head), window split included
constexpr int kMaxK = 64;        // largest DGAP recovery window
constexpr int kMaxHidden = 1024; // largest DGAP hidden width

// Byte sizes inside one 32-token page (see kvq.h).
__host__ __device__ inline int k_codes_bytes(int bits_k) { return 512 * bits_k; }
__host__ __device__ inline int v_codes_bytes(int bits_v) { return 512 * bits_v; }
__host__ __device__ inline int page_bytes(int bits_k, int bits_v) {
  return 512 * (bits_k + bits_v) + 1024;
}
constexpr int page_bytes_c(int bits_k, int bits_v) { return 512 * (bits_k + bits_v) + 1024; }
// Offsets of the four regions of a page.
__host__ __device__ inline int page_off_kmeta(int bits_k) { return 512 * bits_k; }
__host__ __device__ inline int page_off_vcodes(int bits_k) { return 512 * bits_k + 512; }
__host__ __device__ inline int page_off_vmeta(int bits_k, int bits_v) {
  return 512 * (bits_k + bits_v) + 512;
}

// Tokens held in quantized blocks when L tokens are cached.
__host__ __device__ inline int packed_len(int L, int residual) {
  int over = L - residual;
  return over > 0 ? (over / kGroup) * kGroup : 0;
}

// Kernel-facing copy of the configuration (plain ints, passed by value).
struct Dims {
  int batch, hq, hkv, gq, bits_k, bits_v, residual, ring, max_len, max_blocks;
  long long page_bytes;
};

inline Dims make_dims(const kvq_config& c) {
  Dims d;
  d.batch = c.batch;
  d.hq = c.n_q_heads;
  d.hkv = c.n_kv_heads;
  d.gq = c.n_q_heads / c.n_kv_heads;
  d.bits_k = c.bits_k;
  d.bits_v = c.bits_v;
  d.residual = c.residual;
  d.ring = c.residual + kGroup;
  d.max_len = c.max_len;
  d.max_blocks = c.max_len / kGroup;
  d.page_bytes = page_bytes(c.bits_k, c.bits_v);
  return d;
}

// Thread-local error message (api.cu).
void set_error(const char* fmt, ...);

// Launchers (each returns a cudaError_t from cudaGetLastError after launch).
cudaError_t launch_pack(const Dims& d, const kvq_cache& cache, const __half* k_new,
                        const __half* v_new, int n_new, int batch_begin,
                        int batch_count, cudaStream_t stream);
cudaError_t launch_decode_attn(const Dims& d, const kvq_cache& cache, const __half* q,
                               float* out, float scale_log2, int n_splits,
                               void* workspace, cudaStream_t stream);
size_t attn_workspace_bytes(const Dims& d, int n_splits);
int attn_default_splits(const Dims& d, int sm_count);
size_t attn_static_scratch_bytes();
cudaError_t launch_decode_attn_static(const Dims& d, const kvq_cache& cache, const __half* q,
                                      float* out, float scale_log2, int n_splits,
                                      cudaStream_t stream);

struct DgapDims {
  int batch, vocab, K, hidden, n_chunks;
  float logit_tau;  // gate when f > logit_tau
};
size_t dgap_workspace_bytes_impl(int batch, int vocab, int K);
int dgap_chunks(int vocab);
int dgap_max_chunks();
cudaError_t launch_dgap(const DgapDims& d, const dgap_params& p, float* logits,
                        int32_t* topk_idx, float* topk_val, float* risk,
                        uint8_t* gate, int32_t* next_token, float* features,
                        void* workspace, cudaStream_t stream);

}  // namespace kvq
