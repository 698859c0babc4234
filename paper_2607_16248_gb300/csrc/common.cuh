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
constexpr int kMaxSplits = 256;    // bound on n_splits (split plan) and on a flat launch's CTAs
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

// Positions inside a page (layouts documented in kvq.h).
//
// 1-bit codes are stored in mma fragment order: lane L = 4 * gid + tig of the
// consuming warp reads its 128 codes as one 16-byte chunk (4 words) at byte
// 16 * L, and rotating word w left by 4 * r puts the code of fragment row j
// (j = 0..3) and half e at bit 10 + 16 e + j.  Keys: token t = 4 gid + j,
// channel c = 16 ks + 4 tig + 2 h + e, word ks / 2, r = 2 (ks & 1) + h.
// Values: channel c = 32 w + 4 gid + j, token t = 8 tig + r + 4 e.
// The functions return the bit index inside the 512-byte code area.
__host__ __device__ inline int key1_bit(int t, int c) {
  const int gid = t >> 2, j = t & 3, ks = c >> 4, tig = (c >> 2) & 3;
  const int h = (c >> 1) & 1, e = c & 1, r = 2 * (ks & 1) + h;
  return (16 * gid + 4 * tig + (ks >> 1)) * 32 + ((10 + 16 * e + j - 4 * r) & 31);
}
__host__ __device__ inline int val1_bit(int t, int c) {
  const int w = c >> 5, gid = (c >> 2) & 7, j = c & 3, tig = t >> 3, r = t & 3, e = (t >> 2) & 1;
  return (16 * gid + 4 * tig + w) * 32 + ((10 + 16 * e + j - 4 * r) & 31);
}
// Value scale / zero of (group g, token t): tokens of each 8-token run are
// stored in the order 0 4 1 5 2 6 3 7, so a 32-bit word holds tokens (t, t + 4).
__host__ __device__ inline int vmeta_index(int g, int t) {
  return 32 * g + 8 * (t >> 3) + 2 * (t & 3) + ((t >> 2) & 1);
}

// The KbVb quantizer of one 32-element group (Sec. 3.1), each step one IEEE
// float32 operation with the stated rounding:
//   zero  = min x                                   (exact, fp16)
//   scale = RU16(RU32(RU32(max x - min x) / levels)) (stored fp16)
//   code  = clamp(rint(RN32(RN32(x - zero) / scale)), 0, levels); 0 if scale == 0
// Codes fill B little-endian words, element i at bits [(i*B) % 32, +B) of
// word (i*B) / 32.  Used by kvq_pack and by the decode step's flush.
template <int B>
__device__ __forceinline__ void quantize_group(const float (&x)[kGroup], uint32_t (&w)[B],
                                               __half& scale, __half& zero) {
  constexpr float kLevels = float((1 << B) - 1);
  float lo = x[0], hi = x[0];
#pragma unroll
  for (int i = 1; i < kGroup; ++i) {
    lo = fminf(lo, x[i]);
    hi = fmaxf(hi, x[i]);
  }
  const __half s_h = __float2half_ru(__fdiv_ru(__fsub_ru(hi, lo), kLevels));
  const float s = __half2float(s_h);
  // The quotient d / s (d = RN32(x - zero) <= levels * s, so d / s <= 255)
  // comes from one product with RN32(1 / s): the product and RN32(d / s) both
  // lie within 3 * 2^-24 * (d / s) <= 4.6e-5 of d / s, so they round to the
  // same integer unless the product is within 1/8192 of a half-integer, where
  // the exact quotient is taken.  The codes are those of the definition.
  const float r = s > 0.0f ? __frcp_rn(s) : 0.0f;
#pragma unroll
  for (int j = 0; j < B; ++j) w[j] = 0u;
#pragma unroll
  for (int i = 0; i < kGroup; ++i) {
    uint32_t c = 0u;
    if (s > 0.0f) {
      const float dd = __fsub_rn(x[i], lo);
      const float q = __fmul_rn(dd, r);
      float t = rintf(q);
      if (fabsf(fabsf(q - t) - 0.5f) < 1.0f / 8192.0f) t = rintf(__fdiv_rn(dd, s));
      t = fminf(fmaxf(t, 0.0f), kLevels);
      c = (uint32_t)t;
    }
    w[(i * B) / 32] |= c << ((i * B) % 32);
  }
  scale = s_h;
  zero = __float2half_rn(lo);  // lo is an fp16 value: exact
}

// One quarter qi of a 32-token block, quantized by one warp into a page (or
// a page image): key groups of channels 32 qi .. 32 qi + 31 (lane = channel)
// and value group qi of the 32 tokens (lane = token).  row_k(t), row_v(t)
// give the fp16 rows [128] of token t of the block.  The quarters write
// disjoint words, scales and zeros (1-bit codes: words 4 l + qi, l = 0..31,
// assembled from warp ballots in the order key1_bit / val1_bit give), so the
// four may run in different warps.  Used by kvq_pack and by the decode
// step's flush, which are therefore bit-identical.
template <int BK, int BV, typename RowK, typename RowV>
__device__ __forceinline__ void quantize_quarter(RowK row_k, RowV row_v, int qi, char* image) {
  const int lane = threadIdx.x & 31;
  uint32_t* kcodes = reinterpret_cast<uint32_t*>(image);
  uint32_t* vcodes = reinterpret_cast<uint32_t*>(image + page_off_vcodes(BK));
  __half* kmeta = reinterpret_cast<__half*>(image + page_off_kmeta(BK));
  __half* vmeta = reinterpret_cast<__half*>(image + page_off_vmeta(BK, BV));
  const int c = kGroup * qi + lane;  // this lane's key channel
  float xk[kGroup], xv[kGroup];
#pragma unroll
  for (int t = 0; t < kGroup; ++t) xk[t] = __half2float(row_k(t)[c]);
  {
    const uint4* row = reinterpret_cast<const uint4*>(row_v(lane) + kGroup * qi);
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const uint4 u = row[k];
      const uint32_t wd[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float2 f = __half22float2(*reinterpret_cast<const __half2*>(&wd[e]));
        xv[8 * k + 2 * e] = f.x;
        xv[8 * k + 2 * e + 1] = f.y;
      }
    }
  }
  uint32_t wk[BK], wv[BV];
  __half sk, zk, sv, zv;
  quantize_group<BK>(xk, wk, sk, zk);
  quantize_group<BV>(xv, wv, sv, zv);
  kmeta[c] = sk;
  kmeta[kHeadDim + c] = zk;
  vmeta[vmeta_index(qi, lane)] = sv;
  vmeta[kHeadDim + vmeta_index(qi, lane)] = zv;
  // 1-bit codes: lane l = 4 gid + tig assembles word 4 l + qi from ballots
  // (bit positions of key1_bit / val1_bit)
  const int gid = lane >> 2, tig = lane & 3;
  if constexpr (BK == 1) {
    uint32_t mine[4] = {0u, 0u, 0u, 0u};  // ballots of tokens 4 gid + j over channels
#pragma unroll
    for (int t = 0; t < kGroup; ++t) {
      const uint32_t bt = __ballot_sync(0xffffffffu, (wk[0] >> t) & 1u);
      if ((t >> 2) == gid) mine[t & 3] = bt;
    }
    uint32_t word = 0u;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const uint32_t m = mine[j] >> (4 * tig);
#pragma unroll
      for (int ks1 = 0; ks1 < 2; ++ks1)
#pragma unroll
        for (int h = 0; h < 2; ++h)
#pragma unroll
          for (int e = 0; e < 2; ++e)
            word |= ((m >> (16 * ks1 + 2 * h + e)) & 1u) << ((10 + 16 * e + j - 4 * (2 * ks1 + h)) & 31);
    }
    kcodes[4 * lane + qi] = word;
  } else {
#pragma unroll
    for (int j = 0; j < BK; ++j) kcodes[c * BK + j] = wk[j];
  }
  if constexpr (BV == 1) {
    uint32_t mine[4] = {0u, 0u, 0u, 0u};  // ballots of channels 4 gid + j over tokens
#pragma unroll
    for (int ci = 0; ci < kGroup; ++ci) {
      const uint32_t bc = __ballot_sync(0xffffffffu, (wv[0] >> ci) & 1u);
      if ((ci >> 2) == gid) mine[ci & 3] = bc;
    }
    uint32_t word = 0u;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const uint32_t m = mine[j] >> (8 * tig);
#pragma unroll
      for (int e = 0; e < 2; ++e)
#pragma unroll
        for (int r = 0; r < 4; ++r)
          word |= ((m >> (4 * e + r)) & 1u) << ((10 + 16 * e + j - 4 * r) & 31);
    }
    vcodes[4 * lane + qi] = word;
  } else {
#pragma unroll
    for (int j = 0; j < BV; ++j) vcodes[(qi * kGroup + lane) * BV + j] = wv[j];
  }
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

// Pages of one (sequence b, kv-head h).  Contiguous layout: block j at
// base + j * page_bytes.  Paged layout (kvq.h): block j in page set
// row[j] of the pool, at base + row[j] * set_bytes with base = pool + h *
// page_bytes; an entry outside [0, n_pages) maps to no page.
struct PageMap {
  char* base;
  const int32_t* row;  // nullptr: contiguous
  long long page, set_bytes;
  int n_pages, max_blocks;
  __device__ __forceinline__ bool paged() const { return row != nullptr; }
  // address of block j given its table entry (ignored when contiguous);
  // nullptr when the entry is outside the pool
  __device__ __forceinline__ char* at(int j, int entry) const {
    if (!row) return base + (long long)j * page;
    return (entry >= 0 && entry < n_pages) ? base + (long long)entry * set_bytes : nullptr;
  }
  // address of block j, reading its table entry (single-thread use)
  __device__ __forceinline__ char* at(int j) const {
    return at(j, row ? (j < max_blocks ? row[j] : -1) : 0);
  }
};

__device__ __forceinline__ PageMap page_map(const Dims& d, const kvq_cache& c, int b, int h) {
  PageMap m;
  m.page = d.page_bytes;
  m.max_blocks = d.max_blocks;
  m.n_pages = c.n_pages;
  if (c.block_table) {
    m.row = c.block_table + (long long)b * d.max_blocks;
    m.base = static_cast<char*>(c.pages) + (long long)h * d.page_bytes;
    m.set_bytes = (long long)d.hkv * d.page_bytes;
  } else {
    m.row = nullptr;
    m.base = static_cast<char*>(c.pages) + ((long long)b * d.hkv + h) * d.max_blocks * d.page_bytes;
    m.set_bytes = 0;
  }
  return m;
}

// Thread-local error message (api.cu).
void set_error(const char* fmt, ...);

// Launchers (each returns a cudaError_t from cudaGetLastError after launch).
cudaError_t launch_pack(const Dims& d, const kvq_cache& cache, const __half* k_new,
                        const __half* v_new, int n_new, int batch_begin,
                        int batch_count, cudaStream_t stream);
// Decode attention, the flat plan on `ctas` CTAs (attn.cu).  out is fp16
// [batch][n_q_heads][128] when out_f16, else fp32.
cudaError_t launch_decode_attn(const Dims& d, const kvq_cache& cache, const __half* q,
                               void* out, int out_f16, float scale_log2, int ctas,
                               void* workspace, cudaStream_t stream);
// Append one token per sequence (k_new / v_new [batch][n_kv_heads][128]) and
// attend in the same kernel, the flat plan.
cudaError_t launch_decode_step(const Dims& d, const kvq_cache& cache, const __half* k_new,
                               const __half* v_new, const __half* q, void* out, int out_f16,
                               float scale_log2, int ctas, void* workspace,
                               cudaStream_t stream);
size_t attn_workspace_bytes(const Dims& d, int ctas);
// The split plan, n_splits CTAs per (sequence, kv-head) (attn_split.cu).
cudaError_t launch_decode_attn_split(const Dims& d, const kvq_cache& cache, const __half* q,
                                     void* out, int out_f16, float scale_log2, int n_splits,
                                     void* workspace, cudaStream_t stream);
cudaError_t launch_decode_step_split(const Dims& d, const kvq_cache& cache,
                                     const __half* k_new, const __half* v_new,
                                     const __half* q, void* out, int out_f16,
                                     float scale_log2, int n_splits, void* workspace,
                                     cudaStream_t stream);
size_t attn_split_workspace_bytes(const Dims& d, int n_splits);
unsigned* attn_split_tickets(const Dims& d, int n_splits, void* workspace, size_t* bytes);
int attn_default_splits(const Dims& d, int sm_count);
int attn_flat_ctas(int sm_count);
cudaError_t launch_wait_selftest(unsigned* flag, long long limit_cycles, cudaStream_t st);
int attn_splits_for_lengths(const Dims& d, int sm_count, const int32_t* lengths);
size_t attn_static_scratch_bytes();
// n_splits > 0: the split plan; < 0: the flat plan on -n_splits CTAs.
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
// Offline drift metrics (drift.cu).
int drift_max_vocab();
int drift_max_kcov();
cudaError_t launch_drift(const float* z_fp, const float* z_q, int rows, int vocab,
                         const kvq_drift_params& p, int32_t* m_t, float* c_t, float* d_loc,
                         uint8_t* y_t, float* cov, cudaStream_t st);
cudaError_t launch_drift_window(const float* cov, int rows, int k_max, float rho_k,
                                float* mean_cov, int32_t* k_b, cudaStream_t st);
cudaError_t launch_dgap(const DgapDims& d, const dgap_params& p, float* logits,
                        int32_t* topk_idx, float* topk_val, float* risk,
                        uint8_t* gate, int32_t* next_token, float* features,
                        void* workspace, cudaStream_t stream);

}  // namespace kvq
