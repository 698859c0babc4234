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
//
// The codes come from one fused multiply-add, y = RN32(d * r + 1536.5) with
// d = RN32(x - zero) and r = RN32(1 / s): the exact d * r lies within
// 2^-24 * (d / s) of d / s, and so does RN32(d / s), so (d / s <= levels <=
// 255) d * r is within 3.1e-5 of RN32(d / s), and both round to the same
// integer unless d * r lies within 3.1e-5 of a half-integer.  d * r + 1536.5
// lies in [1536.5, 1792.5), where float32 numbers are 2^-13 apart, so the
// bits of y are kCodeBias + floor(q + 0.5) from bit 13 up and the fraction
// of q + 0.5 below, q being d * r on the 2^-13 grid.  A d * r within half a
// grid step (6.1e-5) of a half-integer puts y on an integer, with its 13 low
// bits zero; so does a NaN.  Such an element's code is taken by the
// definition's steps (the exact quotient) and swapped into its word; every
// other element's code is floor(q + 0.5) = rint(RN32(d / s)), which lies in
// [0, levels].  A zero scale takes r = 0, so every code is 0.
constexpr float kCodeMagic = 1536.5f;
constexpr uint32_t kCodeBias = 0x22600u;  // bits of 1536.5 >> 13, plus 512

// Sum of kCodeBias at each code position of a word: a word accumulates
// (y >> 13) << pos = (kCodeBias + code) << pos over its 32 / B codes.
template <int B>
__host__ __device__ constexpr uint32_t code_bias_word() {
  uint32_t c = 0u;
  for (int k = 0; k < 32 / B; ++k) c += kCodeBias << (k * B);
  return c;
}

// RU32(x / L) for a float32 x >= 0 (or +inf) and L = levels: the product
// with RN32(1 / L) lies within two ulps of x / L, and the sign of the exact
// q * L - x (one fused multiply-add) moves it up, then down, to the least
// float32 >= x / L.  L = 1 is exact.
template <int L>
__device__ __forceinline__ float div_ru_levels(float x) {
  if constexpr (L == 1) {
    return x;
  } else {
    float q = __fmul_rn(x, 1.0f / L);
#pragma unroll
    for (int k = 0; k < 2; ++k)
      if (__fmaf_rn(q, float(L), -x) < 0.0f) q = __uint_as_float(__float_as_uint(q) + 1u);
#pragma unroll
    for (int k = 0; k < 2; ++k) {
      const float p = __uint_as_float(__float_as_uint(q) - 1u);
      if (q > 0.0f && __fmaf_rn(p, float(L), -x) >= 0.0f) q = p;
    }
    return q;
  }
}

// Codes and scale of one group from d(i) = RN32(x_i - lo) and the group's
// min lo and max hi.  d2 computes the same values by other instructions, for
// the rare elements near a tie: recomputing them there keeps the compiler
// from holding every element's d and y in registers until then.
template <int B, typename D, typename D2>
__device__ __forceinline__ void quantize_codes(D d, D2 d2, float lo, float hi, uint32_t (&w)[B],
                                               __half& scale) {
  constexpr float kLevels = float((1 << B) - 1);
  const __half s_h = __float2half_ru(div_ru_levels<(1 << B) - 1>(__fsub_ru(hi, lo)));
  const float s = __half2float(s_h);
  const float r = s > 0.0f ? __frcp_rn(s) : 0.0f;
  uint32_t acc[B];
#pragma unroll
  for (int j = 0; j < B; ++j) acc[j] = 0u;
  uint32_t low = 0x1fffu;  // least 13-bit fraction field seen
#pragma unroll
  for (int i = 0; i < kGroup; ++i) {
    const uint32_t y = __float_as_uint(__fmaf_rn(d(i), r, kCodeMagic));
    low = min(low, y & 0x1fffu);
    if constexpr (B == 1) {
      acc[0] |= ((y >> 13) & 1u) << i;  // kCodeBias is even
    } else {
      acc[(i * B) / 32] += (y >> 13) << ((i * B) % 32);
    }
  }
  if constexpr (B > 1) {
#pragma unroll
    for (int j = 0; j < B; ++j) acc[j] -= code_bias_word<B>();
  }
  if (low == 0u) {  // near a tie (or not finite): those elements by the definition's steps
#pragma unroll
    for (int i = 0; i < kGroup; ++i) {
      const float di = d2(i);
      const uint32_t y = __float_as_uint(__fmaf_rn(di, r, kCodeMagic));
      if ((y & 0x1fffu) == 0u) {
        uint32_t c = 0u;
        if (s > 0.0f) c = (uint32_t)fminf(fmaxf(rintf(__fdiv_rn(di, s)), 0.0f), kLevels);
        if constexpr (B == 1) {
          acc[0] = (acc[0] & ~(1u << i)) | (c << i);
        } else {  // the word is a sum of its fields: swap this one's (mod 2^32)
          acc[(i * B) / 32] += (c + kCodeBias - (y >> 13)) << ((i * B) % 32);
        }
      }
    }
  }
#pragma unroll
  for (int j = 0; j < B; ++j) w[j] = acc[j];
  scale = s_h;
}

template <int B>
__device__ __forceinline__ void quantize_group(const float (&x)[kGroup], uint32_t (&w)[B],
                                               __half& scale, __half& zero) {
  float lo = x[0], hi = x[0];
#pragma unroll
  for (int i = 1; i < kGroup; ++i) {
    lo = fminf(lo, x[i]);
    hi = fmaxf(hi, x[i]);
  }
  const auto d = [&](int i) { return __fsub_rn(x[i], lo); };
  quantize_codes<B>(d, d, lo, hi, w, scale);
  zero = __float2half_rn(lo);  // lo is an fp16 value: exact
}

// Min and max of 32 fp16 numbers held as 16 pairs (exact in fp16).
__device__ __forceinline__ void group_range(const __half2 (&x)[kGroup / 2], float& lo, float& hi) {
  __half2 l = x[0], h = x[0];
#pragma unroll
  for (int p = 1; p < kGroup / 2; ++p) {
    l = __hmin2(l, x[p]);
    h = __hmax2(h, x[p]);
  }
  lo = fminf(__low2float(l), __high2float(l));
  hi = fmaxf(__low2float(h), __high2float(h));
}

// RN32(a - c) for an fp16 a (one half of a pair) and a float32 c: one
// mixed-precision subtraction (a is widened exactly, the difference rounded
// once).
template <int kHigh>
__device__ __forceinline__ float sub_half(__half2 pair, float c) {
  float d;
  if constexpr (kHigh)
    asm("{.reg .b16 l, h; mov.b32 {l, h}, %1; sub.rn.f32.f16 %0, h, %2;}"
        : "=f"(d) : "r"(*reinterpret_cast<const uint32_t*>(&pair)), "f"(c));
  else
    asm("{.reg .b16 l, h; mov.b32 {l, h}, %1; sub.rn.f32.f16 %0, l, %2;}"
        : "=f"(d) : "r"(*reinterpret_cast<const uint32_t*>(&pair)), "f"(c));
  return d;
}

// Codes and scale of the group held as 16 pairs (element i = half i & 1 of
// pair i >> 1); lo is the group's min (its zero).
template <int B>
__device__ __forceinline__ void quantize_pairs(const __half2 (&x)[kGroup / 2], uint32_t (&w)[B],
                                               __half& scale, float& lo) {
  float hi;
  group_range(x, lo, hi);
  const float z = lo;
  quantize_codes<B>(
      [&](int i) { return (i & 1) ? sub_half<1>(x[i >> 1], z) : sub_half<0>(x[i >> 1], z); },
      [&](int i) {
        return __fsub_rn((i & 1) ? __high2float(x[i >> 1]) : __low2float(x[i >> 1]), z);
      },
      lo, hi, w, scale);
}

__host__ __device__ constexpr uint32_t rotl_const(uint32_t v, int p) {
  return p == 0 ? v : (v << p) | (v >> (32 - p));
}

// One lane's word of 1-bit codes in fragment order, from the code rows
// (bit i = element i) of eight source lanes: from source k, the nibble at
// bit 4 gid goes to bits p_k .. p_k + 3 (mod 32).
template <typename Src, typename Pos>
__device__ __forceinline__ uint32_t gather_nibbles(uint32_t row, int gid, Src src, Pos pos) {
  uint32_t word = 0u;
#pragma unroll
  for (int k = 0; k < 8; ++k) {
    const uint32_t v = __shfl_sync(0xffffffffu, row, src(k));
    const int p = pos(k) & 31;
    word |= __funnelshift_r(v, v, (4 * gid - p) & 31) & rotl_const(0xfu, p);
  }
  return word;
}

// One quarter qi of a 32-token block, quantized by one warp into a page (or
// a page image): key groups of channels 32 qi .. 32 qi + 31 (lane = channel)
// and value group qi of the 32 tokens (lane = token).  row_k(t), row_v(t)
// give the fp16 rows [128] of token t of the block.  The quarters write
// disjoint words, scales and zeros, so the four may run in different warps.
// Codes of b >= 2 bits: key channel c and value (group qi, token lane) both
// take words (32 qi + lane) * b .. + b - 1 of their code areas.  1-bit
// codes: lane l = 4 gid + tig writes word 4 l + qi, gathered with shuffles
// in the order key1_bit / val1_bit give: keys take tokens 4 gid + j
// (j = 0..3) of channels 16 ks1 + 4 tig + 2 h + e at bit 10 + 16 e + j -
// 4 (2 ks1 + h); values take channels 4 gid + j of tokens 8 tig + 4 e + r
// at bit 10 + 16 e + j - 4 r.  With equal key and value widths one code
// body quantizes both groups in turn (half the instructions to fetch).
// Used by kvq_pack and by the decode step's flush, which are therefore
// bit-identical.
template <int BK, int BV, typename RowK, typename RowV>
__device__ __forceinline__ void quantize_quarter(RowK row_k, RowV row_v, int qi, char* image) {
  const int lane = threadIdx.x & 31;
  const int gid = lane >> 2, tig = lane & 3;
  uint32_t* kcodes = reinterpret_cast<uint32_t*>(image);
  uint32_t* vcodes = reinterpret_cast<uint32_t*>(image + page_off_vcodes(BK));
  __half* kmeta = reinterpret_cast<__half*>(image + page_off_kmeta(BK));
  __half* vmeta = reinterpret_cast<__half*>(image + page_off_vmeta(BK, BV));
  const int c = kGroup * qi + lane;  // this lane's key channel
  const int vm = vmeta_index(qi, lane);
  __half2 xk[kGroup / 2], xv[kGroup / 2];  // tokens 2p, 2p + 1 / channels 2p, 2p + 1
#pragma unroll
  for (int p = 0; p < kGroup / 2; ++p) xk[p] = __halves2half2(row_k(2 * p)[c], row_k(2 * p + 1)[c]);
  {
    const uint4* row = reinterpret_cast<const uint4*>(row_v(lane) + kGroup * qi);
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const uint4 u = row[k];
      const uint32_t wd[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
      for (int e = 0; e < 4; ++e) xv[4 * k + e] = *reinterpret_cast<const __half2*>(&wd[e]);
    }
  }
  uint32_t rk = 0u, rv = 0u;  // 1-bit code rows
  if constexpr (BK == BV) {
#pragma unroll 1
    for (int pass = 0; pass < 2; ++pass) {  // keys from xk, then values moved there
      uint32_t w[BK];
      __half s;
      float lo;
      quantize_pairs<BK>(xk, w, s, lo);
      __half* meta = pass ? vmeta : kmeta;
      const int mi = pass ? vm : c;
      meta[mi] = s;
      meta[kHeadDim + mi] = __float2half_rn(lo);  // an fp16 value: exact
      if constexpr (BK == 1) {
        if (pass) rv = w[0]; else rk = w[0];
      } else {
        uint32_t* codes = (pass ? vcodes : kcodes) + c * BK;
#pragma unroll
        for (int j = 0; j < BK; ++j) codes[j] = w[j];
      }
#pragma unroll
      for (int p = 0; p < kGroup / 2; ++p) xk[p] = xv[p];
    }
  } else {
    uint32_t wk[BK], wv[BV];
    __half sk, sv;
    float lok, lov;
    quantize_pairs<BK>(xk, wk, sk, lok);
    quantize_pairs<BV>(xv, wv, sv, lov);
    kmeta[c] = sk;
    kmeta[kHeadDim + c] = __float2half_rn(lok);
    vmeta[vm] = sv;
    vmeta[kHeadDim + vm] = __float2half_rn(lov);
    if constexpr (BK == 1) rk = wk[0];
    else {
#pragma unroll
      for (int j = 0; j < BK; ++j) kcodes[c * BK + j] = wk[j];
    }
    if constexpr (BV == 1) rv = wv[0];
    else {
#pragma unroll
      for (int j = 0; j < BV; ++j) vcodes[c * BV + j] = wv[j];
    }
  }
  if constexpr (BK == 1)
    kcodes[4 * lane + qi] = gather_nibbles(
        rk, gid, [&](int k) { return 16 * (k >> 2) + 2 * ((k >> 1) & 1) + (k & 1) + 4 * tig; },
        [](int k) { return 10 + 16 * (k & 1) - 8 * (k >> 2) - 4 * ((k >> 1) & 1); });
  if constexpr (BV == 1)
    vcodes[4 * lane + qi] = gather_nibbles(
        rv, gid, [&](int k) { return 8 * tig + 4 * (k >> 2) + (k & 3); },
        [](int k) { return 10 + 16 * (k >> 2) - 4 * (k & 3); });
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
