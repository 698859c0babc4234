// kvq_decode_attn: one decode step of grouped-query attention
// softmax(q K^T * scale) V (Sec. 1 of the paper) over the packed KbVb cache.
//
// Split-K ("flash-decoding") layout: grid (n_splits, n_kv_heads, batch).  The
// work of one (sequence, kv-head) is a list of units — the packed 32-token
// blocks, then the fp16 residual window cut into 32-token chunks — divided
// into n_splits contiguous ranges.  A CTA serves every query head of its
// kv-head, keeps an online softmax per warp, and writes one partial
// (max, sum, unnormalised row) per query head.  The last CTA of a
// (sequence, kv-head) to finish (atomic ticket, no waiting) merges the
// partials:  out = sum_s 2^{m_s - M} o_s / sum_s 2^{m_s - M} l_s.
// Scores are kept in the log2 domain (q is pre-multiplied by scale*log2 e).

#include <float.h>

#include <mutex>

#include "common.cuh"

namespace kvq {
namespace {

constexpr int kThreads = 128;
constexpr int kWarps = kThreads / 32;

struct Ws {
  float* m;       // [B][Hq][S]
  float* l;       // [B][Hq][S]
  float* o;       // [B][Hq][S][128]
  unsigned* tk;   // [B][Hkv]
};

__host__ __device__ inline size_t align256(size_t x) { return (x + 255) / 256 * 256; }

__host__ __device__ inline Ws carve(void* base, int batch, int hq, int hkv, int S) {
  Ws w;
  char* p = static_cast<char*>(base);
  const size_t nml = (size_t)batch * hq * S;
  w.m = reinterpret_cast<float*>(p);
  p += align256(nml * 4);
  w.l = reinterpret_cast<float*>(p);
  p += align256(nml * 4);
  w.o = reinterpret_cast<float*>(p);
  p += align256(nml * kHeadDim * 4);
  w.tk = reinterpret_cast<unsigned*>(p);
  return w;
}

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Per-warp online-softmax state for up to kMaxGq query heads; lane owns
// output channels 4*lane .. 4*lane+3.
struct State {
  float m[kMaxGq], l[kMaxGq], acc[kMaxGq][4];
};

// Fold one 32-token unit's scores (lane = token) and values into the state.
// vrow(t, c4) returns the 4 dequantized values of token t, channels 4*lane..
template <typename VRow>
__device__ __forceinline__ void online_update(State& st, float (&sc)[kMaxGq], int gq,
                                              int n_tok, const VRow& vrow) {
  const int lane = threadIdx.x & 31;
  float p[kMaxGq];
#pragma unroll
  for (int g = 0; g < kMaxGq; ++g) {
    if (g >= gq) break;
    const float s = lane < n_tok ? sc[g] : -INFINITY;
    const float mx = warp_max(s);
    const float mn = fmaxf(st.m[g], mx);
    const float corr = exp2f(st.m[g] - mn);  // m = -inf, mn finite -> 0
    p[g] = exp2f(s - mn);
    st.l[g] = st.l[g] * corr + warp_sum(p[g]);
#pragma unroll
    for (int i = 0; i < 4; ++i) st.acc[g][i] *= corr;
    st.m[g] = mn;
  }
  for (int t = 0; t < n_tok; ++t) {
    float v[4];
    vrow(t, v);
#pragma unroll
    for (int g = 0; g < kMaxGq; ++g) {
      if (g >= gq) break;
      const float pt = __shfl_sync(0xffffffffu, p[g], t);
#pragma unroll
      for (int i = 0; i < 4; ++i) st.acc[g][i] = fmaf(pt, v[i], st.acc[g][i]);
    }
  }
}

template <int BK, int BV>
__device__ void packed_unit(State& st, const float (*qs)[kHeadDim], int gq, const char* page) {
  const int lane = threadIdx.x & 31;
  const uint32_t* kc = reinterpret_cast<const uint32_t*>(page);
  const __half2* km = reinterpret_cast<const __half2*>(page + page_off_kmeta(BK));
  const uint32_t* vc = reinterpret_cast<const uint32_t*>(page + page_off_vcodes(BK));
  const __half2* vm = reinterpret_cast<const __half2*>(page + page_off_vmeta(BK, BV));
  constexpr uint32_t kMaskK = (1u << BK) - 1u, kMaskV = (1u << BV) - 1u;

  float sc[kMaxGq];
#pragma unroll
  for (int g = 0; g < kMaxGq; ++g) sc[g] = 0.0f;
  const int kword = (lane * BK) / 32, kshift = (lane * BK) % 32;
  for (int c = 0; c < kHeadDim; ++c) {
    const uint32_t code = (kc[c * BK + kword] >> kshift) & kMaskK;
    const float2 sz = __half22float2(km[c]);
    const float kh = fmaf(sz.x, (float)code, sz.y);
#pragma unroll
    for (int g = 0; g < kMaxGq; ++g) {
      if (g >= gq) break;
      sc[g] = fmaf(qs[g][c], kh, sc[g]);
    }
  }
  const int grp = lane >> 3;  // channels 4*lane.. lie in group lane / 8
  online_update(st, sc, gq, kGroup, [&](int t, float (&v)[4]) {
    const float2 sz = __half22float2(vm[t * 4 + grp]);
    const uint32_t* w = vc + (t * 4 + grp) * BV;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int cc = (4 * lane + i) & 31;
      const uint32_t code = (w[(cc * BV) / 32] >> ((cc * BV) % 32)) & kMaskV;
      v[i] = fmaf(sz.x, (float)code, sz.y);
    }
  });
}

__device__ void resid_unit(State& st, const float (*qs)[kHeadDim], int gq, const __half* ring_k,
                           const __half* ring_v, int p0, int n_tok, int ring) {
  const int lane = threadIdx.x & 31;
  float sc[kMaxGq];
#pragma unroll
  for (int g = 0; g < kMaxGq; ++g) sc[g] = 0.0f;
  if (lane < n_tok) {
    const uint4* row = reinterpret_cast<const uint4*>(ring_k + (long long)((p0 + lane) % ring) * kHeadDim);
    for (int piece = 0; piece < 16; ++piece) {
      const uint4 u = row[piece];
      const __half2* h2 = reinterpret_cast<const __half2*>(&u);
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float2 f = __half22float2(h2[e]);
        const int c = piece * 8 + 2 * e;
#pragma unroll
        for (int g = 0; g < kMaxGq; ++g) {
          if (g >= gq) break;
          sc[g] = fmaf(qs[g][c], f.x, sc[g]);
          sc[g] = fmaf(qs[g][c + 1], f.y, sc[g]);
        }
      }
    }
  }
  online_update(st, sc, gq, n_tok, [&](int t, float (&v)[4]) {
    const uint2 u = reinterpret_cast<const uint2*>(
        ring_v + (long long)((p0 + t) % ring) * kHeadDim)[lane];
    const float2 a = __half22float2(*reinterpret_cast<const __half2*>(&u.x));
    const float2 b = __half22float2(*reinterpret_cast<const __half2*>(&u.y));
    v[0] = a.x; v[1] = a.y; v[2] = b.x; v[3] = b.y;
  });
}

template <int BK, int BV>
__global__ void __launch_bounds__(kThreads)
    decode_attn_kernel(Dims d, kvq_cache c, const __half* __restrict__ q, __half* __restrict__ out,
                       float scale_log2, int S, Ws ws) {
  __shared__ float qs[kMaxGq][kHeadDim];
  __shared__ float wm[kWarps][kMaxGq], wl[kWarps][kMaxGq];
  __shared__ float wo[kWarps][kMaxGq][kHeadDim];
  __shared__ int last;

  const int s = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
  const int gq = d.gq, warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int L = c.seq_len[b];
  const int Lq = packed_len(L, d.residual);
  const int nb = Lq / kGroup;
  const int units = nb + (L - Lq + kGroup - 1) / kGroup;
  const int per = (units + S - 1) / S;
  const int u0 = min(units, s * per), u1 = min(units, u0 + per);

  const __half* qh = q + ((long long)b * d.hq + (long long)h * gq) * kHeadDim;
  for (int e = threadIdx.x; e < gq * kHeadDim; e += kThreads)
    qs[e / kHeadDim][e % kHeadDim] = __half2float(qh[e]) * scale_log2;
  __syncthreads();

  State st;
#pragma unroll
  for (int g = 0; g < kMaxGq; ++g) {
    st.m[g] = -INFINITY;
    st.l[g] = 0.0f;
#pragma unroll
    for (int i = 0; i < 4; ++i) st.acc[g][i] = 0.0f;
  }
  const long long bh = (long long)b * d.hkv + h;
  const char* pages = static_cast<const char*>(c.pages) + bh * d.max_blocks * d.page_bytes;
  const __half* ring_k = reinterpret_cast<const __half*>(c.k_resid) + bh * d.ring * kHeadDim;
  const __half* ring_v = reinterpret_cast<const __half*>(c.v_resid) + bh * d.ring * kHeadDim;
  for (int u = u0 + warp; u < u1; u += kWarps) {
    if (u < nb) {
      packed_unit<BK, BV>(st, qs, gq, pages + (long long)u * d.page_bytes);
    } else {
      const int p0 = Lq + (u - nb) * kGroup;
      resid_unit(st, qs, gq, ring_k, ring_v, p0, min(kGroup, L - p0), d.ring);
    }
  }

  // Merge the warps' states and publish this split's partials.
#pragma unroll
  for (int g = 0; g < kMaxGq; ++g) {
    if (g >= gq) break;
    if (lane == 0) {
      wm[warp][g] = st.m[g];
      wl[warp][g] = st.l[g];
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) wo[warp][g][4 * lane + i] = st.acc[g][i];
  }
  __syncthreads();
  const int cidx = threadIdx.x;  // one output channel per thread
  for (int g = 0; g < gq; ++g) {
    float M = -INFINITY;
    for (int w = 0; w < kWarps; ++w) M = fmaxf(M, wm[w][g]);
    float l = 0.0f, o = 0.0f;
    if (M != -INFINITY) {
      for (int w = 0; w < kWarps; ++w) {
        const float f = exp2f(wm[w][g] - M);
        l += f * wl[w][g];
        o += f * wo[w][g][cidx];
      }
    }
    const long long row = ((long long)b * d.hq + (long long)h * gq + g) * S + s;
    ws.o[row * kHeadDim + cidx] = o;
    if (cidx == 0) {
      ws.m[row] = M;
      ws.l[row] = l;
    }
  }

  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    const unsigned t = atomicAdd(&ws.tk[bh], 1u);
    last = (t == (unsigned)S - 1);
  }
  __syncthreads();
  if (!last) return;
  __threadfence();

  for (int g = 0; g < gq; ++g) {
    const long long row0 = ((long long)b * d.hq + (long long)h * gq + g) * S;
    float M = -INFINITY;
    for (int k = 0; k < S; ++k) M = fmaxf(M, __ldcg(ws.m + row0 + k));
    float l = 0.0f, o = 0.0f;
    if (M != -INFINITY) {
      for (int k = 0; k < S; ++k) {
        const float f = exp2f(__ldcg(ws.m + row0 + k) - M);
        l += f * __ldcg(ws.l + row0 + k);
        o += f * __ldcg(ws.o + (row0 + k) * kHeadDim + cidx);
      }
    }
    const float r = l > 0.0f ? o / l : 0.0f;
    out[((long long)b * d.hq + (long long)h * gq + g) * kHeadDim + cidx] = __float2half_rn(r);
  }
  if (threadIdx.x == 0) ws.tk[bh] = 0u;
}

template <int BK>
cudaError_t launch_bv(const Dims& d, const kvq_cache& c, const __half* q, __half* out, float sl2,
                      int S, const Ws& ws, cudaStream_t st) {
  dim3 grid(S, d.hkv, d.batch);
  switch (d.bits_v) {
    case 1: decode_attn_kernel<BK, 1><<<grid, kThreads, 0, st>>>(d, c, q, out, sl2, S, ws); break;
    case 2: decode_attn_kernel<BK, 2><<<grid, kThreads, 0, st>>>(d, c, q, out, sl2, S, ws); break;
    case 4: decode_attn_kernel<BK, 4><<<grid, kThreads, 0, st>>>(d, c, q, out, sl2, S, ws); break;
    default: decode_attn_kernel<BK, 8><<<grid, kThreads, 0, st>>>(d, c, q, out, sl2, S, ws); break;
  }
  return cudaGetLastError();
}

}  // namespace

size_t attn_workspace_bytes(const Dims& d, int S) {
  const size_t nml = (size_t)d.batch * d.hq * S;
  return align256(nml * 4) * 2 + align256(nml * kHeadDim * 4) +
         align256((size_t)d.batch * d.hkv * 4);
}

cudaError_t launch_decode_attn(const Dims& d, const kvq_cache& c, const __half* q, __half* out,
                               float scale_log2, int S, void* workspace, cudaStream_t st) {
  const Ws ws = carve(workspace, d.batch, d.hq, d.hkv, S);
  switch (d.bits_k) {
    case 1: return launch_bv<1>(d, c, q, out, scale_log2, S, ws, st);
    case 2: return launch_bv<2>(d, c, q, out, scale_log2, S, ws, st);
    case 4: return launch_bv<4>(d, c, q, out, scale_log2, S, ws, st);
    default: return launch_bv<8>(d, c, q, out, scale_log2, S, ws, st);
  }
}

// ---------------------------------------------------------------------------
// Decode attention without caller-supplied scratch (kvq_decode_attn_noalloc).
//
// Some callers cannot allocate device memory where they run a decode step: a
// host framework whose pool owns every byte of the GPU (a raw allocation would
// fail or fragment it), or a serving loop that must not allocate per step.
// For them the split partials and tickets live in this one file-scope device
// array of fixed size, which every GPU that loads the library holds until the
// process exits.  All calls share it, so calls that overlap on the GPU race.
// ---------------------------------------------------------------------------

namespace {
constexpr size_t kStaticScratchBytes = size_t(4) << 20;  // 4 MiB
constexpr int kMaxDevices = 64;
__device__ __align__(256) unsigned char g_attn_scratch[kStaticScratchBytes];

// Device address of g_attn_scratch on the current device, looked up once per
// device with that device current.  In host code the symbol is only a
// host-side stand-in: passing it to a kernel would fault or silently use the
// wrong memory, so only the looked-up address is ever used.
cudaError_t static_scratch(void** out) {
  static std::mutex mu;
  static void* addr[kMaxDevices] = {};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(mu);
  if (!addr[dev]) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_attn_scratch);
    if (e != cudaSuccess) return e;
    addr[dev] = p;
  }
  *out = addr[dev];
  return cudaSuccess;
}
}  // namespace

size_t attn_static_scratch_bytes() { return kStaticScratchBytes; }

cudaError_t launch_decode_attn_static(const Dims& d, const kvq_cache& c, const __half* q,
                                      __half* out, float scale_log2, int S, cudaStream_t st) {
  void* ws = nullptr;
  cudaError_t e = static_scratch(&ws);
  if (e != cudaSuccess) return e;
  // The array keeps the previous call's contents: the tickets must start at
  // zero, the partials are always written before they are read.
  const Ws w = carve(ws, d.batch, d.hq, d.hkv, S);
  e = cudaMemsetAsync(w.tk, 0, (size_t)d.batch * d.hkv * sizeof(unsigned), st);
  if (e != cudaSuccess) return e;
  return launch_decode_attn(d, c, q, out, scale_log2, S, ws, st);
}

}  // namespace kvq
