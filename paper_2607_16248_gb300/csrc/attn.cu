// kvq_decode_attn: one decode step of grouped-query attention
// softmax(q K^T * scale) V (Sec. 1 of the paper) over the packed KbVb cache.
//
// Split-K ("flash-decoding"): grid (n_splits + 1, n_kv_heads, batch).  Splits
// 0 .. n_splits-1 share the packed 32-token blocks of one (sequence, kv-head);
// the last split takes the fp16 residual window.  Each CTA writes one partial
// (max, sum, unnormalised row) per query head; the last CTA of a
// (sequence, kv-head) to finish (atomic ticket, no waiting) merges them:
//   out = sum_s 2^{m_s - M} o_s / sum_s 2^{m_s - M} l_s.
// Scores are kept in the log2 domain (scaled by softmax_scale * log2 e).
//
// Packed blocks run on the tensor cores (mma.sync m16n8k16, f16 in, f32
// accumulate) with operands built in registers straight from the packed
// codes.  A producer warp streams each split's contiguous pages into shared
// memory with bulk asynchronous copies (cp.async.bulk + mbarrier); four
// consumer warps each take one 32-token block per stage:
//
//   keys    S[t][h] = sum_c code[t][c] * (q_h[c] s_c) + sum_c q_h[c] z_c
//           A = codes (M = tokens, K = channels), B = q*s split into an fp16
//           high part (columns 0..3) and its exact fp16 residual (columns
//           4..7, the padding of the 4 query heads), so the products are
//           exact; the zero-point term is one more MMA with A = z, B = q.
//   values  o[c][h] += sum_t code[t][c] * (p_h[t] s_t,g) + sum_t p_h[t] z_t,g
//           A = codes (M = channels, K = tokens), B = p*s with p split into
//           high / low fp16 parts in columns 0..3 / 4..7; P moves from the
//           score (accumulator) layout to the B layout with movmatrix.
//
// Codes become fp16 values without a table: for 1-bit codes a shifted bit
// lands on an exponent bit (value 2^e), for wider codes the code is OR-ed into
// the mantissa of 1024 and 1024 is subtracted.  The four tokens (keys) or
// channels (values) a lane owns are chosen to sit in one nibble / byte of a
// packed word; the resulting per-row power-of-two factors are undone on the
// fp32 results.  The fp16 residual window takes the same MMAs with operands
// loaded by ldmatrix from rows staged in shared memory.  Query-head groups
// wider than 4 use the SIMT path for every unit.

#include <float.h>

#include <mutex>

#include "common.cuh"

namespace kvq {
namespace {

constexpr int kConsumers = 5;                 // computing warps; the last one also streams
constexpr int kThreads = 32 * kConsumers;
constexpr int kResWarps = kConsumers;         // warps that stage the fp16 window
#ifndef KVQ_ATTN_CTAS_PER_SM
#define KVQ_ATTN_CTAS_PER_SM 2
#endif
#ifndef KVQ_ATTN_UNIT_BLOCKS
#define KVQ_ATTN_UNIT_BLOCKS 2
#endif
constexpr int kCtasPerSm = KVQ_ATTN_CTAS_PER_SM;   // resident CTAs per SM
constexpr int kUnitBlocks = KVQ_ATTN_UNIT_BLOCKS;  // blocks per consumer warp per stage
constexpr int kStageBudget = (kCtasPerSm >= 3 ? 60 : 80) * 1024;  // staged page bytes per CTA
constexpr long long kWaitCycles = 4000000000LL;  // bounded mbarrier waits (~2 s)

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

// Shared-memory areas of one CTA.  The merge area overlaps the stage
// buffers: it is written only after every stage has been consumed.
struct MergeArea {
  float qs[kMaxGq][kHeadDim];           // SIMT path: q * scale * log2 e
  float wm[kConsumers][kMaxGq];
  float wl[kConsumers][kMaxGq];
  float wo[kConsumers][kMaxGq][kHeadDim];
  int last;
};

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

// ---------------------------------------------------------------------------
// PTX helpers: mbarrier, bulk async copy, mma.sync, movmatrix
// ---------------------------------------------------------------------------

__device__ __forceinline__ uint32_t smem_addr(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count)
               : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)),
               "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_addr(bar)) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n"
      " mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
      " selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(smem_addr(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
// Wait for the phase with the given parity to complete; false after ~2 s.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity) {
  if (mbar_try_wait(bar, parity)) return true;
  const long long t0 = clock64();
  while (!mbar_try_wait(bar, parity))
    if (clock64() - t0 > kWaitCycles) return false;
  return true;
}
__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
          smem_addr(dst)),
      "l"(src), "r"(bytes), "r"(smem_addr(bar))
      : "memory");
}
__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
// Programmatic dependent launch: let the next kernel in the stream start
// launching, and wait until the previous one has completed and its writes
// are visible.  Both are no-ops when the kernel was launched without the
// programmatic-serialization attribute.
__device__ __forceinline__ void pdl_launch_dependents() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ int read_len(const int* p) {
  return *reinterpret_cast<const volatile int*>(p);
}

__device__ __forceinline__ void mma16816(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2,
                                         uint32_t a3, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
      "{%8,%9}, {%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}
__device__ __forceinline__ uint32_t movmatrix_t(uint32_t a) {
  uint32_t d;
  asm volatile("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;" : "=r"(d) : "r"(a));
  return d;
}

// 2^x with the SFU (x <= 0 here; -inf gives +0).
__device__ __forceinline__ float fast_exp2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ uint32_t h2u(__half2 h) { return *reinterpret_cast<uint32_t*>(&h); }
__device__ __forceinline__ __half2 u2h(uint32_t u) { return *reinterpret_cast<__half2*>(&u); }
__device__ __forceinline__ uint32_t hsub1024(uint32_t x) {
  return h2u(__hsub2(u2h(x), u2h(0x64006400u)));
}

// ---------------------------------------------------------------------------
// SIMT path: residual window (and every unit when the query group is wider
// than 4).  Lane = token for scores; lane owns channels 4*lane.. for values.
// ---------------------------------------------------------------------------

struct State {
  float m[kMaxGq], l[kMaxGq], acc[kMaxGq][4];
};

template <typename VRow>
__device__ __forceinline__ void online_update(State& st, float (&sc)[kMaxGq], int gq, int n_tok,
                                              const VRow& vrow) {
  const int lane = threadIdx.x & 31;
  float p[kMaxGq];
#pragma unroll
  for (int g = 0; g < kMaxGq; ++g) {
    if (g >= gq) break;
    const float s = lane < n_tok ? sc[g] : -INFINITY;
    const float mx = warp_max(s);
    const float mn = fmaxf(st.m[g], mx);
    const float corr = exp2f(st.m[g] - mn);
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
__device__ void simt_packed_unit(State& st, const float (*qs)[kHeadDim], int gq, const char* page) {
  const int lane = threadIdx.x & 31;
  const uint32_t* kc = reinterpret_cast<const uint32_t*>(page);
  const __half* ksc = reinterpret_cast<const __half*>(page + page_off_kmeta(BK));  // [128] then zeros
  const uint32_t* vc = reinterpret_cast<const uint32_t*>(page + page_off_vcodes(BK));
  const __half* vsc = reinterpret_cast<const __half*>(page + page_off_vmeta(BK, BV));  // [4][32] then zeros
  constexpr uint32_t kMaskK = (1u << BK) - 1u, kMaskV = (1u << BV) - 1u;
  float sc[kMaxGq];
#pragma unroll
  for (int g = 0; g < kMaxGq; ++g) sc[g] = 0.0f;
  const int kword = (lane * BK) / 32, kshift = (lane * BK) % 32;
  for (int c = 0; c < kHeadDim; ++c) {
    const uint32_t code = (kc[c * BK + kword] >> kshift) & kMaskK;
    const float kh = fmaf(__half2float(ksc[c]), (float)code, __half2float(ksc[kHeadDim + c]));
#pragma unroll
    for (int g = 0; g < kMaxGq; ++g) {
      if (g >= gq) break;
      sc[g] = fmaf(qs[g][c], kh, sc[g]);
    }
  }
  const int grp = lane >> 3;
  online_update(st, sc, gq, kGroup, [&](int t, float (&v)[4]) {
    const float sv = __half2float(vsc[grp * 32 + t]), zv = __half2float(vsc[kHeadDim + grp * 32 + t]);
    const uint32_t* w = vc + (grp * 32 + t) * BV;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int cc = (4 * lane + i) & 31;
      const uint32_t code = (w[(cc * BV) / 32] >> ((cc * BV) % 32)) & kMaskV;
      v[i] = fmaf(sv, (float)code, zv);
    }
  });
}

__device__ void simt_resid_unit(State& st, const float (*qs)[kHeadDim], int gq, const __half* ring_k,
                                const __half* ring_v, int p0, int n_tok, int ring) {
  const int lane = threadIdx.x & 31;
  float sc[kMaxGq];
#pragma unroll
  for (int g = 0; g < kMaxGq; ++g) sc[g] = 0.0f;
  if (lane < n_tok) {
    const uint4* row =
        reinterpret_cast<const uint4*>(ring_k + (long long)((p0 + lane) % ring) * kHeadDim);
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
    const uint2 u =
        reinterpret_cast<const uint2*>(ring_v + (long long)((p0 + t) % ring) * kHeadDim)[lane];
    const float2 a = __half22float2(*reinterpret_cast<const __half2*>(&u.x));
    const float2 b = __half22float2(*reinterpret_cast<const __half2*>(&u.y));
    v[0] = a.x;
    v[1] = a.y;
    v[2] = b.x;
    v[3] = b.y;
  });
}

// ---------------------------------------------------------------------------
// Tensor-core path for packed blocks (query groups of up to 4 heads).
// Lane = 4 * gid + tig (mma fragment coordinates).
// ---------------------------------------------------------------------------

// Codes of four rows j = 0..3 of a lane (tokens 4*gid + j for keys, channels
// 4*gid + j of a 32-channel group for values) from two packed words a, b (two
// channels for keys, two tokens for values): v[j] = (f_j code_a, f_j code_b)
// as fp16, exact.  inv(j) = 1 / f_j.
template <int B>
struct Codes;

template <>
struct Codes<1> {
  __device__ static constexpr float inv(int j) {
    return j == 0 ? 16384.0f : j == 1 ? 8192.0f : j == 2 ? 2048.0f : 128.0f;
  }
  __device__ static int word(int gid) { return 0; }
  __device__ static void get(uint32_t a, uint32_t b, uint32_t sel, int sh, uint32_t (&v)[4]) {
    const uint32_t y = __byte_perm(a, b, sel) << sh;  // nibble -> bits 10..13 of each half
    v[0] = y & 0x04000400u;  // exponent bit 0: 2^-14
    v[1] = y & 0x08000800u;  // exponent bit 1: 2^-13
    v[2] = y & 0x10001000u;  // exponent bit 2: 2^-11
    v[3] = y & 0x20002000u;  // exponent bit 3: 2^-7
  }
};
template <>
struct Codes<2> {
  __device__ static constexpr float inv(int j) {
    return j == 0 ? 1.0f : j == 1 ? 0.25f : j == 2 ? 0.0625f : 0.015625f;
  }
  __device__ static int word(int gid) { return gid >> 2; }
  __device__ static void get(uint32_t a, uint32_t b, uint32_t sel, int, uint32_t (&v)[4]) {
    const uint32_t x = __byte_perm(a, b, sel);  // the lane's byte -> bits 0..7 of each half
#pragma unroll
    for (int j = 0; j < 4; ++j) v[j] = hsub1024((x & (0x00030003u << (2 * j))) | 0x64006400u);
  }
};
template <>
struct Codes<4> {
  __device__ static constexpr float inv(int j) { return (j & 1) ? 0.0625f : 1.0f; }
  __device__ static int word(int gid) { return gid >> 1; }
  __device__ static void get(uint32_t a, uint32_t b, uint32_t sel, int, uint32_t (&v)[4]) {
    const uint32_t x = __byte_perm(a, b, sel);  // the lane's 16 bits -> each half
    const uint32_t y = x >> 8;
    v[0] = hsub1024((x & 0x000F000Fu) | 0x64006400u);
    v[1] = hsub1024((x & 0x00F000F0u) | 0x64006400u);
    v[2] = hsub1024((y & 0x000F000Fu) | 0x64006400u);
    v[3] = hsub1024((y & 0x00F000F0u) | 0x64006400u);
  }
};
template <>
struct Codes<8> {
  __device__ static constexpr float inv(int) { return 1.0f; }
  __device__ static int word(int gid) { return gid; }
  __device__ static void get(uint32_t a, uint32_t b, uint32_t, int, uint32_t (&v)[4]) {
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const uint32_t x = __byte_perm(a, b, j | (j << 4) | ((4 + j) << 8) | ((4 + j) << 12));
      v[j] = hsub1024((x & 0x00FF00FFu) | 0x64006400u);
    }
  }
};

template <int B>
__device__ __forceinline__ uint32_t code_selector(int gid) {
  int k;
  if (B == 1) k = gid >> 1;
  else if (B == 2) k = gid & 3;
  else if (B == 4) {
    const int kk = gid & 1;
    return (2 * kk) | ((2 * kk + 1) << 4) | ((4 + 2 * kk) << 8) | ((5 + 2 * kk) << 12);
  } else k = 0;
  return k | (k << 4) | ((4 + k) << 8) | ((4 + k) << 12);
}

struct Lane {
  int gid, tig;
  uint32_t sel_k, sel_v;   // byte-permute selectors for key / value words
  int sh;                   // 1-bit codes: nibble shift to the exponent bits
  int wk, wv;               // word of a group that holds the lane's 4 codes
  uint32_t lo_cols;         // all ones for lanes holding B columns 4..7
  uint32_t row0, row1, rows4;  // all ones for A rows 0 / 1 / 0..3
  float p_lo;               // 1 for lanes holding score columns 4..7
};

struct TcState {
  float acc[8][4];  // o^T[channel][head, part] per value m-tile
  float zv[4];      // sum_t p z per (group, head, part)
  float m[2], l[2]; // heads 2*(tig&1) + {0, 1}
};

// Online softmax over NB 32-token blocks (per block 4 token rows x 2 heads
// per lane; lanes tig and tig^2 hold the same scores), then the
// probabilities as fp16 high / low parts (columns 0..3 / 4..7) moved to the
// B-operand layout of the value MMAs with movmatrix.
template <int NB>
__device__ __forceinline__ void tc_softmax(float (&sc)[NB][4][2], TcState& st, const Lane& ln,
                                           uint32_t (&pt)[NB][2][2]) {
  float mx[2];
#pragma unroll
  for (int hh = 0; hh < 2; ++hh) {
    float x = -INFINITY;
#pragma unroll
    for (int bi = 0; bi < NB; ++bi)
      x = fmaxf(x, fmaxf(fmaxf(sc[bi][0][hh], sc[bi][1][hh]), fmaxf(sc[bi][2][hh], sc[bi][3][hh])));
    x = fmaxf(x, __shfl_xor_sync(0xffffffffu, x, 4));
    x = fmaxf(x, __shfl_xor_sync(0xffffffffu, x, 8));
    x = fmaxf(x, __shfl_xor_sync(0xffffffffu, x, 16));
    mx[hh] = x;
  }
  const bool grow = mx[0] > st.m[0] || mx[1] > st.m[1];
  if (__any_sync(0xffffffffu, grow)) {
    float corr[2];
#pragma unroll
    for (int hh = 0; hh < 2; ++hh) {
      const float mn = fmaxf(st.m[hh], mx[hh]);
      corr[hh] = fast_exp2(st.m[hh] - mn);
      st.m[hh] = mn;
      st.l[hh] *= corr[hh];
    }
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      st.acc[i][0] *= corr[0];
      st.acc[i][1] *= corr[1];
      st.acc[i][2] *= corr[0];
      st.acc[i][3] *= corr[1];
    }
    st.zv[0] *= corr[0];
    st.zv[1] *= corr[1];
    st.zv[2] *= corr[0];
    st.zv[3] *= corr[1];
  }
#pragma unroll
  for (int bi = 0; bi < NB; ++bi)
#pragma unroll
    for (int mt = 0; mt < 2; ++mt)
#pragma unroll
      for (int rh = 0; rh < 2; ++rh) {
        const int j = 2 * mt + rh;
        const float p0 = fast_exp2(sc[bi][j][0] - st.m[0]);
        const float p1 = fast_exp2(sc[bi][j][1] - st.m[1]);
        st.l[0] += p0;
        st.l[1] += p1;
        const float2 hf = __half22float2(__floats2half2_rn(p0, p1));
        const __half2 r = __floats2half2_rn(fmaf(-ln.p_lo, hf.x, p0), fmaf(-ln.p_lo, hf.y, p1));
        pt[bi][mt][rh] = movmatrix_t(h2u(r));
      }
}

// NB packed 32-token blocks (pages in shared memory) for one warp: scores of
// all blocks, one softmax update, then the value MMAs.
template <int BK, int BV, int NB>
__device__ __forceinline__ void tc_unit(const char* const (&pg)[NB], const uint32_t (&qb)[16],
                                        const Lane& ln, float scale_log2, TcState& st) {
  const int gid = ln.gid, tig = ln.tig;

  // ---- keys: S[t][h] ----
  // K slots of k-step ks: lane tig's slots (2tig, 2tig+1) and (2tig+8, 2tig+9)
  // hold channels 16ks + 4tig + (0, 1) and (2, 3), so its four channels are
  // contiguous (one 16-byte load of codes and one of scale/zero).
  float dk[NB][2][4] = {};
  float dz[4] = {};  // zero-point term: row bi of the MMA = block bi
#pragma unroll
  for (int ks = 0; ks < 8; ++ks) {
    const int c = 16 * ks + 4 * tig;
    uint32_t azk[NB][2];
#pragma unroll
    for (int bi = 0; bi < NB; ++bi) {
      const char* kc = pg[bi];
      const char* kmeta = pg[bi] + page_off_kmeta(BK);
      uint32_t w[4];
      if (BK == 1) {
        const uint4 w4 = *reinterpret_cast<const uint4*>(kc + 4 * c);
        w[0] = w4.x;
        w[1] = w4.y;
        w[2] = w4.z;
        w[3] = w4.w;
      } else {
#pragma unroll
        for (int i = 0; i < 4; ++i)
          w[i] = *reinterpret_cast<const uint32_t*>(kc + 4 * ((c + i) * BK + ln.wk));
      }
      // scales of channels c..c+3, then their zeros (two fp16 per word)
      const uint2 sw = *reinterpret_cast<const uint2*>(kmeta + 2 * c);
      const uint2 zw = *reinterpret_cast<const uint2*>(kmeta + 2 * (kHeadDim + c));
      uint32_t a0[4], a1[4], b[2];
#pragma unroll
      for (int half = 0; half < 2; ++half) {
        uint32_t v[4];
        Codes<BK>::get(w[2 * half], w[2 * half + 1], ln.sel_k, ln.sh, v);
        a0[2 * half] = v[0];
        a0[2 * half + 1] = v[1];
        a1[2 * half] = v[2];
        a1[2 * half + 1] = v[3];
        const uint32_t s2 = half ? sw.y : sw.x;
        // q*s as fp16 high part (columns 0..3) or its exact residual (4..7)
        const __half2 hi = __hmul2(u2h(qb[2 * ks + half]), u2h(s2));
        const uint32_t c_in = (h2u(hi) ^ 0x80008000u) & ln.lo_cols;
        b[half] = h2u(__hfma2(u2h(qb[2 * ks + half]), u2h(s2), u2h(c_in)));
        azk[bi][half] = half ? zw.y : zw.x;
      }
      mma16816(dk[bi][0], a0[0], a0[1], a0[2], a0[3], b[0], b[1]);
      mma16816(dk[bi][1], a1[0], a1[1], a1[2], a1[3], b[0], b[1]);
    }
    uint32_t az[2];
#pragma unroll
    for (int half = 0; half < 2; ++half)
      az[half] = NB == 2 ? (azk[0][half] & ln.row0) | (azk[NB - 1][half] & ln.row1)
                         : azk[0][half] & ln.row0;
    mma16816(dz, az[0], 0u, az[1], 0u, qb[2 * ks], qb[2 * ks + 1]);
  }
  // Scores in the log2 domain.  Lanes tig and tig^2 hold the two parts.
  float sc[NB][4][2];
#pragma unroll
  for (int bi = 0; bi < NB; ++bi) {
    const float z0 = __shfl_sync(0xffffffffu, dz[0], 4 * bi + tig) * scale_log2;
    const float z1 = __shfl_sync(0xffffffffu, dz[1], 4 * bi + tig) * scale_log2;
#pragma unroll
    for (int mt = 0; mt < 2; ++mt)
#pragma unroll
      for (int rh = 0; rh < 2; ++rh)
#pragma unroll
        for (int hh = 0; hh < 2; ++hh) {
          const int j = 2 * mt + rh;
          const float d = dk[bi][mt][2 * rh + hh];
          const float full = d + __shfl_xor_sync(0xffffffffu, d, 2);
          sc[bi][j][hh] = fmaf(full, Codes<BK>::inv(j) * scale_log2, hh ? z1 : z0);
        }
  }

  uint32_t pt[NB][2][2];
  tc_softmax<NB>(sc, st, ln, pt);

  // ---- values: o^T[c][h] ----
  // Group-major value pages: group g's (scale, zero) and 1-bit code words of
  // the lane's tokens 8tig .. 8tig+7 are two 16-byte loads each.
#pragma unroll
  for (int bi = 0; bi < NB; ++bi) {
    const char* vc = pg[bi] + page_off_vcodes(BK);
    const char* vmeta = pg[bi] + page_off_vmeta(BK, BV);
    // zeros of group gid & 3 (zero-point MMA rows) for the lane's 8 tokens,
    // two fp16 per word: token 8tig + i is half (i & 1) of word i / 2
    const uint4 z8 = *reinterpret_cast<const uint4*>(vmeta + 2 * (kHeadDim + 32 * (gid & 3) + 8 * tig));
    const uint32_t zw[4] = {z8.x, z8.y, z8.z, z8.w};
#pragma unroll
    for (int ks = 0; ks < 2; ++ks) {
      uint32_t azv[2];
#pragma unroll
      for (int dl = 0; dl < 2; ++dl)  // tokens 8tig + (2ks + dl) and + 4
        azv[dl] = __byte_perm(zw[ks], zw[ks + 2], dl ? 0x7632 : 0x5410) & ln.rows4;
      mma16816(st.zv, azv[0], 0u, azv[1], 0u, pt[bi][ks][0], pt[bi][ks][1]);
    }
#pragma unroll
    for (int g = 0; g < 4; ++g) {
      const uint4 s8 = *reinterpret_cast<const uint4*>(vmeta + 2 * (32 * g + 8 * tig));
      const uint32_t mw[4] = {s8.x, s8.y, s8.z, s8.w};  // scales of tokens 8tig .. 8tig+7
      uint32_t cw[8];
      if (BV == 1) {
        const uint4 cl = *reinterpret_cast<const uint4*>(vc + 4 * (32 * g + 8 * tig));
        const uint4 chh = *reinterpret_cast<const uint4*>(vc + 4 * (32 * g + 8 * tig + 4));
        cw[0] = cl.x; cw[1] = cl.y; cw[2] = cl.z; cw[3] = cl.w;
        cw[4] = chh.x; cw[5] = chh.y; cw[6] = chh.z; cw[7] = chh.w;
      } else {
#pragma unroll
        for (int i = 0; i < 8; ++i)
          cw[i] = *reinterpret_cast<const uint32_t*>(vc + 4 * ((32 * g + 8 * tig + i) * BV + ln.wv));
      }
#pragma unroll
      for (int ks = 0; ks < 2; ++ks) {
        uint32_t am0[4], am1[4], bv[2];
#pragma unroll
        for (int dl = 0; dl < 2; ++dl) {
          const int ia = 2 * ks + dl, ib = ia + 4;  // tokens 8tig + ia, 8tig + ib
          uint32_t v[4];
          Codes<BV>::get(cw[ia], cw[ib], ln.sel_v, ln.sh, v);
          am0[2 * dl] = v[0];
          am0[2 * dl + 1] = v[1];
          am1[2 * dl] = v[2];
          am1[2 * dl + 1] = v[3];
          const uint32_t s2 = __byte_perm(mw[ia >> 1], mw[ib >> 1], (ia & 1) ? 0x7632 : 0x5410);
          bv[dl] = h2u(__hmul2(u2h(pt[bi][ks][dl]), u2h(s2)));
        }
        mma16816(st.acc[2 * g], am0[0], am0[1], am0[2], am0[3], bv[0], bv[1]);
        mma16816(st.acc[2 * g + 1], am1[0], am1[1], am1[2], am1[3], bv[0], bv[1]);
      }
    }
  }
}

template <int BK, int BV>
__device__ __forceinline__ Lane make_lane(int lane) {
  Lane ln;
  ln.gid = lane >> 2;
  ln.tig = lane & 3;
  ln.sel_k = code_selector<BK>(ln.gid);
  ln.sel_v = code_selector<BV>(ln.gid);
  ln.sh = 10 - 4 * (ln.gid & 1);
  ln.wk = Codes<BK>::word(ln.gid);
  ln.wv = Codes<BV>::word(ln.gid);
  ln.lo_cols = ln.gid >= 4 ? 0xffffffffu : 0u;
  ln.row0 = ln.gid == 0 ? 0xffffffffu : 0u;
  ln.row1 = ln.gid == 1 ? 0xffffffffu : 0u;
  ln.rows4 = ln.gid < 4 ? 0xffffffffu : 0u;
  ln.p_lo = ln.tig >= 2 ? 1.0f : 0.0f;
  return ln;
}

// q of head gid & 3 in the B layout (exact fp16), zero beyond the group.
// kPermuted: the packed path's K-slot order (four contiguous channels per
// lane); otherwise slot k of a k-step is channel 16 ks + k.
template <bool kPermuted>
__device__ __forceinline__ void load_qb(uint32_t (&qb)[16], const __half* qh, int gq,
                                        const Lane& ln) {
  const int head = ln.gid & 3;
#pragma unroll
  for (int ks = 0; ks < 8; ++ks)
#pragma unroll
    for (int half = 0; half < 2; ++half) {
      const int c = kPermuted ? 16 * ks + 4 * ln.tig + 2 * half : 16 * ks + 2 * ln.tig + 8 * half;
      qb[2 * ks + half] =
          head < gq ? *reinterpret_cast<const uint32_t*>(qh + head * kHeadDim + c) : 0u;
    }
}

__device__ __forceinline__ void init_state(TcState& st) {
#pragma unroll
  for (int i = 0; i < 8; ++i)
#pragma unroll
    for (int r = 0; r < 4; ++r) st.acc[i][r] = 0.0f;
#pragma unroll
  for (int r = 0; r < 4; ++r) st.zv[r] = 0.0f;
  st.m[0] = st.m[1] = -INFINITY;
  st.l[0] = st.l[1] = 0.0f;
}

// A warp's running state to the merge area: row maximum, row sum and the
// unnormalised output row of heads 0..3.  kPacked: channel rows follow the
// packed layout (nibble of a group, power-of-two factors, zero-point term);
// otherwise channel = 16 * m-tile + row.
template <bool kPacked, int BV>
__device__ __forceinline__ void tc_write_state(const TcState& st, MergeArea& ma, int warp, int lane) {
  const int gid = lane >> 2, tig = lane & 3;
  float l0 = st.l[0], l1 = st.l[1];
#pragma unroll
  for (int o = 4; o < 32; o <<= 1) {
    l0 += __shfl_xor_sync(0xffffffffu, l0, o);
    l1 += __shfl_xor_sync(0xffffffffu, l1, o);
  }
  float zsum[2];
  zsum[0] = st.zv[0] + __shfl_xor_sync(0xffffffffu, st.zv[0], 2);
  zsum[1] = st.zv[1] + __shfl_xor_sync(0xffffffffu, st.zv[1], 2);
  if (gid == 0 && tig < 2) {
    ma.wm[warp][2 * tig] = st.m[0];
    ma.wm[warp][2 * tig + 1] = st.m[1];
    ma.wl[warp][2 * tig] = l0;
    ma.wl[warp][2 * tig + 1] = l1;
  }
#pragma unroll
  for (int g = 0; g < 4; ++g) {
    const float zg0 = kPacked ? __shfl_sync(0xffffffffu, zsum[0], 4 * g + tig) : 0.0f;
    const float zg1 = kPacked ? __shfl_sync(0xffffffffu, zsum[1], 4 * g + tig) : 0.0f;
#pragma unroll
    for (int half = 0; half < 2; ++half) {
      const int mtp = 2 * g + half;
#pragma unroll
      for (int rh = 0; rh < 2; ++rh) {
        const int jp = 2 * half + rh;
        const int cch = kPacked ? 32 * g + 4 * gid + jp : 16 * mtp + gid + 8 * rh;
        const float inv = kPacked ? Codes<BV>::inv(jp) : 1.0f;
#pragma unroll
        for (int hh = 0; hh < 2; ++hh) {
          const float a = st.acc[mtp][2 * rh + hh];
          const float full_v = a + __shfl_xor_sync(0xffffffffu, a, 2);
          if (tig < 2) ma.wo[warp][2 * tig + hh][cch] = fmaf(full_v, inv, hh ? zg1 : zg0);
        }
      }
    }
  }
}

// Blocks per consumer warp and stage: two when pages are small enough that
// two stages of them fit in shared memory.
template <int BK, int BV>
struct Unit {
  static constexpr int kBlocks = (kUnitBlocks > 1 && page_bytes_c(BK, BV) <= 6144) ? kUnitBlocks : 1;
};

// Packed split `split` of one (sequence, kv-head) on the tensor cores: the
// packed blocks nb of the sequence are cut into n_split ranges of
// ceil(nb / n_split) blocks.  A page is written once, when its group leaves
// the window, and never changes afterwards, so before waiting for the
// previous kernel (programmatic dependent launch) the producer already
// streams the full stages of the range given by a length read before the
// wait.  If the length after the wait gives another range start (the
// previous kernel flushed a group of this cache) those stages are discarded.
template <int BK, int BV>
__device__ void tc_split(const Dims& d, const char* pages_bh, int split, int n_split,
                         const int* len_b, int n_bufs, unsigned char* smem, const __half* qh,
                         int gq, float scale_log2, unsigned* flag, MergeArea& ma) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int page = page_bytes(BK, BV);
  constexpr int NB = Unit<BK, BV>::kBlocks;
  constexpr int per_stage = kConsumers * NB;  // blocks per stage
  const int stage = per_stage * page;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + (size_t)n_bufs * stage);
  uint64_t* empty = full + n_bufs;
  __shared__ int issued;
  __shared__ int timed_out;
  __shared__ int hint_len;

  if (threadIdx.x == 0) {
    for (int i = 0; i < n_bufs; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], kConsumers);
    }
    issued = 0;
    timed_out = 0;
    hint_len = read_len(len_b);
    fence_mbar_init();
  }
  __syncthreads();

  auto range = [&](int len, int& lo, int& end) {
    const int nb = packed_len(len, d.residual) / kGroup;
    const int per = (nb + n_split - 1) / n_split;
    lo = min(nb, split * per);
    end = min(nb, lo + per);
  };
  int lo_h, end_h;
  range(hint_len, lo_h, end_h);
  const int pre = min((end_h - lo_h) / per_stage, n_bufs);  // full stages streamed early

  TcState st;
  int consumed = 0;
  const bool streamer = warp == kConsumers - 1 && lane == 0;
  auto issue = [&](int s, int first_blk, int nblk) {
    const int slot = s % n_bufs;
    const uint32_t bytes = (uint32_t)(nblk * page);
    mbar_expect_tx(&full[slot], bytes);
    bulk_g2s(smem + (size_t)slot * stage, pages_bh + (long long)first_blk * page, bytes,
             &full[slot]);
    issued = s + 1;
  };
  if (streamer)
    for (int s = 0; s < pre; ++s) issue(s, lo_h + s * per_stage, per_stage);
  pdl_wait();
  int lo, end;
  range(read_len(len_b), lo, end);
  const int skip = lo == lo_h ? 0 : pre;  // pre-streamed stages of a stale range
  const int nblk = end - lo;
  const int total = skip + (nblk + per_stage - 1) / per_stage;
  auto real_issue = [&](int s) {  // pipeline stage s >= skip
    const int r = s - skip;
    issue(s, lo + r * per_stage, min(per_stage, nblk - r * per_stage));
  };
  if (streamer)
    for (int s = pre; s < min(total, n_bufs); ++s) real_issue(s);

  const Lane ln = make_lane<BK, BV>(lane);
  uint32_t qb[16];
  load_qb<true>(qb, qh, gq, ln);
  init_state(st);
  for (int s = 0; s < total; ++s) {
    const int slot = s % n_bufs;
    if (!mbar_wait(&full[slot], (s / n_bufs) & 1)) {
      if (lane == 0) atomicOr(flag, 2u);
      timed_out = 1;
      break;
    }
    consumed = s + 1;
    if (s >= skip) {
      const int r = s - skip;
      const int blk = r * per_stage + warp * NB;  // first of the warp's blocks
      const char* base = reinterpret_cast<const char*>(smem) + (size_t)slot * stage;
      if (blk + NB <= nblk) {
        const char* pg[NB];
#pragma unroll
        for (int i = 0; i < NB; ++i) pg[i] = base + (warp * NB + i) * page;
        tc_unit<BK, BV, NB>(pg, qb, ln, scale_log2, st);
      } else if (NB > 1 && blk < nblk) {
        const char* pg[1] = {base + warp * NB * page};
        tc_unit<BK, BV, 1>(pg, qb, ln, scale_log2, st);
      }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&empty[slot]);
    // The streaming lane refills this slot once every warp has released it.
    if (streamer && s + n_bufs < total) {
      if (!mbar_wait(&empty[slot], (s / n_bufs) & 1)) {
        atomicOr(flag, 2u);
        timed_out = 1;
      } else {
        real_issue(s + n_bufs);
      }
    }
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    // Copies issued past what the consumers took (the length shrank, or a
    // wait gave up) land before the stage area is reused (bounded waits).
    for (int s = max(consumed, issued - n_bufs); s < issued; ++s)
      mbar_wait(&full[s % n_bufs], (s / n_bufs) & 1);
  }
  __syncthreads();

  tc_write_state<true, BV>(st, ma, warp, lane);
}

// ---------------------------------------------------------------------------
// Tensor-core path for the fp16 residual window: each consumer warp stages a
// 32-token chunk of K and V rows in shared memory and feeds the MMAs with
// ldmatrix (keys as A with tokens as rows; values transposed, channels as
// rows).  Rows past the window are zero and their scores -inf.
// ---------------------------------------------------------------------------

constexpr int kResRow = kHeadDim + 8;  // halves per staged row (16-byte pad)
constexpr int kResWarpBytes = 2 * kGroup * kResRow * 2;
static_assert(kResWarps * kResWarpBytes <= 96 * 1024, "window staging fits");

__device__ __forceinline__ void ldsm_x4(uint32_t (&r)[4], const void* p) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(smem_addr(p)));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t (&r)[4], const void* p) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(smem_addr(p)));
}

__device__ __forceinline__ void tc_resid_chunk(const __half* ks_s, const __half* vs_s, int n_tok,
                                               const uint32_t (&qb)[16], const Lane& ln,
                                               float scale_log2, TcState& st) {
  const int lane = threadIdx.x & 31;
  const int mi = lane >> 3, r8 = lane & 7;
  float dk[2][4] = {};
#pragma unroll
  for (int ks = 0; ks < 8; ++ks)
#pragma unroll
    for (int mt = 0; mt < 2; ++mt) {
      uint32_t a[4];
      ldsm_x4(a, ks_s + (16 * mt + 8 * (mi & 1) + r8) * kResRow + 16 * ks + 8 * (mi >> 1));
      mma16816(dk[mt], a[0], a[1], a[2], a[3], qb[2 * ks], qb[2 * ks + 1]);
    }
  float sc[4][2];
#pragma unroll
  for (int mt = 0; mt < 2; ++mt)
#pragma unroll
    for (int rh = 0; rh < 2; ++rh) {
      const bool ok = 16 * mt + ln.gid + 8 * rh < n_tok;
#pragma unroll
      for (int hh = 0; hh < 2; ++hh)
        sc[2 * mt + rh][hh] = ok ? dk[mt][2 * rh + hh] * scale_log2 : -INFINITY;
    }
  float sc1[1][4][2];
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    sc1[0][j][0] = sc[j][0];
    sc1[0][j][1] = sc[j][1];
  }
  uint32_t pt[1][2][2];
  tc_softmax<1>(sc1, st, ln, pt);
#pragma unroll
  for (int ks = 0; ks < 2; ++ks)
#pragma unroll
    for (int mtp = 0; mtp < 8; ++mtp) {
      uint32_t a[4];
      ldsm_x4_t(a, vs_s + (16 * ks + 8 * (mi >> 1) + r8) * kResRow + 16 * mtp + 8 * (mi & 1));
      mma16816(st.acc[mtp], a[0], a[1], a[2], a[3], pt[0][ks][0], pt[0][ks][1]);
    }
}

__device__ __forceinline__ void cp_async16(void* dst, const void* src, uint32_t src_bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(smem_addr(dst)), "l"(src),
               "r"(src_bytes)
               : "memory");
}

// Residual split: tokens [Lq, L) of one (sequence, kv-head), fp16, from the
// ring.  Warp w takes 32-token chunks w, w + kResWarps, ...; each chunk's K
// and V rows are copied into shared memory with asynchronous 16-byte copies
// (rows past L are zero-filled) before its MMAs.
template <int BK, int BV>
__device__ void tc_resid_split(const Dims& d, const __half* ring_k, const __half* ring_v, int Lq,
                               int L, unsigned char* smem, const __half* qh, int gq,
                               float scale_log2, MergeArea& ma) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n_res = (L - Lq + kGroup - 1) / kGroup;
  TcState st;
  const Lane ln = make_lane<BK, BV>(lane);
  uint32_t qb[16];
  load_qb<false>(qb, qh, gq, ln);
  init_state(st);
  __half* ks_s = reinterpret_cast<__half*>(smem + (size_t)warp * kResWarpBytes);
  __half* vs_s = ks_s + kGroup * kResRow;
  for (int u = warp; u < n_res; u += kResWarps) {
    const int p0 = Lq + u * kGroup;
    const int n_tok = min(kGroup, L - p0);
#pragma unroll 4
    for (int e = lane; e < kGroup * 16; e += 32) {
      const int row = e >> 4, piece = e & 15;
      const bool ok = row < n_tok;
      const long long off = ok ? (long long)((p0 + row) % d.ring) * kHeadDim : 0;
      cp_async16(ks_s + row * kResRow + piece * 8, ring_k + off + piece * 8, ok ? 16u : 0u);
      cp_async16(vs_s + row * kResRow + piece * 8, ring_v + off + piece * 8, ok ? 16u : 0u);
    }
    asm volatile("cp.async.commit_group;\ncp.async.wait_group 0;" ::: "memory");
    __syncwarp();
    tc_resid_chunk(ks_s, vs_s, n_tok, qb, ln, scale_log2, st);
    __syncwarp();
  }
  __syncthreads();  // staging area free: the merge area overlaps it
  tc_write_state<false, BV>(st, ma, warp, lane);
}

// ---------------------------------------------------------------------------
// The kernel
// ---------------------------------------------------------------------------

template <int BK, int BV, bool kTc>
__global__ void __launch_bounds__(kThreads, kCtasPerSm)
    decode_attn_kernel(Dims d, kvq_cache c, const __half* __restrict__ q, float* __restrict__ out,
                       float scale_log2, int S, int n_bufs, unsigned smem_size, Ws ws) {
  extern __shared__ __align__(128) unsigned char smem[];
  MergeArea& ma = *reinterpret_cast<MergeArea*>(smem);

  const int s = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
  const int gq = d.gq, warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  pdl_launch_dependents();
  const long long bh = (long long)b * d.hkv + h;
  const char* pages = static_cast<const char*>(c.pages) + bh * d.max_blocks * d.page_bytes;
  const __half* ring_k = reinterpret_cast<const __half*>(c.k_resid) + bh * d.ring * kHeadDim;
  const __half* ring_v = reinterpret_cast<const __half*>(c.v_resid) + bh * d.ring * kHeadDim;
  const __half* qh = q + ((long long)b * d.hq + (long long)h * gq) * kHeadDim;
  unsigned* flag = reinterpret_cast<unsigned*>(c.seq_len) + d.batch;

  if (kTc && s < S - 1) {
    tc_split<BK, BV>(d, pages, s, S - 1, c.seq_len + b, n_bufs, smem, qh, gq, scale_log2, flag,
                     ma);
  } else {
    pdl_wait();
  }
  const int L = read_len(c.seq_len + b);
  const int Lq = packed_len(L, d.residual);
  const int nb = Lq / kGroup;
  if (kTc && s < S - 1) {
  } else if (kTc) {
    tc_resid_split<BK, BV>(d, ring_k, ring_v, Lq, L, smem, qh, gq, scale_log2, ma);
  } else {
    // SIMT path: every unit, split evenly (query groups wider than 4).
    const int units = nb + (L - Lq + kGroup - 1) / kGroup;
    const int per = (units + S - 1) / S;
    const int u0 = min(units, s * per), u1 = min(units, u0 + per);
    for (int e = threadIdx.x; e < gq * kHeadDim; e += kThreads)
      ma.qs[e / kHeadDim][e % kHeadDim] = __half2float(qh[e]) * scale_log2;
    __syncthreads();
    if (warp < kConsumers) {
      State st;
#pragma unroll
      for (int g = 0; g < kMaxGq; ++g) {
        st.m[g] = -INFINITY;
        st.l[g] = 0.0f;
#pragma unroll
        for (int i = 0; i < 4; ++i) st.acc[g][i] = 0.0f;
      }
      for (int u = u0 + warp; u < u1; u += kConsumers) {
        if (u < nb) {
          simt_packed_unit<BK, BV>(st, ma.qs, gq, pages + (long long)u * d.page_bytes);
        } else {
          const int p0 = Lq + (u - nb) * kGroup;
          simt_resid_unit(st, ma.qs, gq, ring_k, ring_v, p0, min(kGroup, L - p0), d.ring);
        }
      }
#pragma unroll
      for (int g = 0; g < kMaxGq; ++g) {
        if (g >= gq) break;
        if (lane == 0) {
          ma.wm[warp][g] = st.m[g];
          ma.wl[warp][g] = st.l[g];
        }
#pragma unroll
        for (int i = 0; i < 4; ++i) ma.wo[warp][g][4 * lane + i] = st.acc[g][i];
      }
    }
  }
  __syncthreads();

  // Merge the consumer warps and publish this split's partials.
  const int cidx = threadIdx.x;  // one output channel per thread (threads 0..127)
  if (cidx < kHeadDim) {
    for (int g = 0; g < gq; ++g) {
      float M = -INFINITY;
      for (int w = 0; w < kConsumers; ++w) M = fmaxf(M, ma.wm[w][g]);
      float l = 0.0f, o = 0.0f;
      if (M != -INFINITY) {
        for (int w = 0; w < kConsumers; ++w) {
          const float f = exp2f(ma.wm[w][g] - M);
          l += f * ma.wl[w][g];
          o += f * ma.wo[w][g][cidx];
        }
      }
      const long long row = ((long long)b * d.hq + (long long)h * gq + g) * S + s;
      ws.o[row * kHeadDim + cidx] = o;
      if (cidx == 0) {
        ws.m[row] = M;
        ws.l[row] = l;
      }
    }
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    const unsigned t = atomicAdd(&ws.tk[bh], 1u);
    ma.last = (t == (unsigned)S - 1);
  }
  __syncthreads();
  const bool is_last = ma.last;
  __syncthreads();  // the merge below reuses the shared memory that holds `last`
  if (!is_last) return;
  __threadfence();
  // Last CTA: merge the S partials of every query head.  The partial rows of
  // this (sequence, kv-head) are one contiguous range: one bulk copy brings
  // them into shared memory when they fit, while the maxima and sums are
  // loaded; each thread then reduces one (head, 4-channel) slice.
  const long long head0 = (long long)b * d.hq + (long long)h * gq;
  const size_t o_bytes = (size_t)gq * S * kHeadDim * sizeof(float);
  const bool staged = o_bytes + (size_t)(2 * gq * S + gq) * sizeof(float) + 16 <= smem_size;
  float* osm = reinterpret_cast<float*>(smem);
  float* mv = staged ? osm + (size_t)gq * S * kHeadDim : osm;  // [gq][S] maxima, then weights
  float* lv = mv + gq * S;                                      // [gq][S] sums
  float* lsum = lv + gq * S;                                    // [gq]
  uint64_t* mbar = reinterpret_cast<uint64_t*>(smem + smem_size - 16);
  if (staged && threadIdx.x == 0) {
    mbar_init(mbar, 1);
    fence_mbar_init();
    asm volatile("fence.proxy.async.global;" ::: "memory");
    mbar_expect_tx(mbar, (uint32_t)o_bytes);
    bulk_g2s(osm, ws.o + head0 * S * kHeadDim, (uint32_t)o_bytes, mbar);
  }
  for (int i = threadIdx.x; i < gq * S; i += kThreads) {
    mv[i] = __ldcg(ws.m + head0 * S + i);
    lv[i] = __ldcg(ws.l + head0 * S + i);
  }
  __syncthreads();
  for (int g = warp; g < gq; g += kThreads / 32) {
    float M = -INFINITY;
    for (int k = lane; k < S; k += 32) M = fmaxf(M, mv[g * S + k]);
    M = warp_max(M);
    float Ls = 0.0f;
    for (int k = lane; k < S; k += 32) {
      const float m = mv[g * S + k];
      const float w = (m == -INFINITY) ? 0.0f : exp2f(m - M);
      Ls += w * lv[g * S + k];
      mv[g * S + k] = w;
    }
    Ls = warp_sum(Ls);
    if (lane == 0) lsum[g] = Ls;
  }
  bool ok = true;
  if (staged) ok = mbar_wait(mbar, 0);
  __syncthreads();
  for (int i = threadIdx.x; i < gq * (kHeadDim / 4); i += kThreads) {
    const int g = i / (kHeadDim / 4), c4 = i % (kHeadDim / 4);
    const float4* src = staged && ok
                            ? reinterpret_cast<const float4*>(osm + (size_t)g * S * kHeadDim) + c4
                            : reinterpret_cast<const float4*>(ws.o + (head0 + g) * S * kHeadDim) + c4;
    float4 acc = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
#pragma unroll 8
    for (int k = 0; k < S; ++k) {
      const float w = mv[g * S + k];
      const float4 o = staged && ok ? src[(long long)k * (kHeadDim / 4)]
                                    : __ldcg(src + (long long)k * (kHeadDim / 4));
      acc.x = fmaf(w, o.x, acc.x);
      acc.y = fmaf(w, o.y, acc.y);
      acc.z = fmaf(w, o.z, acc.z);
      acc.w = fmaf(w, o.w, acc.w);
    }
    const float Ls = lsum[g];
    const float inv = Ls > 0.0f ? 1.0f / Ls : 0.0f;
    reinterpret_cast<float4*>(out + (head0 + g) * kHeadDim)[c4] =
        make_float4(acc.x * inv, acc.y * inv, acc.z * inv, acc.w * inv);
  }
  if (threadIdx.x == 0) ws.tk[bh] = 0u;
}

int blocks_per_warp(const Dims& d) {
  return (kUnitBlocks > 1 && d.page_bytes <= 6144) ? kUnitBlocks : 1;
}

int stage_buffers(const Dims& d) {
  const int stage = kConsumers * blocks_per_warp(d) * (int)d.page_bytes;
  int n = kStageBudget / stage;
  return n < 2 ? 2 : (n > 8 ? 8 : n);
}

size_t smem_bytes(const Dims& d, bool tc) {
  size_t need = sizeof(MergeArea);
  const size_t merge = (size_t)(2 * kMaxGq * kMaxSplits + kMaxGq) * sizeof(float);
  if (need < merge) need = merge;
  if (tc && need < (size_t)kResWarps * kResWarpBytes) need = (size_t)kResWarps * kResWarpBytes;
  if (tc) {
    const size_t stages = (size_t)stage_buffers(d) * kConsumers * blocks_per_warp(d) * d.page_bytes +
                          16 * stage_buffers(d);
    if (stages > need) need = stages;
  }
  return (need + 16 + 127) / 128 * 128;  // + the final merge's mbarrier
}

template <int BK, int BV, bool kTc>
cudaError_t prepare(const Dims& d) {
  return cudaFuncSetAttribute(decode_attn_kernel<BK, BV, kTc>,
                              cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem_bytes(d, kTc));
}

// Kernel instance for (bits_k, bits_v, query-group width): Op::run<BK, BV, kTc>.
template <typename Op>
cudaError_t dispatch(const Dims& d, const Op& op);

template <int BK, int BV, typename Op>
cudaError_t dispatch_mode(const Dims& d, const Op& op) {
  return d.gq <= 4 ? op.template run<BK, BV, true>() : op.template run<BK, BV, false>();
}
template <int BK, typename Op>
cudaError_t dispatch_bv(const Dims& d, const Op& op) {
  switch (d.bits_v) {
    case 1: return dispatch_mode<BK, 1>(d, op);
    case 2: return dispatch_mode<BK, 2>(d, op);
    case 4: return dispatch_mode<BK, 4>(d, op);
    default: return dispatch_mode<BK, 8>(d, op);
  }
}
template <typename Op>
cudaError_t dispatch(const Dims& d, const Op& op) {
  switch (d.bits_k) {
    case 1: return dispatch_bv<1>(d, op);
    case 2: return dispatch_bv<2>(d, op);
    case 4: return dispatch_bv<4>(d, op);
    default: return dispatch_bv<8>(d, op);
  }
}

struct LaunchOp {
  const Dims& d;
  const kvq_cache& c;
  const __half* q;
  float* out;
  float sl2;
  int S;
  const Ws& ws;
  cudaStream_t st;
  template <int BK, int BV, bool kTc>
  cudaError_t run() const {
    cudaError_t e = prepare<BK, BV, kTc>(d);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(S, d.hkv, d.batch);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = smem_bytes(d, kTc);
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    e = cudaLaunchKernelEx(&cfg, decode_attn_kernel<BK, BV, kTc>, d, c, q, out, sl2, S,
                           stage_buffers(d), (unsigned)smem_bytes(d, kTc), ws);
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
  }
};

struct OccupancyOp {
  const Dims& d;
  int* blocks;
  template <int BK, int BV, bool kTc>
  cudaError_t run() const {
    cudaError_t e = prepare<BK, BV, kTc>(d);
    if (e != cudaSuccess) return e;
    return cudaOccupancyMaxActiveBlocksPerMultiprocessor(blocks, decode_attn_kernel<BK, BV, kTc>,
                                                         kThreads, smem_bytes(d, kTc));
  }
};

}  // namespace

// n_splits counts the packed-block splits; the kernel adds one split for the
// residual window.
size_t attn_workspace_bytes(const Dims& d, int n_splits) {
  const int S = n_splits + 1;
  const size_t nml = (size_t)d.batch * d.hq * S;
  return align256(nml * 4) * 2 + align256(nml * kHeadDim * 4) +
         align256((size_t)d.batch * d.hkv * 4);
}

cudaError_t launch_decode_attn(const Dims& d, const kvq_cache& c, const __half* q, float* out,
                               float scale_log2, int n_splits, void* workspace, cudaStream_t st) {
  const int S = n_splits + 1;
  const Ws ws = carve(workspace, d.batch, d.hq, d.hkv, S);
  return dispatch(d, LaunchOp{d, c, q, out, scale_log2, S, ws, st});
}

// Packed splits per (sequence, kv-head) so that all CTAs (packed splits plus
// the window split) are resident at once; at least ~16 blocks per split.
int attn_default_splits(const Dims& d, int sm_count) {
  int occ = 0;
  if (dispatch(d, OccupancyOp{d, &occ}) != cudaSuccess || occ < 1) {
    cudaGetLastError();
    occ = 1;
  }
  const int bh = d.batch * d.hkv;
  int n = occ * sm_count / bh - 1;
  const int cap = (d.max_blocks + 15) / 16;
  if (n > cap) n = cap;
  if (n > kMaxSplits - 1) n = kMaxSplits - 1;
  if (n < 1) n = 1;
  return n;
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
                                      float* out, float scale_log2, int n_splits,
                                      cudaStream_t st) {
  void* ws = nullptr;
  cudaError_t e = static_scratch(&ws);
  if (e != cudaSuccess) return e;
  // The array keeps the previous call's contents: the tickets must start at
  // zero, the partials are always written before they are read.
  const Ws w = carve(ws, d.batch, d.hq, d.hkv, n_splits + 1);
  e = cudaMemsetAsync(w.tk, 0, (size_t)d.batch * d.hkv * sizeof(unsigned), st);
  if (e != cudaSuccess) return e;
  return launch_decode_attn(d, c, q, out, scale_log2, n_splits, ws, st);
}

}  // namespace kvq
