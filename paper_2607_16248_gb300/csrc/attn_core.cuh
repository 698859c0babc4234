// Shared device code of the two decode-attention kernels (attn.cu, the flat
// plan; attn_split.cu, the split plan): constants, the per-block tensor-core
// arithmetic over packed pages, the fp16 window's MMAs, the page ring and its
// copies.  Included inside each kernel file's anonymous namespace.
#pragma once

#ifndef KVQ_ATTN_WARPS
#define KVQ_ATTN_WARPS 16
#endif
constexpr int kWarps = KVQ_ATTN_WARPS;            // warps per CTA
constexpr int kThreads = 32 * kWarps;
constexpr int kCtasPerSm = kWarps <= 8 ? 2 : 1;   // resident CTAs per SM
constexpr int kRingBudget = (kCtasPerSm == 2 ? 96 : 192) * 1024;  // staged page bytes per CTA
constexpr int kHeads = kMaxGq;  // query heads per CTA (the wide layout's head columns)
constexpr long long kWaitCycles = 4000000000LL;  // bounded mbarrier waits (~2 s)
constexpr int kZeroBytes = 512;                   // all-zero metadata rows
constexpr int kOnesWord0 = 64;                    // ... but for fp16 ones at bytes 256..319

// A warp's final state (row maximum, row sum, unnormalised output row per
// query head of the kv-head), written at the start of the warp's own
// ring as soon as it is done.
struct WarpState {
  float m[kHeads];
  float l[kHeads];
  float o[kHeads][kHeadDim];
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
__device__ __forceinline__ bool mbar_wait_for(uint64_t* bar, uint32_t parity, long long limit) {
  if (mbar_try_wait(bar, parity)) return true;
  const long long t0 = clock64();
  while (!mbar_try_wait(bar, parity))
    if (clock64() - t0 > limit) return false;
  return true;
}
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity) {
  return mbar_wait_for(bar, parity, kWaitCycles);
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
  asm(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
      "{%8,%9}, {%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}
__device__ __forceinline__ uint32_t movmatrix_t(uint32_t a) {
  uint32_t d;
  asm("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;" : "=r"(d) : "r"(a));
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
// Tensor-core path for packed blocks (query groups of up to 4 heads).
// Lane = 4 * gid + tig (mma fragment coordinates).
// ---------------------------------------------------------------------------

// Codes of four rows j = 0..3 of a lane (tokens 4*gid + j for keys, channels
// 4*gid + j of a 32-channel group for values) from two packed words a, b (two
// channels for keys, two tokens for values): v[j] = (f_j code_a, f_j code_b)
// as fp16, exact.  inv(j) = 1 / f_j.
template <int B>
struct Codes;

// 1-bit codes are stored in fragment order (key1_bit / val1_bit): the word
// w of a lane rotated left by 4 r holds, at bit 10 + 16 e + j, the code of
// row j and half e of one fragment register, so each register is one AND
// (an fp16 with a single exponent bit set: 2^-14, 2^-13, 2^-11, 2^-7).
template <>
struct Codes<1> {
  __device__ static constexpr float inv(int j) {
    return j == 0 ? 16384.0f : j == 1 ? 8192.0f : j == 2 ? 2048.0f : 128.0f;
  }
  __device__ static int word(int gid) { return 0; }
  __device__ static void rot(uint32_t w, int r, uint32_t (&v)[4]) {
    // r = 1, 2 only read bits that a plain shift keeps; r = 3 wraps around.
    const uint32_t y = r == 0 ? w : r == 1 ? w << 4 : r == 2 ? w << 8 : __funnelshift_l(w, w, 12);
    v[0] = y & 0x04000400u;
    v[1] = y & 0x08000800u;
    v[2] = y & 0x10001000u;
    v[3] = y & 0x20002000u;
  }
};

__device__ __forceinline__ uint32_t comp(const uint4& u, int i) {
  return i == 0 ? u.x : i == 1 ? u.y : i == 2 ? u.z : u.w;
}
template <>
struct Codes<2> {
  __device__ static constexpr float inv(int j) {
    return j == 0 ? 1.0f : j == 1 ? 0.25f : j == 2 ? 0.0625f : 0.015625f;
  }
  __device__ static int word(int gid) { return gid >> 2; }
  __device__ static void get(uint32_t a, uint32_t b, uint32_t sel, uint32_t (&v)[4]) {
    const uint32_t x = __byte_perm(a, b, sel);  // the lane's byte -> bits 0..7 of each half
#pragma unroll
    for (int j = 0; j < 4; ++j) v[j] = hsub1024((x & (0x00030003u << (2 * j))) | 0x64006400u);
  }
};
template <>
struct Codes<4> {
  __device__ static constexpr float inv(int j) { return (j & 1) ? 0.0625f : 1.0f; }
  __device__ static int word(int gid) { return gid >> 1; }
  __device__ static void get(uint32_t a, uint32_t b, uint32_t sel, uint32_t (&v)[4]) {
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
  __device__ static void get(uint32_t a, uint32_t b, uint32_t, uint32_t (&v)[4]) {
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
  int wk, wv;               // word of a group that holds the lane's 4 codes
  uint32_t neg_lo;          // fp16x2 -1 for lanes holding B columns 4..7, else 0
  float p_lo;               // 1 for lanes holding score columns 4..7
};

struct TcState {
  float acc[8][4];  // o^T[channel][head, part] per value m-tile
  float zv[4];      // sum_t p z per (group, head, part)
  float m[2], l[2]; // heads 2*(tig&1) + {0, 1}
};

// Online softmax over NB 32-token blocks (per block 4 token rows x 2 heads
// per lane), then the probabilities moved to the B-operand layout of the
// value MMAs with movmatrix.  The scores arrive as t = score - m_eff (log2
// domain), m_eff being the lane's running maximum (0 before its first
// block), so the common case (no score above the maximum) costs one exp2 per
// score and a vote; only when some score exceeds it (or before the first
// block) is the new maximum found across the warp, the state rescaled and t
// shifted.
//   exact (kCompact false): p as an fp16 high part and its fp16 residual;
//     narrow (up to 4 heads): columns 0..3 / 4..7 hold the high / low parts
//     of heads 0..3 (lanes tig and tig^2 hold the same scores), pt is one
//     operand whose columns carry both parts; wide (5..8 heads): column =
//     head, pt holds the high parts, pl the low parts, each one operand of
//     its own MMA.
//   compact (1-bit values): the weights are p~ = RN16(p), used alike in the
//     row sum and in the value MMAs (so they are a consistent softmax of
//     scores perturbed by at most 2^-11 relative); pt holds p~ (column =
//     head; narrow: columns 4..7 zero), pl is unused.
// kSumL: add the weights to st.l here (window chunks).  Packed blocks leave
// it: their row sums come out of the value zero-point MMA, whose A row 4 is
// all ones (see tc_unit).
template <int NB, bool kWide, bool kCompact, bool kSumL>
__device__ __forceinline__ void tc_softmax(float (&t)[NB][4][2], TcState& st, const Lane& ln,
                                           uint32_t (&pt)[NB][2][2], uint32_t (&pl)[NB][2][2]) {
  float tm[2];
#pragma unroll
  for (int hh = 0; hh < 2; ++hh) {
    float x = -INFINITY;
#pragma unroll
    for (int bi = 0; bi < NB; ++bi)
      x = fmaxf(x, fmaxf(fmaxf(t[bi][0][hh], t[bi][1][hh]), fmaxf(t[bi][2][hh], t[bi][3][hh])));
    tm[hh] = x;
  }
  const bool fresh = st.m[0] == -INFINITY;
  if (__any_sync(0xffffffffu, tm[0] > 0.0f || tm[1] > 0.0f || fresh)) {
    float corr[2], delta[2];
#pragma unroll
    for (int hh = 0; hh < 2; ++hh) {
      float x = tm[hh];
      x = fmaxf(x, __shfl_xor_sync(0xffffffffu, x, 4));
      x = fmaxf(x, __shfl_xor_sync(0xffffffffu, x, 8));
      x = fmaxf(x, __shfl_xor_sync(0xffffffffu, x, 16));
      const float me = st.m[hh] == -INFINITY ? 0.0f : st.m[hh];
      const float mn = fmaxf(st.m[hh], me + x);
      delta[hh] = mn == -INFINITY ? 0.0f : mn - me;
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
#pragma unroll
    for (int bi = 0; bi < NB; ++bi)
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        t[bi][j][0] -= delta[0];
        t[bi][j][1] -= delta[1];
      }
  }
#pragma unroll
  for (int bi = 0; bi < NB; ++bi)
#pragma unroll
    for (int mt = 0; mt < 2; ++mt)
#pragma unroll
      for (int rh = 0; rh < 2; ++rh) {
        const int j = 2 * mt + rh;
        const float p0 = fast_exp2(t[bi][j][0]);
        const float p1 = fast_exp2(t[bi][j][1]);
        const __half2 h = __floats2half2_rn(p0, p1);
        if constexpr (kCompact) {
          if constexpr (kSumL) {
            const float2 hf = __half22float2(h);
            st.l[0] += hf.x;
            st.l[1] += hf.y;
          }
          pt[bi][mt][rh] = movmatrix_t(kWide || ln.tig < 2 ? h2u(h) : 0u);
          continue;
        }
        if constexpr (kSumL) {
          st.l[0] += p0;
          st.l[1] += p1;
        }
        const float2 hf = __half22float2(h);
        if constexpr (kWide) {
          pt[bi][mt][rh] = movmatrix_t(h2u(h));
          pl[bi][mt][rh] = movmatrix_t(h2u(__floats2half2_rn(p0 - hf.x, p1 - hf.y)));
        } else {
          const __half2 r =
              __floats2half2_rn(fmaf(-ln.p_lo, hf.x, p0), fmaf(-ln.p_lo, hf.y, p1));
          pt[bi][mt][rh] = movmatrix_t(h2u(r));
        }
      }
}

// Offset subtracted from a lane's scores before its softmax update: its
// running maximum, or 0 before the first block.
__device__ __forceinline__ float m_offset(float m) { return m == -INFINITY ? 0.0f : m; }

// NB packed 32-token blocks (pages in shared memory) for one warp: scores of
// all blocks, one softmax update, then the value MMAs.  Narrow: one MMA per
// operand pair, B columns = (head, part); wide: B column = head, and the
// high and low parts of B are two MMAs into the same accumulator.
template <int BK, int BV, int NB, bool kWide>
__device__ __forceinline__ void tc_unit(const char* const (&pg)[NB], const char* zero,
                                        const uint32_t (&qb)[16], const Lane& ln,
                                        float scale_log2, TcState& st) {
  const int gid = ln.gid, tig = ln.tig, lane = 4 * gid + tig;
  // Zero-point MMA rows: row bi (lane group gid = bi) reads block bi's key
  // metadata, the other rows the all-zero area (same 512-byte extent).
  const char* zrow = gid == 0 ? pg[0] + page_off_kmeta(BK)
                     : (NB == 2 && gid == 1) ? pg[NB - 1] + page_off_kmeta(BK) : zero;
  uint4 kw1[NB];
  if constexpr (BK == 1) {
#pragma unroll
    for (int bi = 0; bi < NB; ++bi) kw1[bi] = *reinterpret_cast<const uint4*>(pg[bi] + 16 * lane);
  }

  // ---- keys: S[t][h] ----
  // K slots of k-step ks: lane tig's slots (2tig, 2tig+1) and (2tig+8, 2tig+9)
  // hold channels 16ks + 4tig + (0, 1) and (2, 3), so its four channels are
  // contiguous (one 16-byte load of codes and one of scale/zero).
  // 1-bit codes in the wide layout scale the A operand instead of B: the
  // code of row j is 0 or 2^e_j (e_j = -14, -13, -11, -7), so A = code * s is
  // one fp16 multiply per register and exact unless it falls below the
  // normal range (s < 2^(-14 - e_j), e.g. s < 1 on row 0), where it is
  // rounded to a subnormal: at most 2^-25 * 2^-e_j <= 2^-11 in key units,
  // far below the quantization step s / 2.  B = q then needs no high/low
  // split, which halves the key MMAs (the tensor pipe bounds this layout).
  constexpr bool kScaledA = BK == 1 && kWide;
  float dk[NB][2][4] = {};
  float dz[4] = {};  // zero-point term: row bi of the MMA = block bi
#pragma unroll
  for (int ks = 0; ks < 8; ++ks) {
    const int c = 16 * ks + 4 * tig;
#pragma unroll
    for (int bi = 0; bi < NB; ++bi) {
      const char* kc = pg[bi];
      const char* kmeta = pg[bi] + page_off_kmeta(BK);
      // scales of channels c..c+3 (two fp16 per word)
      const uint2 sw = *reinterpret_cast<const uint2*>(kmeta + 2 * c);
      uint32_t a0[4], a1[4], b[2], bl[2];
#pragma unroll
      for (int half = 0; half < 2; ++half) {
        uint32_t v[4];
        if constexpr (BK == 1) {
          Codes<1>::rot(comp(kw1[bi], ks >> 1), 2 * (ks & 1) + half, v);
        } else {
          const uint32_t wa = *reinterpret_cast<const uint32_t*>(kc + 4 * ((c + 2 * half) * BK + ln.wk));
          const uint32_t wb = *reinterpret_cast<const uint32_t*>(kc + 4 * ((c + 2 * half + 1) * BK + ln.wk));
          Codes<BK>::get(wa, wb, ln.sel_k, v);
        }
        a0[2 * half] = v[0];
        a0[2 * half + 1] = v[1];
        a1[2 * half] = v[2];
        a1[2 * half + 1] = v[3];
        const uint32_t s2 = half ? sw.y : sw.x;
        if constexpr (kScaledA) {
          // 1-bit codes, wide layout: A = code * s (a power of two times the
          // scale, or 0) and B = q, one MMA per tile
#pragma unroll
          for (int i = 0; i < 2; ++i) {
            a0[2 * half + i] = h2u(__hmul2(u2h(a0[2 * half + i]), u2h(s2)));
            a1[2 * half + i] = h2u(__hmul2(u2h(a1[2 * half + i]), u2h(s2)));
          }
          b[half] = qb[2 * ks + half];
        } else if constexpr (kWide) {
          // q*s as its fp16 high part and exact residual, two operands
          const __half2 hi = __hmul2(u2h(qb[2 * ks + half]), u2h(s2));
          b[half] = h2u(hi);
          bl[half] = h2u(__hfma2(u2h(qb[2 * ks + half]), u2h(s2), __hneg2(hi)));
        } else {
          // q*s as fp16 high part (columns 0..3) or its exact residual (4..7):
          // qn = -q on the lanes of columns 4..7 and 0 elsewhere (the same
          // for every block), RN16(qn s) = -RN16(q s) there
          const __half2 qn = __hmul2(u2h(qb[2 * ks + half]), u2h(ln.neg_lo));
          b[half] = h2u(__hfma2(u2h(qb[2 * ks + half]), u2h(s2), __hmul2(qn, u2h(s2))));
        }
      }
      mma16816(dk[bi][0], a0[0], a0[1], a0[2], a0[3], b[0], b[1]);
      mma16816(dk[bi][1], a1[0], a1[1], a1[2], a1[3], b[0], b[1]);
      if constexpr (kWide && !kScaledA) {
        mma16816(dk[bi][0], a0[0], a0[1], a0[2], a0[3], bl[0], bl[1]);
        mma16816(dk[bi][1], a1[0], a1[1], a1[2], a1[3], bl[0], bl[1]);
      }
    }
    const uint2 zw = *reinterpret_cast<const uint2*>(zrow + 2 * (kHeadDim + c));
    mma16816(dz, zw.x, 0u, zw.y, 0u, qb[2 * ks], qb[2 * ks + 1]);
  }
  // Scores in the log2 domain, less the running maximum (one fma each: the
  // zero-point term and the offset are folded into the addend).  Narrow:
  // lanes tig and tig^2 hold the two parts; wide: the accumulator holds the
  // whole score.
  float sc[NB][4][2];
  const float me0 = m_offset(st.m[0]), me1 = m_offset(st.m[1]);
#pragma unroll
  for (int bi = 0; bi < NB; ++bi) {
    const float z0 = fmaf(__shfl_sync(0xffffffffu, dz[0], 4 * bi + tig), scale_log2, -me0);
    const float z1 = fmaf(__shfl_sync(0xffffffffu, dz[1], 4 * bi + tig), scale_log2, -me1);
#pragma unroll
    for (int mt = 0; mt < 2; ++mt)
#pragma unroll
      for (int rh = 0; rh < 2; ++rh)
#pragma unroll
        for (int hh = 0; hh < 2; ++hh) {
          const int j = 2 * mt + rh;
          const float d = dk[bi][mt][2 * rh + hh];
          const float full = kWide ? d : d + __shfl_xor_sync(0xffffffffu, d, 2);
          sc[bi][j][hh] = fmaf(full, Codes<BK>::inv(j) * scale_log2, hh ? z1 : z0);
        }
  }

  constexpr bool kCompact = BV == 1;
  uint32_t pt[NB][2][2], pl[NB][2][2];
  tc_softmax<NB, kWide, kCompact, false>(sc, st, ln, pt, pl);

  // ---- values: o^T[c][h] ----
  // Value scales and zeros are stored in token pairs (t, t + 4), so the
  // B-operand scale of (k-step ks, dl) is word 2ks + dl of the lane's 8-token
  // run; zero-point MMA rows 0..3 = groups, row 4 = ones (the lanes of gid 4
  // read bytes 256..319 of the zero area), so it accumulates the row sum of
  // the weights; rows 5..7 read zeros.  (In the key zero-point MMA above the
  // rows past NB read the same area; their results are never used.)
#pragma unroll
  for (int bi = 0; bi < NB; ++bi) {
    const char* vc = pg[bi] + page_off_vcodes(BK);
    const char* vmeta = pg[bi] + page_off_vmeta(BK, BV);
    const char* vzrow = gid < 4 ? vmeta : zero;
    const uint4 z8 = *reinterpret_cast<const uint4*>(vzrow + 2 * (kHeadDim + 32 * (gid & 3) + 8 * tig));
    mma16816(st.zv, z8.x, 0u, z8.y, 0u, pt[bi][0][0], pt[bi][0][1]);
    mma16816(st.zv, z8.z, 0u, z8.w, 0u, pt[bi][1][0], pt[bi][1][1]);
    if constexpr (kCompact) {
      // 1-bit values: B = RN16(p~ s), one MMA per operand for every head
      const uint4 vw = *reinterpret_cast<const uint4*>(vc + 16 * lane);
#pragma unroll
      for (int g = 0; g < 4; ++g) {
        const uint4 s8 = *reinterpret_cast<const uint4*>(vmeta + 2 * (32 * g + 8 * tig));
        const uint32_t mw[4] = {s8.x, s8.y, s8.z, s8.w};
#pragma unroll
        for (int ks = 0; ks < 2; ++ks) {
          uint32_t am0[4], am1[4], bv[2];
#pragma unroll
          for (int dl = 0; dl < 2; ++dl) {
            const int ia = 2 * ks + dl;
            uint32_t v[4];
            Codes<1>::rot(comp(vw, g), ia, v);
            am0[2 * dl] = v[0];
            am0[2 * dl + 1] = v[1];
            am1[2 * dl] = v[2];
            am1[2 * dl + 1] = v[3];
            bv[dl] = h2u(__hmul2(u2h(pt[bi][ks][dl]), u2h(mw[ia])));
          }
          mma16816(st.acc[2 * g], am0[0], am0[1], am0[2], am0[3], bv[0], bv[1]);
          mma16816(st.acc[2 * g + 1], am1[0], am1[1], am1[2], am1[3], bv[0], bv[1]);
        }
      }
      continue;
    }
    if constexpr (kWide) {
      mma16816(st.zv, z8.x, 0u, z8.y, 0u, pl[bi][0][0], pl[bi][0][1]);
      mma16816(st.zv, z8.z, 0u, z8.w, 0u, pl[bi][1][0], pl[bi][1][1]);
    }
    // B = p * s in two fp16 parts: the high part is RN16(p_hi s); the low
    // part RN16(p_lo s + (p_hi s - RN16(p_hi s))), so rounding the product
    // costs no accuracy.  Narrow: columns 0..3 / 4..7, lanes of columns 4..7
    // hold p_lo after movmatrix and fetch p_hi from lane - 16; wide: every
    // lane has both parts of its head.
    // Narrow: pn = -p_hi on lanes of columns 4..7 and 0 elsewhere, so
    // RN16(pn s) is -RN16(p_hi s) there (rounding is symmetric) and the
    // residual fma needs no separate product.
    uint32_t pa[2][2], pb[2][2], pn[2][2];
#pragma unroll
    for (int ks = 0; ks < 2; ++ks)
#pragma unroll
      for (int dl = 0; dl < 2; ++dl) {
        if constexpr (kWide) {
          pa[ks][dl] = pt[bi][ks][dl];
          pb[ks][dl] = pl[bi][ks][dl];
        } else {
          const uint32_t other = __shfl_xor_sync(0xffffffffu, pt[bi][ks][dl], 16);
          pa[ks][dl] = lane < 16 ? pt[bi][ks][dl] : other;
          pb[ks][dl] = lane < 16 ? 0u : pt[bi][ks][dl];
          pn[ks][dl] = h2u(__hmul2(u2h(pa[ks][dl]), u2h(ln.neg_lo)));
        }
      }
    uint4 vw1;
    if constexpr (BV == 1) vw1 = *reinterpret_cast<const uint4*>(vc + 16 * lane);
#pragma unroll
    for (int g = 0; g < 4; ++g) {
      const uint4 s8 = *reinterpret_cast<const uint4*>(vmeta + 2 * (32 * g + 8 * tig));
      const uint32_t mw[4] = {s8.x, s8.y, s8.z, s8.w};  // scale pairs of tokens (8tig + i, + 4)
      uint32_t cw[8];
      if constexpr (BV != 1) {
#pragma unroll
        for (int i = 0; i < 8; ++i)
          cw[i] = *reinterpret_cast<const uint32_t*>(vc + 4 * ((32 * g + 8 * tig + i) * BV + ln.wv));
      }
#pragma unroll
      for (int ks = 0; ks < 2; ++ks) {
        uint32_t am0[4], am1[4], bv[2], bw[2];
#pragma unroll
        for (int dl = 0; dl < 2; ++dl) {
          const int ia = 2 * ks + dl, ib = ia + 4;  // tokens 8tig + ia, 8tig + ib
          uint32_t v[4];
          if constexpr (BV == 1) Codes<1>::rot(comp(vw1, g), ia, v);
          else Codes<BV>::get(cw[ia], cw[ib], ln.sel_v, v);
          am0[2 * dl] = v[0];
          am0[2 * dl + 1] = v[1];
          am1[2 * dl] = v[2];
          am1[2 * dl + 1] = v[3];
          const __half2 sc = u2h(mw[ia]);
          if constexpr (kWide) {
            const __half2 t = __hmul2(u2h(pa[ks][dl]), sc);
            const __half2 err = __hfma2(u2h(pa[ks][dl]), sc, __hneg2(t));
            bv[dl] = h2u(t);
            bw[dl] = h2u(__hfma2(u2h(pb[ks][dl]), sc, err));
          } else {
            // columns 0..3: RN16(p_hi s); 4..7: RN16(p_lo s + exact residual)
            const __half2 err = __hfma2(u2h(pa[ks][dl]), sc, __hmul2(u2h(pn[ks][dl]), sc));
            bv[dl] = h2u(__hfma2(u2h(pb[ks][dl]), sc, err));
          }
        }
        mma16816(st.acc[2 * g], am0[0], am0[1], am0[2], am0[3], bv[0], bv[1]);
        mma16816(st.acc[2 * g + 1], am1[0], am1[1], am1[2], am1[3], bv[0], bv[1]);
        if constexpr (kWide) {
          mma16816(st.acc[2 * g], am0[0], am0[1], am0[2], am0[3], bw[0], bw[1]);
          mma16816(st.acc[2 * g + 1], am1[0], am1[1], am1[2], am1[3], bw[0], bw[1]);
        }
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
  ln.wk = Codes<BK>::word(ln.gid);
  ln.wv = Codes<BV>::word(ln.gid);
  ln.neg_lo = ln.gid >= 4 ? 0xBC00BC00u : 0u;
  ln.p_lo = ln.tig >= 2 ? 1.0f : 0.0f;
  return ln;
}

// q of head gid & 3 (narrow) or gid (wide) in the B layout (exact fp16),
// zero beyond the group.  kPermuted: the packed path's K-slot order (four
// contiguous channels per lane); otherwise slot k of a k-step is channel
// 16 ks + k.
template <bool kPermuted, bool kWide>
__device__ __forceinline__ void load_qb(uint32_t (&qb)[16], const __half* qh, int gq,
                                        const Lane& ln) {
  const int head = kWide ? ln.gid : ln.gid & 3;
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
// unnormalised output row of heads 0..3 (narrow: the two parts in columns
// tig and tig^2 are added) or 0..7 (wide).  kPacked: channel rows follow the
// packed layout (nibble of a group, power-of-two factors, zero-point term);
// otherwise channel = 16 * m-tile + row.
template <bool kPacked, int BV, bool kWide>
__device__ __forceinline__ void tc_write_state(const TcState& st, WarpState& ws, int lane) {
  const int gid = lane >> 2, tig = lane & 3;
  float l0 = st.l[0], l1 = st.l[1];
#pragma unroll
  for (int o = 4; o < 32; o <<= 1) {
    l0 += __shfl_xor_sync(0xffffffffu, l0, o);
    l1 += __shfl_xor_sync(0xffffffffu, l1, o);
  }
  float zsum[2];
  zsum[0] = kWide ? st.zv[0] : st.zv[0] + __shfl_xor_sync(0xffffffffu, st.zv[0], 2);
  zsum[1] = kWide ? st.zv[1] : st.zv[1] + __shfl_xor_sync(0xffffffffu, st.zv[1], 2);
  if constexpr (kPacked) {
    // packed blocks: the row sum is row 4 of the value zero-point MMA
    l0 += __shfl_sync(0xffffffffu, zsum[0], 16 + tig);
    l1 += __shfl_sync(0xffffffffu, zsum[1], 16 + tig);
  }
  if (gid == 0 && (kWide || tig < 2)) {
    ws.m[2 * tig] = st.m[0];
    ws.m[2 * tig + 1] = st.m[1];
    ws.l[2 * tig] = l0;
    ws.l[2 * tig + 1] = l1;
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
          const float full_v = kWide ? a : a + __shfl_xor_sync(0xffffffffu, a, 2);
          if (kWide || tig < 2) ws.o[2 * tig + hh][cch] = fmaf(full_v, inv, hh ? zg1 : zg0);
        }
      }
    }
  }
}


// ---------------------------------------------------------------------------
// Tensor-core path for the fp16 residual window: a warp stages the K rows of
// a 32-token chunk in shared memory, scores them with ldmatrix-fed MMAs
// (keys as A with tokens as rows), then stages the V rows in the same place
// (values transposed, channels as rows).  Rows past the window are zero and
// their scores -inf.
// ---------------------------------------------------------------------------

constexpr int kResRow = kHeadDim + 8;                    // halves per staged row (16-byte pad)
constexpr int kResRowsBytes = kGroup * kResRow * 2;      // one 32-row K or V chunk

__device__ __forceinline__ void ldsm_x4(uint32_t (&r)[4], const void* p) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(smem_addr(p))
               : "memory");
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t (&r)[4], const void* p) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(smem_addr(p))
               : "memory");
}

template <bool kWide, bool kCompact>
__device__ __forceinline__ void tc_resid_scores(const __half* ks_s, int n_tok,
                                                const uint32_t (&qb)[16], const Lane& ln,
                                                float scale_log2, TcState& st,
                                                uint32_t (&pt)[1][2][2], uint32_t (&pl)[1][2][2]) {
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
  float sc[1][4][2];
  const float me[2] = {m_offset(st.m[0]), m_offset(st.m[1])};
#pragma unroll
  for (int mt = 0; mt < 2; ++mt)
#pragma unroll
    for (int rh = 0; rh < 2; ++rh) {
      const bool ok = 16 * mt + ln.gid + 8 * rh < n_tok;
#pragma unroll
      for (int hh = 0; hh < 2; ++hh)
        sc[0][2 * mt + rh][hh] = ok ? fmaf(dk[mt][2 * rh + hh], scale_log2, -me[hh]) : -INFINITY;
    }
  tc_softmax<1, kWide, kCompact, true>(sc, st, ln, pt, pl);
}

template <bool kWide, bool kCompact>
__device__ __forceinline__ void tc_resid_values(const __half* vs_s, const uint32_t (&pt)[1][2][2],
                                                const uint32_t (&pl)[1][2][2], TcState& st) {
  const int lane = threadIdx.x & 31;
  const int mi = lane >> 3, r8 = lane & 7;
#pragma unroll
  for (int ks = 0; ks < 2; ++ks)
#pragma unroll
    for (int mtp = 0; mtp < 8; ++mtp) {
      uint32_t a[4];
      ldsm_x4_t(a, vs_s + (16 * ks + 8 * (mi >> 1) + r8) * kResRow + 16 * mtp + 8 * (mi & 1));
      mma16816(st.acc[mtp], a[0], a[1], a[2], a[3], pt[0][ks][0], pt[0][ks][1]);
      if constexpr (kWide && !kCompact)
        mma16816(st.acc[mtp], a[0], a[1], a[2], a[3], pl[0][ks][0], pl[0][ks][1]);
    }
}


// Blocks per ring slot and slots per warp for a page size.
__host__ __device__ constexpr int ring_blocks(int page) { return page <= 3072 ? 2 : 1; }
__host__ __device__ constexpr int ring_slots(int page) {
  return kRingBudget / (kWarps * ring_blocks(page) * page) < 1   ? 1
         : kRingBudget / (kWarps * ring_blocks(page) * page) > 4 ? 4
                                                                 : kRingBudget / (kWarps * ring_blocks(page) * page);
}
// A warp's ring: its slots, and at least one 32-row K (or V) chunk of the
// window, which a window warp stages there.
__host__ __device__ constexpr int warp_ring_bytes(int page) {
  return ((ring_slots(page) * ring_blocks(page) * page > kResRowsBytes
               ? ring_slots(page) * ring_blocks(page) * page
               : kResRowsBytes) +
          127) / 128 * 128;
}
static_assert(kWarps * warp_ring_bytes(page_bytes_c(4, 8)) <= kRingBudget + 8 * 1024, "rings fit");


// Packed warps stream their blocks through a private ring of slots.  A page
// is written once, when its group leaves the window, and never changes
// afterwards, so before waiting for the previous kernel (programmatic
// dependent launch) lane 0 already streams the first slots of the range that
// a length read before the wait gives (tc_pre_issue), up to the block before
// the newest.  If the range after the wait does not begin with exactly those
// slots they are consumed without use.
// A warp's window of 32 consecutive block-table entries (paged caches): lane
// i holds the entry of block wb + i, refreshed (one coalesced load) when a
// lookup leaves it.  Lookups are warp-uniform and made by all lanes.
struct TableWin {
  int wb, v;
};
__device__ __forceinline__ void table_win_init(TableWin& w) {
  w.wb = -(1 << 30);
  w.v = -1;
}
__device__ __forceinline__ const char* block_addr(const PageMap& pm, TableWin& w, int j) {
  if (!pm.paged()) return pm.base + (long long)j * pm.page;
  if (j < w.wb || j >= w.wb + 32) {
    w.wb = j;
    const int k = j + (int)(threadIdx.x & 31);
    w.v = k < pm.max_blocks ? __ldg(pm.row + k) : -1;
  }
  return pm.at(j, __shfl_sync(0xffffffffu, w.v, j - w.wb));
}

// Slot s of the ring: blocks [first, first + nblk) (nblk <= blocks per
// slot).  Called by all lanes; lane 0 issues.  Contiguous pages come in one
// bulk copy, paged ones in one copy per page; a block mapped outside the
// pool is not copied (KVQ_FLAG_BAD_PAGE; its slot bytes are stale and the
// call's output is flagged invalid) and the barrier expects only the bytes
// copied.  `fence`: the warp's reads of the slot precede the copies that
// overwrite it.
template <int BK, int BV>
__device__ __forceinline__ void issue_slot(const PageMap& pm, TableWin& tw, char* ring,
                                           uint64_t* full, int R, int s, int first, int nblk,
                                           unsigned* flag, bool fence) {
  constexpr int page = page_bytes_c(BK, BV);
  constexpr int NB = ring_blocks(page);
  const bool lead = (threadIdx.x & 31) == 0;
  uint64_t* bar = full + s % R;
  char* dst = ring + (size_t)(s % R) * NB * page;
  if (!pm.paged()) {
    if (lead) {
      if (fence) asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      const uint32_t bytes = (uint32_t)(nblk * page);
      mbar_expect_tx(bar, bytes);
      bulk_g2s(dst, pm.base + (long long)first * page, bytes, bar);
    }
    return;
  }
  const char* src[NB];
  uint32_t bytes = 0;
#pragma unroll
  for (int i = 0; i < NB; ++i) {
    src[i] = i < nblk ? block_addr(pm, tw, first + i) : nullptr;
    if (src[i]) bytes += page;
  }
  if (lead) {
    if (fence) asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    if (bytes < (uint32_t)(nblk * page)) atomicOr(flag, (unsigned)KVQ_FLAG_BAD_PAGE);
    mbar_expect_tx(bar, bytes);
#pragma unroll
    for (int i = 0; i < NB; ++i)
      if (src[i]) bulk_g2s(dst + i * page, src[i], page, bar);
  }
}

// Units (slots) of the range [lo_h, hi_h) that end at or before hi_safe:
// streams them, returns their count and in `end` the block after them.
template <int BK, int BV>
__device__ __forceinline__ int tc_pre_issue(const PageMap& pm, TableWin& tw, int lo_h, int hi_h,
                                            int hi_safe, char* ring, uint64_t* full, int R,
                                            int& end, unsigned* flag) {
  constexpr int NB = ring_blocks(page_bytes_c(BK, BV));
  int n = 0;
  end = lo_h;
  for (; n < R; ++n) {
    const int b0 = lo_h + n * NB;
    const int nblk = min(NB, hi_h - b0);
    if (nblk <= 0 || b0 + nblk > hi_safe) break;
    issue_slot<BK, BV>(pm, tw, ring, full, R, n, b0, nblk, flag, false);
    end = b0 + nblk;
  }
  return n;
}


// Decode step with a flush: the 32-token block of positions [p0, p0 + 32),
// still fp16 in the ring, leaves the window and is quantized exactly as
// kvq_pack does (quantize_quarter, common.cuh) into a page image in shared
// memory.  The work comes in four quarters (key channels 32 qi .. 32 qi + 31,
// value group qi), so different warps can take them.  Rows are read straight
// from global memory (L2); nothing in this kernel writes them.  Kept out of
// line: it is rare and its registers would otherwise crowd the streaming
// loop.
template <int BK, int BV>
__device__ __noinline__ void flush_quarter(const __half* ring_k, const __half* ring_v, int p0,
                                           int ring, int qi, char* image) {
  const int s0 = p0 % ring;
  quantize_quarter<BK, BV>(
      [&](int t) { return ring_k + (long long)(s0 + t < ring ? s0 + t : s0 + t - ring) * kHeadDim; },
      [&](int t) { return ring_v + (long long)(s0 + t < ring ? s0 + t : s0 + t - ring) * kHeadDim; },
      qi, image);
}

// Copy rows p0 .. p0 + 31 into padded `rows` with one bulk copy per row
// (issued by the row's lane, completing on `bar`); rows at or past n_tok are
// zeroed.  The row of position p_new comes from new_row.  Returns false if
// the bounded wait gave up.
__device__ __forceinline__ bool stage_rows_bulk(__half* rows, const __half* ring_base, int p0,
                                                int n_tok, int ring, int p_new,
                                                const __half* new_row, uint64_t* bar,
                                                uint32_t parity) {
  const int lane = threadIdx.x & 31;
  __syncwarp();
  if (lane >= n_tok) {
    uint4* r = reinterpret_cast<uint4*>(rows + lane * kResRow);
#pragma unroll
    for (int i = 0; i < 16; ++i) r[i] = make_uint4(0u, 0u, 0u, 0u);
  }
  if (lane == 0) {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    mbar_expect_tx(bar, (uint32_t)(n_tok * kHeadDim * 2));
  }
  __syncwarp();
  if (lane < n_tok) {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    const __half* src = p0 + lane == p_new ? new_row
                                           : ring_base + (long long)((p0 + lane) % ring) * kHeadDim;
    bulk_g2s(rows + lane * kResRow, src, kHeadDim * 2, bar);
  }
  const bool ok = __all_sync(0xffffffffu, mbar_wait(bar, parity));
  __syncwarp();
  return ok;

}

// One element of the attention output: the fp32 result, or its fp16
// rounding to nearest even.
__device__ __forceinline__ void store_out(void* out, int out_f16, long long i, float v) {
  if (out_f16) static_cast<__half*>(out)[i] = __float2half_rn(v);
  else static_cast<float*>(out)[i] = v;
}


__device__ __forceinline__ unsigned atom_add_acq_rel(unsigned* p, unsigned v) {
  unsigned old;
  asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(v) : "memory");
  return old;
}

