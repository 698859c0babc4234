// kvq_pack: append new K/V tokens to the fp16 residual window and quantize
// every 32-token group that leaves it (KbVb, Sec. 3.1 of the paper).
//
// Quantizer of one 32-element group x (b bits, levels = 2^b - 1), each step a
// single IEEE float32 operation with the stated rounding:
//   zero  = min x                                   (exact, fp16)
//   scale = RU16(RU32(RU32(max x - min x) / levels)) (stored fp16)
//   code  = clamp(rint(RN32(RN32(x - zero) / scale)), 0, levels); 0 if scale == 0
// Codes of a group fill b little-endian uint32 words, element i at bits
// [(i*b) % 32, +b) of word (i*b) / 32.  Keys group 32 tokens of one channel,
// values 32 channels of one token.  1-bit codes are then scattered into the
// fragment order the attention kernel reads (key1_bit / val1_bit).

#include "common.cuh"

namespace kvq {
namespace {

constexpr int kPackThreads = 256;
constexpr int kRowPad = 136;  // halves per smem row (128 + 8) to spread banks

struct Tile {
  __half k[kGroup][kRowPad];
  __half v[kGroup][kRowPad];
  uint32_t k1[kHeadDim];  // 1-bit key codes in fragment order
  uint32_t v1[kHeadDim];  // 1-bit value codes in fragment order
};

template <int B>
__device__ __forceinline__ void store_words(uint32_t* dst, const uint32_t (&w)[B]) {
#pragma unroll
  for (int j = 0; j < B; ++j) dst[j] = w[j];
}

template <int B>
__device__ __forceinline__ void quantize_key_channel(Tile& t, int c, char* page, int bits_k) {
  float x[kGroup];
#pragma unroll
  for (int i = 0; i < kGroup; ++i) x[i] = __half2float(t.k[i][c]);
  uint32_t w[B];
  __half sc, z;
  quantize_group<B>(x, w, sc, z);
  if (B == 1) {
#pragma unroll 4
    for (int i = 0; i < kGroup; ++i) {
      const int bit = key1_bit(i, c);
      if ((w[0] >> i) & 1u) atomicOr(&t.k1[bit >> 5], 1u << (bit & 31));
    }
  } else {
    store_words<B>(reinterpret_cast<uint32_t*>(page) + c * B, w);
  }
  __half* meta = reinterpret_cast<__half*>(page + page_off_kmeta(bits_k));
  meta[c] = sc;
  meta[kHeadDim + c] = z;
}

// Value codes of b >= 2 bits are stored group-major: group index
// grp * 32 + tok.  Scales and zeros follow vmeta_index; the 128 scales
// precede the 128 zeros.
template <int B>
__device__ __forceinline__ void quantize_value_group(Tile& t, int pair, char* page,
                                                     int bits_k, int bits_v) {
  const int grp = pair >> 5, tok = pair & 31;
  float x[kGroup];
#pragma unroll
  for (int i = 0; i < kGroup; ++i) x[i] = __half2float(t.v[tok][grp * kGroup + i]);
  uint32_t w[B];
  __half sc, z;
  quantize_group<B>(x, w, sc, z);
  if (B == 1) {
#pragma unroll 4
    for (int i = 0; i < kGroup; ++i) {
      const int bit = val1_bit(tok, grp * kGroup + i);
      if ((w[0] >> i) & 1u) atomicOr(&t.v1[bit >> 5], 1u << (bit & 31));
    }
  } else {
    store_words<B>(reinterpret_cast<uint32_t*>(page + page_off_vcodes(bits_k)) + pair * B, w);
  }
  __half* meta = reinterpret_cast<__half*>(page + page_off_vmeta(bits_k, bits_v));
  meta[vmeta_index(grp, tok)] = sc;
  meta[kHeadDim + vmeta_index(grp, tok)] = z;
}

// 256 threads: 0..127 quantize one key channel each, 128..255 one
// (32-channel group, token) value group each.  Called by every thread.
__device__ void quantize_tile(Tile& t, char* page, int bits_k, int bits_v) {
  const int tid = threadIdx.x;
  if (tid < kHeadDim) {
    t.k1[tid] = 0u;
    t.v1[tid] = 0u;
  }
  __syncthreads();
  if (tid < kHeadDim) {
    switch (bits_k) {
      case 1: quantize_key_channel<1>(t, tid, page, bits_k); break;
      case 2: quantize_key_channel<2>(t, tid, page, bits_k); break;
      case 4: quantize_key_channel<4>(t, tid, page, bits_k); break;
      default: quantize_key_channel<8>(t, tid, page, bits_k); break;
    }
  } else {
    const int pair = tid - kHeadDim;
    switch (bits_v) {
      case 1: quantize_value_group<1>(t, pair, page, bits_k, bits_v); break;
      case 2: quantize_value_group<2>(t, pair, page, bits_k, bits_v); break;
      case 4: quantize_value_group<4>(t, pair, page, bits_k, bits_v); break;
      default: quantize_value_group<8>(t, pair, page, bits_k, bits_v); break;
    }
  }
  __syncthreads();
  if (bits_k == 1 && tid < kHeadDim) reinterpret_cast<uint32_t*>(page)[tid] = t.k1[tid];
  if (bits_v == 1 && tid >= kHeadDim)
    reinterpret_cast<uint32_t*>(page + page_off_vcodes(bits_k))[tid - kHeadDim] = t.v1[tid - kHeadDim];
}

// Programmatic dependent launch: let the next kernel of the stream start
// launching at once, then wait for the previous one (and its writes).
__device__ __forceinline__ void pdl_enter() {
  asm volatile("griddepcontrol.launch_dependents;\ngriddepcontrol.wait;" ::: "memory");
}

// Page of block j of (b, h), or nullptr when a paged cache maps it outside
// the pool (then KVQ_FLAG_BAD_PAGE is set and the block is not written).
// Uniform over the CTA.
__device__ __forceinline__ char* page_ptr(const Dims& d, const kvq_cache& c, int b, int h, int j) {
  char* p = page_map(d, c, b, h).at(j);
  if (!p && threadIdx.x == 0)
    atomicOr(reinterpret_cast<unsigned*>(c.seq_len) + d.batch, (unsigned)KVQ_FLAG_BAD_PAGE);
  return p;
}

// Source row (128 fp16) of absolute token p of (b, h): the ring for p < L0,
// the caller's new tokens otherwise.
struct RowSrc {
  const __half* ring_k;
  const __half* ring_v;
  const __half* new_k;
  const __half* new_v;
  int L0, ring;
  __device__ __forceinline__ const uint4* k(int p) const {
    const __half* r = p < L0 ? ring_k + (long long)(p % ring) * kHeadDim
                             : new_k + (long long)(p - L0) * kHeadDim;
    return reinterpret_cast<const uint4*>(r);
  }
  __device__ __forceinline__ const uint4* v(int p) const {
    const __half* r = p < L0 ? ring_v + (long long)(p % ring) * kHeadDim
                             : new_v + (long long)(p - L0) * kHeadDim;
    return reinterpret_cast<const uint4*>(r);
  }
};

// Stage block j's 32 tokens into the smem tile (16 x 16-byte pieces per row).
__device__ void load_tile(Tile& t, const RowSrc& src, int j) {
  for (int e = threadIdx.x; e < kGroup * 16; e += kPackThreads) {
    const int row = e >> 4, piece = e & 15;
    const int p = j * kGroup + row;
    *reinterpret_cast<uint4*>(&t.k[row][piece * 8]) = src.k(p)[piece];
    *reinterpret_cast<uint4*>(&t.v[row][piece * 8]) = src.v(p)[piece];
  }
}

__device__ __forceinline__ RowSrc make_src(const Dims& d, const kvq_cache& c, const __half* k_new,
                                           const __half* v_new, int n_new, int b, int bi, int h,
                                           int L0) {
  RowSrc s;
  const long long bh = (long long)b * d.hkv + h;
  s.ring_k = reinterpret_cast<const __half*>(c.k_resid) + bh * d.ring * kHeadDim;
  s.ring_v = reinterpret_cast<const __half*>(c.v_resid) + bh * d.ring * kHeadDim;
  const long long nh = ((long long)bi * d.hkv + h) * n_new;
  s.new_k = k_new + nh * kHeadDim;
  s.new_v = v_new + nh * kHeadDim;
  s.L0 = L0;
  s.ring = d.ring;
  return s;
}

// Blocks made only of new tokens (prefill): one warp per quarter of a block
// (quantize_quarter: key channels 32 w .. 32 w + 31 and value group w),
// reading the rows straight from the input, so no staging tile and no
// shared-memory atomics; many small CTAs keep the loads of many blocks in
// flight.  grid (blocks, hkv, batch_count) of 128 threads.
constexpr int kInputThreads = 4 * 32;

template <int BK, int BV>
__global__ void __launch_bounds__(kInputThreads)
    pack_input_blocks_kernel(Dims d, kvq_cache c, const __half* __restrict__ k_new,
                             const __half* __restrict__ v_new, int n_new, int batch_begin) {
  pdl_enter();
  const int bi = blockIdx.z, b = batch_begin + bi, h = blockIdx.y;
  const int L0 = c.seq_len[b];
  const int L1 = L0 + n_new;
  if (L1 > d.max_len) return;  // the append kernel reports the overflow
  const int first = max(packed_len(L0, d.residual), ((L0 + kGroup - 1) / kGroup) * kGroup) / kGroup;
  const int j = first + blockIdx.x;
  if (j >= packed_len(L1, d.residual) / kGroup) return;
  char* page = page_ptr(d, c, b, h, j);
  if (!page) return;
  const long long nh = ((long long)bi * d.hkv + h) * n_new;
  const __half* nk = k_new + (nh + (long long)j * kGroup - L0) * kHeadDim;
  const __half* nv = v_new + (nh + (long long)j * kGroup - L0) * kHeadDim;
  quantize_quarter<BK, BV>([&](int t) { return nk + (long long)t * kHeadDim; },
                           [&](int t) { return nv + (long long)t * kHeadDim; },
                           threadIdx.x >> 5, page);
}

template <int BK>
cudaError_t launch_input_blocks_bv(const Dims& d, cudaLaunchConfig_t& cfg, const kvq_cache& cache,
                                   const __half* k_new, const __half* v_new, int n_new,
                                   int batch_begin) {
  switch (d.bits_v) {
    case 1: return cudaLaunchKernelEx(&cfg, pack_input_blocks_kernel<BK, 1>, d, cache, k_new, v_new, n_new, batch_begin);
    case 2: return cudaLaunchKernelEx(&cfg, pack_input_blocks_kernel<BK, 2>, d, cache, k_new, v_new, n_new, batch_begin);
    case 4: return cudaLaunchKernelEx(&cfg, pack_input_blocks_kernel<BK, 4>, d, cache, k_new, v_new, n_new, batch_begin);
    default: return cudaLaunchKernelEx(&cfg, pack_input_blocks_kernel<BK, 8>, d, cache, k_new, v_new, n_new, batch_begin);
  }
}

cudaError_t launch_input_blocks(const Dims& d, cudaLaunchConfig_t& cfg, const kvq_cache& cache,
                                const __half* k_new, const __half* v_new, int n_new,
                                int batch_begin) {
  switch (d.bits_k) {
    case 1: return launch_input_blocks_bv<1>(d, cfg, cache, k_new, v_new, n_new, batch_begin);
    case 2: return launch_input_blocks_bv<2>(d, cfg, cache, k_new, v_new, n_new, batch_begin);
    case 4: return launch_input_blocks_bv<4>(d, cfg, cache, k_new, v_new, n_new, batch_begin);
    default: return launch_input_blocks_bv<8>(d, cfg, cache, k_new, v_new, n_new, batch_begin);
  }
}

// Blocks that touch the ring, the ring append, and the length update.
// grid (hkv, batch_count); the last CTA of a sequence (ticket) publishes L1.
__global__ void __launch_bounds__(kPackThreads)
    pack_append_kernel(Dims d, kvq_cache c, const __half* __restrict__ k_new,
                       const __half* __restrict__ v_new, int n_new, int batch_begin) {
  __shared__ Tile tile;
  pdl_enter();
  const int bi = blockIdx.y, b = batch_begin + bi, h = blockIdx.x;
  const int L0 = c.seq_len[b];
  const int L1 = L0 + n_new;
  if (L1 > d.max_len) {
    if (threadIdx.x == 0 && h == 0) atomicOr(reinterpret_cast<unsigned*>(c.seq_len) + d.batch,
                                             KVQ_FLAG_OVERFLOW);
    return;
  }
  const int Lq0 = packed_len(L0, d.residual), Lq1 = packed_len(L1, d.residual);
  const RowSrc src = make_src(d, c, k_new, v_new, n_new, b, bi, h, L0);

  // 1. Groups leaving the window that start below L0 (they read the ring).
  const int j_end = min(Lq1, ((L0 + kGroup - 1) / kGroup) * kGroup) / kGroup;
  for (int j = Lq0 / kGroup; j < j_end; ++j) {
    char* page = page_ptr(d, c, b, h, j);
    if (!page) continue;
    load_tile(tile, src, j);
    __syncthreads();
    quantize_tile(tile, page, d.bits_k, d.bits_v);
    __syncthreads();
  }

  // 2. New tokens that stay fp16 go to their ring slots (after every ring read).
  const long long bh = (long long)b * d.hkv + h;
  __half* ring_k = reinterpret_cast<__half*>(c.k_resid) + bh * d.ring * kHeadDim;
  __half* ring_v = reinterpret_cast<__half*>(c.v_resid) + bh * d.ring * kHeadDim;
  const int p0 = max(Lq1, L0);
  for (int e = threadIdx.x; e < (L1 - p0) * 16; e += kPackThreads) {
    const int p = p0 + (e >> 4), piece = e & 15;
    reinterpret_cast<uint4*>(ring_k + (long long)(p % d.ring) * kHeadDim)[piece] = src.k(p)[piece];
    reinterpret_cast<uint4*>(ring_v + (long long)(p % d.ring) * kHeadDim)[piece] = src.v(p)[piece];
  }

  // 3. Publish the new length once every kv-head of the sequence has read L0.
  __syncthreads();
  if (threadIdx.x == 0) {
    unsigned* tickets = reinterpret_cast<unsigned*>(c.seq_len) + d.batch + 2;
    __threadfence();
    const unsigned t = atomicAdd(&tickets[b], 1u);
    if (t == (unsigned)d.hkv - 1) {
      c.seq_len[b] = L1;
      tickets[b] = 0u;
      __threadfence();
    }
  }
}

}  // namespace

cudaError_t launch_pack(const Dims& d, const kvq_cache& cache, const __half* k_new,
                        const __half* v_new, int n_new, int batch_begin, int batch_count,
                        cudaStream_t stream) {
  cudaLaunchConfig_t cfg = {};
  cfg.blockDim = dim3(kPackThreads);
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cudaError_t e;
  if (n_new > kGroup) {
    cfg.gridDim = dim3(n_new / kGroup + 1, d.hkv, batch_count);
    cfg.blockDim = dim3(kInputThreads);
    e = launch_input_blocks(d, cfg, cache, k_new, v_new, n_new, batch_begin);
    if (e != cudaSuccess) return e;
    cfg.blockDim = dim3(kPackThreads);
  }
  cfg.gridDim = dim3(d.hkv, batch_count);
  e = cudaLaunchKernelEx(&cfg, pack_append_kernel, d, cache, k_new, v_new, n_new, batch_begin);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace kvq
