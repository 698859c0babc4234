// Host side of the kvq C ABI: argument validation, cache layout, launches.
// Every entry point validates on the host and returns a kvq_status before
// anything is enqueued; no entry point allocates, frees or synchronises.

#include <math.h>
#include <stdarg.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include "common.cuh"

namespace kvq {

static thread_local char g_err[512] = "";

void set_error(const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_err, sizeof(g_err), fmt, ap);
  va_end(ap);
}

static kvq_status fail(kvq_status s, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_err, sizeof(g_err), fmt, ap);
  va_end(ap);
  return s;
}

static kvq_status cuda_status(cudaError_t e, const char* what) {
  if (e == cudaSuccess) {
    g_err[0] = 0;
    return KVQ_OK;
  }
  return fail(KVQ_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

static bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// KVQ_TRACE=1 in the environment: one line per launch on stderr (entry
// point, shapes, grid choices).  Read once per process.
static bool tracing() {
  static const int on = [] {
    const char* v = getenv("KVQ_TRACE");
    return v && v[0] && strcmp(v, "0") != 0 ? 1 : 0;
  }();
  return on != 0;
}
static void trace(const char* fmt, ...) {
  if (!tracing()) return;
  va_list ap;
  va_start(ap, fmt);
  fputs("kvq: ", stderr);
  vfprintf(stderr, fmt, ap);
  fputc('\n', stderr);
  va_end(ap);
}

static size_t round_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

static kvq_status check_config(const kvq_config* c) {
  if (!c) return fail(KVQ_ERR_ARG, "config is NULL");
  if (c->batch < 1) return fail(KVQ_ERR_SHAPE, "batch must be >= 1 (got %d)", c->batch);
  if (c->n_kv_heads < 1 || c->n_q_heads < 1)
    return fail(KVQ_ERR_SHAPE, "head counts must be >= 1");
  if (c->n_q_heads % c->n_kv_heads)
    return fail(KVQ_ERR_SHAPE, "n_q_heads (%d) must be a multiple of n_kv_heads (%d)",
                c->n_q_heads, c->n_kv_heads);
  if (c->n_q_heads / c->n_kv_heads > kMaxGq)
    return fail(KVQ_ERR_UNSUPPORTED, "n_q_heads / n_kv_heads must be <= %d", kMaxGq);
  if (c->head_dim != kHeadDim)
    return fail(KVQ_ERR_UNSUPPORTED, "head_dim must be 128 (got %d)", c->head_dim);
  if (c->group != kGroup) return fail(KVQ_ERR_UNSUPPORTED, "group must be 32 (got %d)", c->group);
  for (int b : {c->bits_k, c->bits_v})
    if (b != 1 && b != 2 && b != 4 && b != 8)
      return fail(KVQ_ERR_UNSUPPORTED, "bits must be 1, 2, 4 or 8 (got %d)", b);
  if (c->residual < kGroup || c->residual % kGroup || c->residual > 4096)
    return fail(KVQ_ERR_UNSUPPORTED, "residual must be a multiple of 32 in [32, 4096] (got %d)",
                c->residual);
  if (c->max_len < kGroup || c->max_len % kGroup)
    return fail(KVQ_ERR_SHAPE, "max_len must be a positive multiple of 32 (got %d)", c->max_len);
  if (c->batch > 65535 || c->n_kv_heads > 65535)
    return fail(KVQ_ERR_SHAPE, "batch and n_kv_heads must be <= 65535");
  g_err[0] = 0;
  return KVQ_OK;
}

struct Layout {
  size_t pages, k_resid, v_resid, seq, total;
};

// paged: the page region is empty (the pages live in the caller's pool).
static Layout layout_of(const kvq_config& c, bool paged = false) {
  Layout l;
  const size_t bh = (size_t)c.batch * c.n_kv_heads;
  const size_t pages =
      paged ? 0 : bh * (size_t)(c.max_len / kGroup) * page_bytes(c.bits_k, c.bits_v);
  const size_t resid = bh * (size_t)(c.residual + kGroup) * kHeadDim * sizeof(__half);
  const size_t seq = (size_t)(c.batch + 2) * 4 + (size_t)c.batch * 4;
  l.pages = 0;
  l.k_resid = round_up(l.pages + pages, 256);
  l.v_resid = round_up(l.k_resid + resid, 256);
  l.seq = round_up(l.v_resid + resid, 256);
  l.total = round_up(l.seq + seq, 256);
  return l;
}

static size_t seq_region_bytes(const kvq_config& c) {
  return (size_t)(c.batch + 2) * 4 + (size_t)c.batch * 4;
}

static kvq_status check_cache(const kvq_config& c, const kvq_cache* cache) {
  if (!cache) return fail(KVQ_ERR_ARG, "cache is NULL");
  if (!cache->pages || !cache->k_resid || !cache->v_resid || !cache->seq_len)
    return fail(KVQ_ERR_ARG, "cache has a NULL pointer");
  if (!aligned16(cache->pages) || !aligned16(cache->k_resid) || !aligned16(cache->v_resid) ||
      (reinterpret_cast<uintptr_t>(cache->seq_len) & 3u))
    return fail(KVQ_ERR_ALIGN, "cache pointers must be 16-byte aligned");
  if (cache->block_table) {
    if (reinterpret_cast<uintptr_t>(cache->block_table) & 3u)
      return fail(KVQ_ERR_ALIGN, "block_table must be 4-byte aligned");
    if (cache->n_pages < 1) return fail(KVQ_ERR_ARG, "a paged cache needs n_pages >= 1");
  }
  (void)c;
  return KVQ_OK;
}

static int sm_count() {
  static int cached = 0;
  if (cached) return cached;
  int dev = 0, n = 0;
  if (cudaGetDevice(&dev) == cudaSuccess &&
      cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess && n > 0) {
    cached = n;
  } else {
    cudaGetLastError();
    n = 152;  // GB300; used only to size the split count when no device is visible
  }
  return n;
}

static int default_splits(const kvq_config& c) {
  return attn_default_splits(make_dims(c), sm_count());
}

// n_splits as the launchers take it: > 0 the split plan, 0 -> the flat plan
// on one CTA per resident slot (a negative count).
static int resolve_splits(int32_t n_splits) {
  return n_splits == 0 ? -attn_flat_ctas(sm_count()) : n_splits;
}
// Workspace bytes of a resolved n_splits.
static size_t attn_ws_bytes(const Dims& d, int n_splits) {
  return n_splits > 0 ? attn_split_workspace_bytes(d, n_splits)
                      : attn_workspace_bytes(d, -n_splits);
}

}  // namespace kvq

using namespace kvq;

extern "C" {

const char* kvq_last_error(void) { return g_err; }

int32_t kvq_version(void) { return 100; }

kvq_status kvq_validate_config(const kvq_config* cfg) { return check_config(cfg); }

size_t kvq_page_bytes(const kvq_config* cfg) {
  if (check_config(cfg) != KVQ_OK) return 0;
  return page_bytes(cfg->bits_k, cfg->bits_v);
}

kvq_status kvq_cache_layout(const kvq_config* cfg, size_t* total_bytes, size_t offsets[4]) {
  kvq_status s = check_config(cfg);
  if (s != KVQ_OK) return s;
  if (!total_bytes || !offsets) return fail(KVQ_ERR_ARG, "output pointer is NULL");
  Layout l = layout_of(*cfg);
  *total_bytes = l.total;
  offsets[0] = l.pages;
  offsets[1] = l.k_resid;
  offsets[2] = l.v_resid;
  offsets[3] = l.seq;
  return KVQ_OK;
}

kvq_status kvq_cache_bind(const kvq_config* cfg, void* base, kvq_cache* cache) {
  kvq_status s = check_config(cfg);
  if (s != KVQ_OK) return s;
  if (!base || !cache) return fail(KVQ_ERR_ARG, "base or cache is NULL");
  if (reinterpret_cast<uintptr_t>(base) & 255u)
    return fail(KVQ_ERR_ALIGN, "cache buffer must be 256-byte aligned");
  Layout l = layout_of(*cfg);
  char* p = static_cast<char*>(base);
  cache->pages = p + l.pages;
  cache->k_resid = reinterpret_cast<uint16_t*>(p + l.k_resid);
  cache->v_resid = reinterpret_cast<uint16_t*>(p + l.v_resid);
  cache->seq_len = reinterpret_cast<int32_t*>(p + l.seq);
  cache->block_table = nullptr;
  cache->n_pages = 0;
  return KVQ_OK;
}

size_t kvq_page_pool_bytes(const kvq_config* cfg, int32_t n_pages) {
  if (check_config(cfg) != KVQ_OK) return 0;
  if (n_pages < 1) {
    set_error("n_pages must be >= 1 (got %d)", n_pages);
    return 0;
  }
  return (size_t)n_pages * cfg->n_kv_heads * page_bytes(cfg->bits_k, cfg->bits_v);
}

kvq_status kvq_paged_cache_layout(const kvq_config* cfg, size_t* total_bytes,
                                  size_t offsets[4]) {
  kvq_status s = check_config(cfg);
  if (s != KVQ_OK) return s;
  if (!total_bytes || !offsets) return fail(KVQ_ERR_ARG, "output pointer is NULL");
  Layout l = layout_of(*cfg, true);
  *total_bytes = l.total;
  offsets[0] = l.pages;
  offsets[1] = l.k_resid;
  offsets[2] = l.v_resid;
  offsets[3] = l.seq;
  return KVQ_OK;
}

kvq_status kvq_paged_cache_bind(const kvq_config* cfg, void* base, void* pool, int32_t n_pages,
                                const int32_t* block_table, kvq_cache* cache) {
  kvq_status s = check_config(cfg);
  if (s != KVQ_OK) return s;
  if (!base || !pool || !block_table || !cache)
    return fail(KVQ_ERR_ARG, "base, pool, block_table or cache is NULL");
  if (reinterpret_cast<uintptr_t>(base) & 255u)
    return fail(KVQ_ERR_ALIGN, "cache buffer must be 256-byte aligned");
  if (!aligned16(pool)) return fail(KVQ_ERR_ALIGN, "page pool must be 16-byte aligned");
  if (reinterpret_cast<uintptr_t>(block_table) & 3u)
    return fail(KVQ_ERR_ALIGN, "block_table must be 4-byte aligned");
  if (n_pages < 1) return fail(KVQ_ERR_ARG, "n_pages must be >= 1 (got %d)", n_pages);
  Layout l = layout_of(*cfg, true);
  char* p = static_cast<char*>(base);
  cache->pages = pool;
  cache->k_resid = reinterpret_cast<uint16_t*>(p + l.k_resid);
  cache->v_resid = reinterpret_cast<uint16_t*>(p + l.v_resid);
  cache->seq_len = reinterpret_cast<int32_t*>(p + l.seq);
  cache->block_table = block_table;
  cache->n_pages = n_pages;
  return KVQ_OK;
}

kvq_status kvq_cache_reset(const kvq_config* cfg, const kvq_cache* cache, void* stream) {
  kvq_status s = check_config(cfg);
  if (s != KVQ_OK) return s;
  if ((s = check_cache(*cfg, cache)) != KVQ_OK) return s;
  return cuda_status(cudaMemsetAsync(cache->seq_len, 0, seq_region_bytes(*cfg),
                                     static_cast<cudaStream_t>(stream)),
                     "kvq_cache_reset");
}

kvq_status kvq_pack(const kvq_config* cfg, const kvq_cache* cache, const uint16_t* k_new,
                    const uint16_t* v_new, int32_t n_new, int32_t batch_begin,
                    int32_t batch_count, void* stream) {
  kvq_status s = check_config(cfg);
  if (s != KVQ_OK) return s;
  if ((s = check_cache(*cfg, cache)) != KVQ_OK) return s;
  if (!k_new || !v_new) return fail(KVQ_ERR_ARG, "k_new / v_new is NULL");
  if (!aligned16(k_new) || !aligned16(v_new))
    return fail(KVQ_ERR_ALIGN, "k_new / v_new must be 16-byte aligned");
  if (n_new < 1) return fail(KVQ_ERR_ARG, "n_new must be >= 1 (got %d)", n_new);
  if (n_new > cfg->max_len)
    return fail(KVQ_ERR_CAPACITY, "n_new (%d) exceeds max_len (%d)", n_new, cfg->max_len);
  if (batch_begin < 0 || batch_count < 1 || batch_begin + batch_count > cfg->batch)
    return fail(KVQ_ERR_SHAPE, "batch range [%d, %d) outside [0, %d)", batch_begin,
                batch_begin + batch_count, cfg->batch);
  Dims d = make_dims(*cfg);
  trace("kvq_pack batch [%d, %d) n_new %d bits K%dV%d", batch_begin, batch_begin + batch_count,
        n_new, d.bits_k, d.bits_v);
  return cuda_status(launch_pack(d, *cache, reinterpret_cast<const __half*>(k_new),
                                 reinterpret_cast<const __half*>(v_new), n_new, batch_begin,
                                 batch_count, static_cast<cudaStream_t>(stream)),
                     "kvq_pack launch");
}

int32_t kvq_attn_splits_for_lengths(const kvq_config* cfg, const int32_t* lengths) {
  if (check_config(cfg) != KVQ_OK) return -1;
  if (!lengths) {
    fail(KVQ_ERR_ARG, "lengths is NULL");
    return -1;
  }
  for (int b = 0; b < cfg->batch; ++b)
    if (lengths[b] < 0 || lengths[b] > cfg->max_len) {
      fail(KVQ_ERR_ARG, "lengths[%d] = %d outside [0, max_len]", b, lengths[b]);
      return -1;
    }
  return attn_splits_for_lengths(make_dims(*cfg), sm_count(), lengths);
}

int32_t kvq_attn_default_splits(const kvq_config* cfg) {
  if (check_config(cfg) != KVQ_OK) return 0;
  return default_splits(*cfg);
}

size_t kvq_attn_workspace_bytes(const kvq_config* cfg, int32_t n_splits) {
  if (check_config(cfg) != KVQ_OK) return 0;
  if (n_splits < 0 || n_splits > kMaxSplits - 1) {
    set_error("n_splits must be in [0, %d] (got %d)", kMaxSplits - 1, n_splits);
    return 0;
  }
  return attn_ws_bytes(make_dims(*cfg), resolve_splits(n_splits));
}

kvq_status kvq_workspace_init(void* workspace, size_t ws_bytes, void* stream) {
  if (!workspace || ws_bytes == 0) return fail(KVQ_ERR_ARG, "workspace is NULL or empty");
  return cuda_status(cudaMemsetAsync(workspace, 0, ws_bytes, static_cast<cudaStream_t>(stream)),
                     "kvq_workspace_init");
}

}  // extern "C"

namespace kvq {

// Shared host validation of the decode-attention calls; on success *scale_log2
// holds softmax_scale (0 -> 1/sqrt(128)) times log2(e) and *n_splits the
// split count to launch.
static kvq_status check_attn_call(const kvq_config* cfg, const kvq_cache* cache,
                                  const void* q, const void* out, float softmax_scale,
                                  int32_t* n_splits, void* workspace, size_t ws_bytes,
                                  float* scale_log2) {
  kvq_status s = check_config(cfg);
  if (s != KVQ_OK) return s;
  if ((s = check_cache(*cfg, cache)) != KVQ_OK) return s;
  if (!q || !out) return fail(KVQ_ERR_ARG, "q / out is NULL");
  if (!aligned16(q) || !aligned16(out)) return fail(KVQ_ERR_ALIGN, "q / out must be 16-byte aligned");
  if (!(softmax_scale >= 0.0f) || isinf(softmax_scale))
    return fail(KVQ_ERR_ARG, "softmax_scale must be finite and >= 0");
  if (*n_splits < 0 || *n_splits > kMaxSplits - 1)
    return fail(KVQ_ERR_ARG, "n_splits must be in [0, %d] (got %d)", kMaxSplits - 1, *n_splits);
  *n_splits = resolve_splits(*n_splits);
  const size_t need = attn_ws_bytes(make_dims(*cfg), *n_splits);
  if (!workspace) return fail(KVQ_ERR_ARG, "workspace is NULL");
  if (!aligned16(workspace)) return fail(KVQ_ERR_ALIGN, "workspace must be 16-byte aligned");
  if (ws_bytes < need)
    return fail(KVQ_ERR_CAPACITY, "workspace too small: %zu < %zu bytes", ws_bytes, need);
  const float scale = softmax_scale == 0.0f ? 1.0f / sqrtf((float)kHeadDim) : softmax_scale;
  *scale_log2 = scale * 1.4426950408889634f;
  return KVQ_OK;
}

static kvq_status decode_attn(const kvq_config* cfg, const kvq_cache* cache, const uint16_t* q,
                              void* out, int out_f16, float softmax_scale, int32_t n_splits,
                              void* workspace, size_t ws_bytes, void* stream) {
  float sl2 = 0.0f;
  kvq_status s = check_attn_call(cfg, cache, q, out, softmax_scale, &n_splits, workspace,
                                 ws_bytes, &sl2);
  if (s != KVQ_OK) return s;
  Dims d = make_dims(*cfg);
  trace("kvq_decode_attn%s batch %d heads %d/%d bits K%dV%d grid (%d) x 512, %s %d",
        out_f16 ? "" : "_f32", d.batch, d.hq, d.hkv, d.bits_k, d.bits_v,
        n_splits > 0 ? n_splits * d.batch * d.hkv : -n_splits,
        n_splits > 0 ? "splits" : "flat plan, CTAs", n_splits > 0 ? n_splits : -n_splits);
  const cudaStream_t st = static_cast<cudaStream_t>(stream);
  const __half* qh = reinterpret_cast<const __half*>(q);
  return cuda_status(n_splits > 0
                         ? launch_decode_attn_split(d, *cache, qh, out, out_f16, sl2, n_splits,
                                                    workspace, st)
                         : launch_decode_attn(d, *cache, qh, out, out_f16, sl2, -n_splits,
                                              workspace, st),
                     "kvq_decode_attn launch");
}

static kvq_status decode_step(const kvq_config* cfg, const kvq_cache* cache,
                              const uint16_t* k_new, const uint16_t* v_new, const uint16_t* q,
                              void* out, int out_f16, float softmax_scale, int32_t n_splits,
                              void* workspace, size_t ws_bytes, void* stream) {
  if (!k_new || !v_new) return fail(KVQ_ERR_ARG, "k_new / v_new is NULL");
  if (!aligned16(k_new) || !aligned16(v_new))
    return fail(KVQ_ERR_ALIGN, "k_new / v_new must be 16-byte aligned");
  float sl2 = 0.0f;
  kvq_status s = check_attn_call(cfg, cache, q, out, softmax_scale, &n_splits, workspace,
                                 ws_bytes, &sl2);
  if (s != KVQ_OK) return s;
  Dims d = make_dims(*cfg);
  trace("kvq_decode_step%s batch %d heads %d/%d bits K%dV%d grid (%d) x 512, %s %d",
        out_f16 ? "" : "_f32", d.batch, d.hq, d.hkv, d.bits_k, d.bits_v,
        n_splits > 0 ? n_splits * d.batch * d.hkv : -n_splits,
        n_splits > 0 ? "splits" : "flat plan, CTAs", n_splits > 0 ? n_splits : -n_splits);
  const cudaStream_t st = static_cast<cudaStream_t>(stream);
  const __half* kh = reinterpret_cast<const __half*>(k_new);
  const __half* vh = reinterpret_cast<const __half*>(v_new);
  const __half* qh = reinterpret_cast<const __half*>(q);
  return cuda_status(n_splits > 0
                         ? launch_decode_step_split(d, *cache, kh, vh, qh, out, out_f16, sl2,
                                                    n_splits, workspace, st)
                         : launch_decode_step(d, *cache, kh, vh, qh, out, out_f16, sl2,
                                              -n_splits, workspace, st),
                     "kvq_decode_step launch");
}

}  // namespace kvq

extern "C" {

kvq_status kvq_decode_attn(const kvq_config* cfg, const kvq_cache* cache, const uint16_t* q,
                           uint16_t* out, float softmax_scale, int32_t n_splits,
                           void* workspace, size_t ws_bytes, void* stream) {
  return decode_attn(cfg, cache, q, out, 1, softmax_scale, n_splits, workspace, ws_bytes, stream);
}

kvq_status kvq_decode_attn_f32(const kvq_config* cfg, const kvq_cache* cache, const uint16_t* q,
                               float* out, float softmax_scale, int32_t n_splits,
                               void* workspace, size_t ws_bytes, void* stream) {
  return decode_attn(cfg, cache, q, out, 0, softmax_scale, n_splits, workspace, ws_bytes, stream);
}

kvq_status kvq_decode_step(const kvq_config* cfg, const kvq_cache* cache, const uint16_t* k_new,
                           const uint16_t* v_new, const uint16_t* q, uint16_t* out,
                           float softmax_scale, int32_t n_splits, void* workspace,
                           size_t ws_bytes, void* stream) {
  return decode_step(cfg, cache, k_new, v_new, q, out, 1, softmax_scale, n_splits, workspace,
                     ws_bytes, stream);
}

kvq_status kvq_decode_step_f32(const kvq_config* cfg, const kvq_cache* cache,
                               const uint16_t* k_new, const uint16_t* v_new, const uint16_t* q,
                               float* out, float softmax_scale, int32_t n_splits,
                               void* workspace, size_t ws_bytes, void* stream) {
  return decode_step(cfg, cache, k_new, v_new, q, out, 0, softmax_scale, n_splits, workspace,
                     ws_bytes, stream);
}

kvq_status kvq_decode_attn_noalloc(const kvq_config* cfg, const kvq_cache* cache,
                                   const uint16_t* q, float* out, float softmax_scale,
                                   int32_t n_splits, void* stream) {
  kvq_status s = check_config(cfg);
  if (s != KVQ_OK) return s;
  if ((s = check_cache(*cfg, cache)) != KVQ_OK) return s;
  if (!q || !out) return fail(KVQ_ERR_ARG, "q / out is NULL");
  if (!aligned16(q) || !aligned16(out)) return fail(KVQ_ERR_ALIGN, "q / out must be 16-byte aligned");
  if (!(softmax_scale >= 0.0f) || isinf(softmax_scale))
    return fail(KVQ_ERR_ARG, "softmax_scale must be finite and >= 0");
  if (n_splits < 0 || n_splits > kMaxSplits - 1)
    return fail(KVQ_ERR_ARG, "n_splits must be in [0, %d] (got %d)", kMaxSplits - 1, n_splits);
  n_splits = resolve_splits(n_splits);
  Dims d = make_dims(*cfg);
  const size_t need = attn_ws_bytes(d, n_splits);
  if (need > attn_static_scratch_bytes())
    return fail(KVQ_ERR_CAPACITY,
                "this config needs %zu bytes of scratch but the built-in array holds %zu; "
                "use kvq_decode_attn with a workspace, or fewer splits",
                need, attn_static_scratch_bytes());
  const float scale = softmax_scale == 0.0f ? 1.0f / sqrtf((float)kHeadDim) : softmax_scale;
  return cuda_status(launch_decode_attn_static(d, *cache, reinterpret_cast<const __half*>(q),
                                               out,
                                               scale * 1.4426950408889634f, n_splits,
                                               static_cast<cudaStream_t>(stream)),
                     "kvq_decode_attn_noalloc launch");
}

static kvq_status check_dgap(const dgap_params* p, int32_t batch, int32_t vocab) {
  if (!p) return fail(KVQ_ERR_ARG, "params is NULL");
  if (batch < 1 || vocab < 1) return fail(KVQ_ERR_SHAPE, "batch and vocab must be >= 1");
  if (p->K < 2 || p->K > kMaxK)
    return fail(KVQ_ERR_UNSUPPORTED, "K must be in [2, %d] (got %d)", kMaxK, p->K);
  if (p->K >= vocab) return fail(KVQ_ERR_SHAPE, "K (%d) must be < vocab (%d)", p->K, vocab);
  if (p->hidden < 1 || p->hidden > kMaxHidden)
    return fail(KVQ_ERR_UNSUPPORTED, "hidden must be in [1, %d] (got %d)", kMaxHidden, p->hidden);
  if (isnan(p->tau)) return fail(KVQ_ERR_ARG, "tau is NaN");
  if ((long long)batch * vocab > (1LL << 40)) return fail(KVQ_ERR_SHAPE, "logits too large");
  if (dgap_chunks(vocab) > dgap_max_chunks())
    return fail(KVQ_ERR_UNSUPPORTED, "vocab must be <= %d", dgap_max_chunks() * 4096);
  return KVQ_OK;
}

size_t dgap_workspace_bytes(int32_t batch, int32_t vocab, const dgap_params* p) {
  if (check_dgap(p, batch, vocab) != KVQ_OK) return 0;
  return dgap_workspace_bytes_impl(batch, vocab, p->K);
}

kvq_status dgap_restore(const dgap_params* p, float* logits, int32_t batch, int32_t vocab,
                        int32_t* topk_idx, float* topk_val, float* risk, uint8_t* gate,
                        int32_t* next_token, float* features, void* workspace, size_t ws_bytes,
                        void* stream) {
  kvq_status s = check_dgap(p, batch, vocab);
  if (s != KVQ_OK) return s;
  if (!p->det_w1 || !p->det_b1 || !p->det_w2 || !p->det_b2 || !p->cor_w1 || !p->cor_b1 ||
      !p->cor_w2 || !p->cor_b2)
    return fail(KVQ_ERR_ARG, "a DGAP weight pointer is NULL");
  if (!logits || !topk_idx || !topk_val || !risk || !gate)
    return fail(KVQ_ERR_ARG, "an output pointer is NULL");
  if (!aligned16(logits)) return fail(KVQ_ERR_ALIGN, "logits must be 16-byte aligned");
  if (!workspace) return fail(KVQ_ERR_ARG, "workspace is NULL");
  if (!aligned16(workspace)) return fail(KVQ_ERR_ALIGN, "workspace must be 16-byte aligned");
  const size_t need = dgap_workspace_bytes_impl(batch, vocab, p->K);
  if (ws_bytes < need)
    return fail(KVQ_ERR_CAPACITY, "workspace too small: %zu < %zu bytes", ws_bytes, need);
  DgapDims d;
  d.batch = batch;
  d.vocab = vocab;
  d.K = p->K;
  d.hidden = p->hidden;
  d.n_chunks = dgap_chunks(vocab);
  if (p->tau >= 1.0f)
    d.logit_tau = INFINITY;
  else if (p->tau <= 0.0f)
    d.logit_tau = -INFINITY;
  else
    d.logit_tau = (float)log((double)p->tau / (1.0 - (double)p->tau));
  trace("dgap_restore batch %d vocab %d K %d hidden %d tau %g grid (%d, %d) x 256", batch, vocab,
        p->K, p->hidden, (double)p->tau, d.n_chunks, batch);
  return cuda_status(launch_dgap(d, *p, logits, topk_idx, topk_val, risk, gate, next_token,
                                 features, workspace, static_cast<cudaStream_t>(stream)),
                     "dgap_restore launch");
}

kvq_status kvq_selftest_wait_timeout(uint32_t* flag, void* stream) {
  if (!flag) return fail(KVQ_ERR_ARG, "flag is NULL");
  if ((reinterpret_cast<uintptr_t>(flag) & 3u) != 0) return fail(KVQ_ERR_ALIGN, "flag must be 4-byte aligned");
  // about 10 ms at the SM clock: the copy waits' loop with a short limit
  return cuda_status(launch_wait_selftest(reinterpret_cast<unsigned*>(flag), 20000000LL,
                                          static_cast<cudaStream_t>(stream)),
                     "kvq_selftest_wait_timeout launch");
}

int32_t kvq_drift_max_vocab(void) { return drift_max_vocab(); }

kvq_status kvq_drift_metrics(const float* z_fp, const float* z_q, int32_t rows, int32_t vocab,
                             const kvq_drift_params* p, int32_t* m_t, float* c_t, float* d_loc,
                             uint8_t* y_t, float* cov, void* stream) {
  if (!p) return fail(KVQ_ERR_ARG, "params is NULL");
  if (!z_fp || !z_q) return fail(KVQ_ERR_ARG, "z_fp / z_q is NULL");
  if (!m_t || !c_t || !d_loc || !y_t || !cov) return fail(KVQ_ERR_ARG, "an output pointer is NULL");
  if (rows < 1 || rows > 65535) return fail(KVQ_ERR_SHAPE, "rows must be in [1, 65535] (got %d)", rows);
  if (vocab < 1) return fail(KVQ_ERR_SHAPE, "vocab must be >= 1 (got %d)", vocab);
  if (vocab > drift_max_vocab())
    return fail(KVQ_ERR_UNSUPPORTED, "vocab must be <= %d (got %d)", drift_max_vocab(), vocab);
  if (!(p->alpha > 0.0f && p->alpha <= 1.0f))
    return fail(KVQ_ERR_ARG, "alpha must be in (0, 1] (got %g)", (double)p->alpha);
  if (p->k_max < 1 || p->k_max > drift_max_kcov() || p->k_max > vocab)
    return fail(KVQ_ERR_ARG, "k_max must be in [1, min(%d, vocab)] (got %d)", drift_max_kcov(),
                p->k_max);
  if (p->window < 1 || p->window > p->k_max)
    return fail(KVQ_ERR_ARG, "window must be in [1, k_max] (got %d)", p->window);
  if (!isfinite(p->eps) || !isfinite(p->rho_c))
    return fail(KVQ_ERR_ARG, "eps and rho_c must be finite");
  trace("kvq_drift_metrics rows %d vocab %d alpha %g window %d k_max %d grid (8, %d) x 512, "
        "clusters of 8", rows, vocab, (double)p->alpha, p->window, p->k_max, rows);
  return cuda_status(launch_drift(z_fp, z_q, rows, vocab, *p, m_t, c_t, d_loc, y_t, cov,
                                  static_cast<cudaStream_t>(stream)),
                     "kvq_drift_metrics launch");
}

kvq_status kvq_drift_window(const float* cov, int32_t rows, int32_t k_max, float rho_k,
                            float* mean_cov, int32_t* k_b, void* stream) {
  if (!cov || !mean_cov || !k_b) return fail(KVQ_ERR_ARG, "a pointer is NULL");
  if (rows < 1) return fail(KVQ_ERR_SHAPE, "rows must be >= 1 (got %d)", rows);
  if (k_max < 1 || k_max > drift_max_kcov())
    return fail(KVQ_ERR_ARG, "k_max must be in [1, %d] (got %d)", drift_max_kcov(), k_max);
  if (!isfinite(rho_k)) return fail(KVQ_ERR_ARG, "rho_k must be finite");
  return cuda_status(launch_drift_window(cov, rows, k_max, rho_k, mean_cov, k_b,
                                         static_cast<cudaStream_t>(stream)),
                     "kvq_drift_window launch");
}

}  // extern "C"
