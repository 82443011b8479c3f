// C ABI of libglide (declared in include/glide.h): host-side argument checks,
// workspace sizing and dispatch to the kernels.  Nothing here computes any
// part of the path; every step runs in the kernels.
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include "../../include/glide.h"
#include "common.cuh"
#include "kernels.h"

namespace glide {

int sm_count() {
  static int cached_dev = -1;
  static int cached = 0;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 1;
  if (dev != cached_dev) {
    int v = 0;
    if (cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || v < 1) v = 1;
    cached = v;
    cached_dev = dev;
  }
  return cached;
}

}  // namespace glide

namespace {

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Cached (key/value) heads: H_kv, or H when it is 0.
int hkv(const glide_attn_desc* d) { return d->H_kv > 0 ? d->H_kv : d->H; }

bool desc_ok(const glide_attn_desc* d) {
  if (!d) return false;
  if (d->B < 1 || d->B > glide::kMaxBatch) return false;
  if (d->H < 1 || d->H > 65535) return false;
  if (d->H_kv < 0 || d->H_kv > d->H || d->H % hkv(d) != 0) return false;
  if (d->D != 64 && d->D != 128) return false;
  if (d->S_cap < 1) return false;
  if (d->dtype != GLIDE_BF16 && d->dtype != GLIDE_F32) return false;
  if (!(d->scale >= 0.f) || isinf(d->scale)) return false;  // rejects NaN and negatives
  if (d->max_ctas < 0) return false;
  // every element offset must fit comfortably in 63 bits
  const double elems = (double)d->B * d->H * (double)d->S_cap * d->D;  // >= the cache (H_kv <= H)
  if (elems > 4.0e18) return false;
  return true;
}

size_t attn_ws_bytes(const glide_attn_desc* d, int nq) {
  // partial slots: one per (share or chunk, b, h) pair index; a tree slot holds
  // nq query rows, a cross-attention slot one row per consumer warp
  // (with grouped-query attention a slab is a (b, cached head) and holds
  // nq x group query rows)
  const size_t slots = (size_t)glide::kMaxCtas + (size_t)d->B * hkv(d);
  const size_t q_rows = (size_t)nq * (d->H / hkv(d));
  const size_t rows = q_rows > (size_t)glide::kCrossPartials ? q_rows : (size_t)glide::kCrossPartials;
  return glide::WsLayout::partials_off(d->B, d->H) + slots * rows * (d->D + 2) * sizeof(float);
}

glide::AttnArgs make_args(const glide_attn_desc* d, const void* q, const void* K, const void* V,
                          const int32_t* kv_len, const int32_t* parent, float* out, void* ws, int nq,
                          int max_kv_len) {
  glide::AttnArgs a;
  a.q = q; a.K = K; a.V = V; a.kv_len = kv_len; a.parent = parent; a.out = out; a.ws = ws;
  a.B = d->B; a.H = d->H; a.D = d->D; a.S_cap = d->S_cap; a.nq = nq; a.max_kv_len = max_kv_len;
  a.Hkv = hkv(d);
  a.tree = parent != nullptr ? 1 : 0;
  a.block_L = 0;
  a.T = 0;
  a.dtype = d->dtype == GLIDE_BF16 ? 0 : 1;
  a.scale = d->scale > 0.f ? d->scale : 1.0f / sqrtf((float)d->D);
  a.flags = d->flags;
  a.max_ctas = d->max_ctas;
  return a;
}

glide_status from_cuda(cudaError_t e) { return e == cudaSuccess ? GLIDE_OK : GLIDE_ERR_CUDA; }

}  // namespace

extern "C" {

int32_t glide_abi_version(void) { return GLIDE_ABI_VERSION; }

const char* glide_status_str(glide_status s) {
  switch (s) {
    case GLIDE_OK: return "ok";
    case GLIDE_ERR_INVALID: return "invalid argument";
    case GLIDE_ERR_UNSUPPORTED: return "unsupported shape or type";
    case GLIDE_ERR_CUDA: return "CUDA error";
    case GLIDE_ERR_DEVICE_TIMEOUT: return "kernel wait timed out";
  }
  return "unknown status";
}

size_t glide_attn_workspace_bytes(const glide_attn_desc* desc, int32_t n_queries) {
  if (!desc_ok(desc) || n_queries < 1 || n_queries > glide::kMaxTree) return 0;
  if (n_queries * (desc->H / hkv(desc)) > glide::kMaxRows) return 0;
  return attn_ws_bytes(desc, n_queries);
}

size_t glide_accept_workspace_bytes(int32_t B, int32_t n) {
  if (B < 1 || n < 1 || n > glide::kMaxTree) return 0;
  return glide::accept_workspace_bytes(B, n);
}

size_t glide_cape_workspace_bytes(int32_t B, int32_t gamma, int32_t V) {
  if (B < 1 || gamma < 1 || gamma > glide::kMaxTree - 1 || V < 1) return 0;
  return glide::cape_workspace_bytes(B, gamma, V);
}

glide_status glide_cross_attn(const glide_attn_desc* desc, const void* q_draft, const void* K_cache,
                              const void* V_cache, const int32_t* kv_len, int32_t max_kv_len, float* out,
                              void* workspace, size_t workspace_bytes, glide_stream_t stream) {
  if (!desc_ok(desc)) return GLIDE_ERR_INVALID;
  if (!q_draft || !K_cache || !V_cache || !kv_len || !out || !workspace) return GLIDE_ERR_INVALID;
  if (!aligned16(q_draft) || !aligned16(K_cache) || !aligned16(V_cache) || !aligned16(out) ||
      !aligned16(workspace) || (reinterpret_cast<uintptr_t>(kv_len) & 3u))
    return GLIDE_ERR_INVALID;
  if (max_kv_len < 1 || max_kv_len > desc->S_cap) return GLIDE_ERR_INVALID;
  if (workspace_bytes < attn_ws_bytes(desc, 1)) return GLIDE_ERR_INVALID;
  glide::AttnArgs a = make_args(desc, q_draft, K_cache, V_cache, kv_len, nullptr, out, workspace, 1, max_kv_len);
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  if (a.Hkv == a.H) return from_cuda(glide::launch_cross_attn(a, st));
  // Grouped-query attention: a cached head serves H / H_kv draft queries, so
  // one pass over its keys is a small dense contraction -- the verification
  // kernels without tree keys, with the group's queries as their rows.
  if (a.H / a.Hkv > glide::kMaxRows) return GLIDE_ERR_UNSUPPORTED;
  if (!(a.flags & GLIDE_FLAG_FORCE_FMA)) {
    if (!(a.flags & GLIDE_FLAG_TILE64)) {
      cudaError_t e = glide::launch_tree_attn_wide(a, st);
      if (e != cudaErrorNotSupported) return from_cuda(e);
    }
    cudaError_t e = glide::launch_tree_attn_tc(a, st);
    if (e != cudaErrorNotSupported) return from_cuda(e);
  }
  return from_cuda(glide::launch_tree_attn_fma(a, st));
}

glide_status tree_verify_attn(const glide_attn_desc* desc, const void* q_tree, int32_t n, const int32_t* parent_idx,
                              const void* K_cache, const void* V_cache, const int32_t* kv_len, int32_t max_kv_len,
                              float* out, void* workspace, size_t workspace_bytes, glide_stream_t stream) {
  if (!desc_ok(desc)) return GLIDE_ERR_INVALID;
  if (n < 1 || n > glide::kMaxTree) return GLIDE_ERR_INVALID;
  if (!q_tree || !parent_idx || !K_cache || !V_cache || !kv_len || !out || !workspace) return GLIDE_ERR_INVALID;
  if (!aligned16(q_tree) || !aligned16(K_cache) || !aligned16(V_cache) || !aligned16(out) ||
      !aligned16(workspace) || (reinterpret_cast<uintptr_t>(kv_len) & 3u) ||
      (reinterpret_cast<uintptr_t>(parent_idx) & 3u))
    return GLIDE_ERR_INVALID;
  if (max_kv_len < 0 || (long long)max_kv_len + n > desc->S_cap) return GLIDE_ERR_INVALID;
  if (n * (desc->H / hkv(desc)) > glide::kMaxRows) return GLIDE_ERR_UNSUPPORTED;  // query rows of a slab
  if (workspace_bytes < attn_ws_bytes(desc, n)) return GLIDE_ERR_INVALID;
  glide::AttnArgs a = make_args(desc, q_tree, K_cache, V_cache, kv_len, parent_idx, out, workspace, n, max_kv_len);
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  if (!(a.flags & GLIDE_FLAG_FORCE_FMA)) {
    if (!(a.flags & GLIDE_FLAG_TILE64)) {  // grouped-query slabs and slabs of more than 64 rows: 128-row tiles
      cudaError_t e = glide::launch_tree_attn_wide(a, st);
      if (e != cudaErrorNotSupported) return from_cuda(e);
    }
    cudaError_t e = glide::launch_tree_attn_tc(a, st);
    if (e != cudaErrorNotSupported) return from_cuda(e);
  }
  return from_cuda(glide::launch_tree_attn_fma(a, st));
}

glide_status tree_accept(const int32_t* draft_tokens, const int32_t* parent_idx, const float* target_logits,
                         int32_t B, int32_t n, int32_t V, int32_t* path, int32_t* len, int32_t* bonus,
                         void* workspace, size_t workspace_bytes, glide_stream_t stream) {
  if (B < 1 || n < 1 || n > glide::kMaxTree || V < 1) return GLIDE_ERR_INVALID;
  if (!draft_tokens || !parent_idx || !target_logits || !path || !len || !bonus || !workspace)
    return GLIDE_ERR_INVALID;
  if (!aligned16(target_logits) || !aligned16(workspace) || (reinterpret_cast<uintptr_t>(draft_tokens) & 3u) ||
      (reinterpret_cast<uintptr_t>(parent_idx) & 3u) || (reinterpret_cast<uintptr_t>(path) & 3u) ||
      (reinterpret_cast<uintptr_t>(len) & 3u) || (reinterpret_cast<uintptr_t>(bonus) & 3u))
    return GLIDE_ERR_INVALID;
  if (workspace_bytes < glide::accept_workspace_bytes(B, n)) return GLIDE_ERR_INVALID;
  glide::AcceptArgs a;
  a.draft = draft_tokens; a.parent = parent_idx; a.logits = target_logits;
  a.B = B; a.n = n; a.V = V; a.path = path; a.len = len; a.bonus = bonus; a.ws = workspace;
  return from_cuda(glide::launch_tree_accept(a, reinterpret_cast<cudaStream_t>(stream)));
}

glide_status cape_expand(const float* probs, const int32_t* root_token, int32_t B, int32_t gamma, int32_t V,
                         int32_t max_tokens, int32_t fixed_k, int32_t* draft_tokens, int32_t* parent_idx,
                         int32_t* n_nodes, float* conf, void* workspace, size_t workspace_bytes,
                         glide_stream_t stream) {
  if (B < 1 || gamma < 1 || V < 1) return GLIDE_ERR_INVALID;
  if (max_tokens < gamma || max_tokens > glide::kMaxTree - 1) return GLIDE_ERR_INVALID;
  if (fixed_k < -1) return GLIDE_ERR_INVALID;
  if (fixed_k > glide::kCapeMaxSet) return GLIDE_ERR_UNSUPPORTED;
  if (!probs || !root_token || !draft_tokens || !parent_idx || !n_nodes || !workspace) return GLIDE_ERR_INVALID;
  if (!aligned16(probs) || !aligned16(workspace) || (reinterpret_cast<uintptr_t>(root_token) & 3u) ||
      (reinterpret_cast<uintptr_t>(draft_tokens) & 3u) || (reinterpret_cast<uintptr_t>(parent_idx) & 3u) ||
      (reinterpret_cast<uintptr_t>(n_nodes) & 3u) || (reinterpret_cast<uintptr_t>(conf) & 3u))
    return GLIDE_ERR_INVALID;
  if (workspace_bytes < glide::cape_workspace_bytes(B, gamma, V)) return GLIDE_ERR_INVALID;
  glide::CapeArgs a;
  a.probs = probs; a.root = root_token; a.B = B; a.gamma = gamma; a.V = V;
  a.max_tokens = max_tokens; a.fixed_k = fixed_k;
  a.tokens = draft_tokens; a.parent = parent_idx; a.n_nodes = n_nodes; a.conf = conf; a.ws = workspace;
  return from_cuda(glide::launch_cape_expand(a, reinterpret_cast<cudaStream_t>(stream)));
}

glide_status glide_kv_compact(const glide_attn_desc* desc, int32_t n_layers, int64_t layer_stride, void* K_cache,
                              void* V_cache, const int32_t* kv_len, int32_t n, const int32_t* path,
                              const int32_t* len, int32_t* new_kv_len, glide_stream_t stream) {
  if (!desc_ok(desc)) return GLIDE_ERR_INVALID;
  if (n < 1 || n > glide::kMaxTree || n > desc->S_cap) return GLIDE_ERR_INVALID;
  if (n_layers < 1) return GLIDE_ERR_INVALID;
  const int64_t layer_elems = (int64_t)desc->B * hkv(desc) * desc->S_cap * desc->D;  // the cache's heads
  if (n_layers > 1 && layer_stride < layer_elems) return GLIDE_ERR_INVALID;
  if ((double)n_layers * (double)(n_layers > 1 ? layer_stride : layer_elems) > 4.0e18) return GLIDE_ERR_INVALID;
  const int elt = desc->dtype == GLIDE_BF16 ? 2 : 4;
  if (n_layers > 1 && ((layer_stride * elt) & 15)) return GLIDE_ERR_INVALID;
  if (!K_cache || !V_cache || !kv_len || !path || !len || !new_kv_len) return GLIDE_ERR_INVALID;
  if (!aligned16(K_cache) || !aligned16(V_cache) || (reinterpret_cast<uintptr_t>(kv_len) & 3u) ||
      (reinterpret_cast<uintptr_t>(path) & 3u) || (reinterpret_cast<uintptr_t>(len) & 3u) ||
      (reinterpret_cast<uintptr_t>(new_kv_len) & 3u))
    return GLIDE_ERR_INVALID;
  if (new_kv_len == kv_len) return GLIDE_ERR_INVALID;
  glide::CompactArgs a;
  a.K = K_cache; a.V = V_cache; a.kv_len = kv_len; a.path = path; a.len = len; a.new_kv_len = new_kv_len;
  a.layers = n_layers; a.layer_stride = n_layers > 1 ? layer_stride : layer_elems;
  a.B = desc->B; a.H = hkv(desc); a.D = desc->D; a.S_cap = desc->S_cap; a.n = n;
  a.dtype = desc->dtype == GLIDE_BF16 ? 0 : 1;
  return from_cuda(glide::launch_kv_compact(a, reinterpret_cast<cudaStream_t>(stream)));
}

size_t glide_sample_workspace_bytes(int32_t B, int32_t gamma) {
  if (B < 1 || gamma < 1 || gamma > glide::kMaxTree - 1) return 0;
  return glide::sample_workspace_bytes(B, gamma);
}

glide_status spec_sample_accept(const int32_t* draft_tokens, const float* draft_probs, const float* target_logits,
                                const float* uniforms, int32_t B, int32_t gamma, int32_t V, int32_t* n_accepted,
                                int32_t* next_token, void* workspace, size_t workspace_bytes,
                                glide_stream_t stream) {
  if (B < 1 || gamma < 1 || gamma > glide::kMaxTree - 1 || V < 1) return GLIDE_ERR_INVALID;
  if ((double)B * (gamma + 1) * V > 4.0e18) return GLIDE_ERR_INVALID;
  if (!draft_tokens || !draft_probs || !target_logits || !uniforms || !n_accepted || !next_token || !workspace)
    return GLIDE_ERR_INVALID;
  if (!aligned16(target_logits) || !aligned16(workspace) || (reinterpret_cast<uintptr_t>(draft_probs) & 3u) ||
      (reinterpret_cast<uintptr_t>(draft_tokens) & 3u) || (reinterpret_cast<uintptr_t>(uniforms) & 3u) ||
      (reinterpret_cast<uintptr_t>(n_accepted) & 3u) || (reinterpret_cast<uintptr_t>(next_token) & 3u))
    return GLIDE_ERR_INVALID;
  if (workspace_bytes < glide::sample_workspace_bytes(B, gamma)) return GLIDE_ERR_INVALID;
  glide::SampleArgs a;
  a.draft = draft_tokens; a.q = draft_probs; a.logits = target_logits; a.u = uniforms;
  a.B = B; a.gamma = gamma; a.V = V; a.n_acc = n_accepted; a.next_tok = next_token; a.ws = workspace;
  return from_cuda(glide::launch_spec_sample(a, reinterpret_cast<cudaStream_t>(stream)));
}

size_t glide_block_attn_workspace_bytes(const glide_attn_desc* desc, int32_t T) {
  if (!desc_ok(desc) || T < 1 || T > desc->S_cap) return 0;
  return glide::WsLayout::kHeader;  // the status word
}

glide_status glide_block_cross_attn(const glide_attn_desc* desc, const void* q, int32_t T, int32_t L,
                                    const void* K_cache, const void* V_cache, const int32_t* seq_len, float* out,
                                    void* workspace, size_t workspace_bytes, glide_stream_t stream) {
  if (!desc_ok(desc)) return GLIDE_ERR_INVALID;
  if (T < 1 || T > desc->S_cap || L < 1) return GLIDE_ERR_INVALID;
  if (!q || !K_cache || !V_cache || !seq_len || !out || !workspace) return GLIDE_ERR_INVALID;
  if (!aligned16(q) || !aligned16(K_cache) || !aligned16(V_cache) || !aligned16(out) || !aligned16(workspace) ||
      (reinterpret_cast<uintptr_t>(seq_len) & 3u))
    return GLIDE_ERR_INVALID;
  if (desc->dtype != GLIDE_BF16) return GLIDE_ERR_UNSUPPORTED;
  if (workspace_bytes < glide::WsLayout::kHeader) return GLIDE_ERR_INVALID;
  glide::AttnArgs a = make_args(desc, q, K_cache, V_cache, seq_len, nullptr, out, workspace, 1, T);
  a.block_L = L;
  a.T = T;
  cudaError_t e = glide::launch_block_attn(a, reinterpret_cast<cudaStream_t>(stream));
  if (e == cudaErrorNotSupported) return GLIDE_ERR_UNSUPPORTED;
  return from_cuda(e);
}

glide_status glide_validate_tree(const int32_t* parent_idx_host, int32_t B, int32_t n, int32_t require_root0) {
  if (!parent_idx_host || B < 1 || n < 1) return GLIDE_ERR_INVALID;
  for (int32_t b = 0; b < B; ++b) {
    const int32_t* p = parent_idx_host + (size_t)b * n;
    for (int32_t i = 0; i < n; ++i) {
      if (p[i] < -1 || p[i] >= i) return GLIDE_ERR_INVALID;
      if (require_root0 && i > 0 && p[i] < 0) return GLIDE_ERR_INVALID;
    }
    if (require_root0 && p[0] != -1) return GLIDE_ERR_INVALID;
  }
  return GLIDE_OK;
}

glide_status glide_read_device_status(void* workspace, glide_stream_t stream) {
  if (!workspace || !aligned16(workspace)) return GLIDE_ERR_INVALID;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  unsigned word = 0;
  if (cudaMemcpyAsync(&word, workspace, sizeof(word), cudaMemcpyDeviceToHost, st) != cudaSuccess)
    return GLIDE_ERR_CUDA;
  if (cudaStreamSynchronize(st) != cudaSuccess) return GLIDE_ERR_CUDA;
  if (word == 0) return GLIDE_OK;
  const unsigned zero = 0;
  if (cudaMemcpyAsync(workspace, &zero, sizeof(zero), cudaMemcpyHostToDevice, st) != cudaSuccess)
    return GLIDE_ERR_CUDA;
  if (cudaStreamSynchronize(st) != cudaSuccess) return GLIDE_ERR_CUDA;
  return word == (unsigned)GLIDE_ERR_DEVICE_TIMEOUT ? GLIDE_ERR_DEVICE_TIMEOUT : GLIDE_ERR_CUDA;
}

}  // extern "C"
