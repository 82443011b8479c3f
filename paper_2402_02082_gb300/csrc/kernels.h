// Host-side launch interface between the C ABI (abi.cu) and the kernels.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace glide {

constexpr int kMaxBatch = 1024;   // sequences per call (per-CTA tile table lives in shared memory)
constexpr int kMaxTree = 64;      // tree nodes (one 64-bit ancestor mask per node)
constexpr int kRowTile = 64;      // query rows of a slab one verification CTA serves
constexpr int kMaxRows = 256;     // query rows per slab (n nodes x H / H_kv heads): up to four row tiles
constexpr int kMaxCtas = 1024;    // CTAs (or claimed chunks) per attention launch (bounds the partial slots)
constexpr int kCrossPartials = 8; // cross-attention partials per slot: one per consumer warp
constexpr int kCapeMaxSet = 7;    // largest expansion set: S(p) <= 7, fixed sizes up to 7

struct AttnArgs {
  const void* q;
  const void* K;
  const void* V;
  const int32_t* kv_len;
  const int32_t* parent;  // tree only
  float* out;
  void* ws;
  int B, H, D, S_cap;
  int nq;                 // queries per (b, h): 1 for cross-attention, n for the tree
  int Hkv;                // cached (key/value) heads; H % Hkv == 0, H / Hkv query heads per cached head
  int tree;               // 1: the nq tree keys follow the prefix (verification); 0: prefix only
  int block_L;            // > 0: the training-time block mask with blocks of block_L positions
  int T;                  // block mask: positions per sequence (queries [B, T, H, D]); kv_len = lengths
  int max_kv_len;
  int dtype;              // 0 bf16, 1 f32
  float scale;            // already resolved (never 0)
  unsigned flags;
  int max_ctas;           // 0 = automatic
};

struct AcceptArgs {
  const int32_t* draft;
  const int32_t* parent;
  const float* logits;
  int B, n, V;
  int32_t* path;
  int32_t* len;
  int32_t* bonus;
  void* ws;
};

struct CapeArgs {
  const float* probs;     // [B, gamma, V]
  const int32_t* root;    // [B]
  int B, gamma, V;
  int max_tokens;         // gamma .. kMaxTree - 1
  int fixed_k;            // -1: S(p); else 0 .. kCapeMaxSet
  int32_t* tokens;        // [B, 1 + max_tokens]
  int32_t* parent;        // [B, 1 + max_tokens]
  int32_t* n_nodes;       // [B]
  float* conf;            // [B, gamma] or null
  void* ws;
};

struct CompactArgs {
  void* K;
  void* V;
  const int32_t* kv_len;
  const int32_t* path;
  const int32_t* len;
  int32_t* new_kv_len;
  int layers;
  long long layer_stride;  // elements between layers
  int B, H, D, S_cap, n;
  int dtype;               // 0 bf16, 1 f32
};

struct SampleArgs {
  const int32_t* draft;   // [B, gamma]
  const float* q;         // [B, gamma, V]
  const float* logits;    // [B, gamma + 1, V]
  const float* u;         // [B, gamma + 1]
  int B, gamma, V;
  int32_t* n_acc;         // [B]
  int32_t* next_tok;      // [B]
  void* ws;
};

int sm_count();  // multiprocessors of the current device (cached per device)

cudaError_t launch_cross_attn(const AttnArgs& a, cudaStream_t st);
cudaError_t launch_tree_attn_fma(const AttnArgs& a, cudaStream_t st);
// Returns cudaErrorNotSupported when the tensor-core kernel does not apply to `a`.
cudaError_t launch_tree_attn_tc(const AttnArgs& a, cudaStream_t st);
// Tree verification in 128-row tiles (slabs of more than 64 query rows whose
// head group divides 128); cudaErrorNotSupported where it does not apply.
cudaError_t launch_tree_attn_wide(const AttnArgs& a, cudaStream_t st);
cudaError_t launch_tree_accept(const AcceptArgs& a, cudaStream_t st);
// Training-time block-mask cross-attention (block_L > 0, T positions per sequence).
cudaError_t launch_block_attn(const AttnArgs& a, cudaStream_t st);

cudaError_t launch_cape_expand(const CapeArgs& a, cudaStream_t st);
cudaError_t launch_kv_compact(const CompactArgs& a, cudaStream_t st);
cudaError_t launch_spec_sample(const SampleArgs& a, cudaStream_t st);

size_t accept_workspace_bytes(int B, int n);
size_t cape_workspace_bytes(int B, int gamma, int V);
size_t sample_workspace_bytes(int B, int gamma);

}  // namespace glide
