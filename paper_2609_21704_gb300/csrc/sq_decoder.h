// sq_decoder.h -- declarations of the decoder around the linear stack
// (sq_attention.cu): RMSNorm, RoPE + KV append, decode attention, cache
// rollback, embedding gather and the speculative bookkeeping.
#pragma once

#include "sq_internal.h"

namespace sq {

// sq_attention.cu: RMSNorm, RoPE + KV append, decode attention, rollback
cudaError_t launch_rmsnorm(const __half* x, const __half* gamma, int M, int64_t H, float eps, __half* y,
                           cudaStream_t st);
cudaError_t launch_kv_append(const __half* qkv, int B, int T, int Hq, int Hkv, const int32_t* pos0,
                             double theta, __half* kc, __half* vc, int64_t max_ctx, cudaStream_t st);
size_t attention_workspace_bytes(int B, int T, int Hq, int Hkv, int64_t max_ctx);
size_t attention_smem_bytes(int Q);
int attention_max_tokens();  // T limit of sq_kv_append / sq_attention
// kc_append / vc_append (the same caches as kc / vc, or null): append the
// new tokens' rotated keys and values in the same launch.
cudaError_t launch_attention(const __half* qkv, int B, int T, int Hq, int Hkv, const int32_t* pos0,
                             double theta, const __half* kc, const __half* vc, int64_t max_ctx,
                             __half* out, void* ws, cudaStream_t st, __half* kc_append = nullptr,
                             __half* vc_append = nullptr);
cudaError_t launch_kv_rollback(const int32_t* base, const int32_t* n, int B, int limit, int32_t* len,
                               cudaStream_t st);
cudaError_t launch_embed(const int32_t* ids, int M, int64_t ids_stride, const __half* table, int64_t V,
                         int64_t H, __half* out, cudaStream_t st);
cudaError_t launch_spec_commit(const int32_t* n, const int32_t* tokens, int ldt, int B, int K, int32_t* hist,
                               int cap, int32_t* len, int32_t* pos, int32_t* last2, cudaStream_t st);
cudaError_t launch_spec_drafts(const int32_t* samples, const int32_t* last2, int B, int K, int32_t* verify,
                               int32_t* draft, cudaStream_t st);
cudaError_t take_attn_status(uint32_t* bits);

}  // namespace sq
