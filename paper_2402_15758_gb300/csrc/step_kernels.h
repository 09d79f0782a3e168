// Launchers of the step-assembly kernels (internal to the library).
#pragma once

#include <cuda_runtime.h>

namespace chimera {

cudaError_t launch_trigram_gather(int dtype, const void* E, int d, int V, const int* n, const int* tok,
                                  int tok_stride, const int* topk, int K, int KMAX, int k, void* out,
                                  int B, int* err, float* zero, cudaStream_t s, float* zero2 = nullptr,
                                  long long zero2_floats = 0);
cudaError_t launch_hfull_store(int dtype, const float* dres, int d, void* headin, void* headin_lo, float* hlog,
                               float* zero, int V, int B, cudaStream_t s);
cudaError_t launch_tree_expand(const int* n, const int* tok, int tok_stride, const int* topk, int K, int KMAX,
                               const int* depth, const int* rank, int N, const int* ovr_flag, const int* ovr,
                               int* node_tok, int B, cudaStream_t s);
cudaError_t launch_accept(const int* n, int* tok, int tok_stride, const int* node_tok, const int* amax,
                          const int* child_start, const int* child, int N, int D1, int* path, int* Lacc,
                          int* bonus, int B, cudaStream_t s);
// Trigram cache: look up the trigram of draft sub-step k for every sequence (hits fill
// dres and set *skip when all hit), then store the misses after the encoder ran.
cudaError_t launch_trigram_lookup(const int* n, const int* tok, int tok_stride, const int* topk, int K, int KMAX, int k,
                                  int B, int d, int nsets, const unsigned long long* keys, int* stamp,
                                  const float* vals, float* dres, int* hit, int* slot, int* skip, int* clock,
                                  int* hit_log, cudaStream_t s);
cudaError_t launch_trigram_insert(const int* n, const int* tok, int tok_stride, const int* topk, int K, int KMAX, int k,
                                  int B, int d, unsigned long long* keys, int* stamp, float* vals, const float* dres,
                                  const int* hit, const int* slot, const int* clock, float* htri_log, cudaStream_t s);
// Typical acceptance over the verify logits (stats: per row max, log-sum-exp, entropy).
cudaError_t launch_accept_typical(const int* n, int* tok, int tok_stride, const int* node_tok, const int* amax,
                                  const float* logits, int V, const float* stats, const int* parent, const int* depth,
                                  int N, int D1, float eps, float delta, int* path, int* Lacc, int* bonus, int B,
                                  cudaStream_t s);
cudaError_t launch_compact(void* pool, long long layer_stride_bytes, int n_layers, int H, int planes, int row_bytes,
                           const int* n, const int* path, const int* Lacc, int D1, const int* page_table,
                           int max_pages, int B, cudaStream_t s);
cudaError_t launch_gather_hidden(int dtype, const float* hfin, int d, int N, const int* path, const int* Lacc,
                                 int D1, float* hsel, void* headin, void* headin_lo, int B, cudaStream_t s);
cudaError_t launch_finalize(int* n, int* tok, int tok_stride, const int* Lacc, const int* bonus, int* count_log,
                            int log_cap, int* step, int B, cudaStream_t s);
cudaError_t launch_prefill_advance(int dtype, const float* hfin, int d, int rows_per_seq, const int* valid,
                                   const int* last, int* n, void* headin, void* headin_lo, int B, cudaStream_t s);
cudaError_t launch_set_root(const int* n, int* tok, int tok_stride, const int* amax, int B, cudaStream_t s);

}  // namespace chimera
