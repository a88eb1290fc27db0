// Host-side launchers of the kvc kernels (defined in the .cu files) and the
// argument blocks they pass by value.
#pragma once

#include "kvc_internal.cuh"

namespace kvc {

// ---------------------------------------------------------------------------
// Launchers (defined in the .cu files).
// ---------------------------------------------------------------------------
struct AppendArgs {
  int32_t n_seq;
  int32_t total;
  int32_t pf_target;       // desired item count of the binary32 prefill's chunk list
  int32_t pf_min_blocks;
  int32_t sessions[MAX_SEQ];
  int32_t cu[MAX_SEQ + 1];
};

struct SeqArgs {
  int32_t n_seq;
  int32_t sessions[MAX_SEQ];
};

cudaError_t launch_init(const Dev& d, double rope_base, cudaStream_t s);
// single: every session of the call gets exactly one token (plan and K/V write in
// one launch).
cudaError_t launch_append(const Dev& d, const AppendArgs& a, const uint8_t* types, const void* k,
                          const void* v, bool single, cudaStream_t s);
cudaError_t launch_append_layers(const Dev& d, int total, int layer0, int n_layers, const void* k,
                                 const void* v, cudaStream_t s);
cudaError_t launch_evict(const Dev& d, const SeqArgs& a, int64_t* resident_out, cudaStream_t s);
cudaError_t launch_release(const Dev& d, const SeqArgs& a, cudaStream_t s);
cudaError_t launch_transcript(const Dev& d, int session, int cap, int32_t* pos_out, void* k_out,
                              void* v_out, int32_t* count, cudaStream_t s);
// new_k / new_v (optional): the fused per-layer write of the new tokens' K/V.
// epoch: tag of this launch's partial states (nonzero, never reused while tags
// of it may remain in the slots); 0 selects the fenced arrival instead.
cudaError_t launch_attn_decode(const Dev& d, int layer, const void* q, void* out, int n_seq,
                               bool pdl, cudaStream_t s, uint32_t epoch,
                               const void* new_k = nullptr, const void* new_v = nullptr);
// Stream-K decode kernel (kvc_attn_decode.cu): its grid (resident CTAs, capped by
// the partial slots) and its launch.
int decode_stream_k_grid(const Dev& d);
cudaError_t launch_attn_decode_streamk(const Dev& d, int layer, const CUtensorMap& map_lo,
                                       const CUtensorMap& map_hi, const void* q, void* out,
                                       float scale, int grid, int min_units, const void* new_k,
                                       const void* new_v, bool pdl, cudaStream_t s);
// Pair-split decode kernel (kvc_attn_decode_split.cu).  wide: the 16-warp shape
// (one CTA per SM; tensor-core pages for bfloat16), else the 4-warp shape.
int decode_split_slots(int esz, bool wide);          // resident CTAs in one wave
bool decode_split_uses_tma(int esz, bool wide);      // needs the pool's tensor maps
cudaError_t launch_attn_decode_split(const Dev& d, bool wide, int layer, const CUtensorMap& map_lo,
                                     const CUtensorMap& map_hi, const void* q, void* out,
                                     float scale, int k, uint32_t epoch, const void* new_k,
                                     const void* new_v, int n_pairs, bool pdl, cudaStream_t s);
// new_k / new_v (optional, bfloat16 only): the chunk's rows of this layer, written
// into the pool by the launch itself (the per-layer order).
cudaError_t launch_attn_prefill(const Dev& d, int layer, const void* q, void* out, int n_seq,
                                int max_t, bool pdl, cudaStream_t s, const void* new_k = nullptr,
                                const void* new_v = nullptr);
cudaError_t launch_attn_prefill_tc(const Dev& d, int layer, const CUtensorMap& lo,
                                   const CUtensorMap& hi, const void* q, void* out, int grid,
                                   bool pdl, cudaStream_t s, const void* new_k, const void* new_v);
const void* prefill_tc_kernel_ptr();
// Two 2-D views of the bfloat16 pool as rows of 128 elements (columns 0-63 and
// 64-127), 16-row boxes, 128-byte swizzle; cached per pool.  False if the driver
// entry point is missing or the encoding fails.
bool pool_tensor_maps(const Dev& d, CUtensorMap* lo, CUtensorMap* hi);
int prefill_tc_smem();
int prefill_tc_threads();
int noalloc_max_pairs();
cudaError_t launch_attn_decode_noalloc(const Dev& d, int layer, const void* q, void* out,
                                       int n_seq, cudaStream_t s);
int prefill_grid_ctas(const Dev& d);

}  // namespace kvc
