// Dispatch of a decode attention call (one token per session) between the three
// kernel shapes, by the number of (session, KV head) pairs it has:
//   - pair split, 16-warp CTAs (one per SM): every pair gets k >= 5 CTAs in one
//     wave (at most 3 sessions of 8 KV heads on 152 SMs); for bfloat16 the pages run
//     on the tensor cores;
//   - pair split, 4-warp CTAs (three per SM, tensor-core pages for bfloat16): every
//     pair gets k >= 1 CTAs in one wave (with k = 1 a pair needs no merge);
//   - stream-K over (session, KV head, page) units, tensor-core pages for bfloat16:
//     the rest (more pairs than the 4-warp shape's resident CTAs, e.g. the full-batch
//     rounds of 64 sessions).
#include <cstring>

#include "kvc_launch.cuh"

namespace kvc {

namespace {

constexpr int MAX_PARTS = 64;      // partial states per pair (both pair-split shapes)
constexpr float LOG2E = 1.4426950408889634f;
// Minimum (session, kv head, page) units per CTA of the stream-K split.
constexpr int DEC_MIN_UNITS = 12;
// The pair-split kernel takes calls whose pairs each get at least this many CTAs
// in one wave: with 16-warp CTAs (one per SM) first, else with stream-K's 4-warp
// CTAs (three per SM).  Only the 16-warp shape uses tagged partial states: with
// 4-warp CTAs the fenced arrival measured faster.  Against stream-K (CUDA-core
// pages), the 4-warp tensor-core split measured faster at 20-28 sessions with two
// slices per pair (56.1 against 60.8 us at 20, 71.1 against 79.0 at 28) and, with one,
// at 29-57 sessions except near 36 (73.2 against 81.7 at 29, 99.6 against 97.7 at
// 36, 138.4 against 148.2 at 57).  Against the 16-warp shape, the 4-warp one measured
// faster from 4 sessions on (15.4 against 16.7 us at 4, 26.4 against 28.1 at 9) and
// slower below (11.7 against 8.1 at 1).
constexpr int SPLIT_MIN_K = 5, SPLIT4_MIN_K = 1;

}  // namespace

cudaError_t launch_attn_decode(const Dev& d, int layer, const void* q, void* out, int n_seq,
                               bool pdl, cudaStream_t s, uint32_t epoch, const void* new_k,
                               const void* new_v) {
  const int esz = d.esz;
  // Grid sizes of the three shapes, per element type (their CTA shapes differ), worked
  // out on a thread's first call with that type.
  struct Shapes {
    int grid = 0, slots = 0, slots4 = 0;
  };
  static thread_local Shapes shapes[2];
  Shapes& sh = shapes[esz == 2 ? 1 : 0];
  if (sh.grid == 0) {
    sh.grid = decode_stream_k_grid(d);
    sh.slots = decode_split_slots(esz, true);
    sh.slots4 = decode_split_slots(esz, false);
  }
  const int grid = sh.grid, slots = sh.slots, slots4 = sh.slots4;
  const float scale = LOG2E / sqrtf((float)d.head_dim);
  const int n_pairs = n_seq * d.kv_heads;
  const int k = n_pairs * SPLIT_MIN_K <= slots ? min(MAX_PARTS, slots / n_pairs) : 0;
  const int k4 = k == 0 && n_pairs * SPLIT4_MIN_K <= slots4 ? min(MAX_PARTS, slots4 / n_pairs) : 0;
  // Tensor maps of the pool for the tensor-core page loop (bfloat16).
  CUtensorMap map_lo, map_hi;
  memset(&map_lo, 0, sizeof(map_lo));
  memset(&map_hi, 0, sizeof(map_hi));
  // (The stream-K kernel's bfloat16 pages also run on the tensor cores.)
  if (((k > 0 && decode_split_uses_tma(esz, true)) ||
       (k4 > 0 && decode_split_uses_tma(esz, false)) || (k == 0 && k4 == 0 && esz == 2)) &&
      !pool_tensor_maps(d, &map_lo, &map_hi))
    return cudaErrorInvalidValue;
  if (k > 0) {
    const uint32_t tag = n_pairs * k <= d.dec_tag_slots ? epoch : 0u;
    return launch_attn_decode_split(d, true, layer, map_lo, map_hi, q, out, scale, k, tag, new_k,
                                    new_v, n_pairs, pdl, s);
  }
  if (k4 > 0)
    return launch_attn_decode_split(d, false, layer, map_lo, map_hi, q, out, scale, k4, 0u, new_k,
                                    new_v, n_pairs, pdl, s);
  return launch_attn_decode_streamk(d, layer, map_lo, map_hi, q, out, scale, grid, DEC_MIN_UNITS,
                                    new_k, new_v, pdl, s);
}

}  // namespace kvc
