// dard_internal.h - launch parameter blocks shared by the C-ABI layer and the kernels.
#pragma once
#include <cuda_runtime.h>
#include <cstddef>
#include <cstdint>

#include "dard.h"

namespace dard {

constexpr int kStateM = 0, kStateC = 1, kStateU = 2;

// ------------------------------------------------------------------ attention
// Per-sequence layout, copied by value into the kernel parameters (no device metadata).
struct SeqDesc {
  int32_t row_base;   // first row of the sequence in Q/K/V/O
  int32_t n_orig;     // N
  int32_t b0;         // block start
  int32_t blen;       // B
  int32_t slen;       // S
  int32_t blk_off;    // offset of the block in state / prev_conf
  int32_t sh_off;     // offset of the shadow rows in shadow_src
  int32_t q_start;    // first query row (rows before it are keys only)
  int32_t n_qtiles;   // ceil((N + S - q_start) / 128)
};

// Keys per tile of the tensor-core attention kernels.
constexpr int kKeyTile = 128;
// CTAs of the fp32 CUDA-core kernel per 128-row query tile (32 rows each).
constexpr int kSimtCtasPerTile = 4;

// Key tiles that query rows [r0, r1) of a sequence need. Original queries of positions after
// the block (query block 1 of Sec. 3.2: M positions attend the x copy of every position) never
// see a shadow key, so a run of such rows stops before the tiles that hold shadow keys only;
// every other run of rows needs all tiles of the sequence.
__host__ __device__ inline int key_tiles(const SeqDesc& sd, int r0, int r1) {
  if (r0 >= sd.b0 + sd.blen && r1 <= sd.n_orig) return (sd.n_orig + kKeyTile - 1) / kKeyTile;
  return (sd.n_orig + sd.slen + kKeyTile - 1) / kKeyTile;
}

struct AttnParams {
  const uint8_t* state;
  const float* prev_conf;
  const int32_t* shadow_src;
  void* o;
  const void* q;
  const void* k;
  const void* v;
  uint32_t* status;
  float scale;               // softmax scale
  float scale_log2;          // scale * log2(e)
  long long wait_cycles;     // bound of every in-kernel wait in SM cycles (0: the default)
  int32_t test_drop_kv;      // test hook: the key tile (the CTA-pair kernel: the K stage use)
                             // whose K copy is never issued
                             // (a wait then runs out); -1 in normal operation
  // RoPE (rope != 0): k is the rotated copy the key pass writes (k_rope of the call), k_src
  // the keys as given; the attention kernels rotate q as they load it.
  const void* k_src;
  int32_t rope;
  int32_t rope_style;        // DARD_ROPE_INTERLEAVED or DARD_ROPE_HALF
  float rope_f[2 * 64];      // f_i = theta^(-2i/D) for i < D/2 as (float, remainder) pairs
  int32_t hq, hkv, head_dim, num_seqs;
  int32_t total_rows;
  int32_t total_work;        // number of (sequence, q-tile, head) work items
  // Work items in longest-first order: sequence order[r] owns items
  // [work_prefix[r], work_prefix[r+1]), laid out q-tile major, head minor.
  int32_t total_pairs;       // number of (sequence, pair of q-tiles, head) work items
  int32_t order[DARD_MAX_SEQS];
  int32_t work_prefix[DARD_MAX_SEQS + 1];
  int32_t pair_prefix[DARD_MAX_SEQS + 1];  // the same over pairs of q-tiles
  SeqDesc seq[DARD_MAX_SEQS];
};

// The kernel a validated call launches: 1 or 2 (the tensor-core kernel with one or two
// query tiles per CTA), 3 (the fp32 CUDA-core kernel). Shared by the launcher and by
// dard_attention_kernel(); reads DARD_ATTN_TC and the current device's SM count.
int attention_kernel_choice(const dard_attn_args& a, const AttnParams& p);

// The pair kernel (two CTAs per 256-row work item, tcgen05 cta_group::2, head_dim 128,
// persistent over work items): launch, and the number of clusters a launch uses.
cudaError_t launch_pair_attention(const AttnParams& p, cudaStream_t stream);
// The fp32 CUDA-core attention kernel (dard_attention_simt.cu); kSimtCtasPerTile CTAs per
// 128-row query tile.
cudaError_t launch_simt_attention(const AttnParams& p, cudaStream_t stream);
int pair_clusters_for(const AttnParams& p);

dard_status launch_attention(const dard_attn_args& a, AttnParams& p, cudaStream_t stream,
                             char* err, size_t err_len);

// The RoPE pass over the key rows (rope != 0): k_src rotated into k. The attention kernel
// launched after it on the same stream waits for it (programmatic dependent launch).
cudaError_t launch_rope_keys(const AttnParams& p, int dtype, cudaStream_t stream);

// ------------------------------------------------------------------ scoring
struct ScoreParams {
  const void* lx;
  const void* ls;
  const uint8_t* state_in;
  float* conf;
  int32_t* token;
  uint8_t* state_out;
  float* w_out;
  int32_t* counts;
  const int32_t* cur_token;  // optional: p_cur of this token
  float* p_cur;              // optional
  int32_t* tokens;           // optional: next step's tokens (x^, or mask_token for M)
  int32_t mask_token;
  int32_t state_in_place;    // state_out is the state_in buffer
  float* entropy;            // optional
  float* margin;             // optional
  float* order_key;          // optional: next step's key per order_mode
  int32_t order_mode;
  uint32_t* status;
  // workspace
  uint32_t* ready;     // [num_seqs] C rows of the block that published their outcome
  uint32_t* departed;  // [num_seqs] M-row CTAs of the block past their wait
  uint32_t* fin;       // [num_seqs] rows of the block that finished (counts, in-place states)
  uint8_t* pd_flag;    // [rows] 1 = promoted (C -> U), 2 = demoted (C -> M), 3 = an M row
                       // (scored in pass 2), 0 otherwise
  uint8_t* new_state;  // [rows] the state each row ends in
  int64_t row_stride;
  int32_t vocab, rows, num_seqs, nsplit, chunk;
  float tau_c, tau_u, lambda, p0;
  float log2_lambda;  // lambda^k = 2^(k log2 lambda) (Eq. 5 kernel)
  int32_t blk_off[DARD_MAX_SEQS + 1];
};

constexpr int kScoreThreads = 256;
constexpr int kScoreMaxSplit = 16;  // CTAs per row = thread-block cluster size
constexpr int kScoreCtasPerSm = 12;  // target CTAs per SM when choosing the split

// Validates a scoring call and fills its kernel parameters; touches no device memory.
dard_status prepare_score(const dard_score_args* a, ScoreParams& p);
size_t score_workspace_bytes(int32_t rows, int32_t num_seqs);
size_t score_counter_bytes(int32_t num_seqs);  // the counters at the start of the workspace
dard_status launch_score(const dard_score_args& a, ScoreParams& p, cudaStream_t stream,
                         char* err, size_t err_len);
// Records the message returned by dard_last_error() on this thread and returns `s`.
dard_status report(dard_status s, const char* fmt, ...);

}  // namespace dard
