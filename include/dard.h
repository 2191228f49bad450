/*
 * dard.h - C ABI of the GB300 (sm_103a) DARD step library, libdard.so.
 *
 * DARD (Dependency-Aware Revocable Decoding, arXiv 2608.26574) adds two pieces of compute
 * to every denoising step of a diffusion LLM:
 *
 *   dard_step_attention        bidirectional softmax attention over the augmented sequence
 *                              x~_t = (x_t; s_t) under the state-specific mask of Sec. 3
 *                              (Eq. 2, Eq. 3 and query blocks 1-6 of Sec. 3.2), one layer;
 *   dard_score_and_transition  vocabulary-wide confidence and argmax (Eq. 1), verification
 *                              outcomes and guidance weights (Eq. 5, Eq. 6), logit mixing
 *                              (Eq. 7) and the three-state transition (Eq. 8), in the order
 *                              of Algorithm 1.
 *
 * Conventions shared by every entry point
 *   - Pointers named "device" are CUDA device memory owned by the caller; pointers named
 *     "host" are ordinary host memory owned by the caller and read during the call only.
 *   - Every call is asynchronous on the given stream; nothing is synchronised.
 *   - The library never allocates memory. Scratch space is passed in by the caller, or
 *     (dard_score_and_transition_noalloc) is a fixed array inside the library.
 *   - Argument and shape errors are detected on the host and returned before any launch;
 *     nothing is launched when a call returns an error. A failed launch returns
 *     DARD_ERR_CUDA (the CUDA error string is available from dard_last_error()).
 *   - Problems found only on the device (a state byte above 2, a shadow row that points
 *     outside its block, a row whose softmax normaliser is not finite) never trap: they set
 *     bits of the optional device status word (DARD_STATUS_*) and the affected outputs follow
 *     the documented fallback.
 *
 * Sequence layout (per sequence i of a ragged batch, everything stored back to back):
 *   rows      N_i original rows (prompt + full generation length, positions 0..N_i-1),
 *             then S_i shadow rows. Row N_i + k is the shadow copy s^j, j = shadow_src[k].
 *   block     positions [b0_i, b0_i + B_i) are the block being decoded. Positions before
 *             it are decoded context (state U); positions after it are still masked
 *             (state M) and have no shadow row.
 *   states    one byte per block position: 0 = M (masked), 1 = C (candidate),
 *             2 = U (unmasked), the three states of Sec. 3.2.
 */
#ifndef DARD_H_
#define DARD_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  DARD_OK = 0,
  DARD_ERR_NULL = 1,         /* a required pointer is NULL                              */
  DARD_ERR_SHAPE = 2,        /* inconsistent sizes / offsets                            */
  DARD_ERR_VALUE = 3,        /* a parameter out of its range (tau, lambda, p0, scale)   */
  DARD_ERR_UNSUPPORTED = 4,  /* valid but not implemented (e.g. head_dim not 64 or 128) */
  DARD_ERR_CUDA = 5,         /* a CUDA runtime call failed                              */
  DARD_ERR_ALIGN = 6,        /* a pointer or stride breaks the alignment rule           */
  DARD_ERR_WORKSPACE = 7     /* workspace missing or smaller than required              */
} dard_status;

typedef enum { DARD_F32 = 0, DARD_BF16 = 1 } dard_dtype;

/* Orderings of candidate tokens in the mask (Eq. 3 compares one key per block position).
 * The attention-mask ablation of Sec. 5 compares DARD's confidence ordering with a
 * bidirectional mask and with left-to-right, entropy and margin orderings; each is a choice
 * of key, which the scoring call can write for the next step (dard_score_args.order_key):
 *   CONFIDENCE  c_t (the paper's DARD)          BIDIR   0 (equal keys: every C pair attends
 *   L2R         minus the block position          both ways, Eq. 3 ties being mutual)
 *   ENTROPY     minus the entropy (nats)        MARGIN  p(x^) minus the second probability */
typedef enum {
  DARD_ORDER_CONFIDENCE = 0,
  DARD_ORDER_BIDIR = 1,
  DARD_ORDER_L2R = 2,
  DARD_ORDER_ENTROPY = 3,
  DARD_ORDER_MARGIN = 4
} dard_order_mode;

/* Bits of the optional device status word (OR-ed in, never cleared by the library). */
#define DARD_STATUS_BAD_STATE 0x1u     /* a state byte > 2 (treated as M)                    */
#define DARD_STATUS_BAD_SHADOW 0x2u    /* shadow_src outside its block or repeated (row
                                          treated as a masked-out key and left unwritten)    */
#define DARD_STATUS_INVALID_ROW 0x4u   /* softmax normaliser not finite or zero (NaN, +inf or
                                          all -inf logits): conf 0, token -1, state M        */
#define DARD_STATUS_TIMEOUT 0x8u       /* a bounded in-kernel wait gave up (the launch's
                                          outputs are incomplete)                             */

#define DARD_MAX_SEQS 256       /* sequences per call                                     */
#define DARD_MAX_BLOCK 128      /* block length B_i                                       */

/* ------------------------------------------------------------------------------------- *
 * Masked attention (Sec. 3.1 Eq. 2; Sec. 3.2 query blocks 1-6 and Eq. 3).
 *
 * For every sequence, head h and row r:
 *     O[r,h,:] = sum_j softmax_j(scale * <Q[r,h,:], K[key(r,j),g,:]>) V[key(r,j),g,:]
 * where j runs over the N_i original positions, key(r,j) is the row of x^j or of s^j as
 * the mask selects (exactly one per position, Eq. 2), and g = h / (hq / hkv) (grouped-query
 * heads share a key/value head). The mask is built inside the kernel from the state vector
 * and prev_conf; no L x L tensor exists anywhere. Selection rule (q = query copy):
 *   key j state U : x^j, except a shadow query s^i takes s^i for j = i;
 *   key j state M : x^j for original queries of M positions, s^j for every other query;
 *   key j state C : original query of an M position       -> x^j
 *                   query of a C position i (x or s)      -> x^j if c_i <= c_j, else s^j
 *                                                            (a shadow query takes s^i at j=i)
 *                   query of a U position, or s^i of an M -> s^j
 *   and x^j whenever j has no shadow row (positions outside the block, or a block position
 *   the caller gave no shadow row). Out-of-block queries are original queries of U (before
 *   the block) or M (after it) positions.
 * Arithmetic: bf16 operands on the tcgen05 tensor cores with fp32 accumulation and an fp32
 * online softmax (dtype BF16); fp32 CUDA cores throughout (dtype F32).
 * ------------------------------------------------------------------------------------- */
typedef struct {
  const void* q;             /* device [total_rows, hq,  head_dim] row-major              */
  const void* k;             /* device [total_rows, hkv, head_dim]                        */
  const void* v;             /* device [total_rows, hkv, head_dim]                        */
  void* o;                   /* device [total_rows, hq,  head_dim], same dtype as q       */
  int32_t dtype;             /* dard_dtype of q, k, v and o                                */
  int32_t hq, hkv;           /* query heads, key/value heads; hq % hkv == 0                */
  int32_t head_dim;          /* 64 or 128                                                  */
  int32_t num_seqs;          /* 1 .. DARD_MAX_SEQS                                         */
  const int32_t* n_orig;     /* host [num_seqs] N_i >= 1                                   */
  const int32_t* block_start;/* host [num_seqs] b0_i, 0 <= b0_i, b0_i + B_i <= N_i         */
  const int32_t* block_len;  /* host [num_seqs] B_i in 0 .. DARD_MAX_BLOCK                 */
  const int32_t* shadow_len; /* host [num_seqs] S_i in 0 .. B_i                            */
  const uint8_t* state;      /* device [sum B_i] states of block positions, seq by seq     */
  const float* prev_conf;    /* device [sum B_i] c_{t-1} of block positions (Eq. 3 order)  */
  const int32_t* shadow_src; /* device [sum S_i] original position of each shadow row,
                                in [b0_i, b0_i + B_i), distinct within a sequence          */
  float scale;               /* softmax scale; 0 means 1/sqrt(head_dim)                    */
  uint32_t* status;          /* optional device word, DARD_STATUS_* bits OR-ed in          */
  const int32_t* query_start;/* optional host [num_seqs] q_i in 0 .. N_i + S_i: only rows
                                q_i .. N_i + S_i - 1 of sequence i are queries (prefix
                                caching: the prompt's outputs are not recomputed, its
                                K/V rows still serve as keys); rows before q_i of o are
                                left untouched. NULL means 0 for every sequence.           */
  /* Rotary position embedding inside the call (Sec. 3.1: x^i and s^i share the positional
   * embedding of position i). rope_theta = 0: q and k already carry their positions (no
   * rotation here, k_rope unused). rope_theta >= 1: q and k arrive before RoPE and the call
   * rotates them, original row r of a sequence at position r and shadow row N_i + k at
   * position shadow_src[k]; see "RoPE" below. */
  float rope_theta;          /* 0, or the RoPE base theta >= 1                             */
  int32_t rope_style;        /* dard_rope_style: which elements form a rotated pair        */
  void* k_rope;              /* device [total_rows, hkv, head_dim], dtype: receives k after
                                RoPE, the keys the attention reads (a key cache may take
                                it); may be k itself (rotated in place). Required when
                                rope_theta > 0, 16-byte aligned.                           */
} dard_attn_args;

/* RoPE (rotary position embedding, Su et al., RoFormer, 2021) as dard_step_attention applies
 * it when rope_theta > 0. For head dimension D and frequency index i in 0 .. D/2 - 1 the
 * pair (a, b) of a row at position p is replaced by
 *     (a cos(p f_i) - b sin(p f_i),  a sin(p f_i) + b cos(p f_i)),   f_i = theta^(-2i/D),
 * in every head of q and of k. DARD_ROPE_INTERLEAVED pairs elements (2i, 2i + 1);
 * DARD_ROPE_HALF pairs (i, i + D/2). The call first rotates k into k_rope (one pass over the
 * key rows, launched on the stream ahead of the attention kernel, which waits for it with
 * programmatic dependent launch), then the attention kernel rotates each query tile as it
 * loads it; the rotated q is not written out. Arithmetic: the angle p f_i is carried in two
 * floats (f_i split into a float and its remainder), reduced modulo 2 pi with a two-constant
 * additive (Cody-Waite) split of 2 pi, and its cosine and sine taken by the hardware
 * approximations on the reduced angle (absolute error near 1e-6 in all); rotated values are
 * rounded to dtype. Every N_i must be at most 2^20 (DARD_ERR_SHAPE). A shadow row whose
 * shadow_src is invalid (DARD_STATUS_BAD_SHADOW) is rotated by an unspecified angle; it is a
 * masked-out key and an unwritten query row anyway. */
typedef enum { DARD_ROPE_INTERLEAVED = 0, DARD_ROPE_HALF = 1 } dard_rope_style;
#define DARD_ROPE_MAX_POSITIONS (1 << 20)

/* Rows are total_rows = sum_i (N_i + S_i). q, k, v, o must be 16-byte aligned; with dtype
 * BF16 a tensor-core kernel runs (head_dim 64 or 128), with F32 the CUDA-core kernel.
 * Of the two tensor-core kernels (one or two 128-row query tiles per CTA) the library
 * picks the one a cost model of the batch (query tiles, key tiles, SM count) predicts to be
 * faster; the environment variable DARD_ATTN_TC=1 or 2 forces one of them (results agree
 * within rounding).
 * Errors: DARD_ERR_NULL (also: k_rope NULL with rope_theta > 0), _SHAPE, _VALUE (scale < 0
 * or not finite; rope_theta neither 0 nor a finite value >= 1; rope_style not a
 * dard_rope_style), _UNSUPPORTED, _ALIGN, _CUDA. */
dard_status dard_step_attention(const dard_attn_args* args, void* stream /* cudaStream_t */);

/* The attention kernel dard_step_attention would launch for these arguments, without
 * launching anything: *kernel = 1 or 2 (the tensor-core kernel with one or two 128-row
 * query tiles per CTA, as the cost model or DARD_ATTN_TC picks), 4 (the kernel on CTA
 * pairs, head_dim 128, chosen only by DARD_ATTN_TC=4), 3 (the fp32 CUDA-core kernel), or 0
 * (no query rows, no launch). The arguments go through the same host
 * validation as dard_step_attention and fail with the same codes; device pointers are
 * checked but never read. The cost model uses the current device's SM count (148 when no
 * device is visible, so that the choice can be planned on a host without one). An
 * interface addition: the paper has no counterpart. */
dard_status dard_attention_kernel(const dard_attn_args* args, int32_t* kernel);

/* The launch plan of dard_step_attention for these arguments, computed on the host without
 * launching anything (an interface addition: the paper has no counterpart). The arguments
 * go through the same host validation as dard_step_attention and fail with the same codes.
 *   kernel              as dard_attention_kernel (0: no query rows, nothing launched)
 *   ctas                CTAs of the launch (the CTA-pair kernel: two per cluster, as many
 *                       clusters as fit on the current device, or SMs / 2 without one)
 *   tile_pairs          (query tile, key tile) pairs a tensor-core kernel computes: 128 query
 *                       rows of one head against 128 key rows, over every head and sequence
 *   tile_pairs_skipped  pairs it leaves out because no query of the rows a CTA (or CTA pair)
 *                       handles attends any key of the tile: tiles holding only shadow keys,
 *                       for rows that are all original queries of positions after the block
 *                       (Sec. 3.2, query block 1 attends x copies only). The fp32 kernel,
 *                       which masks key by key, reports 0 for both.                         */
typedef struct {
  int32_t kernel;
  int64_t ctas;
  int64_t tile_pairs;
  int64_t tile_pairs_skipped;
} dard_attn_plan;
dard_status dard_attention_plan(const dard_attn_args* args, dard_attn_plan* plan);

/* ------------------------------------------------------------------------------------- *
 * Confidence scoring and state transition (Eq. 1, Eq. 5-8, Algorithm 1).
 *
 * Rows are the block positions of all sequences, seq by seq (sum B_i rows). For row i of a
 * sequence with incoming state s_i:
 *   s_i in {C, U}: (c_i, x^_i) = (max softmax, argmax) of logits_s row i          (Eq. 1)
 *   then every C row that moves to U joins P, every C row that moves to M joins D (Eq. 8);
 *   s_i = M: P_i = sum_{j in P} lambda^|i-j|, D_i likewise over D                  (Eq. 5)
 *            w_i = (P_i + p0) / (P_i + D_i + p0)                                  (Eq. 6)
 *            mix = ls + w_i (lx - ls), each operation rounded to fp32              (Eq. 7)
 *            (c_i, x^_i) = (max softmax, argmax) of mix
 *   new state: c <= tau_c -> M, c <= tau_u -> C, else U                            (Eq. 8)
 * Argmax ties go to the lowest index. Softmax sums and w accumulate in fp32 (the terms
 * lambda^k as 2^(k log2 lambda)); w then enters Eq. 7 as an fp32 value.
 * Invalid rows (normaliser not finite or 0): conf 0, token -1, state M, status bit.
 * ------------------------------------------------------------------------------------- */
typedef struct {
  const void* logits_x;      /* device [rows, row_stride] logits of the original copies   */
  const void* logits_s;      /* device [rows, row_stride] logits of the shadow copies     */
  int32_t dtype;             /* dard_dtype of both logit tensors                           */
  int32_t vocab;             /* V >= 1                                                     */
  int64_t row_stride;        /* elements between consecutive rows, >= vocab               */
  int32_t num_seqs;          /* 1 .. DARD_MAX_SEQS                                         */
  const int32_t* block_len;  /* host [num_seqs] B_i in 0 .. DARD_MAX_BLOCK                 */
  const uint8_t* state_in;   /* device [rows] incoming states                              */
  float tau_c, tau_u;        /* 0 <= tau_c <= tau_u <= 1                                   */
  float lambda;              /* 0 < lambda < 1 (paper: 0.5^(1/8))                          */
  float p0;                  /* p0 > 0 (paper: 0.1)                                        */
  float* conf;               /* device [rows] out: c_t                                     */
  int32_t* token;            /* device [rows] out: x^_t (or -1 for an invalid row)         */
  uint8_t* state_out;        /* device [rows] out: state after Eq. 8                       */
  float* w_out;              /* optional device [rows] out: w for M rows, NaN otherwise    */
  int32_t* counts;           /* optional device [num_seqs * 3] out: M, C, U counts         */
  uint32_t* status;          /* optional device word, DARD_STATUS_* bits OR-ed in          */
  void* workspace;           /* device scratch of dard_score_workspace_size() bytes: three
                                counters per sequence, then two bytes per block row (each
                                C row's promotion / demotion outcome, each row's new
                                state). Fill it with zeros before its first use; every
                                call leaves the counters at zero again, except a call that
                                sets DARD_STATUS_TIMEOUT, after which it must be zeroed
                                again. Calls that overlap on the GPU need separate
                                workspaces.                                                */
  size_t workspace_bytes;
  /* Optional, the end of a step (each may be NULL):                                       */
  const int32_t* cur_token;  /* device [rows] the token currently at each block position   */
  float* p_cur;              /* device [rows] out: the probability the scored distribution
                                (shadow logits for C/U rows, mixed logits for M rows) gives
                                to cur_token; 0 for a token outside [0, vocab) or an invalid
                                row. Needs cur_token.                                      */
  int32_t* tokens;           /* device [rows] out: the next step's tokens, as the last line
                                of Algorithm 1's step fills them: x^ where the new state is
                                C or U, mask_token where it is M                           */
  int32_t mask_token;        /* the mask token id written by `tokens`                      */
  float* entropy;            /* device [rows] out: entropy (nats) of the scored
                                distribution; 0 for an invalid row                         */
  float* margin;             /* device [rows] out: p(x^) minus the second-largest
                                probability (a repeated maximum gives 0); 0 if invalid     */
  float* order_key;          /* device [rows] out: the next step's ordering key, to pass as
                                dard_attn_args.prev_conf, per order_mode                   */
  int32_t order_mode;        /* dard_order_mode of order_key                               */
} dard_score_args;

/* In place: state_out may be the state_in buffer (the next step's states replace this
 * step's), and conf can serve directly as the next step's prev_conf of dard_step_attention;
 * tokens may be the buffer cur_token points to. */

/* Bytes of workspace a call with these sizes needs (0 on invalid sizes). */
size_t dard_score_workspace_size(int32_t rows, int32_t vocab, int32_t num_seqs);

/* Logits pointers must be 16-byte aligned and row_stride * element size a multiple of 16.
 * Two launches (C and U rows, then M rows: Algorithm 1's order), the second a programmatic
 * dependent of the first. DARD_SCORE_PATH=fused selects one launch instead, whose M rows
 * wait (bounded) for their block's C rows of the same launch, when every row's group of
 * CTAs fits on the device at once. Errors: DARD_ERR_NULL, _SHAPE, _VALUE, _ALIGN,
 * _WORKSPACE, _CUDA. */
dard_status dard_score_and_transition(const dard_score_args* args, void* stream);

/* ------------------------------------------------------------------------------------- *
 * dard_score_and_transition_noalloc: the same scoring and transition, with the scratch
 * inside the library. The paper has no counterpart: this is an interface addition.
 *
 * Who needs it: a caller that only holds the buffers another component handed to it (a
 * plug-in inside an inference server, a C host program driving a model it did not load)
 * and has no device allocator, or one whose device memory is planned in advance so that no
 * call may ask for more. Such a caller cannot provide `workspace`; this entry point needs
 * none and neither allocates nor frees device memory.
 *
 * Arguments, outputs and errors are those of dard_score_and_transition, except that
 * `workspace` and `workspace_bytes` are ignored. The scratch is a fixed array in the
 * library's device memory sized for DARD_SCORE_NOALLOC_MAX_ROWS block rows and DARD_MAX_SEQS
 * sequences (the workspace layout of dard_score_and_transition). A call with more block
 * rows (sum of block_len) than that returns DARD_ERR_WORKSPACE before any launch; use
 * dard_score_and_transition with a workspace for it. Each call clears the array's counters
 * on its stream (cudaMemsetAsync, which allocates nothing) before the kernels run, so no
 * call depends on what an earlier one left.
 *
 * The first call on each device (the device current at the call) looks up the array's
 * address there (cudaGetSymbolAddress) and caches it with the current context; a later call
 * in another context of the device (after a device reset, say) looks it up again. Make the
 * first call in a context before any stream capture there. A failed lookup returns
 * DARD_ERR_CUDA.
 *
 * There is one array per device, shared by every call on it: calls whose kernels can
 * overlap on one device (different streams, different host threads) race on it and may
 * return wrong results. Order them (one stream, or events between streams).
 * ------------------------------------------------------------------------------------- */
#define DARD_SCORE_NOALLOC_MAX_ROWS 8192
dard_status dard_score_and_transition_noalloc(const dard_score_args* args, void* stream);

/* Human-readable name of a status code; never NULL. */
const char* dard_status_string(dard_status s);

/* The message of the last DARD_ERR_CUDA / validation failure on this thread; never NULL. */
const char* dard_last_error(void);

/* Library version as major * 10000 + minor * 100 + patch. */
int32_t dard_version(void);

#ifdef __cplusplus
}
#endif
#endif /* DARD_H_ */
