// dard_api.cu - C-ABI entry points of libdard: host-side validation, the ragged-batch
// launch plan (longest sequences first) and dispatch to the kernels.
#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <numeric>
#include <vector>

#include "dard_internal.h"

namespace {

thread_local char g_err[512] = "";

dard_status fail(dard_status s, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_err, sizeof(g_err), fmt, ap);
  va_end(ap);
  return s;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace

dard_status dard::report(dard_status s, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_err, sizeof(g_err), fmt, ap);
  va_end(ap);
  return s;
}

extern "C" {

const char* dard_status_string(dard_status s) {
  switch (s) {
    case DARD_OK: return "DARD_OK";
    case DARD_ERR_NULL: return "DARD_ERR_NULL";
    case DARD_ERR_SHAPE: return "DARD_ERR_SHAPE";
    case DARD_ERR_VALUE: return "DARD_ERR_VALUE";
    case DARD_ERR_UNSUPPORTED: return "DARD_ERR_UNSUPPORTED";
    case DARD_ERR_CUDA: return "DARD_ERR_CUDA";
    case DARD_ERR_ALIGN: return "DARD_ERR_ALIGN";
    case DARD_ERR_WORKSPACE: return "DARD_ERR_WORKSPACE";
  }
  return "DARD_ERR_UNKNOWN";
}

const char* dard_last_error(void) { return g_err; }

int32_t dard_version(void) { return 20100; }

}  // extern "C"

namespace {

// Host-side validation of an attention call and its launch plan (the per-sequence
// descriptors, the longest-first work order and the kernel parameters). Touches no device.
dard_status prepare_attention(const dard_attn_args* a, dard::AttnParams& p) {
  using namespace dard;
  if (!a) return fail(DARD_ERR_NULL, "args is NULL");
  if (!a->q || !a->k || !a->v || !a->o) return fail(DARD_ERR_NULL, "q, k, v or o is NULL");
  if (!a->n_orig || !a->block_start || !a->block_len || !a->shadow_len)
    return fail(DARD_ERR_NULL, "a per-sequence host array is NULL");
  if (a->dtype != DARD_BF16 && a->dtype != DARD_F32)
    return fail(DARD_ERR_VALUE, "dtype %d is neither DARD_F32 nor DARD_BF16", a->dtype);
  if (a->num_seqs < 1 || a->num_seqs > DARD_MAX_SEQS)
    return fail(DARD_ERR_SHAPE, "num_seqs %d outside 1..%d", a->num_seqs, DARD_MAX_SEQS);
  if (a->hq < 1 || a->hkv < 1 || a->hq % a->hkv != 0)
    return fail(DARD_ERR_SHAPE, "hq %d / hkv %d: need hq %% hkv == 0", a->hq, a->hkv);
  if (a->head_dim != 64 && a->head_dim != 128)
    return fail(DARD_ERR_UNSUPPORTED, "head_dim %d (supported: 64, 128)", a->head_dim);
  if (!(a->scale >= 0.f) || !std::isfinite(a->scale))
    return fail(DARD_ERR_VALUE, "scale must be finite and >= 0");
  if (!aligned16(a->q) || !aligned16(a->k) || !aligned16(a->v) || !aligned16(a->o))
    return fail(DARD_ERR_ALIGN, "q, k, v and o must be 16-byte aligned");
  const bool rope = a->rope_theta != 0.f;
  if (rope) {
    if (!(a->rope_theta >= 1.f) || !std::isfinite(a->rope_theta))
      return fail(DARD_ERR_VALUE, "rope_theta must be 0 or a finite value >= 1");
    if (a->rope_style != DARD_ROPE_INTERLEAVED && a->rope_style != DARD_ROPE_HALF)
      return fail(DARD_ERR_VALUE, "rope_style %d is not a dard_rope_style", a->rope_style);
    if (!a->k_rope) return fail(DARD_ERR_NULL, "k_rope is NULL with rope_theta > 0");
    if (!aligned16(a->k_rope)) return fail(DARD_ERR_ALIGN, "k_rope must be 16-byte aligned");
  }

  memset(&p, 0, sizeof(p));
  long long rows = 0, blk = 0, sh = 0;
  std::vector<long long> cost(a->num_seqs);
  for (int s = 0; s < a->num_seqs; ++s) {
    const int n = a->n_orig[s], b0 = a->block_start[s], B = a->block_len[s], S = a->shadow_len[s];
    if (n < 1) return fail(DARD_ERR_SHAPE, "seq %d: n_orig %d < 1", s, n);
    if (B < 0 || B > DARD_MAX_BLOCK)
      return fail(DARD_ERR_SHAPE, "seq %d: block_len %d outside 0..%d", s, B, DARD_MAX_BLOCK);
    if (b0 < 0 || static_cast<long long>(b0) + B > n)
      return fail(DARD_ERR_SHAPE, "seq %d: block [%d, %d) outside [0, %d)", s, b0, b0 + B, n);
    if (S < 0 || S > B) return fail(DARD_ERR_SHAPE, "seq %d: shadow_len %d outside 0..%d", s, S, B);
    if (rope && n > DARD_ROPE_MAX_POSITIONS)
      return fail(DARD_ERR_SHAPE, "seq %d: n_orig %d exceeds the %d positions RoPE supports", s,
                  n, DARD_ROPE_MAX_POSITIONS);
    const int qs = a->query_start ? a->query_start[s] : 0;
    if (qs < 0 || qs > n + S)
      return fail(DARD_ERR_SHAPE, "seq %d: query_start %d outside 0..%d", s, qs, n + S);
    SeqDesc& d = p.seq[s];
    d.row_base = static_cast<int32_t>(rows);
    d.n_orig = n;
    d.b0 = b0;
    d.blen = B;
    d.slen = S;
    d.blk_off = static_cast<int32_t>(blk);
    d.sh_off = static_cast<int32_t>(sh);
    d.q_start = qs;
    d.n_qtiles = (n + S - qs + 127) / 128;
    cost[s] = static_cast<long long>(n) + S;
    rows += n + S;
    blk += B;
    sh += S;
    if (rows > (1ll << 31) - 1) return fail(DARD_ERR_SHAPE, "total rows exceed 2^31 - 1");
  }
  if (blk > 0 && (!a->state || !a->prev_conf))
    return fail(DARD_ERR_NULL, "state / prev_conf is NULL with block rows present");
  if (sh > 0 && !a->shadow_src) return fail(DARD_ERR_NULL, "shadow_src is NULL with shadow rows");
  if (rows * a->hq * a->head_dim > (1ll << 40))
    return fail(DARD_ERR_SHAPE, "tensor too large");

  // Longest-first order of the sequences; each owns n_qtiles * hq consecutive work items.
  std::vector<int> order(a->num_seqs);
  std::iota(order.begin(), order.end(), 0);
  std::stable_sort(order.begin(), order.end(), [&](int x, int y) { return cost[x] > cost[y]; });
  long long work = 0, pairs = 0;
  for (int r = 0; r < a->num_seqs; ++r) {
    p.order[r] = order[r];
    p.work_prefix[r] = static_cast<int32_t>(work);
    p.pair_prefix[r] = static_cast<int32_t>(pairs);
    work += static_cast<long long>(p.seq[order[r]].n_qtiles) * a->hq;
    pairs += static_cast<long long>((p.seq[order[r]].n_qtiles + 1) / 2) * a->hq;
    if (work > (1ll << 31) - 1) return fail(DARD_ERR_SHAPE, "too many work items");
  }
  p.work_prefix[a->num_seqs] = static_cast<int32_t>(work);
  p.pair_prefix[a->num_seqs] = static_cast<int32_t>(pairs);
  p.total_work = static_cast<int32_t>(work);
  p.total_pairs = static_cast<int32_t>(pairs);
  p.total_rows = static_cast<int32_t>(rows);
  p.state = a->state;
  p.prev_conf = a->prev_conf;
  p.shadow_src = a->shadow_src;
  p.q = a->q;
  p.k = a->k;
  p.v = a->v;
  p.o = a->o;
  p.status = a->status;
  p.hq = a->hq;
  p.hkv = a->hkv;
  p.head_dim = a->head_dim;
  p.num_seqs = a->num_seqs;
  p.scale = a->scale > 0.f ? a->scale : 1.0f / std::sqrt(static_cast<float>(a->head_dim));
  p.scale_log2 = p.scale * 1.4426950408889634f;
  p.wait_cycles = 0;
  p.test_drop_kv = -1;
  p.k_src = a->k;
  p.rope = rope ? 1 : 0;
  if (rope) {
    // f_i = theta^(-2i/D) in double, passed as a float and the float of its remainder
    p.k = a->k_rope;
    p.rope_style = a->rope_style;
    for (int i = 0; i < a->head_dim / 2; ++i) {
      const double f = std::pow(static_cast<double>(a->rope_theta),
                                -2.0 * i / static_cast<double>(a->head_dim));
      const float hi = static_cast<float>(f);
      p.rope_f[2 * i] = hi;
      p.rope_f[2 * i + 1] = static_cast<float>(f - static_cast<double>(hi));
    }
  }
  return DARD_OK;
}

}  // namespace

// Host-side validation of a scoring call and its kernel parameters (no device access).
dard_status dard::prepare_score(const dard_score_args* a, dard::ScoreParams& p) {
  using namespace dard;
  if (!a) return fail(DARD_ERR_NULL, "args is NULL");
  if (!a->block_len) return fail(DARD_ERR_NULL, "block_len is NULL");
  if (a->dtype != DARD_BF16 && a->dtype != DARD_F32)
    return fail(DARD_ERR_VALUE, "dtype %d is neither DARD_F32 nor DARD_BF16", a->dtype);
  if (a->num_seqs < 1 || a->num_seqs > DARD_MAX_SEQS)
    return fail(DARD_ERR_SHAPE, "num_seqs %d outside 1..%d", a->num_seqs, DARD_MAX_SEQS);
  if (a->vocab < 1) return fail(DARD_ERR_SHAPE, "vocab %d < 1", a->vocab);
  if (a->row_stride < a->vocab) return fail(DARD_ERR_SHAPE, "row_stride < vocab");
  if (!(a->tau_c >= 0.f && a->tau_c <= a->tau_u && a->tau_u <= 1.f))
    return fail(DARD_ERR_VALUE, "need 0 <= tau_c <= tau_u <= 1");
  if (!(a->lambda > 0.f && a->lambda < 1.f)) return fail(DARD_ERR_VALUE, "need 0 < lambda < 1");
  if (!(a->p0 > 0.f) || !std::isfinite(a->p0)) return fail(DARD_ERR_VALUE, "need p0 > 0");
  memset(&p, 0, sizeof(p));
  long long rows = 0;
  for (int s = 0; s < a->num_seqs; ++s) {
    const int B = a->block_len[s];
    if (B < 0 || B > DARD_MAX_BLOCK)
      return fail(DARD_ERR_SHAPE, "seq %d: block_len %d outside 0..%d", s, B, DARD_MAX_BLOCK);
    p.blk_off[s] = static_cast<int32_t>(rows);
    rows += B;
  }
  p.blk_off[a->num_seqs] = static_cast<int32_t>(rows);
  if (rows > 0 && (!a->logits_x || !a->logits_s || !a->state_in || !a->conf || !a->token ||
                   !a->state_out))
    return fail(DARD_ERR_NULL, "a logits, state or output pointer is NULL");
  if (a->p_cur && !a->cur_token) return fail(DARD_ERR_NULL, "p_cur needs cur_token");
  if (a->order_mode < DARD_ORDER_CONFIDENCE || a->order_mode > DARD_ORDER_MARGIN)
    return fail(DARD_ERR_VALUE, "order_mode %d is not a dard_order_mode", a->order_mode);
  const int esz = a->dtype == DARD_BF16 ? 2 : 4;
  if (rows > 0 && (!aligned16(a->logits_x) || !aligned16(a->logits_s) ||
                   (a->row_stride * esz) % 16 != 0))
    return fail(DARD_ERR_ALIGN, "logits must be 16-byte aligned with a 16-byte row pitch");
  const size_t need = dard_score_workspace_size(static_cast<int32_t>(rows), a->vocab, a->num_seqs);
  if (rows > 0 && (!a->workspace || a->workspace_bytes < need))
    return fail(DARD_ERR_WORKSPACE, "workspace of %zu bytes needed", need);
  if (rows > 0 && !aligned16(a->workspace))
    return fail(DARD_ERR_ALIGN, "workspace must be 16-byte aligned");
  p.lx = a->logits_x;
  p.ls = a->logits_s;
  p.state_in = a->state_in;
  p.conf = a->conf;
  p.token = a->token;
  p.state_out = a->state_out;
  p.w_out = a->w_out;
  p.counts = a->counts;
  p.status = a->status;
  p.cur_token = a->cur_token;
  p.p_cur = a->p_cur;
  p.tokens = a->tokens;
  p.mask_token = a->mask_token;
  p.state_in_place = static_cast<const void*>(a->state_out) == static_cast<const void*>(a->state_in);
  p.entropy = a->entropy;
  p.margin = a->margin;
  p.order_key = a->order_key;
  p.order_mode = a->order_mode;
  p.row_stride = a->row_stride;
  p.vocab = a->vocab;
  p.rows = static_cast<int32_t>(rows);
  p.num_seqs = a->num_seqs;
  p.tau_c = a->tau_c;
  p.tau_u = a->tau_u;
  p.lambda = a->lambda;
  p.p0 = a->p0;
  return DARD_OK;
}


extern "C" {

dard_status dard_step_attention(const dard_attn_args* a, void* stream) {
  using namespace dard;
  g_err[0] = '\0';
  AttnParams p;
  const dard_status st = prepare_attention(a, p);
  if (st != DARD_OK) return st;
  if (p.total_work == 0) return DARD_OK;  // no query rows (every query_start at the end)
  return launch_attention(*a, p, static_cast<cudaStream_t>(stream), g_err, sizeof(g_err));
}

dard_status dard_attention_kernel(const dard_attn_args* a, int32_t* kernel) {
  using namespace dard;
  g_err[0] = '\0';
  if (!kernel) return fail(DARD_ERR_NULL, "kernel is NULL");
  AttnParams p;
  const dard_status st = prepare_attention(a, p);
  if (st != DARD_OK) return st;
  *kernel = p.total_work == 0 ? 0 : attention_kernel_choice(*a, p);
  return DARD_OK;
}

dard_status dard_attention_plan(const dard_attn_args* a, dard_attn_plan* plan) {
  using namespace dard;
  g_err[0] = '\0';
  if (!plan) return fail(DARD_ERR_NULL, "plan is NULL");
  AttnParams p;
  const dard_status st = prepare_attention(a, p);
  if (st != DARD_OK) return st;
  memset(plan, 0, sizeof(*plan));
  if (p.total_work == 0) return DARD_OK;
  plan->kernel = attention_kernel_choice(*a, p);
  if (plan->kernel == 3) {
    plan->ctas = static_cast<int64_t>(p.total_work) * kSimtCtasPerTile;
    return DARD_OK;
  }
  plan->ctas = plan->kernel == 1 ? p.total_work
             : plan->kernel == 2 ? p.total_pairs
                                 : 2ll * pair_clusters_for(p);
  // rows handled together: one query tile (kernel 1), or two (kernels 2 and 4)
  const int unit = plan->kernel == 1 ? kKeyTile : 2 * kKeyTile;
  for (int s = 0; s < p.num_seqs; ++s) {
    const SeqDesc& sd = p.seq[s];
    const int rows = sd.n_orig + sd.slen;
    const long long all_kt = (rows + kKeyTile - 1) / kKeyTile;
    for (int r0 = sd.q_start; r0 < rows; r0 += unit) {
      const int r1 = std::min(r0 + unit, rows);
      const long long qtiles = (r1 - r0 + kKeyTile - 1) / kKeyTile;
      const long long used = key_tiles(sd, r0, r1);
      plan->tile_pairs += qtiles * used * p.hq;
      plan->tile_pairs_skipped += qtiles * (all_kt - used) * p.hq;
    }
  }
  return DARD_OK;
}

size_t dard_score_workspace_size(int32_t rows, int32_t vocab, int32_t num_seqs) {
  if (rows < 0 || vocab < 1 || num_seqs < 1 || num_seqs > DARD_MAX_SEQS) return 0;
  return dard::score_workspace_bytes(rows, num_seqs);
}

dard_status dard_score_and_transition(const dard_score_args* a, void* stream) {
  using namespace dard;
  g_err[0] = '\0';
  ScoreParams p;
  const dard_status st = prepare_score(a, p);
  if (st != DARD_OK) return st;
  return launch_score(*a, p, static_cast<cudaStream_t>(stream), g_err, sizeof(g_err));
}

}  // extern "C"
