// C ABI of the BAG sampler: context (weights, activation arena, device state), the
// per-sample conditioning precompute, one denoising step as a CUDA graph whose
// full-network body and residual-reuse body hang off a conditional node that the gate
// kernel sets on the device, and the single-operation entry points.
//
// One step, as enqueued (Algorithm 2, one iteration):
//   prefix : patch embed  h_in = x W_pe^T + b  (also seeds the image stream)
//            signal       m_t = LN-mod of h_in with block 0's first modulation (or h_in
//                         itself, the paper's post-patch-embedding observable), fused
//                         with the per-row partial sums of |m_t - m_last| and |m_last|;
//                         after a full step it also takes m_last <- m_{t-1}
//            gate         drift, gate MLP, forced rules, counters, log, decision
//   full   : text tokens -> stream, every block, R = h_out - h_in
//   reuse  : h_out = h_in + R
//   suffix : final LN-mod + projection fused with the Euler update, t += 1
#include <algorithm>
#include <cmath>
#include <cstdlib>
#include <cstdio>
#include <cstring>
#include <map>
#include <string>
#include <vector>

#include "bag.h"
#include "kernels.h"

using namespace bag;

namespace {

struct Tensor {
  void* p = nullptr;
  long n = 0;
  int bf16 = 0;
};

enum BlockType { BT_SINGLE = 0, BT_DOUBLE = 1, BT_WAN = 2 };

struct Block {
  int type = BT_SINGLE;
  std::map<std::string, Tensor> w;
  long mod_off = 0;  // column of this block's first modulation vector in a mod_all row
};

// ----- the seeded generator, host side (SplitMix64; same definition as the device fill)
uint64_t sm_mix(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}
uint64_t sm_start(uint64_t seed, uint64_t key) {
  return sm_mix((seed * 0x9E3779B97F4A7C15ull) ^ sm_mix(key));
}
void sm_uniform(uint64_t seed, uint64_t key, int n, double lo, double hi, float* out) {
  const uint64_t s = sm_start(seed, key);
  const float lo32 = (float)lo, hi32 = (float)hi;
  const float span = hi32 - lo32;
  for (int i = 0; i < n; ++i) {
    const uint64_t u = sm_mix(s + (uint64_t)(i + 1) * 0x9E3779B97F4A7C15ull);
    const float f = (float)(u >> 40) * (1.0f / 16777216.0f);
    const float prod = span * f;
    out[i] = lo32 + prod;
  }
}

// Tensor ids of the generator's inventory (key = slot * 256 + id).
const std::map<std::string, int> kGlobalIds = {
    {"pe_w", 0}, {"pe_b", 1}, {"t1_w", 2}, {"t1_b", 3}, {"t2_w", 4}, {"t2_b", 5},
    {"fmod_w", 6}, {"fmod_b", 7}, {"fin_w", 8}, {"fin_b", 9}, {"tproj_w", 10}, {"tproj_b", 11}};
const std::map<std::string, int> kSingleIds = {{"mod_w", 0},  {"mod_b", 1},  {"lin1_w", 2},
                                               {"lin1_b", 3}, {"lin2_w", 4}, {"lin2_b", 5},
                                               {"q_norm", 6}, {"k_norm", 7}};
std::map<std::string, int> double_ids() {
  std::map<std::string, int> m;
  const char* st[2] = {"img", "txt"};
  const char* nm[5] = {"mod", "qkv", "proj", "up", "down"};
  for (int i = 0; i < 2; ++i)
    for (int j = 0; j < 5; ++j) {
      m[std::string(st[i]) + "_" + nm[j] + "_w"] = i * 10 + 2 * j;
      m[std::string(st[i]) + "_" + nm[j] + "_b"] = i * 10 + 2 * j + 1;
    }
  for (int i = 0; i < 2; ++i) {
    m[std::string(st[i]) + "_q_norm"] = 20 + 2 * i;
    m[std::string(st[i]) + "_k_norm"] = 21 + 2 * i;
  }
  return m;
}
const std::map<std::string, int> kWanIds = {
    {"mod_tab", 0}, {"sa_qkv_w", 1}, {"sa_qkv_b", 2}, {"sa_o_w", 3}, {"sa_o_b", 4},
    {"ca_q_w", 5}, {"ca_q_b", 6}, {"ca_kv_w", 7}, {"ca_kv_b", 8}, {"ca_o_w", 9}, {"ca_o_b", 10},
    {"ffn_up_w", 11}, {"ffn_up_b", 12}, {"ffn_down_w", 13}, {"ffn_down_b", 14}};

constexpr int kTembDim = 256;

}  // namespace

struct bag_ctx {
  bag_arch arch{};
  int T = 0, B = 0;
  int d = 0, H = 0, dh = 0, F = 0, C = 0, ni = 0, nx = 0, N = 0, nrope = 0, nblk = 0;
  int act_bf16 = 0;
  size_t act_size = 4;
  cudaStream_t stream = nullptr;       // internal stream: all work and graph capture
  cudaStream_t user_stream = nullptr;  // caller's stream (bag_set_stream), bridged by events
  cudaEvent_t ev_in = nullptr, ev_out = nullptr;
  std::string err;

  // weights
  void* warena = nullptr;
  std::map<std::string, Tensor> G;
  std::vector<Block> blocks;
  Tensor wmod;        // [n_mod, d]: every modulation projection, concatenated
  float* bmod = nullptr;
  long n_mod = 0;
  long mod_stride = 0;  // floats per step in mod_all
  long fmod_off = 0;    // final-layer modulation column in mod_all
  float* wan_tabs = nullptr;  // [nblk][6d]

  // gate
  float* d_gate = nullptr;
  float thr = 0.f;
  int policy = BAG_POLICY_BAG;
  float delta = 0.f;  // threshold of BAG_POLICY_THRESHOLD
  uint8_t* d_pmask = nullptr;

  // activations
  void* aarena = nullptr;
  float *x = nullptr, *h_in = nullptr, *hj = nullptr, *R = nullptr;
  void *m_cur = nullptr, *m_last = nullptr;
  float* sig_partial = nullptr;
  __nv_bfloat16* xb = nullptr;
  void *xn = nullptr, *q = nullptr, *k = nullptr, *vt = nullptr, *cat = nullptr;
  void *qc = nullptr, *kc = nullptr, *vtc = nullptr;
  long vpad = 0, vpad_c = 0;
  void* txt_stage = nullptr;
  float* pooled_stage = nullptr;
  float2* rope = nullptr;
  float* dsig = nullptr;
  double* d_sigma = nullptr;  // [T + 1] noise levels (time embedding, samplers)
  float* uni_coef = nullptr;  // UniPC: [T][kUniCoefs]
  float *uni_xl = nullptr, *uni_m0 = nullptr, *uni_m1 = nullptr;
  float *sin_all = nullptr, *t1o = nullptr, *svec = nullptr;  // fp32 conditioning chain
  __nv_bfloat16* splitbuf = nullptr;  // [T, 2 * max(256, d)] hi|lo halves (bf16 configs)
  float *vec_all = nullptr, *mod_all = nullptr, *wan_shared = nullptr;
  // classifier-free guidance: the unconditional branch's stream, cached residual, staged
  // conditioning and modulation (Wan: mod_all_u aliases mod_all, its modulation does not
  // depend on the text), and the conditional velocity of the current step
  float *R_u = nullptr, *vcond = nullptr;
  void* txt_stage_u = nullptr;
  float *pooled_stage_u = nullptr, *vec_all_u = nullptr, *svec_u = nullptr, *mod_all_u = nullptr;
  DevState* st = nullptr;     // sampler state
  DevState* st_op = nullptr;  // state for single-operation calls
  float* log = nullptr;
  float* tmp_f32 = nullptr;   // staging for bag_run_host text conversion
  long tmp_f32_n = 0;

  // step graph
  cudaGraph_t graph = nullptr;
  cudaGraphExec_t exec = nullptr;
  cudaStream_t cap_stream = nullptr;
  int use_graph = 1;
  bool pdl = true;  // programmatic dependent launch between the kernels of a segment
  long n_prefix = 0, n_full = 0, n_skip = 0, n_suffix = 0, n_prepare = 0;
  long launches = 0;

  int next_t = 0;
  bool prepared = false;

  // per-launch profiling (direct launches only)
  struct ProfRec {
    int kind;
    double flops, bytes;
    int e0, e1;
    int m, n, k;
    int variant;
  };
  std::vector<ProfRec> prof;
  std::vector<cudaEvent_t> ev_pool;
  size_t ev_used = 0;
  bool profiling = false;
};

// Errors of calls without a context (bag_create, bag_rel_l1_noalloc) are kept per host
// thread, so that one thread's failure never overwrites or frees the text another thread
// is reading through bag_last_error(NULL).
static thread_local std::string g_create_error;
thread_local bool bag::g_pdl = false;

void bag::set_global_error(const std::string& msg) { g_create_error = msg; }

#define CK(expr)                                                                     \
  do {                                                                               \
    cudaError_t _e = (expr);                                                         \
    if (_e != cudaSuccess) {                                                         \
      ctx->err = std::string(#expr) + ": " + cudaGetErrorString(_e);                 \
      return BAG_ECUDA;                                                              \
    }                                                                                \
  } while (0)

#define CKS(expr)                                  \
  do {                                             \
    bag_status _s = (expr);                        \
    if (_s != BAG_OK) return _s;                   \
  } while (0)

static bag_status fail(bag_ctx* ctx, bag_status s, const std::string& msg) {
  if (ctx)
    ctx->err = msg;
  else
    g_create_error = msg;
  return s;
}

// ---------------------------------------------------------------------------
// creation
// ---------------------------------------------------------------------------
static size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

namespace {
struct Arena {
  size_t off = 0;
  std::vector<std::pair<void**, size_t>> items;
  void add(void** slot, size_t bytes) {
    items.push_back({slot, off});
    off += align256(bytes);
  }
  void bind(char* base) {
    for (auto& it : items) *it.first = base + it.second;
  }
};
}  // namespace

static bag_status validate_arch(const bag_arch* a, int T, int B) {
  if (!a) return fail(nullptr, BAG_EINVAL, "arch is null");
  if (T < 1 || B < 1 || B > T) return fail(nullptr, BAG_EINVAL, "need 1 <= B <= T");
  if (a->kind < 0 || a->kind > 2) return fail(nullptr, BAG_EINVAL, "unknown kind");
  if (a->hidden <= 0 || a->heads <= 0 || a->hidden % a->heads) return fail(nullptr, BAG_EINVAL, "hidden % heads");
  const int dh = a->hidden / a->heads;
  if (dh != 64 && dh != 128) return fail(nullptr, BAG_EUNSUPPORTED, "head_dim must be 64 or 128");
  if (a->hidden % 64 || a->mlp % 64 || a->mlp <= 0) return fail(nullptr, BAG_EUNSUPPORTED, "hidden and mlp must be multiples of 64");
  if (a->hidden > 6144) return fail(nullptr, BAG_EUNSUPPORTED, "hidden > 6144");
  if (a->patch_ch != 64) return fail(nullptr, BAG_EUNSUPPORTED, "patch_ch must be 64");
  if (a->grid[0] < 1 || a->grid[1] < 1 || a->grid[2] < 1 || a->n_txt < 1) return fail(nullptr, BAG_EINVAL, "empty grid or text");
  int s = 0;
  for (int i = 0; i < 3; ++i) {
    if (a->rope_axes[i] < 0 || a->rope_axes[i] % 2) return fail(nullptr, BAG_EINVAL, "rope axes must be even");
    s += a->rope_axes[i];
  }
  if (s != dh) return fail(nullptr, BAG_EINVAL, "rope axes must sum to head_dim");
  const int nb = a->kind == BAG_KIND_WAN ? a->n_wan : a->n_double + a->n_single;
  if (nb < 1) return fail(nullptr, BAG_EINVAL, "no blocks");
  if (a->kind == BAG_KIND_SINGLE && a->n_double) return fail(nullptr, BAG_EINVAL, "SINGLE kind has no double blocks");
  if (!(a->tau > 0.f && a->tau < 1.f)) return fail(nullptr, BAG_EINVAL, "tau must be in (0, 1)");
  if (a->dtype != BAG_F32 && a->dtype != BAG_BF16) return fail(nullptr, BAG_EINVAL, "dtype");
  if (a->dtype == BAG_BF16 && dh != 128)
    return fail(nullptr, BAG_EUNSUPPORTED, "bf16 backbones need head_dim 128 (tensor-core attention)");
  if (a->gate_kind < BAG_GATE_MLP3 || a->gate_kind > BAG_GATE_WAN6) return fail(nullptr, BAG_EINVAL, "gate_kind");
  if (a->cfg != 0 && a->cfg != 1) return fail(nullptr, BAG_EINVAL, "cfg must be 0 or 1");
  if (a->cfg && !std::isfinite(a->guidance)) return fail(nullptr, BAG_EINVAL, "guidance must be finite");
  if (a->qk_norm != 0 && a->qk_norm != 1) return fail(nullptr, BAG_EINVAL, "qk_norm must be 0 or 1");
  if (a->qk_norm && (a->kind == BAG_KIND_WAN || a->dtype != BAG_BF16))
    return fail(nullptr, BAG_EUNSUPPORTED, "qk_norm needs a bf16 SINGLE or MMDIT backbone");
  if (a->qk_norm && a->mlp % dh)
    return fail(nullptr, BAG_EUNSUPPORTED, "qk_norm needs mlp to be a multiple of head_dim");
  if (a->sampler != BAG_SAMPLER_EULER && a->sampler != BAG_SAMPLER_UNIPC) return fail(nullptr, BAG_EINVAL, "sampler");
  if (a->observable != BAG_OBS_MODULATED && a->observable != BAG_OBS_EMBEDDED)
    return fail(nullptr, BAG_EINVAL, "observable");
  if (!(a->shift == 0.f || (std::isfinite(a->shift) && a->shift > 0.f)))
    return fail(nullptr, BAG_EINVAL, "shift must be positive (0 = no shift)");
  return BAG_OK;
}

static std::map<std::string, std::vector<long>> global_shapes(const bag_ctx* c) {
  const long d = c->d, C = c->C;
  std::map<std::string, std::vector<long>> s = {
      {"pe_w", {d, C}}, {"pe_b", {d}}, {"t1_w", {d, kTembDim}}, {"t1_b", {d}}, {"t2_w", {d, d}},
      {"t2_b", {d}}, {"fmod_w", {2 * d, d}}, {"fmod_b", {2 * d}}, {"fin_w", {C, d}}, {"fin_b", {C}}};
  if (c->arch.kind == BAG_KIND_WAN) {
    s["tproj_w"] = {6 * d, d};
    s["tproj_b"] = {6 * d};
  }
  return s;
}

static std::map<std::string, std::vector<long>> block_shapes(const bag_ctx* c, int type) {
  const long d = c->d, F = c->F, dh = c->dh;
  const bool qkn = c->arch.qk_norm != 0;
  if (type == BT_SINGLE) {
    std::map<std::string, std::vector<long>> s = {
        {"mod_w", {3 * d, d}}, {"mod_b", {3 * d}}, {"lin1_w", {3 * d + F, d}},
        {"lin1_b", {3 * d + F}}, {"lin2_w", {d, d + F}}, {"lin2_b", {d}}};
    if (qkn) {
      s["q_norm"] = {dh};
      s["k_norm"] = {dh};
    }
    return s;
  }
  if (type == BT_DOUBLE) {
    std::map<std::string, std::vector<long>> s;
    for (const char* st : {"img", "txt"}) {
      std::string p(st);
      s[p + "_mod_w"] = {6 * d, d};
      s[p + "_mod_b"] = {6 * d};
      s[p + "_qkv_w"] = {3 * d, d};
      s[p + "_qkv_b"] = {3 * d};
      s[p + "_proj_w"] = {d, d};
      s[p + "_proj_b"] = {d};
      s[p + "_up_w"] = {F, d};
      s[p + "_up_b"] = {F};
      s[p + "_down_w"] = {d, F};
      s[p + "_down_b"] = {d};
      if (qkn) {
        s[p + "_q_norm"] = {dh};
        s[p + "_k_norm"] = {dh};
      }
    }
    return s;
  }
  return {{"mod_tab", {6 * d}}, {"sa_qkv_w", {3 * d, d}}, {"sa_qkv_b", {3 * d}},
          {"sa_o_w", {d, d}}, {"sa_o_b", {d}}, {"ca_q_w", {d, d}}, {"ca_q_b", {d}},
          {"ca_kv_w", {2 * d, d}}, {"ca_kv_b", {2 * d}}, {"ca_o_w", {d, d}}, {"ca_o_b", {d}},
          {"ffn_up_w", {F, d}}, {"ffn_up_b", {F}}, {"ffn_down_w", {d, F}}, {"ffn_down_b", {d}}};
}

static bool is_mod_weight(const std::string& n) {
  return n == "mod_w" || n == "img_mod_w" || n == "txt_mod_w";
}
static bool is_mod_bias(const std::string& n) {
  return n == "mod_b" || n == "img_mod_b" || n == "txt_mod_b";
}

static bag_status alloc_weights(bag_ctx* ctx) {
  const int act = ctx->act_bf16;
  const long d = ctx->d;
  // modulation projections first, contiguous: [blocks..., final] (Wan: [tproj, final])
  std::vector<std::pair<std::string, int>> mod_order;  // (name, block or -1)
  long nmod = 0;
  for (int b = 0; b < ctx->nblk; ++b) {
    Block& blk = ctx->blocks[b];
    if (blk.type == BT_DOUBLE) {
      blk.mod_off = nmod;
      mod_order.push_back({"img_mod", b});
      mod_order.push_back({"txt_mod", b});
      nmod += 12 * d;
    } else if (blk.type == BT_SINGLE) {
      blk.mod_off = nmod;
      mod_order.push_back({"mod", b});
      nmod += 3 * d;
    } else {
      blk.mod_off = (long)b * 6 * d;
    }
  }
  if (ctx->arch.kind == BAG_KIND_WAN) {
    mod_order.push_back({"tproj", -1});
    ctx->fmod_off = (long)ctx->nblk * 6 * d;
    ctx->mod_stride = ctx->fmod_off + 2 * d;
    nmod = 6 * d;
  } else {
    ctx->fmod_off = nmod;
    ctx->mod_stride = nmod + 2 * d;
  }
  mod_order.push_back({"fmod", -1});
  nmod += 2 * d;
  ctx->n_mod = nmod;

  // sizes
  size_t total = 0;
  const size_t es = act ? 2 : 4;
  total += align256((size_t)nmod * d * es) + align256((size_t)nmod * 4);
  auto gs = global_shapes(ctx);
  for (auto& kv : gs) {
    if (kv.first == "fmod_w" || kv.first == "fmod_b" || kv.first == "tproj_w" || kv.first == "tproj_b") continue;
    long n = 1;
    for (long v : kv.second) n *= v;
    total += align256((size_t)n * (kv.second.size() == 2 ? es : 4));
  }
  for (int b = 0; b < ctx->nblk; ++b) {
    for (auto& kv : block_shapes(ctx, ctx->blocks[b].type)) {
      if (is_mod_weight(kv.first) || is_mod_bias(kv.first)) continue;
      long n = 1;
      for (long v : kv.second) n *= v;
      total += align256((size_t)n * (kv.second.size() == 2 ? es : 4));
    }
  }
  if (cudaMalloc(&ctx->warena, total) != cudaSuccess)
    return fail(ctx, BAG_ENOMEM, "weight allocation of " + std::to_string(total) + " bytes failed");
  char* base = (char*)ctx->warena;
  size_t off = 0;
  ctx->wmod = {base, nmod * d, act};
  off += align256((size_t)nmod * d * es);
  ctx->bmod = (float*)(base + off);
  off += align256((size_t)nmod * 4);
  // bind modulation pieces into the concatenated buffers
  long row = 0;
  for (auto& it : mod_order) {
    const std::string& stem = it.first;
    const long rows = stem == "fmod" ? 2 * d : (stem == "mod" ? 3 * d : 6 * d);
    Tensor w{(char*)ctx->wmod.p + (size_t)row * d * es, rows * d, act};
    Tensor bb{ctx->bmod + row, rows, 0};
    if (it.second < 0) {
      ctx->G[stem + "_w"] = w;
      ctx->G[stem + "_b"] = bb;
    } else {
      ctx->blocks[it.second].w[stem + "_w"] = w;
      ctx->blocks[it.second].w[stem + "_b"] = bb;
    }
    row += rows;
  }
  for (auto& kv : gs) {
    if (ctx->G.count(kv.first)) continue;
    long n = 1;
    for (long v : kv.second) n *= v;
    const int is_mat = kv.second.size() == 2;
    ctx->G[kv.first] = {base + off, n, is_mat ? act : 0};
    off += align256((size_t)n * (is_mat ? es : 4));
  }
  // Wan per-block tables go contiguous for the expansion kernel
  if (ctx->arch.kind == BAG_KIND_WAN) {
    ctx->wan_tabs = (float*)(base + off);
    for (int b = 0; b < ctx->nblk; ++b) ctx->blocks[b].w["mod_tab"] = {ctx->wan_tabs + (size_t)b * 6 * d, 6 * d, 0};
    off += align256((size_t)ctx->nblk * 6 * d * 4);
  }
  for (int b = 0; b < ctx->nblk; ++b) {
    for (auto& kv : block_shapes(ctx, ctx->blocks[b].type)) {
      if (ctx->blocks[b].w.count(kv.first)) continue;
      long n = 1;
      for (long v : kv.second) n *= v;
      const int is_mat = kv.second.size() == 2;
      ctx->blocks[b].w[kv.first] = {base + off, n, is_mat ? act : 0};
      off += align256((size_t)n * (is_mat ? es : 4));
    }
  }
  if (off > total) return fail(ctx, BAG_ESTATE, "weight arena overflow");
  return BAG_OK;
}

static bag_status seed_weights(bag_ctx* ctx) {
  const uint64_t seed = ctx->arch.weight_seed;
  // weights and biases N(0, 0.02) (Irwin-Hall(4) approximation); QK-norm scales
  // 1 + N(0, 0.02)
  auto fill = [&](const Tensor& t, int slot, int id, bool is_norm) -> bag_status {
    const double sd = 0.02;
    const float c32 = (float)(sd * std::sqrt(3.0) / 65536.0);
    cudaError_t e = fill_synth(t.p, t.n, sm_start(seed, (uint64_t)slot * 256 + id), is_norm ? 1.f : 0.f,
                               c32, t.bf16, ctx->stream);
    if (e != cudaSuccess) return fail(ctx, BAG_ECUDA, std::string("fill: ") + cudaGetErrorString(e));
    return BAG_OK;
  };
  for (auto& kv : ctx->G) {
    auto it = kGlobalIds.find(kv.first);
    if (it == kGlobalIds.end()) return fail(ctx, BAG_ESTATE, "unknown global " + kv.first);
    CKS(fill(kv.second, 0, it->second, false));
  }
  const auto dids = double_ids();
  for (int b = 0; b < ctx->nblk; ++b) {
    const Block& blk = ctx->blocks[b];
    const std::map<std::string, int>& ids =
        blk.type == BT_SINGLE ? kSingleIds : (blk.type == BT_DOUBLE ? dids : kWanIds);
    for (auto& kv : blk.w) {
      auto it = ids.find(kv.first);
      if (it == ids.end()) return fail(ctx, BAG_ESTATE, "unknown block tensor " + kv.first);
      const bool is_norm = kv.first.size() > 5 && kv.first.compare(kv.first.size() - 5, 5, "_norm") == 0;
      CKS(fill(kv.second, 1 + b, it->second, is_norm));
    }
  }
  return BAG_OK;
}

// Layer shapes (out, in) of each gate kind, in evaluation / storage order (Eq. 1; the
// six-input architectures are App. A.2's: 449 and 785 parameters).
static std::vector<std::pair<int, int>> gate_shapes(int kind) {
  if (kind == BAG_GATE_FLUX6) return {{8, 6}, {8, 8}, {32, 8}, {1, 32}};
  if (kind == BAG_GATE_WAN6) return {{8, 3}, {8, 8}, {8, 3}, {8, 8}, {32, 16}, {1, 32}};
  return {{16, 3}, {1, 16}};
}
static int gate_param_count(int kind) {
  int n = 0;
  for (auto& s : gate_shapes(kind)) n += s.first * s.second + s.first;
  return n;
}
static int gate_inputs(int kind) { return kind == BAG_GATE_MLP3 ? 3 : 6; }

static bag_status seed_gate(bag_ctx* ctx) {
  // per layer W ~ U(-a, a), a = sqrt(6 / (in + out)) and b ~ U(-0.1, 0.1); generator keys
  // 1, 2, ... in storage order; z-score statistics 0 and 1
  std::vector<float> g(kGateFloats, 0.f);
  const uint64_t s = ctx->arch.gate_seed;
  uint64_t key = 1;
  int off = 0;
  for (auto& sh : gate_shapes(ctx->arch.gate_kind)) {
    const double a = std::sqrt(6.0 / (sh.first + sh.second));
    sm_uniform(s, key, sh.first * sh.second, -a, a, g.data() + off);
    off += sh.first * sh.second;
    sm_uniform(s, key + 1, sh.first, -0.1, 0.1, g.data() + off);
    off += sh.first;
    key += 2;
  }
  for (int i = 0; i < 6; ++i) g[kGateSd + i] = 1.f;
  CK(cudaMemcpy(ctx->d_gate, g.data(), g.size() * 4, cudaMemcpyHostToDevice));
  return BAG_OK;
}

static void rope_table(const bag_ctx* ctx, std::vector<float2>& tab) {
  // angle of pair j (axes laid out one after another) at token position p:
  // p_axis * theta^(-2 jj / d_axis)
  const int half = ctx->dh / 2;
  tab.assign((size_t)ctx->nrope * half, make_float2(1.f, 0.f));
  const int f = ctx->arch.grid[0], r = ctx->arch.grid[1], c = ctx->arch.grid[2];
  const int txt_rows = ctx->arch.kind == BAG_KIND_WAN ? 0 : ctx->nx;
  for (int row = 0; row < ctx->nrope; ++row) {
    double pos[3] = {0, 0, 0};
    if (row >= txt_rows) {
      const int i = row - txt_rows;
      pos[0] = i / (r * c);
      pos[1] = (i / c) % r;
      pos[2] = i % c;
    }
    int j = 0;
    for (int a = 0; a < 3; ++a) {
      const int da = ctx->arch.rope_axes[a];
      for (int jj = 0; jj < da / 2; ++jj, ++j) {
        const double ang = pos[a] * std::pow(10000.0, -2.0 * jj / da);
        tab[(size_t)row * half + j] = make_float2((float)std::cos(ang), (float)std::sin(ang));
      }
    }
  }
  (void)f;
}

// Noise levels sigma_i, i = 0..T: u_i = 1 - i/T, time-shifted s u / (1 + (s - 1) u).
static std::vector<double> sigma_grid(int T, float shift) {
  const double s = shift == 0.f ? 1.0 : (double)shift;
  std::vector<double> g(T + 1);
  for (int i = 0; i <= T; ++i) {
    const double u = 1.0 - (double)i / T;
    g[i] = s == 1.0 ? u : s * u / (1.0 + (s - 1.0) * u);
  }
  return g;
}

// UniPC (Zhao et al. 2023) of order 2 with its corrector, data-prediction form with
// B(h) = e^{-h} - 1, on a flow-matching grid (alpha = 1 - sigma, lambda = log(alpha /
// sigma)).  A move s -> t is x_t = (sigma_t / sigma_s) x_s - alpha_t psi m_s -
// alpha_t B sum_k rho_k D_k, psi = B = e^{-h} - 1, D_k = (m_k - m_s) / r_k,
// r_k = (lambda_k - lambda_s) / h; the corrector adds the new point (r = 1, D = m_t -
// m_s).  One coefficient: rho = 1/2; two: R rho = b with R = [[1, 1], [r_1, 1]],
// b_j = j! psi_{j+1} / B, psi_{j+1} = psi_j / (-h) - 1 / j!.  Predictor order
// min(2, i + 1, T - i); earlier points at sigma = 1 are not used.  The step's update is
// folded into fixed weights of x_i, the previous corrected sample and m_i, m_{i-1},
// m_{i-2} (UC_* layout).
static std::vector<float> unipc_table(const std::vector<double>& sig) {
  const int T = (int)sig.size() - 1;
  auto lam = [&](int i) { return std::log1p(-sig[i]) - std::log(sig[i]); };
  struct Move {
    double ratio, at, psi, hh;
  };
  auto move = [&](int s, int t) {
    const double at = 1.0 - sig[t], as = 1.0 - sig[s];
    const double emh = (sig[t] * as) / (at * sig[s]);
    return Move{sig[t] / sig[s], at, emh - 1.0, std::log(emh)};
  };
  std::vector<float> tab((size_t)T * kUniCoefs, 0.f);
  bool prev_hist = false;  // did the predictor of the previous step use m_{i-2}?
  for (int i = 0; i < T; ++i) {
    float* k = tab.data() + (size_t)i * kUniCoefs;
    k[UC_SIG] = (float)sig[i];
    if (i == 0) {
      k[UC_CX] = 1.f;
    } else {
      const Move mv = move(i - 1, i);
      const double B = mv.psi, aB = mv.at * B;
      double cm1 = -mv.at * mv.psi, cm2 = 0.0, cmt;
      if (!prev_hist) {
        cm1 += aB * 0.5;
        cmt = -aB * 0.5;
      } else {
        const double r1 = (lam(i - 2) - lam(i - 1)) / (-mv.hh);
        double p = mv.psi, b[2];
        double fact = 1.0;
        for (int j = 1; j <= 2; ++j) {
          p = (std::isfinite(mv.hh) ? p / mv.hh : 0.0) - 1.0 / fact;
          b[j - 1] = fact * p / B;
          fact *= j + 1;
        }
        const double rho1 = (b[0] - b[1]) / (1.0 - r1), rho2 = b[0] - rho1;
        cm1 += aB * (rho1 / r1 + rho2);
        cm2 = -aB * rho1 / r1;
        cmt = -aB * rho2;
      }
      k[UC_CLAST] = (float)mv.ratio;
      k[UC_CM1] = (float)cm1;
      k[UC_CM2] = (float)cm2;
      k[UC_CMT] = (float)cmt;
    }
    const int p = std::min(std::min(2, i + 1), T - i);
    const bool hist = p >= 2 && sig[i - 1] < 1.0;
    const Move mv = move(i, i + 1);
    double dm0 = -mv.at * mv.psi, dm1 = 0.0;
    if (hist) {
      const double r = (lam(i - 1) - lam(i)) / (-mv.hh);
      const double aB = mv.at * mv.psi;
      dm0 += aB * 0.5 / r;
      dm1 = -aB * 0.5 / r;
    }
    k[UC_DX] = (float)mv.ratio;
    k[UC_DM0] = (float)dm0;
    k[UC_DM1] = (float)dm1;
    prev_hist = hist;
  }
  return tab;
}

static bag_status alloc_activations(bag_ctx* ctx) {
  const size_t es = ctx->act_size;
  const long d = ctx->d, F = ctx->F, ni = ctx->ni, nx = ctx->nx, N = ctx->N, T = ctx->T;
  const bool wan = ctx->arch.kind == BAG_KIND_WAN;
  ctx->vpad = ((long)ctx->nrope + 127) / 128 * 128;
  ctx->vpad_c = ((long)nx + 127) / 128 * 128;
  // under guidance both branches share one stream and one set of activation buffers
  // (rows of both branches, see enq_block)
  const long nb = ctx->arch.cfg ? 2 : 1;
  const long rows = (wan ? ni : N) * nb;
  Arena A;
  A.add((void**)&ctx->x, (size_t)ni * ctx->C * 4);
  A.add((void**)&ctx->xb, (size_t)ni * ctx->C * 2 * 2);  // bf16 hi | lo halves of x
  A.add((void**)&ctx->h_in, (size_t)ni * d * 4);
  A.add((void**)&ctx->hj, (size_t)rows * d * 4);
  A.add((void**)&ctx->R, (size_t)ni * d * 4);
  // the signal's observable: in the operand precision for block 0's modulated input, in
  // fp32 for the post-patch-embedding tokens (a small drift is a difference of two nearly
  // equal tensors, which bf16 storage would bias)
  const size_t obs_es = ctx->arch.observable == BAG_OBS_EMBEDDED ? 4 : es;
  A.add(&ctx->m_cur, (size_t)ni * d * obs_es);
  A.add(&ctx->m_last, (size_t)ni * d * obs_es);
  A.add((void**)&ctx->sig_partial, (size_t)ni * 4 * 4);
  A.add(&ctx->xn, (size_t)rows * d * es);
  A.add(&ctx->q, (size_t)rows * d * es);
  A.add(&ctx->k, (size_t)rows * d * es);
  A.add(&ctx->vt, std::max((size_t)rows * d, (size_t)nb * d * ctx->vpad) * es);
  A.add(&ctx->cat, (size_t)rows * (d + F) * es);
  if (wan) {
    A.add(&ctx->qc, (size_t)nb * ni * d * es);
    A.add(&ctx->kc, (size_t)nb * nx * d * es);
    A.add(&ctx->vtc, std::max((size_t)nb * nx * d, (size_t)nb * d * ctx->vpad_c) * es);
  }
  A.add(&ctx->txt_stage, (size_t)nb * nx * d * es);  // [text_c; text_u]
  A.add((void**)&ctx->pooled_stage, (size_t)d * 4);
  A.add((void**)&ctx->rope, (size_t)ctx->nrope * (ctx->dh / 2) * sizeof(float2));
  A.add((void**)&ctx->dsig, (size_t)T * 4);
  A.add((void**)&ctx->d_sigma, (size_t)(T + 1) * 8);
  if (ctx->arch.sampler == BAG_SAMPLER_UNIPC) {
    A.add((void**)&ctx->uni_coef, (size_t)T * kUniCoefs * 4);
    A.add((void**)&ctx->uni_xl, (size_t)ni * ctx->C * 4);
    A.add((void**)&ctx->uni_m0, (size_t)ni * ctx->C * 4);
    A.add((void**)&ctx->uni_m1, (size_t)ni * ctx->C * 4);
  }
  A.add((void**)&ctx->sin_all, (size_t)T * kTembDim * 4);
  A.add((void**)&ctx->t1o, (size_t)T * d * 4);
  A.add((void**)&ctx->svec, (size_t)T * d * 4);
  A.add((void**)&ctx->splitbuf, (size_t)T * 2 * std::max<long>(kTembDim, d) * 2);
  A.add((void**)&ctx->vec_all, (size_t)T * d * 4);
  A.add((void**)&ctx->mod_all, (size_t)T * ctx->mod_stride * 4);
  if (wan) A.add((void**)&ctx->wan_shared, (size_t)T * 8 * d * 4);
  if (ctx->arch.cfg) {
    A.add((void**)&ctx->R_u, (size_t)ni * d * 4);
    A.add((void**)&ctx->vcond, (size_t)ni * ctx->C * 4);
    if (!wan) {
      A.add((void**)&ctx->pooled_stage_u, (size_t)d * 4);
      A.add((void**)&ctx->vec_all_u, (size_t)T * d * 4);
      A.add((void**)&ctx->svec_u, (size_t)T * d * 4);
      A.add((void**)&ctx->mod_all_u, (size_t)T * ctx->mod_stride * 4);
    }
  }
  A.add((void**)&ctx->st, sizeof(DevState));
  A.add((void**)&ctx->st_op, sizeof(DevState));
  A.add((void**)&ctx->log, (size_t)T * kLogFloats * 4);
  A.add((void**)&ctx->d_gate, kGateFloats * 4);
  A.add((void**)&ctx->d_pmask, (size_t)T);
  ctx->tmp_f32_n = (long)nx * d;
  A.add((void**)&ctx->tmp_f32, (size_t)ctx->tmp_f32_n * 4);
  if (cudaMalloc(&ctx->aarena, A.off) != cudaSuccess)
    return fail(ctx, BAG_ENOMEM, "activation allocation of " + std::to_string(A.off) + " bytes failed");
  A.bind((char*)ctx->aarena);
  if (ctx->arch.cfg) ctx->txt_stage_u = (char*)ctx->txt_stage + (size_t)nx * d * es;
  if (ctx->arch.cfg && wan) ctx->mod_all_u = ctx->mod_all;
  CK(cudaMemset(ctx->aarena, 0, A.off));
  std::vector<float2> tab;
  rope_table(ctx, tab);
  CK(cudaMemcpy(ctx->rope, tab.data(), tab.size() * sizeof(float2), cudaMemcpyHostToDevice));
  const std::vector<double> sg = sigma_grid(T, ctx->arch.shift);
  std::vector<float> ds(T);
  for (int t = 0; t < T; ++t) ds[t] = (float)(sg[t + 1] - sg[t]);
  CK(cudaMemcpy(ctx->dsig, ds.data(), T * 4, cudaMemcpyHostToDevice));
  CK(cudaMemcpy(ctx->d_sigma, sg.data(), (T + 1) * 8, cudaMemcpyHostToDevice));
  if (ctx->arch.sampler == BAG_SAMPLER_UNIPC) {
    const std::vector<float> tab = unipc_table(sg);
    CK(cudaMemcpy(ctx->uni_coef, tab.data(), tab.size() * 4, cudaMemcpyHostToDevice));
  }
  return BAG_OK;
}

// ---------------------------------------------------------------------------
// enqueue helpers
// ---------------------------------------------------------------------------
static int prof_event(bag_ctx* ctx) {
  if (ctx->ev_used == ctx->ev_pool.size()) {
    cudaEvent_t ev;
    if (cudaEventCreate(&ev) != cudaSuccess) return -1;
    ctx->ev_pool.push_back(ev);
  }
  return (int)ctx->ev_used++;
}

// One enqueued segment of kernels on one stream (a step's prefix, a body of the
// conditional, the suffix, a block, the per-sample preparation).  Every launch after
// the segment's first is made with programmatic stream serialization unless profiling
// (whose events sit between the kernels) or the context turned it off.
struct Enq {
  bag_ctx* ctx;
  cudaStream_t s;
  long* count;
  cudaError_t e = cudaSuccess;
  Enq(bag_ctx* c, cudaStream_t st, long* n) : ctx(c), s(st), count(n) { g_pdl = false; }
  ~Enq() { g_pdl = false; }
  Enq(const Enq&) = delete;
  Enq& operator=(const Enq&) = delete;
  int pk = -1, pe0 = -1, pm = 0, pn = 0, pkk = 0, pv = 0;
  double pf = 0, pb = 0;
  // announce the next launch (kind, algorithmic flops and bytes, shape, kernel variant)
  // for profiling
  void pre(int kind, double flops, double bytes, int m = 0, int n = 0, int k = 0, int variant = 0) {
    if (!ctx->profiling) return;
    pv = variant;
    pe0 = prof_event(ctx);
    if (pe0 < 0) return;
    cudaEventRecord(ctx->ev_pool[pe0], s);
    pk = kind;
    pf = flops;
    pb = bytes;
    pm = m;
    pn = n;
    pkk = k;
  }
  void chk(cudaError_t r) {
    if (e == cudaSuccess && r != cudaSuccess) e = r;
    if (count) ++*count;
    g_pdl = ctx->pdl && !ctx->profiling;
    if (pk >= 0) {
      const int pe1 = prof_event(ctx);
      if (pe1 >= 0) {
        cudaEventRecord(ctx->ev_pool[pe1], s);
        ctx->prof.push_back({pk, pf, pb, pe0, pe1, pm, pn, pkk, pv});
      }
      pk = -1;
    }
  }
};

static Epi base_epi(const bag_ctx* ctx, const DevState* st, int flag_want) {
  Epi e;
  e.st = st;
  e.flag_want = flag_want;
  e.act_bf16 = ctx->act_bf16;
  // attention operands of bf16 backbones are fp16 (see the attention kernel)
  e.qkv_type = ctx->act_bf16 ? kStoreF16 : kStoreF32;
  return e;
}

static inline void* off_act(const bag_ctx* ctx, void* p, long elems) {
  return (char*)p + elems * (long)ctx->act_size;
}

static void enq_gemm(Enq& q, const void* A, long lda, const Tensor& W, long ldw, int M, int N,
                     int K, const Epi& e) {
  {
    const double es = (double)q.ctx->act_size;
    double out = (double)M * N * 4;
    if (e.kind == EPI_GATED_RES || e.kind == EPI_RES_ADD) out = (double)M * N * 8;
    else if (e.kind == EPI_QKV || e.kind == EPI_GELU) out = (double)M * N * es;
    q.pre(BAG_PROF_GEMM, 2.0 * M * N * K, ((double)M + N) * K * es + out, M, N, K,
          q.ctx->act_bf16 ? gemm_uses_pair(M, 0, N) : 0);
  }
  q.chk(gemm(A, lda, W.p, ldw, M, N, K, q.ctx->act_bf16, e, q.ctx->st ? &q.ctx->st->err : nullptr, q.s));
}

// Two projections with the same N and K (image and text stream of a double-stream
// block) in one tensor-core launch; fp32 configurations run them one after the other.
static void enq_gemm2(Enq& q, const void* A0, long lda0, const Tensor& W0, long ldw0, int M0,
                      const Epi& e0, const void* A1, long lda1, const Tensor& W1, long ldw1,
                      int M1, const Epi& e1, int N, int K) {
  if (!q.ctx->act_bf16) {
    enq_gemm(q, A0, lda0, W0, ldw0, M0, N, K, e0);
    enq_gemm(q, A1, lda1, W1, ldw1, M1, N, K, e1);
    return;
  }
  const double es = 2.0;
  double out = (double)(M0 + M1) * N * 4;
  if (e0.kind == EPI_GATED_RES || e0.kind == EPI_RES_ADD) out = (double)(M0 + M1) * N * 8;
  else if (e0.kind == EPI_QKV || e0.kind == EPI_GELU) out = (double)(M0 + M1) * N * es;
  q.pre(BAG_PROF_GEMM, 2.0 * (M0 + M1) * N * K, ((double)M0 + M1 + 2.0 * N) * K * es + out,
        M0 + M1, N, K, gemm_uses_pair(M0, M1, N));
  q.chk(gemm2(A0, lda0, W0.p, ldw0, M0, e0, A1, lda1, W1.p, ldw1, M1, e1, N, K,
              q.ctx->st ? &q.ctx->st->err : nullptr, q.s));
}

static void enq_ln(Enq& q, const float* x, long ldx, void* y, long ldy, int rows, int split,
                   const float* sh_a, const float* sc_a, const float* sh_b, const float* sc_b,
                   const DevState* st, int flag_want) {
  LnArgs a{};
  a.x = x;
  a.ldx = ldx;
  a.y = y;
  a.ldy = ldy;
  a.y_bf16 = q.ctx->act_bf16;
  a.rows = rows;
  a.cols = q.ctx->d;
  a.split = split;
  a.shift_a = sh_a;
  a.scale_a = sc_a;
  a.shift_b = sh_b;
  a.scale_b = sc_b;
  a.mod_step = q.ctx->mod_stride;
  a.st = st;
  a.flag_want = flag_want;
  q.pre(BAG_PROF_NORM, 0.0, (double)rows * q.ctx->d * (4.0 + q.ctx->act_size));
  q.chk(ln_mod(a, q.s));
}

// LayerNorm + modulation with four row segments [0, s1), [s1, s2), [s2, s3), [s3, rows),
// each under its own modulation (shift at m, scale at m + d).
static void enq_ln4(Enq& q, const float* x, long ldx, void* y, long ldy, int rows, int s1, int s2, int s3,
                    const float* ma, const float* mb, const float* mc, const float* md, const DevState* st,
                    int flag_want) {
  const long d = q.ctx->d;
  LnArgs a{};
  a.x = x;
  a.ldx = ldx;
  a.y = y;
  a.ldy = ldy;
  a.y_bf16 = q.ctx->act_bf16;
  a.rows = rows;
  a.cols = (int)d;
  a.split = s1;
  a.split2 = s2;
  a.split3 = s3;
  a.shift_a = ma;
  a.scale_a = ma + d;
  a.shift_b = mb;
  a.scale_b = mb + d;
  a.shift_c = mc;
  a.scale_c = mc + d;
  a.shift_d = md;
  a.scale_d = md + d;
  a.mod_step = q.ctx->mod_stride;
  a.st = st;
  a.flag_want = flag_want;
  q.pre(BAG_PROF_NORM, 0.0, (double)rows * d * (4.0 + q.ctx->act_size));
  q.chk(ln_mod(a, q.s));
}

static void enq_qkv_epi(const bag_ctx* ctx, Epi& e, int row_off, bool rope) {
  e.kind = EPI_QKV;
  e.q = ctx->q;
  e.k = ctx->k;
  e.v = ctx->vt;
  e.v_mode = ctx->act_bf16 ? 1 : 0;
  e.vpad = ctx->vpad;
  e.ldqk = ctx->d;
  e.d = ctx->d;
  e.dh = ctx->dh;
  e.row_off = row_off;
  e.col_base = 0;
  e.rope = rope ? ctx->rope : nullptr;
  e.mlp = off_act(ctx, ctx->cat, ctx->d);
  e.ldm = ctx->d + ctx->F;
}

// Attention of one branch, or of both guidance branches in one launch (nbr = 2, bf16
// backbones): branch 1's q / k rows br_q / br_k rows further, its V^T block right after
// branch 0's, its output to O_b1 / O2_b1.
struct AttnBranch {
  int nbr = 1;
  long br_q = 0, br_k = 0;
  void* o_b1 = nullptr;
  void* o2_b1 = nullptr;
};

static void enq_attn(Enq& q, const void* Q, const void* K, const void* V, long vpad, void* O,
                     long ldo, int nq, int nk, const DevState* st, int flag_want,
                     void* O2 = nullptr, int o_split = 0, const AttnBranch& ab = AttnBranch()) {
  const bag_ctx* ctx = q.ctx;
  AttnArgs a{};
  a.q = Q;
  a.ldq = ctx->d;
  a.k = K;
  a.ldk = ctx->d;
  a.v = V;
  a.v_mode = ctx->act_bf16 ? 1 : 0;
  a.ldv = ctx->d;
  a.vpad = vpad;
  a.o = O;
  a.ldo = ldo;
  a.o2 = O2;
  a.o_split = o_split;
  a.nbr = ab.nbr;
  a.br_q_rows = ab.br_q;
  a.br_k_rows = ab.br_k;
  a.o_b1 = ab.o_b1;
  a.o2_b1 = ab.o2_b1;
  a.nq = nq;
  a.nk = nk;
  a.heads = ctx->H;
  a.dh = ctx->dh;
  a.bf16 = ctx->act_bf16;
  a.f16 = ctx->act_bf16;  // q, k, v fp16 (written so by the projections' epilogues)
  a.st = st;
  a.flag_want = flag_want;
  q.pre(BAG_PROF_ATTN, 4.0 * nq * nk * ctx->H * ctx->dh * ab.nbr,
        ((double)nq * 2 + 2.0 * nk) * ctx->d * ctx->act_size * ab.nbr, nq, nk, ctx->H);
  q.chk(attention(a, ctx->st ? &ctx->st->err : nullptr, q.s));
}

// Per-branch buffers: branch 0 is the conditional (or only) branch, branch 1 the
// unconditional branch of classifier-free guidance.  Under guidance both branches live
// in one stream, ordered [text_c; text_u; image_c; image_u] (Wan: [image_c; image_u]),
// so that every projection takes both branches' rows in one launch; the q / k / v,
// attention-output and MLP buffers hold each branch's joint sequence [text; image].
static const float* br_mod(const bag_ctx* ctx, int br) { return br ? ctx->mod_all_u : ctx->mod_all; }
static const void* br_txt(const bag_ctx* ctx, int br) { return br ? ctx->txt_stage_u : ctx->txt_stage; }
static int n_branches(const bag_ctx* ctx) { return ctx->arch.cfg ? 2 : 1; }

// Branch-map fields of an epilogue whose problem holds nb branches of `rows` rows each.
static void epi_branches(const bag_ctx* ctx, Epi& e, int nb, int rows, long qk_rows, long vpad) {
  if (nb < 2) return;
  e.br_rows = rows;
  e.br_qk = qk_rows;
  e.br_vt = (long)ctx->H * ctx->dh * vpad;  // used only for transposed V (v_mode 1)
}

// One block of the stack on the stream h for nb branches (1: the joint [N, d] sequence
// with text rows first, or the Wan image stream [ni, d]; 2: both guidance branches in
// the order above), with each branch's modulation and (Wan) context.
static void enq_block(Enq& q, int b, float* h, const DevState* st, int fw, int nb = 1) {
  bag_ctx* ctx = q.ctx;
  const Block& blk = ctx->blocks[b];
  const long d = ctx->d, F = ctx->F, ldc = d + F;
  const int ni = ctx->ni, nx = ctx->nx, N = ctx->N;
  const float* mod = ctx->mod_all + blk.mod_off;                     // branch 0
  const float* modu = br_mod(ctx, nb > 1 ? 1 : 0) + blk.mod_off;      // branch 1 (or 0)
  const long ms = ctx->mod_stride;
  // element offset of branch 1's V: transposed per head for the tensor-core attention
  // (H x dh x vpad), else row-major like k (rows x d)
  auto v_br = [&](long rows, long vpad) { return ctx->act_bf16 ? (long)ctx->H * ctx->dh * vpad : rows * d; };
  const long vt_br = v_br(N, ctx->vpad);
  // QK-norm scales of a stream (pre = "", "img_" or "txt_"), when the block has them
  auto qk_norm = [&](Epi& e, const std::string& pre) {
    auto it = blk.w.find(pre + "q_norm");
    if (it == blk.w.end()) return;
    e.qn_q = (const float*)it->second.p;
    e.qn_k = (const float*)blk.w.at(pre + "k_norm").p;
  };
  // LayerNorm + modulation of the joint stream (nb * N rows) with the text rows of each
  // branch under (sh_t, sc_t) + offset and the image rows under (sh_i, sc_i) + offset
  auto ln_joint = [&](const float* mt_c, const float* mt_u, const float* mi_c, const float* mi_u,
                      long off) {
    if (nb == 1) {
      enq_ln(q, h, d, ctx->xn, d, N, nx, mt_c + off, mt_c + off + d, mi_c + off, mi_c + off + d, st, fw);
      return;
    }
    enq_ln4(q, h, d, ctx->xn, d, 2 * N, nx, 2 * nx, 2 * nx + ni, mt_c + off, mt_u + off, mi_c + off,
            mi_u + off, st, fw);
  };
  // attention of every branch: q / k / v of branch br at row br * N (transposed V at
  // br * vt_br); the output rows go back in stream order (text rows of branch br at
  // br * nx, its image rows at nb * nx + br * ni)
  auto attn_joint = [&]() {
    if (nb > 1 && ctx->act_bf16) {  // both branches in one launch
      AttnBranch ab;
      ab.nbr = 2;
      ab.br_q = ab.br_k = N;
      ab.o_b1 = off_act(ctx, ctx->cat, (long)nx * ldc);
      ab.o2_b1 = off_act(ctx, ctx->cat, ((long)nb * nx + ni - nx) * ldc);
      enq_attn(q, ctx->q, ctx->k, ctx->vt, ctx->vpad, ctx->cat, ldc, N, N, st, fw,
               off_act(ctx, ctx->cat, ((long)nb * nx - nx) * ldc), nx, ab);
      return;
    }
    for (int br = 0; br < nb; ++br) {
      void* o = off_act(ctx, ctx->cat, (long)br * nx * ldc);
      void* o2 = off_act(ctx, ctx->cat, ((long)nb * nx + (long)br * ni - nx) * ldc);
      enq_attn(q, off_act(ctx, ctx->q, (long)br * N * d), off_act(ctx, ctx->k, (long)br * N * d),
               off_act(ctx, ctx->vt, br * vt_br), ctx->vpad, o, ldc, N, N, st, fw,
               nb > 1 ? o2 : nullptr, nx);
    }
  };
  if (blk.type == BT_SINGLE) {
    ln_joint(mod, modu, mod, modu, 0);
    Epi e = base_epi(ctx, st, fw);
    enq_qkv_epi(ctx, e, 0, true);
    qk_norm(e, "");
    e.bias = (const float*)blk.w.at("lin1_b").p;
    Epi r = base_epi(ctx, st, fw);
    r.kind = EPI_GATED_RES;
    r.bias = (const float*)blk.w.at("lin2_b").p;
    r.resid = h;
    r.ldr = d;
    r.gate = mod + 2 * d;
    r.gate_u = modu + 2 * d;
    r.gate_step = ms;
    if (nb == 1) {
      enq_gemm(q, ctx->xn, d, blk.w.at("lin1_w"), d, N, (int)(3 * d + F), (int)d, e);
      attn_joint();
      enq_gemm(q, ctx->cat, ldc, blk.w.at("lin2_w"), ldc, N, (int)d, (int)(d + F), r);
      return;
    }
    // both branches: the text rows and the image rows as two problems of one launch
    // (the same weight), each covering the two branches
    Epi ei = e;
    ei.row_off = nx;
    ei.mlp = off_act(ctx, ctx->cat, 2L * nx * ldc + d);
    epi_branches(ctx, ei, nb, ni, N, ctx->vpad);
    epi_branches(ctx, e, nb, nx, N, ctx->vpad);
    enq_gemm2(q, off_act(ctx, ctx->xn, 2L * nx * d), d, blk.w.at("lin1_w"), d, 2 * ni, ei,
              ctx->xn, d, blk.w.at("lin1_w"), d, 2 * nx, e, (int)(3 * d + F), (int)d);
    attn_joint();
    Epi ri = r;
    ri.resid = h + 2L * nx * d;
    ri.br_rows = ni;
    r.br_rows = nx;
    enq_gemm2(q, off_act(ctx, ctx->cat, 2L * nx * ldc), ldc, blk.w.at("lin2_w"), ldc, 2 * ni, ri,
              ctx->cat, ldc, blk.w.at("lin2_w"), ldc, 2 * nx, r, (int)d, (int)(d + F));
    return;
  }
  if (blk.type == BT_DOUBLE) {
    const float* mi = mod;              // image stream modulation (6d), branch 0
    const float* mt = mod + 6 * d;      // text stream modulation (6d), branch 0
    const float* miu = modu;            // branch 1
    const float* mtu = modu + 6 * d;
    const long ti = (long)nb * nx;      // first image row of the stream
    float* h_img = h + ti * d;
    // attention half
    ln_joint(mt, mtu, mi, miu, 0);
    {
      Epi e = base_epi(ctx, st, fw);
      enq_qkv_epi(ctx, e, nx, true);
      e.bias = (const float*)blk.w.at("img_qkv_b").p;
      qk_norm(e, "img_");
      epi_branches(ctx, e, nb, ni, N, ctx->vpad);
      Epi e2 = base_epi(ctx, st, fw);
      enq_qkv_epi(ctx, e2, 0, true);
      e2.bias = (const float*)blk.w.at("txt_qkv_b").p;
      qk_norm(e2, "txt_");
      epi_branches(ctx, e2, nb, nx, N, ctx->vpad);
      enq_gemm2(q, off_act(ctx, ctx->xn, ti * d), d, blk.w.at("img_qkv_w"), d, nb * ni, e,
                ctx->xn, d, blk.w.at("txt_qkv_w"), d, nb * nx, e2, (int)(3 * d), (int)d);
    }
    attn_joint();
    {
      Epi r = base_epi(ctx, st, fw);
      r.kind = EPI_GATED_RES;
      r.bias = (const float*)blk.w.at("img_proj_b").p;
      r.resid = h_img;
      r.ldr = d;
      r.gate = mi + 2 * d;
      r.gate_u = miu + 2 * d;
      r.gate_step = ms;
      if (nb > 1) r.br_rows = ni;
      Epi r2 = r;
      r2.bias = (const float*)blk.w.at("txt_proj_b").p;
      r2.resid = h;
      r2.gate = mt + 2 * d;
      r2.gate_u = mtu + 2 * d;
      if (nb > 1) r2.br_rows = nx;
      enq_gemm2(q, off_act(ctx, ctx->cat, ti * ldc), ldc, blk.w.at("img_proj_w"), d, nb * ni, r,
                ctx->cat, ldc, blk.w.at("txt_proj_w"), d, nb * nx, r2, (int)d, (int)d);
    }
    // MLP half
    ln_joint(mt, mtu, mi, miu, 3 * d);
    {
      Epi u = base_epi(ctx, st, fw);
      u.kind = EPI_GELU;
      u.out_bf16 = ctx->act_bf16;
      u.ldo = ldc;
      u.bias = (const float*)blk.w.at("img_up_b").p;
      u.out = off_act(ctx, ctx->cat, ti * ldc + d);
      Epi u2 = u;
      u2.bias = (const float*)blk.w.at("txt_up_b").p;
      u2.out = off_act(ctx, ctx->cat, d);
      enq_gemm2(q, off_act(ctx, ctx->xn, ti * d), d, blk.w.at("img_up_w"), d, nb * ni, u,
                ctx->xn, d, blk.w.at("txt_up_w"), d, nb * nx, u2, (int)F, (int)d);
      Epi r = base_epi(ctx, st, fw);
      r.kind = EPI_GATED_RES;
      r.bias = (const float*)blk.w.at("img_down_b").p;
      r.resid = h_img;
      r.ldr = d;
      r.gate = mi + 5 * d;
      r.gate_u = miu + 5 * d;
      r.gate_step = ms;
      if (nb > 1) r.br_rows = ni;
      Epi r2 = r;
      r2.bias = (const float*)blk.w.at("txt_down_b").p;
      r2.resid = h;
      r2.gate = mt + 5 * d;
      r2.gate_u = mtu + 5 * d;
      if (nb > 1) r2.br_rows = nx;
      enq_gemm2(q, off_act(ctx, ctx->cat, ti * ldc + d), ldc, blk.w.at("img_down_w"), F, nb * ni, r,
                off_act(ctx, ctx->cat, d), ldc, blk.w.at("txt_down_w"), F, nb * nx, r2, (int)d, (int)F);
    }
    return;
  }
  // Wan block: self-attention, cross-attention, FFN; under guidance the stream holds
  // [image_c; image_u] and the staged contexts [context_c; context_u]
  const int R = nb * ni;
  const long vtw_br = v_br(ni, ctx->vpad), vtc_br = v_br(nx, ctx->vpad_c);
  enq_ln(q, h, d, ctx->xn, d, R, ni, mod, mod + d, modu, modu + d, st, fw);
  {
    Epi e = base_epi(ctx, st, fw);
    enq_qkv_epi(ctx, e, 0, true);
    e.bias = (const float*)blk.w.at("sa_qkv_b").p;
    epi_branches(ctx, e, nb, ni, ni, ctx->vpad);
    enq_gemm(q, ctx->xn, d, blk.w.at("sa_qkv_w"), d, R, (int)(3 * d), (int)d, e);
  }
  AttnBranch ab;  // Wan, both branches in one launch (bf16 backbones)
  const int nl = (nb > 1 && ctx->act_bf16) ? 1 : nb;
  if (nl < nb) {
    ab.nbr = 2;
    ab.br_q = ab.br_k = ni;
    ab.o_b1 = off_act(ctx, ctx->cat, (long)ni * ldc);
  }
  for (int br = 0; br < nl; ++br)
    enq_attn(q, off_act(ctx, ctx->q, (long)br * ni * d), off_act(ctx, ctx->k, (long)br * ni * d),
             off_act(ctx, ctx->vt, br * vtw_br), ctx->vpad, off_act(ctx, ctx->cat, (long)br * ni * ldc),
             ldc, ni, ni, st, fw, nullptr, 0, ab);
  {
    Epi r = base_epi(ctx, st, fw);
    r.kind = EPI_GATED_RES;
    r.bias = (const float*)blk.w.at("sa_o_b").p;
    r.resid = h;
    r.ldr = d;
    r.gate = mod + 2 * d;
    r.gate_u = modu + 2 * d;
    r.gate_step = ms;
    if (nb > 1) r.br_rows = ni;
    enq_gemm(q, ctx->cat, ldc, blk.w.at("sa_o_w"), d, R, (int)d, (int)d, r);
  }
  enq_ln(q, h, d, ctx->xn, d, R, 0, nullptr, nullptr, nullptr, nullptr, st, fw);
  {
    Epi e = base_epi(ctx, st, fw);
    e.kind = EPI_STORE;
    e.out = ctx->qc;
    e.ldo = d;
    e.out_bf16 = ctx->act_bf16 ? kStoreF16 : kStoreF32;  // an attention operand
    e.bias = (const float*)blk.w.at("ca_q_b").p;
    enq_gemm(q, ctx->xn, d, blk.w.at("ca_q_w"), d, R, (int)d, (int)d, e);
    Epi kv = base_epi(ctx, st, fw);
    kv.kind = EPI_QKV;
    kv.q = nullptr;
    kv.k = ctx->kc;
    kv.v = ctx->vtc;
    kv.v_mode = ctx->act_bf16 ? 1 : 0;
    kv.vpad = ctx->vpad_c;
    kv.ldqk = d;
    kv.d = (int)d;
    kv.dh = ctx->dh;
    kv.row_off = 0;
    kv.col_base = (int)d;
    kv.rope = nullptr;
    kv.bias = (const float*)blk.w.at("ca_kv_b").p;
    epi_branches(ctx, kv, nb, nx, nx, ctx->vpad_c);
    enq_gemm(q, ctx->txt_stage, d, blk.w.at("ca_kv_w"), d, nb * nx, (int)(2 * d), (int)d, kv);
  }
  AttnBranch abc = ab;
  abc.br_k = nx;
  for (int br = 0; br < nl; ++br)
    enq_attn(q, off_act(ctx, ctx->qc, (long)br * ni * d), off_act(ctx, ctx->kc, (long)br * nx * d),
             off_act(ctx, ctx->vtc, br * vtc_br), ctx->vpad_c, off_act(ctx, ctx->cat, (long)br * ni * ldc),
             ldc, ni, nx, st, fw, nullptr, 0, abc);
  {
    Epi r = base_epi(ctx, st, fw);
    r.kind = EPI_RES_ADD;
    r.bias = (const float*)blk.w.at("ca_o_b").p;
    r.resid = h;
    r.ldr = d;
    enq_gemm(q, ctx->cat, ldc, blk.w.at("ca_o_w"), d, R, (int)d, (int)d, r);
  }
  enq_ln(q, h, d, ctx->xn, d, R, ni, mod + 3 * d, mod + 4 * d, modu + 3 * d, modu + 4 * d, st, fw);
  {
    Epi u = base_epi(ctx, st, fw);
    u.kind = EPI_GELU;
    u.out_bf16 = ctx->act_bf16;
    u.ldo = ldc;
    u.bias = (const float*)blk.w.at("ffn_up_b").p;
    u.out = off_act(ctx, ctx->cat, d);
    enq_gemm(q, ctx->xn, d, blk.w.at("ffn_up_w"), d, R, (int)F, (int)d, u);
    Epi r = base_epi(ctx, st, fw);
    r.kind = EPI_GATED_RES;
    r.bias = (const float*)blk.w.at("ffn_down_b").p;
    r.resid = h;
    r.ldr = d;
    r.gate = mod + 5 * d;
    r.gate_u = modu + 5 * d;
    r.gate_step = ms;
    if (nb > 1) r.br_rows = ni;
    enq_gemm(q, off_act(ctx, ctx->cat, d), ldc, blk.w.at("ffn_down_w"), F, R, (int)d, (int)F, r);
  }
}

// Image rows of branch br in the stream (text rows of branch br start at br * nx).
static float* img_stream(bag_ctx* ctx, int br = 0) {
  if (ctx->arch.kind == BAG_KIND_WAN) return ctx->hj + (long)br * ctx->ni * ctx->d;
  return ctx->hj + ((long)n_branches(ctx) * ctx->nx + (long)br * ctx->ni) * ctx->d;
}

static void enq_prefix(Enq& q, int use_cond, unsigned long long handle) {
  bag_ctx* ctx = q.ctx;
  const long d = ctx->d;
  Epi pe = base_epi(ctx, ctx->st, -1);
  pe.kind = EPI_DUAL_F32;
  pe.bias = (const float*)ctx->G.at("pe_b").p;
  pe.out = ctx->h_in;
  pe.ldo = d;
  pe.out2 = img_stream(ctx);
  pe.ldo2 = d;
  if (ctx->act_bf16) {
    // the latent enters as bf16 hi + lo halves (split A): the patch embedding, and with
    // it the post-patch-embedding observable, carries no bf16 rounding of x
    q.pre(BAG_PROF_GEMM, 4.0 * ctx->ni * d * ctx->C,
          ((double)ctx->ni * 2 + d) * ctx->C * 2 + (double)ctx->ni * d * 8, ctx->ni, (int)d, 2 * ctx->C,
          gemm_uses_pair(ctx->ni, 0, (int)d));
    q.chk(gemm(ctx->xb, 2L * ctx->C, ctx->G.at("pe_w").p, ctx->C, ctx->ni, (int)d, ctx->C, 1, pe,
               ctx->st ? &ctx->st->err : nullptr, q.s, 0, 1));
  } else {
    enq_gemm(q, ctx->x, ctx->C, ctx->G.at("pe_w"), ctx->C, ctx->ni, (int)d, ctx->C, pe);
  }
  // signal (Eq. 3 drift and step change) on the observable: block 0's first modulated
  // input on the image stream, or the post-patch-embedding tokens themselves
  const Block& b0 = ctx->blocks[0];
  const float* m0 = ctx->mod_all + b0.mod_off;  // image-stream modulation comes first
  LnArgs a{};
  a.x = ctx->h_in;
  a.ldx = d;
  a.y = ctx->m_cur;
  a.ldy = d;
  a.y_bf16 = ctx->act_bf16;
  a.rows = ctx->ni;
  a.cols = (int)d;
  a.split = 0;
  if (ctx->arch.observable == BAG_OBS_EMBEDDED) {
    a.identity = 1;
    a.y_bf16 = 0;
    a.shift_a = a.shift_b = a.scale_a = a.scale_b = nullptr;
  } else {
    a.shift_a = a.shift_b = m0;
    a.scale_a = a.scale_b = m0 + d;
  }
  a.mod_step = ctx->mod_stride;
  a.sig_ref = ctx->m_last;
  a.sig_ref_w = ctx->m_last;  // refreshed here after a full step (m_last <- m_{t-1})
  a.sig_ref2 = ctx->m_cur;    // still the previous step's observable; replaced in place
  a.sig_partial = ctx->sig_partial;
  a.sig_on = 1;
  a.st = ctx->st;
  a.flag_want = -1;
  q.pre(BAG_PROF_SIGNAL, 0.0, (double)ctx->ni * d * (4.0 + 3.0 * (a.y_bf16 ? 2.0 : 4.0)));
  q.chk(ln_mod(a, q.s));
  q.pre(BAG_PROF_GATE, 0.0, (double)ctx->ni * 8);
  q.chk(gate_step(ctx->st, ctx->sig_partial, ctx->ni, ctx->d_gate, ctx->arch.gate_kind, ctx->thr, ctx->T, ctx->B,
                  ctx->policy, ctx->d_pmask, ctx->delta, ctx->log, handle, use_cond, q.s));
}

// Full step: the whole stack for every branch, then each branch's residual is cached
// (and the conditional branch's signal observable m_t becomes m_last).
static void enq_full(Enq& q, int fw) {
  bag_ctx* ctx = q.ctx;
  const long d = ctx->d;
  const int nb = n_branches(ctx);
  for (int br = 0; br < nb; ++br) {
    if (ctx->arch.kind != BAG_KIND_WAN)
      q.chk(copy_rows_f32(ctx->st, fw, ctx->hj + (long)br * ctx->nx * d, d, br_txt(ctx, br), d, ctx->act_bf16,
                          ctx->nx, (int)d, q.s));
    if (br) {  // the patch-embed epilogue filled only the conditional stream's image rows
      q.pre(BAG_PROF_CACHE, 0.0, (double)ctx->ni * d * 8.0);
      q.chk(copy_rows_f32(ctx->st, fw, img_stream(ctx, br), d, ctx->h_in, d, 0, ctx->ni, (int)d, q.s));
    }
  }
  // the stack once for all branches (every projection takes both branches' rows)
  for (int b = 0; b < ctx->nblk; ++b) enq_block(q, b, ctx->hj, ctx->st, fw, nb);
  for (int br = 0; br < nb; ++br) {
    q.pre(BAG_PROF_CACHE, 0.0, (double)ctx->ni * d * 12.0);
    q.chk(cache_refresh(ctx->st, img_stream(ctx, br), ctx->h_in, br ? ctx->R_u : ctx->R,
                        (long)ctx->ni * d, fw, q.s));
  }
}

// Cached step: every branch adds its own cached residual (one shared mask, App. A.1).
static void enq_skip(Enq& q, int fw) {
  bag_ctx* ctx = q.ctx;
  for (int br = 0; br < n_branches(ctx); ++br) {
    q.pre(BAG_PROF_CACHE, 0.0, (double)ctx->ni * ctx->d * 12.0);
    q.chk(cache_reuse(ctx->st, img_stream(ctx, br), ctx->h_in, br ? ctx->R_u : ctx->R,
                      (long)ctx->ni * ctx->d, fw, q.s));
  }
}

// Final layer and Euler update.  Under guidance the conditional velocity is stored and
// the unconditional branch's final GEMM applies v_u + g (v_c - v_u) in its epilogue.
static void enq_suffix(Enq& q) {
  bag_ctx* ctx = q.ctx;
  const long d = ctx->d;
  const int nb = n_branches(ctx);
  for (int br = 0; br < nb; ++br) {
    const float* fm = br_mod(ctx, br) + ctx->fmod_off;
    enq_ln(q, img_stream(ctx, br), d, ctx->xn, d, ctx->ni, 0, fm, fm + d, fm, fm + d, ctx->st, -1);
    Epi e = base_epi(ctx, ctx->st, -1);
    e.bias = (const float*)ctx->G.at("fin_b").p;
    if (br + 1 < nb) {
      e.kind = EPI_STORE;
      e.out = ctx->vcond;
      e.ldo = ctx->C;
      e.out_bf16 = 0;
    } else {
      e.kind = EPI_EULER;
      e.x = ctx->x;
      e.xb = ctx->act_bf16 ? ctx->xb : nullptr;
      e.ldx = ctx->C;
      e.dsig = ctx->dsig;
      if (br) {
        e.vcond = ctx->vcond;
        e.guidance = ctx->arch.guidance;
      }
      if (ctx->arch.sampler == BAG_SAMPLER_UNIPC) {
        e.uni_coef = ctx->uni_coef;
        e.uni_xl = ctx->uni_xl;
        e.uni_m0 = ctx->uni_m0;
        e.uni_m1 = ctx->uni_m1;
      }
    }
    enq_gemm(q, ctx->xn, d, ctx->G.at("fin_w"), d, ctx->ni, ctx->C, (int)d, e);
  }
  q.chk(advance_step(ctx->st, q.s));
}

// Per-sample conditioning: time embedding and every modulation vector for all T steps
// in three GEMMs (the modulation weights are read once per sample).
static bag_status enq_prepare(bag_ctx* ctx, const bag_cond* cond) {
  const bool wan = ctx->arch.kind == BAG_KIND_WAN;
  if (!cond || !cond->txt) return fail(ctx, BAG_EINVAL, "cond->txt is null");
  if (!wan && !cond->pooled) return fail(ctx, BAG_EINVAL, "cond->pooled is null");
  if (ctx->arch.cfg && !cond->txt_uncond) return fail(ctx, BAG_EINVAL, "cond->txt_uncond is null (cfg context)");
  if (ctx->arch.cfg && !wan && !cond->pooled_uncond)
    return fail(ctx, BAG_EINVAL, "cond->pooled_uncond is null (cfg context)");
  const long d = ctx->d;
  cudaStream_t s = ctx->stream;
  const size_t tbytes = (size_t)ctx->nx * d * ctx->act_size;
  if (cond->txt != ctx->txt_stage) CK(cudaMemcpyAsync(ctx->txt_stage, cond->txt, tbytes, cudaMemcpyDeviceToDevice, s));
  if (!wan && cond->pooled != ctx->pooled_stage)
    CK(cudaMemcpyAsync(ctx->pooled_stage, cond->pooled, (size_t)d * 4, cudaMemcpyDeviceToDevice, s));
  if (ctx->arch.cfg) {
    if (cond->txt_uncond != ctx->txt_stage_u)
      CK(cudaMemcpyAsync(ctx->txt_stage_u, cond->txt_uncond, tbytes, cudaMemcpyDeviceToDevice, s));
    if (!wan && cond->pooled_uncond != ctx->pooled_stage_u)
      CK(cudaMemcpyAsync(ctx->pooled_stage_u, cond->pooled_uncond, (size_t)d * 4, cudaMemcpyDeviceToDevice, s));
  }
  long cnt = 0;
  Enq q{ctx, s, &cnt};
  // The conditioning chain stays fp32: for bf16 configs each GEMM takes its fp32
  // activation as bf16 hi + lo halves (split A), so the modulation vectors carry no
  // bf16 rounding of the activations (an error that would be the same for every token
  // and every block and so would not average out).
  const int bf = ctx->act_bf16;
  auto gemm_f32_act = [&](const float* act, int K, const Tensor& W, int N, const Epi& e) {
    if (bf) {
      q.chk(split_bf16(ctx->splitbuf, act, ctx->T, K, s));
      q.pre(BAG_PROF_GEMM, 4.0 * ctx->T * N * K, (double)N * K * 2, ctx->T, N, 2 * K,
            gemm_uses_pair(ctx->T, 0, N));
      q.chk(gemm(ctx->splitbuf, 2L * K, W.p, K, ctx->T, N, K, 1, e, &ctx->st->err, s, 0, 1));
    } else {
      enq_gemm(q, act, K, W, K, ctx->T, N, K, e);
    }
  };
  q.chk(sinusoid_all(ctx->sin_all, 0, ctx->d_sigma, ctx->T, kTembDim, s));
  Epi e1 = base_epi(ctx, nullptr, -1);
  e1.kind = EPI_SILU;
  e1.bias = (const float*)ctx->G.at("t1_b").p;
  e1.out = ctx->t1o;
  e1.ldo = d;
  e1.out_bf16 = 0;
  gemm_f32_act(ctx->sin_all, kTembDim, ctx->G.at("t1_w"), (int)d, e1);
  // vec = t2(t1) + pooled and every modulation vector, per branch (the time embedding
  // t1 is shared; a Wan modulation has no text term, so its unconditional branch
  // reads the conditional one's)
  const int nb = wan ? 1 : n_branches(ctx);
  for (int br = 0; br < nb; ++br) {
    float* svec = br ? ctx->svec_u : ctx->svec;
    Epi e2 = base_epi(ctx, nullptr, -1);
    e2.kind = EPI_VEC;
    e2.bias = (const float*)ctx->G.at("t2_b").p;
    e2.out = br ? ctx->vec_all_u : ctx->vec_all;
    e2.ldo = d;
    e2.addend = wan ? nullptr : (br ? ctx->pooled_stage_u : ctx->pooled_stage);
    e2.out2 = svec;
    e2.ldo2 = d;
    e2.out2_bf16 = 0;
    gemm_f32_act(ctx->t1o, (int)d, ctx->G.at("t2_w"), (int)d, e2);
    Epi e3 = base_epi(ctx, nullptr, -1);
    e3.kind = EPI_STORE;
    e3.bias = ctx->bmod;
    e3.out_bf16 = 0;
    if (wan) {
      e3.out = ctx->wan_shared;
      e3.ldo = 8 * d;
      gemm_f32_act(svec, (int)d, ctx->wmod, (int)ctx->n_mod, e3);
      q.chk(expand_wan_mod(ctx->mod_all, ctx->wan_shared, ctx->wan_tabs, ctx->T, ctx->nblk, (int)d, s));
    } else {
      e3.out = br ? ctx->mod_all_u : ctx->mod_all;
      e3.ldo = ctx->mod_stride;
      gemm_f32_act(svec, (int)d, ctx->wmod, (int)ctx->n_mod, e3);
    }
  }
  if (q.e != cudaSuccess) return fail(ctx, BAG_ECUDA, std::string("prepare: ") + cudaGetErrorString(q.e));
  ctx->n_prepare = cnt;
  ctx->prepared = true;
  return BAG_OK;
}

static void destroy_graph(bag_ctx* ctx) {
  if (ctx->exec) cudaGraphExecDestroy(ctx->exec);
  if (ctx->graph) cudaGraphDestroy(ctx->graph);
  ctx->exec = nullptr;
  ctx->graph = nullptr;
}

// Capture one step: prefix, conditional node (body 0: full network; body 1: reuse),
// suffix.  The gate kernel sets the condition on the device.
static bag_status build_graph(bag_ctx* ctx) {
  destroy_graph(ctx);
  cudaStream_t s = ctx->stream;
  if (!ctx->cap_stream) CK(cudaStreamCreateWithFlags(&ctx->cap_stream, cudaStreamNonBlocking));
  CK(cudaGraphCreate(&ctx->graph, 0));
  cudaGraphConditionalHandle handle;
  CK(cudaGraphConditionalHandleCreate(&handle, ctx->graph, 0, 0));
  CK(cudaStreamBeginCaptureToGraph(s, ctx->graph, nullptr, nullptr, 0, cudaStreamCaptureModeThreadLocal));
  long cnt = 0;
  Enq q{ctx, s, &cnt};
  enq_prefix(q, 1, (unsigned long long)handle);
  ctx->n_prefix = cnt;
  cudaStreamCaptureStatus cs;
  const cudaGraphNode_t* deps = nullptr;
  size_t ndeps = 0;
  cudaGraph_t cg = nullptr;
  cudaError_t e = cudaStreamGetCaptureInfo(s, &cs, nullptr, &cg, &deps, nullptr, &ndeps);
  cudaGraphNode_t cnode = nullptr;
  cudaGraphNodeParams p = {};
  if (e == cudaSuccess && q.e == cudaSuccess) {
    p.type = cudaGraphNodeTypeConditional;
    p.conditional.handle = handle;
    p.conditional.type = cudaGraphCondTypeIf;
    p.conditional.size = 2;
    e = cudaGraphAddNode(&cnode, cg, deps, nullptr, ndeps, &p);
  }
  if (e == cudaSuccess) e = cudaStreamUpdateCaptureDependencies(s, &cnode, nullptr, 1, cudaStreamSetCaptureDependencies);
  if (e == cudaSuccess) {
    cudaGraph_t bodies[2] = {p.conditional.phGraph_out[0], p.conditional.phGraph_out[1]};
    for (int bi = 0; bi < 2 && e == cudaSuccess; ++bi) {
      e = cudaStreamBeginCaptureToGraph(ctx->cap_stream, bodies[bi], nullptr, nullptr, 0,
                                        cudaStreamCaptureModeThreadLocal);
      if (e != cudaSuccess) break;
      long c2 = 0;
      Enq qb{ctx, ctx->cap_stream, &c2};
      if (bi == 0)
        enq_full(qb, 1);
      else
        enq_skip(qb, 0);
      cudaGraph_t tmp;
      cudaError_t e2 = cudaStreamEndCapture(ctx->cap_stream, &tmp);
      if (qb.e != cudaSuccess) e = qb.e;
      if (e2 != cudaSuccess && e == cudaSuccess) e = e2;
      if (bi == 0)
        ctx->n_full = c2;
      else
        ctx->n_skip = c2;
    }
  }
  cnt = 0;
  if (e == cudaSuccess) {
    Enq qs{ctx, s, &cnt};
    enq_suffix(qs);
    e = qs.e;
  }
  ctx->n_suffix = cnt;
  cudaGraph_t out = nullptr;
  cudaError_t e3 = cudaStreamEndCapture(s, &out);
  if (e == cudaSuccess) e = e3;
  if (e == cudaSuccess) e = cudaGraphInstantiate(&ctx->exec, ctx->graph, 0);
  if (e != cudaSuccess) {
    destroy_graph(ctx);
    cudaGetLastError();
    return fail(ctx, BAG_ECUDA, std::string("step graph capture: ") + cudaGetErrorString(e));
  }
  return BAG_OK;
}

// Enqueue one step.  Graph mode replays the captured step; direct mode launches every
// kernel and the two bodies' kernels skip themselves on the device flag.
static bag_status launch_step(bag_ctx* ctx) {
  if (ctx->use_graph) {
    if (!ctx->exec) CKS(build_graph(ctx));
    CK(cudaGraphLaunch(ctx->exec, ctx->stream));
    return BAG_OK;
  }
  long cnt = 0;
  Enq q{ctx, ctx->stream, &cnt};
  enq_prefix(q, 0, 0);
  enq_full(q, 1);
  enq_skip(q, 0);
  enq_suffix(q);
  if (q.e != cudaSuccess) return fail(ctx, BAG_ECUDA, std::string("step: ") + cudaGetErrorString(q.e));
  return BAG_OK;
}

// Profiled sample: direct launches, each bracketed by events; the decision is read back
// after every gate so that only the taken branch is launched (and timed).
static bag_status profile_run_impl(bag_ctx* ctx, float* x_inout, const bag_cond* cond,
                                   bag_stats* stats, bag_prof_entry* out) {
  if (!x_inout || !out) return fail(ctx, BAG_EINVAL, "null argument");
  if (ctx->next_t != 0) return fail(ctx, BAG_ESTATE, "needs a fresh sample (bag_reset)");
  ctx->prof.clear();
  ctx->ev_used = 0;
  ctx->profiling = true;
  bag_status s = enq_prepare(ctx, cond);
  const size_t xbytes = (size_t)ctx->ni * ctx->C * 4;
  int nfe = 0;
  std::vector<float> lg((size_t)ctx->T * kLogFloats);
  if (s == BAG_OK) {
    cudaMemcpyAsync(ctx->x, x_inout, xbytes, cudaMemcpyDeviceToDevice, ctx->stream);
    if (ctx->act_bf16) split_bf16(ctx->xb, ctx->x, ctx->ni, ctx->C, ctx->stream);
    for (int t = 0; t < ctx->T && s == BAG_OK; ++t) {
      long cnt = 0;
      Enq q{ctx, ctx->stream, &cnt};
      enq_prefix(q, 0, 0);
      int flag = 0;
      if (cudaMemcpyAsync(&flag, &ctx->st->flag, 4, cudaMemcpyDeviceToHost, ctx->stream) != cudaSuccess ||
          cudaStreamSynchronize(ctx->stream) != cudaSuccess) {
        s = fail(ctx, BAG_ECUDA, "profile sync failed");
        break;
      }
      nfe += flag;
      if (flag)
        enq_full(q, 1);
      else
        enq_skip(q, 0);
      enq_suffix(q);
      if (q.e != cudaSuccess) s = fail(ctx, BAG_ECUDA, std::string("profile step: ") + cudaGetErrorString(q.e));
    }
    cudaMemcpyAsync(x_inout, ctx->x, xbytes, cudaMemcpyDeviceToDevice, ctx->stream);
    cudaMemcpyAsync(lg.data(), ctx->log, lg.size() * 4, cudaMemcpyDeviceToHost, ctx->stream);
    if (cudaStreamSynchronize(ctx->stream) != cudaSuccess && s == BAG_OK) s = fail(ctx, BAG_ECUDA, "profile sync");
  }
  ctx->profiling = false;
  ctx->next_t = ctx->T;
  for (int k = 0; k < BAG_PROF_KINDS; ++k) out[k] = bag_prof_entry{0, 0.0, 0.0, 0.0};
  for (auto& r : ctx->prof) {
    float ms = 0.f;
    cudaEventElapsedTime(&ms, ctx->ev_pool[r.e0], ctx->ev_pool[r.e1]);
    bag_prof_entry& o = out[r.kind];
    o.launches += 1;
    o.ms += ms;
    o.flops += r.flops;
    o.bytes += r.bytes;
  }
  if (stats) {
    stats->T = ctx->T;
    stats->B = ctx->B;
    stats->nfe = nfe;
    if (stats->mask)
      for (int t = 0; t < ctx->T; ++t) stats->mask[t] = lg[(size_t)t * kLogFloats + 5] != 0.f;
    if (stats->log) std::memcpy(stats->log, lg.data(), lg.size() * 4);
  }
  return s;
}

static bag_status check_device_error(bag_ctx* ctx) {
  DevState h;
  CK(cudaMemcpyAsync(&h, ctx->st, sizeof(h), cudaMemcpyDeviceToHost, ctx->stream));
  CK(cudaStreamSynchronize(ctx->stream));
  if (h.err) return fail(ctx, BAG_EDEVICE_TIMEOUT, "a kernel's bounded wait expired");
  return BAG_OK;
}

static bag_status reset_state(bag_ctx* ctx) {
  DevState h{};
  h.t = 0;
  h.c = 0;
  h.t_last = -1;
  CK(cudaMemcpyAsync(ctx->st, &h, sizeof(h), cudaMemcpyHostToDevice, ctx->stream));
  ctx->next_t = 0;
  ctx->prepared = false;
  return BAG_OK;
}

// Order the internal stream after the caller's stream, and the caller's stream after
// the work just enqueued.
static bag_status enter(bag_ctx* ctx) {
  CK(cudaEventRecord(ctx->ev_in, ctx->user_stream));
  CK(cudaStreamWaitEvent(ctx->stream, ctx->ev_in, 0));
  return BAG_OK;
}
static bag_status leave(bag_ctx* ctx, bag_status s) {
  if (cudaEventRecord(ctx->ev_out, ctx->stream) == cudaSuccess)
    cudaStreamWaitEvent(ctx->user_stream, ctx->ev_out, 0);
  return s;
}

// ---------------------------------------------------------------------------
// C ABI
// ---------------------------------------------------------------------------
static bag_status bag_reset_impl(bag_ctx* ctx) {
  if (!ctx) return BAG_EINVAL;
  CKS(reset_state(ctx));
  return BAG_OK;
}

static bag_status bag_prepare_impl(bag_ctx* ctx, const bag_cond* cond) {
  if (!ctx) return BAG_EINVAL;
  return enq_prepare(ctx, cond);
}

static bag_status bag_step_impl(bag_ctx* ctx, const float* x, int t, const bag_cond* cond, float* x_out,
                    int32_t* full_or_cached) {
  if (!ctx) return BAG_EINVAL;
  if (!x || !x_out) return fail(ctx, BAG_EINVAL, "x / x_out is null");
  if (t != ctx->next_t || t >= ctx->T)
    return fail(ctx, BAG_EORDER, "step " + std::to_string(t) + " called, expected " + std::to_string(ctx->next_t));
  if (t == 0) CKS(enq_prepare(ctx, cond));
  if (!ctx->prepared) return fail(ctx, BAG_ESTATE, "sample not prepared");
  const size_t xbytes = (size_t)ctx->ni * ctx->C * 4;
  CK(cudaMemcpyAsync(ctx->x, x, xbytes, cudaMemcpyDeviceToDevice, ctx->stream));
  if (ctx->act_bf16) CK(split_bf16(ctx->xb, ctx->x, ctx->ni, ctx->C, ctx->stream));
  CKS(launch_step(ctx));
  CK(cudaMemcpyAsync(x_out, ctx->x, xbytes, cudaMemcpyDeviceToDevice, ctx->stream));
  if (full_or_cached)
    CK(cudaMemcpyAsync(full_or_cached, &ctx->st->flag, 4, cudaMemcpyDeviceToDevice, ctx->stream));
  ctx->next_t++;
  return BAG_OK;
}

static bag_status bag_run_impl(bag_ctx* ctx, float* x_inout, const bag_cond* cond, bag_stats* stats) {
  if (!ctx) return BAG_EINVAL;
  if (!x_inout) return fail(ctx, BAG_EINVAL, "x is null");
  if (ctx->next_t != 0) return fail(ctx, BAG_ESTATE, "bag_run needs a fresh sample (bag_reset)");
  CKS(enq_prepare(ctx, cond));
  const size_t xbytes = (size_t)ctx->ni * ctx->C * 4;
  CK(cudaMemcpyAsync(ctx->x, x_inout, xbytes, cudaMemcpyDeviceToDevice, ctx->stream));
  if (ctx->act_bf16) CK(split_bf16(ctx->xb, ctx->x, ctx->ni, ctx->C, ctx->stream));
  for (int t = 0; t < ctx->T; ++t) CKS(launch_step(ctx));
  CK(cudaMemcpyAsync(x_inout, ctx->x, xbytes, cudaMemcpyDeviceToDevice, ctx->stream));
  ctx->next_t = ctx->T;
  DevState h;
  CK(cudaMemcpyAsync(&h, ctx->st, sizeof(h), cudaMemcpyDeviceToHost, ctx->stream));
  std::vector<float> lg;
  if (stats) {
    lg.resize((size_t)ctx->T * kLogFloats);
    CK(cudaMemcpyAsync(lg.data(), ctx->log, lg.size() * 4, cudaMemcpyDeviceToHost, ctx->stream));
  }
  CK(cudaStreamSynchronize(ctx->stream));
  const long per_step = ctx->n_prefix + ctx->n_suffix;
  ctx->launches = ctx->n_prepare + 2 + (long)ctx->T * per_step + (long)h.c * ctx->n_full +
                  (long)(ctx->T - h.c) * ctx->n_skip;
  if (stats) {
    stats->T = ctx->T;
    stats->B = ctx->B;
    stats->nfe = h.c;
    if (stats->mask)
      for (int t = 0; t < ctx->T; ++t) stats->mask[t] = lg[(size_t)t * kLogFloats + 5] != 0.f;
    if (stats->log) std::memcpy(stats->log, lg.data(), lg.size() * 4);
  }
  if (h.err) return fail(ctx, BAG_EDEVICE_TIMEOUT, "a kernel's bounded wait expired");
  return BAG_OK;
}

static bag_status bag_run_host_impl(bag_ctx* ctx, float* x_host, const bag_cond* ch, bag_stats* stats) {
  if (!ctx) return BAG_EINVAL;
  const bool wan = ctx->arch.kind == BAG_KIND_WAN;
  if (!x_host || !ch || !ch->txt) return fail(ctx, BAG_EINVAL, "host buffer is null");
  if (!wan && !ch->pooled) return fail(ctx, BAG_EINVAL, "pooled is null");
  if (ctx->arch.cfg && (!ch->txt_uncond || (!wan && !ch->pooled_uncond)))
    return fail(ctx, BAG_EINVAL, "unconditional text / pooled is null (cfg context)");
  if (ctx->next_t != 0) return fail(ctx, BAG_ESTATE, "bag_run_host needs a fresh sample (bag_reset)");
  const long d = ctx->d;
  const size_t xbytes = (size_t)ctx->ni * ctx->C * 4;
  // stage: latent into the working buffer, each text (fp32) into the scratch then
  // converted into its staging buffer
  CK(cudaMemcpyAsync(ctx->x, x_host, xbytes, cudaMemcpyHostToDevice, ctx->stream));
  for (int br = 0; br < n_branches(ctx); ++br) {
    void* stage = br ? ctx->txt_stage_u : ctx->txt_stage;
    float* pstage = br ? ctx->pooled_stage_u : ctx->pooled_stage;
    const float* pooled = (const float*)(br ? ch->pooled_uncond : ch->pooled);
    CK(cudaMemcpyAsync(ctx->tmp_f32, br ? ch->txt_uncond : ch->txt, (size_t)ctx->nx * d * 4,
                       cudaMemcpyHostToDevice, ctx->stream));
    if (!wan) CK(cudaMemcpyAsync(pstage, pooled, (size_t)d * 4, cudaMemcpyHostToDevice, ctx->stream));
    if (ctx->act_bf16)
      CK(to_bf16((__nv_bfloat16*)stage, ctx->tmp_f32, (long)ctx->nx * d, ctx->stream));
    else
      CK(cudaMemcpyAsync(stage, ctx->tmp_f32, (size_t)ctx->nx * d * 4, cudaMemcpyDeviceToDevice, ctx->stream));
  }
  bag_cond cond{ctx->txt_stage, wan ? nullptr : ctx->pooled_stage, ctx->txt_stage_u,
                wan ? nullptr : ctx->pooled_stage_u};
  CKS(bag_run_impl(ctx, ctx->x, &cond, stats));
  CK(cudaMemcpyAsync(x_host, ctx->x, xbytes, cudaMemcpyDeviceToHost, ctx->stream));
  CK(cudaStreamSynchronize(ctx->stream));
  return BAG_OK;
}

static bag_status bag_forward_block_impl(bag_ctx* ctx, int block, int t_mod, float* h) {
  if (!ctx || !h) return BAG_EINVAL;
  if (block < 0 || block >= ctx->nblk) return fail(ctx, BAG_EINVAL, "block out of range");
  if (t_mod < 0 || t_mod >= ctx->T) return fail(ctx, BAG_EINVAL, "t_mod out of range");
  if (!ctx->prepared) return fail(ctx, BAG_ESTATE, "call bag_prepare first");
  DevState hs{};
  hs.t = t_mod;
  hs.flag = 1;
  CK(cudaMemcpyAsync(ctx->st_op, &hs, sizeof(hs), cudaMemcpyHostToDevice, ctx->stream));
  long cnt = 0;
  Enq q{ctx, ctx->stream, &cnt};
  enq_block(q, block, h, ctx->st_op, -1);
  if (q.e != cudaSuccess) return fail(ctx, BAG_ECUDA, std::string("block: ") + cudaGetErrorString(q.e));
  ctx->launches = cnt;
  return BAG_OK;
}

static bag_status bag_gemm_bf16_impl(bag_ctx* ctx, const void* A, long lda, const void* W, long ldw,
                         const float* bias, float* C, long ldc, int M, int N, int K, int epilogue,
                         int force_simt) {
  if (!ctx || !A || !W || !C) return BAG_EINVAL;
  if (M < 0 || N <= 0 || K <= 0 || N % 64 || K % 64 || lda < K || ldw < K || ldc < N)
    return fail(ctx, BAG_EINVAL, "bad gemm shape");
  Epi e;
  e.kind = epilogue == 1 ? EPI_GELU : EPI_STORE;
  e.bias = bias;
  e.out = C;
  e.ldo = ldc;
  e.out_bf16 = 0;
  CK(gemm(A, lda, W, ldw, M, N, K, 1, e, &ctx->st_op->err, ctx->stream, force_simt));
  return BAG_OK;
}

static bag_status attention_op(bag_ctx* ctx, const void* q, const void* k, const void* v, void* o,
                               long ld, int nq, int nk, int heads, int dh, long vpad, int force_simt,
                               int f16) {
  if (!ctx || !q || !k || !v || !o) return BAG_EINVAL;
  if (nq < 0 || nk <= 0 || heads <= 0 || (dh != 64 && dh != 128) || ld < (long)heads * dh)
    return fail(ctx, BAG_EINVAL, "bad attention shape");
  AttnArgs a{};
  a.q = q;
  a.ldq = ld;
  a.k = k;
  a.ldk = ld;
  a.v = v;
  a.v_mode = vpad > 0 ? 1 : 0;
  a.ldv = ld;
  a.vpad = vpad;
  if (vpad > 0 && (vpad < nk || vpad % 8)) return fail(ctx, BAG_EINVAL, "vpad must be >= nk and a multiple of 8");
  a.o = o;
  a.ldo = ld;
  a.nq = nq;
  a.nk = nk;
  a.heads = heads;
  a.dh = dh;
  a.bf16 = 1;
  a.f16 = f16;
  a.st = nullptr;
  a.flag_want = -1;
  if (f16 && force_simt) return fail(ctx, BAG_EUNSUPPORTED, "fp16 attention runs on the tensor cores only");
  if (!force_simt && !attention_tc_supported(a))
    return fail(ctx, BAG_EUNSUPPORTED, "tensor-core attention needs dh 128, transposed V and 16-byte alignment");
  CK(attention(a, &ctx->st_op->err, ctx->stream, force_simt));
  return BAG_OK;
}

static bag_status bag_ln_mod_impl(bag_ctx* ctx, const float* x, const float* shift, const float* scale, void* y,
                      int rows, int cols) {
  if (!ctx || !x || !y) return BAG_EINVAL;
  if (rows < 0 || cols <= 0 || cols % 4) return fail(ctx, BAG_EINVAL, "bad ln shape");
  LnArgs a{};
  a.x = x;
  a.ldx = cols;
  a.y = y;
  a.ldy = cols;
  a.y_bf16 = 1;
  a.rows = rows;
  a.cols = cols;
  a.split = 0;
  a.shift_a = a.shift_b = shift;
  a.scale_a = a.scale_b = scale;
  a.mod_step = 0;
  a.flag_want = -1;
  CK(ln_mod(a, ctx->stream));
  return BAG_OK;
}

static bag_status bag_rel_l1_impl(bag_ctx* ctx, const void* a, const void* b, int dtype, long rows,
                                   long cols, float* scratch, float* out) {
  if (!a || !b || !scratch || !out) return fail(ctx, BAG_EINVAL, "null pointer");
  if (rows <= 0 || cols <= 0 || (dtype != BAG_F32 && dtype != BAG_BF16))
    return fail(ctx, BAG_EINVAL, "bad rel_l1 shape or dtype");
  CK(rel_l1_partials(a, b, dtype == BAG_BF16, rows, cols, scratch, ctx->stream));
  CK(rel_l1_finalize(scratch, rows, out, ctx->stream));
  return BAG_OK;
}

static bag_status bag_residual_add_impl(bag_ctx* ctx, float* out, const float* h_in, const float* R, long n) {
  if (!ctx || !out || !h_in || !R) return BAG_EINVAL;
  if (n < 0 || n % 4) return fail(ctx, BAG_EINVAL, "n must be a multiple of 4");
  CK(residual_add(out, h_in, R, n, ctx->stream));
  return BAG_OK;
}

extern "C" {

bag_status bag_create(const bag_arch* arch, int T, int B, bag_ctx** out) {
  if (!out) return fail(nullptr, BAG_EINVAL, "out is null");
  *out = nullptr;
  CKS(validate_arch(arch, T, B));
  bag_ctx* ctx = new bag_ctx();
  ctx->arch = *arch;
  ctx->T = T;
  ctx->B = B;
  ctx->d = arch->hidden;
  ctx->H = arch->heads;
  ctx->dh = arch->hidden / arch->heads;
  ctx->F = arch->mlp;
  ctx->C = arch->patch_ch;
  ctx->ni = arch->grid[0] * arch->grid[1] * arch->grid[2];
  ctx->nx = arch->n_txt;
  ctx->N = ctx->ni + ctx->nx;
  ctx->nrope = arch->kind == BAG_KIND_WAN ? ctx->ni : ctx->N;
  ctx->act_bf16 = arch->dtype == BAG_BF16;
  ctx->act_size = ctx->act_bf16 ? 2 : 4;
  ctx->thr = (float)std::log((double)arch->tau / (1.0 - (double)arch->tau));
  if (const char* v = std::getenv("BAG_PDL")) ctx->pdl = std::atoi(v) != 0;
  if (arch->kind == BAG_KIND_WAN) {
    ctx->nblk = arch->n_wan;
    ctx->blocks.assign(ctx->nblk, Block{});
    for (auto& b : ctx->blocks) b.type = BT_WAN;
  } else {
    ctx->nblk = arch->n_double + arch->n_single;
    ctx->blocks.assign(ctx->nblk, Block{});
    for (int i = 0; i < ctx->nblk; ++i) ctx->blocks[i].type = i < arch->n_double ? BT_DOUBLE : BT_SINGLE;
  }
  bag_status s = BAG_OK;
  if (cudaStreamCreateWithFlags(&ctx->stream, cudaStreamNonBlocking) != cudaSuccess ||
      cudaEventCreateWithFlags(&ctx->ev_in, cudaEventDisableTiming) != cudaSuccess ||
      cudaEventCreateWithFlags(&ctx->ev_out, cudaEventDisableTiming) != cudaSuccess)
    s = fail(ctx, BAG_ECUDA, "stream/event creation failed");
  if (s == BAG_OK && kernels_init() != cudaSuccess) s = fail(ctx, BAG_ECUDA, "kernel attribute setup failed");
  if (s == BAG_OK) s = alloc_weights(ctx);
  if (s == BAG_OK) s = alloc_activations(ctx);
  if (s == BAG_OK) s = seed_weights(ctx);
  if (s == BAG_OK) s = seed_gate(ctx);
  if (s == BAG_OK) s = reset_state(ctx);
  if (s == BAG_OK && cudaStreamSynchronize(ctx->stream) != cudaSuccess) s = fail(ctx, BAG_ECUDA, "create sync failed");
  if (s != BAG_OK) {
    g_create_error = ctx->err;
    bag_destroy(ctx);
    return s;
  }
  *out = ctx;
  return BAG_OK;
}

void bag_destroy(bag_ctx* ctx) {
  if (!ctx) return;
  destroy_graph(ctx);
  if (ctx->cap_stream) cudaStreamDestroy(ctx->cap_stream);
  if (ctx->warena) cudaFree(ctx->warena);
  if (ctx->aarena) cudaFree(ctx->aarena);
  if (ctx->ev_in) cudaEventDestroy(ctx->ev_in);
  if (ctx->ev_out) cudaEventDestroy(ctx->ev_out);
  for (auto ev : ctx->ev_pool) cudaEventDestroy(ev);
  if (ctx->stream) cudaStreamDestroy(ctx->stream);
  delete ctx;
}

const char* bag_last_error(bag_ctx* ctx) { return ctx ? ctx->err.c_str() : g_create_error.c_str(); }

bag_status bag_set_stream(bag_ctx* ctx, void* stream) {
  if (!ctx) return BAG_EINVAL;
  ctx->user_stream = (cudaStream_t)stream;
  return BAG_OK;
}

bag_status bag_load_gate(bag_ctx* ctx, const float* theta, int n, const float* mu, const float* sd) {
  if (!ctx) return BAG_EINVAL;
  if (!theta) return fail(ctx, BAG_EINVAL, "theta is null");
  const int kind = ctx->arch.gate_kind;
  if (n != gate_param_count(kind))
    return fail(ctx, BAG_EINVAL, "gate kind " + std::to_string(kind) + " has " +
                                     std::to_string(gate_param_count(kind)) + " parameters, got " +
                                     std::to_string(n));
  std::vector<float> g(kGateFloats, 0.f);
  std::memcpy(g.data(), theta, (size_t)n * sizeof(float));
  for (int i = 0; i < 6; ++i) g[kGateSd + i] = 1.f;
  for (int i = 0; i < gate_inputs(kind); ++i) {
    g[kGateMu + i] = mu ? mu[i] : 0.f;
    g[kGateSd + i] = sd ? sd[i] : 1.f;
    if (!(g[kGateSd + i] != 0.f)) return fail(ctx, BAG_EINVAL, "sd must be nonzero");
  }
  CK(cudaMemcpyAsync(ctx->d_gate, g.data(), g.size() * 4, cudaMemcpyHostToDevice, ctx->stream));
  CK(cudaStreamSynchronize(ctx->stream));
  return BAG_OK;
}

bag_status bag_set_policy(bag_ctx* ctx, int policy, const uint8_t* host_mask, float delta) {
  if (!ctx) return BAG_EINVAL;
  if (policy < BAG_POLICY_BAG || policy > BAG_POLICY_THRESHOLD) return fail(ctx, BAG_EINVAL, "unknown policy");
  if (policy == BAG_POLICY_MASK || policy == BAG_POLICY_STATIC_UNIFORM) {
    std::vector<uint8_t> m(ctx->T, 0);
    if (policy == BAG_POLICY_MASK) {
      if (!host_mask) return fail(ctx, BAG_EINVAL, "mask policy needs host_mask");
      std::memcpy(m.data(), host_mask, ctx->T);
    } else {
      // static paradigm: B steps evenly spaced, floor(i * T / B) for i < B
      for (int i = 0; i < ctx->B; ++i) m[(long)i * ctx->T / ctx->B] = 1;
    }
    CK(cudaMemcpyAsync(ctx->d_pmask, m.data(), ctx->T, cudaMemcpyHostToDevice, ctx->stream));
    CK(cudaStreamSynchronize(ctx->stream));
  }
  if (policy == BAG_POLICY_THRESHOLD && !(delta == delta)) return fail(ctx, BAG_EINVAL, "delta is NaN");
  // policy and delta are kernel arguments of the captured gate launch; a new mask is
  // device data the same graph reads
  if (policy != ctx->policy || delta != ctx->delta) destroy_graph(ctx);
  ctx->policy = policy;
  ctx->delta = delta;
  return BAG_OK;
}

bag_status bag_check_wait_timeout(bag_ctx* ctx) {
  if (!ctx) return BAG_EINVAL;
  CKS(enter(ctx));
  cudaError_t e = wait_timeout_probe(ctx->st, ctx->stream);
  if (e != cudaSuccess) return leave(ctx, fail(ctx, BAG_ECUDA, std::string("probe: ") + cudaGetErrorString(e)));
  return leave(ctx, check_device_error(ctx));
}

bag_status bag_set_budget(bag_ctx* ctx, int B) {
  if (!ctx) return BAG_EINVAL;
  if (B < 1 || B > ctx->T) return fail(ctx, BAG_EINVAL, "need 1 <= B <= T");
  ctx->B = B;
  destroy_graph(ctx);  // B is a kernel argument of the captured gate launch
  if (ctx->policy == BAG_POLICY_STATIC_UNIFORM) return bag_set_policy(ctx, ctx->policy, nullptr, ctx->delta);
  return BAG_OK;
}

bag_status bag_reset(bag_ctx* ctx) {
  if (!ctx) return BAG_EINVAL;
  CKS(enter(ctx));
  return leave(ctx, bag_reset_impl(ctx));
}

bag_status bag_prepare(bag_ctx* ctx, const bag_cond* cond) {
  if (!ctx) return BAG_EINVAL;
  CKS(enter(ctx));
  return leave(ctx, bag_prepare_impl(ctx, cond));
}

bag_status bag_step(bag_ctx* ctx, const float* x, int t, const bag_cond* cond, float* x_out,
                    int32_t* full_or_cached) {
  if (!ctx) return BAG_EINVAL;
  CKS(enter(ctx));
  return leave(ctx, bag_step_impl(ctx, x, t, cond, x_out, full_or_cached));
}

bag_status bag_run(bag_ctx* ctx, float* x_inout, const bag_cond* cond, bag_stats* stats) {
  if (!ctx) return BAG_EINVAL;
  CKS(enter(ctx));
  return leave(ctx, bag_run_impl(ctx, x_inout, cond, stats));
}

bag_status bag_run_host(bag_ctx* ctx, float* x_host, const bag_cond* cond_host, bag_stats* stats) {
  if (!ctx) return BAG_EINVAL;
  CKS(enter(ctx));
  return leave(ctx, bag_run_host_impl(ctx, x_host, cond_host, stats));
}

bag_status bag_get_weight(bag_ctx* ctx, int block, const char* name, float* out, size_t n) {
  if (!ctx || !name || !out) return BAG_EINVAL;
  const std::map<std::string, Tensor>* m = nullptr;
  if (block < 0)
    m = &ctx->G;
  else if (block < ctx->nblk)
    m = &ctx->blocks[block].w;
  else
    return fail(ctx, BAG_EINVAL, "block out of range");
  auto it = m->find(name);
  if (it == m->end()) return fail(ctx, BAG_EINVAL, std::string("no tensor ") + name);
  const Tensor& t = it->second;
  if ((long)n != t.n) return fail(ctx, BAG_EINVAL, "size mismatch: tensor has " + std::to_string(t.n));
  if (t.bf16) {
    std::vector<uint16_t> tmp(n);
    CK(cudaMemcpyAsync(tmp.data(), t.p, n * 2, cudaMemcpyDeviceToHost, ctx->stream));
    CK(cudaStreamSynchronize(ctx->stream));
    for (size_t i = 0; i < n; ++i) {
      uint32_t u = (uint32_t)tmp[i] << 16;
      std::memcpy(out + i, &u, 4);
    }
  } else {
    CK(cudaMemcpyAsync(out, t.p, n * 4, cudaMemcpyDeviceToHost, ctx->stream));
    CK(cudaStreamSynchronize(ctx->stream));
  }
  return BAG_OK;
}

bag_status bag_forward_block(bag_ctx* ctx, int block, int t_mod, float* h) {
  if (!ctx) return BAG_EINVAL;
  CKS(enter(ctx));
  return leave(ctx, bag_forward_block_impl(ctx, block, t_mod, h));
}

bag_status bag_profile_run(bag_ctx* ctx, float* x_inout, const bag_cond* cond, bag_stats* stats,
                           bag_prof_entry* out) {
  if (!ctx) return BAG_EINVAL;
  CKS(enter(ctx));
  return leave(ctx, profile_run_impl(ctx, x_inout, cond, stats, out));
}

bag_status bag_profile_launches(bag_ctx* ctx, bag_prof_launch* out, long max, long* n) {
  if (!ctx || !n) return BAG_EINVAL;
  *n = (long)ctx->prof.size();
  if (!out) return BAG_OK;
  const long m = std::min<long>(max, (long)ctx->prof.size());
  for (long i = 0; i < m; ++i) {
    const auto& r = ctx->prof[i];
    float ms = 0.f;
    cudaEventElapsedTime(&ms, ctx->ev_pool[r.e0], ctx->ev_pool[r.e1]);
    out[i] = bag_prof_launch{r.kind, r.m, r.n, r.k, ms, r.flops, r.bytes, r.variant};
  }
  return BAG_OK;
}

bag_status bag_launch_count(bag_ctx* ctx, long* out) {
  if (!ctx || !out) return BAG_EINVAL;
  *out = ctx->launches;
  return BAG_OK;
}

bag_status bag_gemm_bf16(bag_ctx* ctx, const void* A, long lda, const void* W, long ldw,
                         const float* bias, float* C, long ldc, int M, int N, int K, int epilogue,
                         int force_simt) {
  if (!ctx) return BAG_EINVAL;
  CKS(enter(ctx));
  return leave(ctx, bag_gemm_bf16_impl(ctx, A, lda, W, ldw, bias, C, ldc, M, N, K, epilogue, force_simt));
}

bag_status bag_attention_bf16(bag_ctx* ctx, const void* q, const void* k, const void* v, void* o,
                              long ld, int nq, int nk, int heads, int dh, long vpad, int force_simt) {
  if (!ctx) return BAG_EINVAL;
  CKS(enter(ctx));
  return leave(ctx, attention_op(ctx, q, k, v, o, ld, nq, nk, heads, dh, vpad, force_simt, 0));
}

bag_status bag_attention_f16(bag_ctx* ctx, const void* q, const void* k, const void* v, void* o,
                             long ld, int nq, int nk, int heads, int dh, long vpad) {
  if (!ctx) return BAG_EINVAL;
  CKS(enter(ctx));
  return leave(ctx, attention_op(ctx, q, k, v, o, ld, nq, nk, heads, dh, vpad, 0, 1));
}

bag_status bag_ln_mod(bag_ctx* ctx, const float* x, const float* shift, const float* scale, void* y,
                      int rows, int cols) {
  if (!ctx) return BAG_EINVAL;
  CKS(enter(ctx));
  return leave(ctx, bag_ln_mod_impl(ctx, x, shift, scale, y, rows, cols));
}

bag_status bag_rel_l1(bag_ctx* ctx, const void* a, const void* b, int dtype, long rows, long cols,
                      float* scratch, float* out) {
  if (!ctx) return BAG_EINVAL;
  CKS(enter(ctx));
  return leave(ctx, bag_rel_l1_impl(ctx, a, b, dtype, rows, cols, scratch, out));
}

bag_status bag_residual_add(bag_ctx* ctx, float* out, const float* h_in, const float* R, long n) {
  if (!ctx) return BAG_EINVAL;
  CKS(enter(ctx));
  return leave(ctx, bag_residual_add_impl(ctx, out, h_in, R, n));
}

}  // extern "C"
