// Layer entry points (Eq. 7, Eq. 10 with mean aggregation, Eq. 11, optional LayerNorm), status
// strings, thread-local error text and the optional per-kernel event timing.
#include <stdarg.h>
#include <stdio.h>
#include <string.h>

#include <algorithm>
#include <map>
#include <mutex>
#include <string>
#include <vector>

#include "layer_kernels.cuh"

namespace hg {


// ---------------------------------------------------------------------------------------------
// errors
// ---------------------------------------------------------------------------------------------
static thread_local char g_err[1024];

void set_error(const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_err, sizeof(g_err), fmt, ap);
  va_end(ap);
}
void clear_error() { g_err[0] = 0; }

// ---------------------------------------------------------------------------------------------
// timing
// ---------------------------------------------------------------------------------------------
struct TimingRec {
  const char* name;
  cudaEvent_t a, b;
};
static std::mutex g_tmu;
static bool g_timing = false;
static std::vector<TimingRec> g_recs;
static std::vector<cudaEvent_t> g_pool;

static cudaEvent_t take_event() {
  if (!g_pool.empty()) {
    cudaEvent_t e = g_pool.back();
    g_pool.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  cudaEventCreate(&e);
  return e;
}

int timing_begin(const char* name, cudaStream_t s) {
  if (!g_timing) return -1;
  std::lock_guard<std::mutex> lk(g_tmu);
  TimingRec r{name, take_event(), take_event()};
  cudaEventRecord(r.a, s);
  g_recs.push_back(r);
  return (int)g_recs.size() - 1;
}

void timing_end(int slot, cudaStream_t s) {
  if (slot < 0) return;
  std::lock_guard<std::mutex> lk(g_tmu);
  cudaEventRecord(g_recs[slot].b, s);
}

static size_t elem_size(hg_dtype dt) { return dt == HG_F32 ? 4 : 2; }

void carve_layer(const hg_graph* g, int d, hg_dtype dt, void* saved, void* scratch, LayerLayout* L,
                 size_t* saved_bytes, size_t* scratch_bytes, bool fused) {
  const GraphMeta& m = g->meta;
  const int64_t N = m.type_off[m.num_types];
  const size_t b = elem_size(dt);
  const bool tc = dt == HG_BF16;
  const size_t dd = (size_t)d * d;
  Carve s(saved), k(scratch);
  *L = LayerLayout{};
  if (fused) {
    L->Mlong = s.take<char>((size_t)std::max<int64_t>(g->long_cap, 1) * d * b);
  } else {
    L->M = s.take<char>((size_t)g->csr_rows * d * b);
  }
  if (!tc) L->Z = s.take<char>((size_t)N * d * b);
  L->U = s.take<char>((size_t)N * d * b);
  L->stats = s.take<float2>(std::max<int64_t>(N, 1));
  if (tc) {
    L->V = s.take<char>(2 * m.num_rels * dd * b);  // hi and lo halves of each fused weight
    L->Vt = s.take<char>(2 * m.num_rels * dd * b);
  }
  L->agg_part = k.take<float>((size_t)std::max(g->chunk_cap_csr, g->chunk_cap_node) * d);
  L->work = k.take<int32_t>(64);
  L->dY = k.take<char>((size_t)N * d * b);
  L->dU = k.take<char>((size_t)N * d * b);
  if (!tc) L->dZ = k.take<char>((size_t)N * d * b);
  L->dMs = k.take<char>((size_t)g->csr_rows * d * b);
  int64_t max_rows = 1;
  for (int t = 0; t < m.num_types; ++t) max_rows = std::max(max_rows, m.type_off[t + 1] - m.type_off[t]);
  const int cblocks = (int)std::max<int64_t>(ceil_div(max_rows, 64), std::min<int64_t>(ceil_div(max_rows, 8), 152 * 8));
  L->cpart = k.take<float>((size_t)cblocks * 3 * d);
  const int wsplits = std::max(wgrad_splits(max_rows), wgrad_tc_splits(max_rows, d));
  L->wpart = k.take<float>((size_t)wsplits * dd * (tc ? wgrad_tc_max_rels(d) : 1));
  L->rtmp = k.take<float>(std::max(reduce_tmp_floats(cblocks, d), reduce_tmp_floats(wsplits, (int64_t)dd)));
  if (tc) {
    L->G = k.take<float>(m.num_rels * dd);
  } else {
    L->WrelT = k.take<char>(m.num_rels * dd * b);
    L->WaggT = k.take<char>(m.num_types * dd * b);
  }
  if (saved_bytes) *saved_bytes = s.used;
  if (scratch_bytes) *scratch_bytes = k.used;
}

RelDst rel_dst_of(const GraphMeta& m) {
  RelDst rd{};
  for (int r = 0; r < m.num_rels; ++r) rd.v[r] = m.rel_dst[r];
  return rd;
}

static hg_status check_params(const hg_graph* g, const hg_layer_params* p) {
  HG_REQUIRE(g != nullptr && p != nullptr, "graph and params must be non-null");
  if (!(p->d == 64 || p->d == 128 || p->d == 256)) {
    set_error("d=%d not supported (64, 128, 256)", p->d);
    return HG_ERR_UNSUPPORTED;
  }
  if (!(p->dtype == HG_F32 || p->dtype == HG_BF16)) {
    set_error("dtype %d not supported", (int)p->dtype);
    return HG_ERR_UNSUPPORTED;
  }
  HG_REQUIRE(p->act == HG_ACT_RELU || p->act == HG_ACT_GELU_TANH || p->act == HG_ACT_NONE, "unknown activation %d",
             (int)p->act);
  HG_REQUIRE(p->W_rel && p->W_agg && p->b_agg, "W_rel, W_agg and b_agg must be non-null");
  HG_REQUIRE(!p->layernorm || (p->ln_gamma && p->ln_beta), "layernorm needs ln_gamma and ln_beta");
  HG_REQUIRE(!p->layernorm || p->ln_eps > 0.f, "ln_eps must be > 0");
  if (p->fused && !(p->dtype == HG_BF16 && p->d == 128)) {
    set_error("the fused mean layer needs bf16 and d = 128 (dtype %d, d = %d)", (int)p->dtype, p->d);
    return HG_ERR_UNSUPPORTED;
  }
  return HG_OK;
}

static hg_status check_buf(const void* p, const char* name) {
  HG_REQUIRE(p != nullptr, "%s must be non-null", name);
  HG_REQUIRE(((uintptr_t)p & 255) == 0, "%s must be 256-byte aligned", name);
  return HG_OK;
}

}  // namespace hg

using namespace hg;

extern "C" const char* hg_status_string(hg_status s) {
  switch (s) {
    case HG_OK: return "ok";
    case HG_ERR_INVALID_ARG: return "invalid argument";
    case HG_ERR_UNSUPPORTED: return "unsupported";
    case HG_ERR_WORKSPACE: return "workspace too small";
    case HG_ERR_CUDA: return "CUDA error";
    case HG_ERR_DEVICE_CHECK: return "device-side input check failed";
    case HG_ERR_TIMEOUT: return "timeout";
  }
  return "unknown status";
}

extern "C" const char* hg_last_error(void) { return g_err; }
extern "C" int32_t hg_abi_version(void) { return 2; }

extern "C" hg_status hg_device_status(int32_t* flags) {
  clear_error();
  HG_TRY(device_guard());
  int* p = device_status_ptr();
  HG_REQUIRE(p != nullptr, "device status word unavailable");
  int v = 0;
  HG_CUDA(cudaDeviceSynchronize());
  HG_CUDA(cudaMemcpy(&v, p, sizeof(int), cudaMemcpyDeviceToHost));
  if (flags) *flags = v;
  if (v != 0) {
    const int zero = 0;
    HG_CUDA(cudaMemcpy(p, &zero, sizeof(int), cudaMemcpyHostToDevice));
    set_error("a bounded wait in a tensor-core kernel gave up (flags %d); its results are invalid", v);
    return HG_ERR_TIMEOUT;
  }
  return HG_OK;
}

extern "C" hg_status hg_timing_enable(int32_t on) {
  std::lock_guard<std::mutex> lk(g_tmu);
  g_timing = on != 0;
  return HG_OK;
}

extern "C" hg_status hg_timing_report(char* buf, size_t len) {
  clear_error();
  std::lock_guard<std::mutex> lk(g_tmu);
  std::map<std::string, std::pair<long, double>> acc;
  hg_status st = HG_OK;
  for (auto& r : g_recs) {
    float ms = 0.f;
    if (cudaEventSynchronize(r.b) != cudaSuccess || cudaEventElapsedTime(&ms, r.a, r.b) != cudaSuccess) {
      set_error("event timing failed: %s", cudaGetErrorString(cudaGetLastError()));
      st = HG_ERR_CUDA;
    }
    auto& e = acc[r.name];
    e.first += 1;
    e.second += ms;
    g_pool.push_back(r.a);
    g_pool.push_back(r.b);
  }
  g_recs.clear();
  std::string out;
  char line[256];
  for (auto& kv : acc) {
    snprintf(line, sizeof(line), "%s %ld %.6f\n", kv.first.c_str(), kv.second.first, kv.second.second);
    out += line;
  }
  if (buf && len) {
    size_t n = std::min(len - 1, out.size());
    memcpy(buf, out.data(), n);
    buf[n] = 0;
  }
  return st;
}

extern "C" hg_status hg_layer_workspace_size(const hg_graph* graph, const hg_layer_params* params,
                                             size_t* saved_bytes, size_t* scratch_bytes) {
  clear_error();
  HG_TRY(check_params(graph, params));
  HG_REQUIRE(saved_bytes && scratch_bytes, "saved_bytes and scratch_bytes must be non-null");
  LayerLayout L;
  carve_layer(graph, params->d, params->dtype, nullptr, nullptr, &L, saved_bytes, scratch_bytes, params->fused != 0);
  return HG_OK;
}

extern "C" hg_status hg_layer_fwd(const hg_graph* graph, const hg_layer_params* p, const void* H_in, void* H_out,
                                  void* saved, void* scratch, hg_stream stream) {
  clear_error();
  HG_TRY(device_guard());
  HG_TRY(check_params(graph, p));
  HG_TRY(check_buf(H_in, "H_in"));
  HG_TRY(check_buf(H_out, "H_out"));
  HG_TRY(check_buf(saved, "saved"));
  HG_TRY(check_buf(scratch, "scratch"));
  HG_REQUIRE(H_in != H_out, "H_in and H_out must not alias");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const int d = p->d;
  LayerLayout L;
  carve_layer(graph, d, p->dtype, saved, scratch, &L, nullptr, nullptr, p->fused != 0);
  if (p->fused) {  // only the long rows' means are formed here; the projection sums the others
    HG_TRY(aggregate_forward_long(graph, d, H_in, L.Mlong, L.agg_part, L.work, s));
  } else {
    HG_TRY(aggregate_forward(graph, p->dtype, d, H_in, L.M, L.agg_part, L.work, s));
  }
  return project_forward(graph, p, H_in, H_out, L, true, s);
}

namespace hg {

// Eq. 7 and Eq. 11 from the relation rows in L.M: U = sum_r M_r W_r W_agg + b, activation,
// residual, optional LayerNorm.
hg_status project_forward(const hg_graph* graph, const hg_layer_params* p, const void* H_in, void* H_out,
                          const LayerLayout& L, bool compact, cudaStream_t s) {
  const GraphMeta& m = graph->meta;
  const int d = p->d;
  const size_t b = elem_size(p->dtype);
  if (p->dtype == HG_BF16) {
    // tensor-core path: U = sum_r M_r V_r with the fused weights V_r = W_r W_agg[t_r]
    HG_TRY(tc_fuse_weights(d, p->W_rel, p->W_agg, rel_dst_of(m), m.num_rels, L.V, L.Vt, s));
    for (int t = 0; t < m.num_types; ++t) {
      TcFwdArgs a{};
      for (int r = 0; r < m.num_rels; ++r) {
        if (m.rel_dst[r] != t) continue;
        a.rel[a.nrel] = r;
        a.mrow0[a.nrel] = m.row_base[r];
        ++a.nrel;
      }
      a.type = t;
      a.mrow = compact ? graph->mrow : nullptr;
      a.msent = graph->csr_rows;
      a.perm = compact ? graph->nperm + m.type_off[t] : nullptr;
      a.tmask = compact ? graph->tmask + graph->tile_base[t] : nullptr;
      a.b = (const __nv_bfloat16*)p->b_agg + (size_t)t * d;
      a.gamma = p->layernorm ? (const __nv_bfloat16*)p->ln_gamma + (size_t)t * d : nullptr;
      a.beta = p->layernorm ? (const __nv_bfloat16*)p->ln_beta + (size_t)t * d : nullptr;
      a.H_in = (const __nv_bfloat16*)H_in;
      a.H_out = (__nv_bfloat16*)H_out;
      a.U = (__nv_bfloat16*)L.U;
      a.stats = L.stats;
      a.off = m.type_off[t];
      a.n = m.type_off[t + 1] - m.type_off[t];
      a.act = p->act;
      a.ln = p->layernorm;
      a.eps = p->ln_eps;
      a.status = device_status_ptr();
      if (a.n == 0) continue;
      if (p->fused) {
        a.agg_ptr = graph->agg_ptr;
        a.agg_col = graph->agg_col;
        a.agg_cnt = graph->agg_cnt;
        a.csr_ptr = graph->csr_ptr;
        a.long_ofs = graph->long_ofs;
        a.Mlong = (const __nv_bfloat16*)L.Mlong;
        HG_TRY(tc_proj_forward_gather(d, a, L.Vt, m.num_rels, s));
      } else {
        HG_TRY(tc_proj_forward(d, a, L.M, graph->csr_rows, L.Vt, m.num_rels, s));
      }
    }
    return HG_OK;
  }
  for (int t = 0; t < m.num_types; ++t) {
    FwdArgs a{};
    a.M = L.M;
    a.mrow = compact ? graph->mrow : nullptr;
    a.msent = graph->csr_rows;
    for (int r = 0; r < m.num_rels; ++r) {
      if (m.rel_dst[r] != t) continue;
      a.mrow0[a.nrel] = m.row_base[r];
      a.W_rel[a.nrel] = (const char*)p->W_rel + (size_t)r * d * d * b;
      ++a.nrel;
    }
    a.W_agg = (const char*)p->W_agg + (size_t)t * d * d * b;
    a.b = (const char*)p->b_agg + (size_t)t * d * b;
    a.gamma = p->layernorm ? (const char*)p->ln_gamma + (size_t)t * d * b : nullptr;
    a.beta = p->layernorm ? (const char*)p->ln_beta + (size_t)t * d * b : nullptr;
    a.H_in = H_in;
    a.H_out = H_out;
    a.Z = L.Z;
    a.U = L.U;
    a.stats = L.stats;
    a.off = m.type_off[t];
    a.n = m.type_off[t + 1] - m.type_off[t];
    a.act = p->act;
    a.ln = p->layernorm;
    a.eps = p->ln_eps;
    if (a.n > 0) HG_TRY(proj_forward(p->dtype, d, a, s));
  }
  return HG_OK;
}

}  // namespace hg

extern "C" hg_status hg_layer_bwd(const hg_graph* graph, const hg_layer_params* p, const void* H_in, const void* saved,
                                  const void* dH_out, void* dH_in, const hg_layer_grads* grads, void* scratch,
                                  hg_stream stream) {
  clear_error();
  HG_TRY(device_guard());
  HG_TRY(check_params(graph, p));
  HG_TRY(check_buf(H_in, "H_in"));
  HG_TRY(check_buf(saved, "saved"));
  HG_TRY(check_buf(dH_out, "dH_out"));
  HG_TRY(check_buf(scratch, "scratch"));
  HG_REQUIRE(dH_in == nullptr || ((uintptr_t)dH_in & 255) == 0, "dH_in must be 256-byte aligned");
  HG_REQUIRE(grads && grads->dW_rel && grads->dW_agg && grads->db_agg, "grads and its dW_rel, dW_agg, db_agg must be non-null");
  HG_REQUIRE(!p->layernorm || (grads->dln_gamma && grads->dln_beta), "layernorm needs dln_gamma and dln_beta");
  HG_REQUIRE(dH_in != dH_out, "dH_in and dH_out must not alias");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  LayerLayout L;
  carve_layer(graph, p->d, p->dtype, const_cast<void*>(saved), scratch, &L, nullptr, nullptr, p->fused != 0);
  HG_TRY(project_backward(graph, p, H_in, dH_out, grads, L, true, true, s));
  if (dH_in) HG_TRY(aggregate_backward(graph, p->dtype, p->d, L.dMs, L.dY, dH_in, L.agg_part, L.work, s));
  return HG_OK;
}

namespace hg {

// Backward of project_forward: L.dY = the residual path's dL/dH_in, L.dMs = dL/dM_r (divided by
// deg_r when deg_scale is set, for the mean's transposed gather), and every weight gradient.
hg_status project_backward(const hg_graph* graph, const hg_layer_params* p, const void* H_in, const void* dH_out,
                           const hg_layer_grads* grads, const LayerLayout& L, bool deg_scale, bool compact,
                           cudaStream_t s) {
  const GraphMeta& m = graph->meta;
  const int d = p->d;
  const size_t b = elem_size(p->dtype);
  const bool tc = p->dtype == HG_BF16;
  if (!tc) {
    HG_TRY(transpose_weights(p->dtype, d, p->W_rel, L.WrelT, m.num_rels, s));
    HG_TRY(transpose_weights(p->dtype, d, p->W_agg, L.WaggT, m.num_types, s));
  }
  for (int t = 0; t < m.num_types; ++t) {
    const int64_t n = m.type_off[t + 1] - m.type_off[t];
    float* db = grads->db_agg + (size_t)t * d;
    if (n == 0) {
      HG_CUDA(cudaMemsetAsync(db, 0, d * sizeof(float), s));
      if (p->layernorm) {
        HG_CUDA(cudaMemsetAsync(grads->dln_gamma + (size_t)t * d, 0, d * sizeof(float), s));
        HG_CUDA(cudaMemsetAsync(grads->dln_beta + (size_t)t * d, 0, d * sizeof(float), s));
      }
      HG_CUDA(cudaMemsetAsync(grads->dW_agg + (size_t)t * d * d, 0, (size_t)d * d * sizeof(float), s));
      continue;
    }
    int blocks;
    if (tc) {
      TcBwdArgs a{};
      for (int r = 0; r < m.num_rels; ++r) {
        if (m.rel_dst[r] != t) continue;
        a.rel[a.nrel] = r;
        a.mrow0[a.nrel] = m.row_base[r];
        ++a.nrel;
      }
      a.type = t;
      a.dH_out = (const __nv_bfloat16*)dH_out;
      a.H_in = (const __nv_bfloat16*)H_in;
      a.U = (const __nv_bfloat16*)L.U;
      a.stats = L.stats;
      a.gamma = p->layernorm ? (const __nv_bfloat16*)p->ln_gamma + (size_t)t * d : nullptr;
      a.b = (const __nv_bfloat16*)p->b_agg + (size_t)t * d;
      a.csr_ptr = deg_scale ? graph->csr_ptr : nullptr;
      a.mlist = compact ? graph->mlist : nullptr;
      a.mbase = compact ? graph->mbase : nullptr;
      a.dY = (__nv_bfloat16*)L.dY;
      a.dU = (__nv_bfloat16*)L.dU;
      a.dMs = (__nv_bfloat16*)L.dMs;
      a.part = L.cpart;
      a.off = m.type_off[t];
      a.n = n;
      a.act = p->act;
      a.ln = p->layernorm;
      a.status = device_status_ptr();
      HG_TRY(tc_ln_act_backward(d, a, &blocks, s));
      HG_TRY(tc_proj_backward(d, a, L.V, m.num_rels, s));
    } else {
      BwdArgs a{};
      a.dH_out = dH_out;
      a.H_in = H_in;
      a.U = L.U;
      a.stats = L.stats;
      a.gamma = p->layernorm ? (const char*)p->ln_gamma + (size_t)t * d * b : nullptr;
      a.W_aggT = (const char*)L.WaggT + (size_t)t * d * d * b;
      for (int r = 0; r < m.num_rels; ++r) {
        if (m.rel_dst[r] != t) continue;
        a.mrow0[a.nrel] = m.row_base[r];
        a.W_relT[a.nrel] = (const char*)L.WrelT + (size_t)r * d * d * b;
        ++a.nrel;
      }
      a.csr_ptr = deg_scale ? graph->csr_ptr : nullptr;
      a.mrow = compact ? graph->mrow : nullptr;
      a.msent = graph->csr_rows;
      a.dY = L.dY;
      a.dU = L.dU;
      a.dZ = L.dZ;
      a.dMs = L.dMs;
      a.part = L.cpart;
      a.off = m.type_off[t];
      a.n = n;
      a.act = p->act;
      a.ln = p->layernorm;
      HG_TRY(proj_backward(p->dtype, d, a, s));
      blocks = (int)ceil_div(n, 64);
    }
    HG_TRY(reduce_partials3(L.cpart, 3LL * d, blocks, d, db,
                            p->layernorm ? grads->dln_gamma + (size_t)t * d : nullptr,
                            p->layernorm ? grads->dln_beta + (size_t)t * d : nullptr, s));
    const int64_t off = m.type_off[t];
    if (!tc)
      HG_TRY(weight_grad(p->dtype, d, L.Z, off, L.dU, off, n, L.wpart, grads->dW_agg + (size_t)t * d * d, L.rtmp, s));
  }
  if (tc && p->fused) {  // G_r = M_r^T dU, the rows of M_r summed again from H_in
    for (int r = 0; r < m.num_rels; ++r) {
      const int t = m.rel_dst[r];
      HG_TRY(tc_weight_grad_gather(d, graph, H_in, L.Mlong, r, m.row_base[r], L.dU, m.type_off[t],
                                   m.type_off[t + 1] - m.type_off[t], L.wpart, L.G + (size_t)r * d * d, L.rtmp,
                                   s));
    }
  } else if (tc && compact) {  // G_r = M_r^T dU over each relation's stored rows (dU rows gathered)
    for (int r = 0; r < m.num_rels; ++r) {
      const int t = m.rel_dst[r];
      HG_TRY(tc_weight_grad_rows(d, L.M, graph->csr_rows, graph->mlist, graph->mbase, r, m.row_base[r], L.dU,
                                 m.type_off[t], m.type_off[t + 1] - m.type_off[t], L.wpart, L.G + (size_t)r * d * d,
                                 L.rtmp, s));
    }
  } else if (tc) {  // G_r = M_r^T dU, the relations into one type sharing the loads of dU
    for (int t = 0; t < m.num_types; ++t) {
      const int64_t n = m.type_off[t + 1] - m.type_off[t];
      int64_t x0[kMaxRels];
      float* outs[kMaxRels];
      int R = 0;
      for (int r = 0; r <= m.num_rels; ++r) {
        if (r < m.num_rels && m.rel_dst[r] == t) {
          x0[R] = m.row_base[r];
          outs[R] = L.G + (size_t)r * d * d;
          ++R;
        }
        if (R > 0 && (R == wgrad_tc_max_rels(d) || r == m.num_rels)) {
          HG_TRY(tc_weight_grad(d, L.M, x0, R, L.dU, m.type_off[t], n, L.wpart, outs, L.rtmp, s));
          R = 0;
        }
      }
    }
  } else {
    for (int r = 0; r < m.num_rels; ++r) {
      const int t = m.rel_dst[r];
      const int64_t n = m.type_off[t + 1] - m.type_off[t];
      HG_TRY(weight_grad(p->dtype, d, L.M, m.row_base[r], L.dZ, m.type_off[t], n, L.wpart,
                         grads->dW_rel + (size_t)r * d * d, L.rtmp, s, compact ? graph->mrow : nullptr,
                         graph->csr_rows));
    }
  }
  if (tc)  // dW_r = G_r W_agg^T, dW_agg[t] = sum_{r -> t} W_r^T G_r
    HG_TRY(tc_wgrad_finish(d, L.G, p->W_rel, p->W_agg, rel_dst_of(m), m.num_rels, m.num_types, grads->dW_rel,
                           grads->dW_agg, s));
  return HG_OK;
}

}  // namespace hg
