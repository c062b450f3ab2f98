// Per-launch CUDA-event timing of the library's kernels (measurement utility,
// see pf_timing_* in proxyformer.h).
#include <map>
#include <string>
#include <vector>

#include "kernels.h"
#include "proxyformer.h"

namespace pf {
namespace {

struct Record {
  const char* label;
  int ev;  // index of the start event; stop is ev + 1
  double flops, bytes;
};

struct Agg {
  std::string label;
  double ms = 0, flops = 0, bytes = 0;
  int n = 0;
};

bool g_on = false;
std::vector<cudaEvent_t> g_events;  // pool, reused across collections
int g_used = 0;
std::vector<Record> g_recs;
std::vector<Agg> g_aggs;
const char* g_tag = "gemm";
double g_tag_bytes = 0;

int next_event() {
  if (g_used == (int)g_events.size()) {
    cudaEvent_t e;
    if (cudaEventCreate(&e) != cudaSuccess) return -1;
    g_events.push_back(e);
  }
  return g_used++;
}

}  // namespace

void set_gemm_tag(const char* label, double epi_bytes) {
  g_tag = label;
  g_tag_bytes = epi_bytes;
}
const char* gemm_tag_label() { return g_tag; }
double gemm_tag_bytes() { return g_tag_bytes; }

LaunchTimer::LaunchTimer(const char* label, cudaStream_t s, double flops, double bytes)
    : idx(-1), st(s) {
  if (!g_on) return;
  const int a = next_event(), b = next_event();
  if (a < 0 || b < 0 || b != a + 1) return;
  cudaEventRecord(g_events[a], st);
  g_recs.push_back({label, a, flops, bytes});
  idx = a;
}

LaunchTimer::~LaunchTimer() {
  if (idx >= 0) cudaEventRecord(g_events[idx + 1], st);
}

}  // namespace pf

using namespace pf;

extern "C" {

void pf_timing_enable(int on) {
  g_on = on != 0;
  g_recs.clear();
  g_used = 0;
}

int pf_timing_collect(void) {
  std::map<std::string, int> pos;
  g_aggs.clear();
  for (const Record& r : g_recs) {
    float ms = 0.f;
    if (cudaEventElapsedTime(&ms, g_events[r.ev], g_events[r.ev + 1]) != cudaSuccess) ms = 0.f;
    auto it = pos.find(r.label);
    if (it == pos.end()) {
      pos[r.label] = (int)g_aggs.size();
      g_aggs.push_back(Agg{r.label});
      it = pos.find(r.label);
    }
    Agg& a = g_aggs[it->second];
    a.ms += ms;
    a.flops += r.flops;
    a.bytes += r.bytes;
    a.n += 1;
  }
  return (int)g_aggs.size();
}

const char* pf_timing_label(int i) {
  return (i >= 0 && i < (int)g_aggs.size()) ? g_aggs[i].label.c_str() : "";
}
double pf_timing_ms(int i) { return (i >= 0 && i < (int)g_aggs.size()) ? g_aggs[i].ms : 0.0; }
int pf_timing_launches(int i) { return (i >= 0 && i < (int)g_aggs.size()) ? g_aggs[i].n : 0; }
double pf_timing_flops(int i) {
  return (i >= 0 && i < (int)g_aggs.size() && g_aggs[i].n) ? g_aggs[i].flops / g_aggs[i].n : 0.0;
}
double pf_timing_bytes(int i) {
  return (i >= 0 && i < (int)g_aggs.size() && g_aggs[i].n) ? g_aggs[i].bytes / g_aggs[i].n : 0.0;
}

}  // extern "C"

// ------------------------------------------------------------ FFMA probe
// Peak of the fp32 FMA pipe, measured: every thread runs 8 independent FMA
// chains of `iters` steps (8 chains hide the FMA latency at 16 warps per SM
// sub-partition), then stores one value so the chains are not dead code.
namespace pf {
namespace {
__global__ void __launch_bounds__(512) ffma_probe_kernel(float* out, int iters, float a0) {
  float v[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) v[j] = a0 + 0.001f * (float)(threadIdx.x + j);
  const float b = 0.999f, c = 0.001f;
  for (int i = 0; i < iters; ++i) {
#pragma unroll
    for (int j = 0; j < 8; ++j) v[j] = fmaf(v[j], b, c);
  }
  float acc = 0.f;
#pragma unroll
  for (int j = 0; j < 8; ++j) acc += v[j];
  out[(long)blockIdx.x * blockDim.x + threadIdx.x] = acc;
}
}  // namespace
}  // namespace pf

extern "C" pf_status pf_probe_ffma(void* out, int blocks, int iters, void* stream) {
  if (out == nullptr || blocks < 1 || iters < 1) return PF_ERR_INVALID_ARG;
  pf::ffma_probe_kernel<<<blocks, 512, 0, static_cast<cudaStream_t>(stream)>>>(
      static_cast<float*>(out), iters, 1.0f);
  return cudaGetLastError() == cudaSuccess ? PF_OK : PF_ERR_CUDA;
}

