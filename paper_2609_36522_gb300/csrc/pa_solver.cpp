// Host side of the C ABI: argument checks, the call-order state machine,
// workspace carving, DDIM drift coefficients and kernel dispatch.
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <string>
#include <vector>

#include "../../include/paraanya.h"
#include "pa_internal.h"
#include "pa_loop.h"

namespace pa {

static thread_local std::string g_err;
void set_error(const std::string& msg) { g_err = msg; }

bool pdl_enabled() {
  static const bool on = [] {
    const char* v = std::getenv("PA_DISABLE_PDL");
    return !(v && v[0] == '1');
  }();
  return on;
}

}  // namespace pa

namespace {

enum class St { Created, Ready, Stepped, Done };

}  // namespace

struct pa_solver {
  pa::Dev d;
  pa::Layout L;
  char* ws;
  cudaStream_t st;
  St state;
  int update_kind;   // requested: 0 plain, 1 bulk pipeline, 2 lean register form, 3 fused step
  int lean_shape;    // launch shape of the lean register form
  int last_kind;     // kernel the last pa_submit_eps actually launched (-1: none yet)
  int64_t k;         // pa_submit_eps calls since pa_init: the plan of iteration k is copy k mod 2
  int64_t launches;
  pa::Ctl* host_ctl; // pinned mirror of the device Ctl
  pa::Ctl* host_ring;        // pinned: two more mirrors, one per pending pa_poll_begin
  cudaEvent_t poll_ev[2];    // recorded behind each pending poll's copies
  int poll_head, poll_count;  // the oldest pending poll's mirror, polls pending
  // the device-driven generation loop (pa_loop_*): a graph [clear the pass
  // counter] -> [WHILE node; body: two iterations and the loop test]
  cudaGraph_t loop_graph;
  cudaGraphExec_t loop_exec;
  cudaGraphConditionalHandle loop_cond;
  bool loop_capturing;     // between pa_loop_capture_begin and _end
  bool looped;             // a loop was launched since pa_init: host-side stepping is closed
  int64_t loop_k0, loop_launches0;  // s->k and s->launches when the capture began
  std::vector<double> alphas;  // the schedule, kept for pa_set_noise
  double eta;
  // optional CUDA-event timing of the Picard-update kernel
  bool timing;
  std::vector<cudaEvent_t> ev;  // pairs: [2k] before, [2k+1] after launch k
  size_t ev_next;               // pairs recorded since the last read
};

namespace {

// DDIM step i -> i+1 with noise scale sigma_i = eta sqrt((1 - a') / (1 - a))
// sqrt(1 - a / a'), written as x + s(x, eps, z) with
// s = (c_i - 1) x + e_i eps + sigma_i z, c_i = sqrt(a' / a),
// e_i = sqrt(1 - a' - sigma_i^2) - sqrt(a' (1 - a) / a); c_i - 1 is formed
// without cancellation. fp64 on the host, stored as fp32 [3][T].
std::vector<float> step_coefficients(const std::vector<double>& al, double eta) {
  const int T = (int)al.size() - 1;
  std::vector<float> hc(3 * (size_t)T);
  for (int i = 0; i < T; ++i) {
    const double a = al[i], an = al[i + 1];
    const double r = an / a;
    const double c = std::sqrt(r);
    const double cm1 = (r - 1.0) / (c + 1.0);
    const double sig = eta * std::sqrt((1.0 - an) / (1.0 - a)) * std::sqrt(1.0 - a / an);
    const double e = std::sqrt(std::max(0.0, 1.0 - an - sig * sig)) - std::sqrt(an) * std::sqrt(1.0 - a) / std::sqrt(a);
    hc[i] = (float)cm1;
    hc[T + i] = (float)e;
    hc[2 * (size_t)T + i] = (float)sig;
  }
  return hc;
}

pa_status cuda_fail(const char* where, cudaError_t e) {
  pa::set_error(std::string(where) + ": " + cudaGetErrorString(e));
  return PA_ERR_CUDA;
}

pa_status arg_fail(const std::string& msg) {
  pa::set_error(msg);
  return PA_ERR_ARG;
}

pa_status state_fail(const char* where) {
  pa::set_error(std::string(where) + ": call out of order");
  return PA_ERR_STATE;
}

bool sizes_ok(int T, int P, int64_t D, int B) {
  return T >= 1 && P >= 1 && P <= pa::kMaxWindow && D >= 1 && B >= 1 && B <= pa::kMaxBatch &&
         D <= ((int64_t)1 << 40);
}

// The device status word of a copied Ctl as a status.
pa_status check_ctl(const pa::Ctl& c, const char* where) {
  const int ds = c.status;
  if (ds == pa::kDevTimeout) {
    pa::set_error(std::string(where) + ": a device-side bounded wait ran out");
    return PA_ERR_TIMEOUT;
  }
  if (ds != pa::kDevOk) {
    pa::set_error(std::string(where) + ": device-side check failed (code " + std::to_string(ds) + ")");
    return PA_ERR_DEVICE;
  }
  return PA_OK;
}

// Copy the device Ctl into the pinned mirror and wait. Returns a status for
// a CUDA failure or a device-side error.
pa_status sync_ctl(pa_solver* s, const char* where) {
  cudaError_t e = cudaMemcpyAsync(s->host_ctl, s->d.ctl, sizeof(pa::Ctl), cudaMemcpyDeviceToHost, s->st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s->st);
  if (e != cudaSuccess) return cuda_fail(where, e);
  return check_ctl(*s->host_ctl, where);
}

// Inside a stream capture the event becomes an event-record node of the graph
// (recorded again at every replay); outside it is an ordinary record.
cudaError_t record_timing_event(cudaEvent_t ev, cudaStream_t st) {
  cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
  cudaError_t e = cudaStreamIsCapturing(st, &cs);
  if (e != cudaSuccess) return e;
  if (cs == cudaStreamCaptureStatusActive) return cudaEventRecordWithFlags(ev, st, cudaEventRecordExternal);
  return cudaEventRecord(ev, st);
}

// Enqueue the copy of the states in the slot of t = T ([batch][D]) into x_out.
cudaError_t copy_xt(pa_solver* s, float* x_out) {
  const pa::Dev& d = s->d;
  const float* src = d.X + (int64_t)(d.T % (d.P + 1)) * d.D;
  return cudaMemcpy2DAsync(x_out, (size_t)d.D * sizeof(float), src, (size_t)(d.P + 1) * d.D * sizeof(float),
                           (size_t)d.D * sizeof(float), d.B, cudaMemcpyDefault, s->st);
}

// Let go of a loop graph whose capture the runtime invalidated, without
// destroying it: destroying such a graph crashed the host process inside the
// CUDA runtime. The graph leaks; the handle can capture again.
void forget_loop(pa_solver* s) {
  s->loop_exec = nullptr;
  s->loop_graph = nullptr;
  s->loop_cond = 0;
}

// Forget the captured generation loop (its launches carry the settings of
// the capture). Not while a capture is open.
void drop_loop(pa_solver* s) {
  if (s->loop_exec) cudaGraphExecDestroy(s->loop_exec);
  if (s->loop_graph) cudaGraphDestroy(s->loop_graph);  // and the body the conditional node owns
  s->loop_exec = nullptr;
  s->loop_graph = nullptr;
  s->loop_cond = 0;
}

// Setters that change what the captured launches would be drop the loop;
// none may run while one is being captured.
bool loop_busy(pa_solver* s, const char* where) {
  if (!s->loop_capturing) {
    drop_loop(s);
    return false;
  }
  pa::set_error(std::string(where) + ": a generation loop is being captured");
  return true;
}

// Enqueue the copy of x_init ([batch][D], host or device) into state 0 of
// every trajectory; the rest of the first window is lazy.
cudaError_t copy_x_init(pa_solver* s, const float* x_init) {
  const pa::Dev& d = s->d;
  return cudaMemcpy2DAsync(d.X, (size_t)(d.P + 1) * d.D * sizeof(float), x_init, (size_t)d.D * sizeof(float),
                           (size_t)d.D * sizeof(float), d.B, cudaMemcpyDefault, s->st);
}

}  // namespace

extern "C" {

const char* pa_last_error(void) { return pa::g_err.c_str(); }

const char* pa_status_string(int status) {
  switch (status) {
    case PA_OK: return "PA_OK";
    case PA_DONE: return "PA_DONE";
    case PA_ERR_ARG: return "PA_ERR_ARG";
    case PA_ERR_STATE: return "PA_ERR_STATE";
    case PA_ERR_CUDA: return "PA_ERR_CUDA";
    case PA_ERR_WORKSPACE: return "PA_ERR_WORKSPACE";
    case PA_ERR_TIMEOUT: return "PA_ERR_TIMEOUT";
    case PA_ERR_DEVICE: return "PA_ERR_DEVICE";
    default: return "PA_UNKNOWN";
  }
}

size_t pa_workspace_bytes(int T, int window, int64_t D, int batch) {
  if (!sizes_ok(T, window, D, batch)) return 0;
  const int P = window < T ? window : T;
  return pa::make_layout(T, P, D, batch).total;
}

pa_status pa_create(pa_solver** out, int T, int window, const int64_t* latent_shape, int ndim,
                    const double* alphas_cumprod, double tol, double cache_thresh, int batch,
                    void* workspace_dev, size_t workspace_bytes, void* stream) {
  if (!out) return arg_fail("pa_create: out is NULL");
  *out = nullptr;
  if (!latent_shape || ndim < 1 || ndim > 8) return arg_fail("pa_create: latent_shape/ndim invalid");
  int64_t D = 1;
  for (int k = 0; k < ndim; ++k) {
    if (latent_shape[k] < 1) return arg_fail("pa_create: latent_shape entries must be >= 1");
    D *= latent_shape[k];
    if (D > ((int64_t)1 << 40)) return arg_fail("pa_create: latent too large");
  }
  if (!sizes_ok(T, window, D, batch))
    return arg_fail("pa_create: need T >= 1, 1 <= window <= 1024, 1 <= batch <= 64");
  if (!alphas_cumprod) return arg_fail("pa_create: alphas_cumprod is NULL");
  for (int i = 0; i <= T; ++i) {
    const double a = alphas_cumprod[i];
    if (!(a > 0.0 && a <= 1.0)) return arg_fail("pa_create: alphas_cumprod entries must be in (0, 1]");
  }
  if (!(tol >= 0.0) || !std::isfinite(tol)) return arg_fail("pa_create: tol must be finite and >= 0");
  if (!(cache_thresh >= 0.0) || std::isnan(cache_thresh))
    return arg_fail("pa_create: cache_thresh must be >= 0");
  const int P = window < T ? window : T;
  const pa::Layout L = pa::make_layout(T, P, D, batch);
  if (!workspace_dev || (reinterpret_cast<uintptr_t>(workspace_dev) % pa::kAlign) != 0 ||
      workspace_bytes < L.total) {
    pa::set_error("pa_create: workspace NULL, not 256-byte aligned, or smaller than pa_workspace_bytes()");
    return PA_ERR_WORKSPACE;
  }

  pa_solver* s = new pa_solver{};
  s->L = L;
  s->ws = static_cast<char*>(workspace_dev);
  s->st = static_cast<cudaStream_t>(stream);
  s->state = St::Created;
  s->launches = 0;
  s->k = 0;
  s->last_kind = -1;
  s->lean_shape = 0;
  char* w = s->ws;
  pa::Dev& d = s->d;
  d.X = reinterpret_cast<float*>(w + L.X);
  d.Xhat = reinterpret_cast<float*>(w + L.Xhat);
  d.Ehat = reinterpret_cast<float*>(w + L.Ehat);
  d.batch_x = reinterpret_cast<float*>(w + L.batch_x);
  float* coef = reinterpret_cast<float*>(w + L.coef);
  d.cm1 = coef;
  d.ecoef = coef + T;
  d.sigma = coef + 2 * (size_t)T;
  d.noise = nullptr;
  s->alphas.assign(alphas_cumprod, alphas_cumprod + T + 1);
  s->eta = 0.0;
  d.traj = reinterpret_cast<pa::Traj*>(w + L.traj);
  d.pc = reinterpret_cast<pa::PlanCtr*>(w + L.pc);
  d.ctl = reinterpret_cast<pa::Ctl*>(w + L.ctl);
  d.rank = reinterpret_cast<int32_t*>(w + L.rank);
  d.miss_bt = reinterpret_cast<int32_t*>(w + L.miss_bt);
  d.acc = reinterpret_cast<double*>(w + L.acc);
  d.red_err = reinterpret_cast<float*>(w + L.red_err);
  d.red_del = reinterpret_cast<float*>(w + L.red_del);
  d.iter_log = reinterpret_cast<int32_t*>(w + L.iter_log);
  d.gbar = reinterpret_cast<unsigned long long*>(w + L.gbar);
  d.taa_g = nullptr;
  d.taa_r = nullptr;
  d.taa_acc = nullptr;
  d.taa_xe = nullptr;
  d.taa = 0;
  d.tau = reinterpret_cast<double*>(w + L.tau);
  d.adapt = 0;
  d.adapt_up = 1.0;
  d.adapt_target = 0.0;
  d.tau_min = 0.0;
  d.tau_max = 0.0;
  d.T = T; d.P = P; d.B = batch; d.D = D;
  d.tol = tol;
  d.cache_thresh = cache_thresh;
  d.tol_d = tol * (double)D;
  d.thr_d = cache_thresh * (double)D;
  d.inv_d = 1.0 / (double)D;
  d.wait_limit = pa::kWaitLimit;
  d.cache_bf16 = 0;
  // the lean register form and the planning kernel, else the bulk forms, else
  // plain loads; the fused step (3) is an option: at the 4x64x64 shape it
  // takes as long per solver step as the pair and a generation with the
  // denoiser is slower with it (its 16-warp CTAs hold every SM's register
  // file through the grid barrier, so nothing overlaps their tail)
  s->update_kind = (D % 4 == 0) ? 2 : 0;

  const std::vector<float> hc = step_coefficients(s->alphas, 0.0);  // DDIM (eta = 0)
  s->poll_ev[0] = s->poll_ev[1] = nullptr;
  s->poll_head = s->poll_count = 0;
  s->loop_graph = nullptr;
  s->loop_exec = nullptr;
  s->loop_cond = 0;
  s->loop_capturing = s->looped = false;
  s->loop_k0 = s->loop_launches0 = 0;
  cudaError_t e = cudaHostAlloc(reinterpret_cast<void**>(&s->host_ctl), 3 * sizeof(pa::Ctl), cudaHostAllocDefault);
  if (e != cudaSuccess) {
    delete s;
    return cuda_fail("pa_create: cudaHostAlloc", e);
  }
  std::memset(s->host_ctl, 0, 3 * sizeof(pa::Ctl));
  s->host_ring = s->host_ctl + 1;
  e = cudaEventCreateWithFlags(&s->poll_ev[0], cudaEventDisableTiming);
  if (e == cudaSuccess) e = cudaEventCreateWithFlags(&s->poll_ev[1], cudaEventDisableTiming);
  if (e != cudaSuccess) {
    for (cudaEvent_t x : s->poll_ev)
      if (x) cudaEventDestroy(x);
    cudaFreeHost(s->host_ctl);
    delete s;
    return cuda_fail("pa_create: cudaEventCreate", e);
  }
  e = cudaMemcpyAsync(coef, hc.data(), hc.size() * sizeof(float), cudaMemcpyHostToDevice, s->st);
  if (e == cudaSuccess) e = cudaMemsetAsync(d.ctl, 0, sizeof(pa::Ctl), s->st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s->st);
  if (e != cudaSuccess) {
    for (cudaEvent_t x : s->poll_ev) cudaEventDestroy(x);
    cudaFreeHost(s->host_ctl);
    delete s;
    return cuda_fail("pa_create", e);
  }
  *out = s;
  return PA_OK;
}

pa_status pa_set_noise(pa_solver* s, double eta, const float* noise_dev) {
  if (!s) return arg_fail("pa_set_noise: solver is NULL");
  if (loop_busy(s, "pa_set_noise")) return PA_ERR_STATE;
  if (s->state == St::Stepped) return state_fail("pa_set_noise");
  if (!(eta >= 0.0 && eta <= 1.0)) return arg_fail("pa_set_noise: eta must be in [0, 1]");
  if (eta > 0.0 && !noise_dev) return arg_fail("pa_set_noise: eta > 0 needs the draws (noise_dev)");
  if (eta > 0.0 && (reinterpret_cast<uintptr_t>(noise_dev) & 15) != 0)
    return arg_fail("pa_set_noise: noise_dev must be 16-byte aligned");
  const std::vector<float> hc = step_coefficients(s->alphas, eta);
  cudaError_t e = cudaMemcpyAsync(s->ws + s->L.coef, hc.data(), hc.size() * sizeof(float), cudaMemcpyHostToDevice,
                                  s->st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s->st);  // hc is a local buffer
  if (e != cudaSuccess) return cuda_fail("pa_set_noise", e);
  s->eta = eta;
  s->d.noise = eta > 0.0 ? noise_dev : nullptr;
  return PA_OK;
}

pa_status pa_init(pa_solver* s, const float* x_init) {
  if (!s) return arg_fail("pa_init: solver is NULL");
  if (!x_init) return arg_fail("pa_init: x_init is NULL");
  cudaError_t e = copy_x_init(s, x_init);
  if (e != cudaSuccess) return cuda_fail("pa_init: copy x_init", e);
  // the first plan (every timestep a first entry), its batch, both sets of the
  // reductions' (and the Anderson Gram sums') accumulators cleared: one kernel
  e = pa::launch_init(s->d, s->st);
  s->launches += 1;
  if (e != cudaSuccess) return cuda_fail("pa_init: launch", e);
  s->k = 0;
  s->looped = false;
  s->state = St::Ready;
  return PA_OK;
}

pa_status pa_step_async(pa_solver* s, const float** batch_x_dev, const int32_t** miss_bt_dev,
                        const int32_t** n_miss_dev) {
  if (!s) return arg_fail("pa_step_async: solver is NULL");
  if (s->state != St::Ready || s->looped) return state_fail("pa_step_async");
  // the batch was gathered by the kernel that planned this iteration
  if (batch_x_dev) *batch_x_dev = s->d.batch_x;
  if (miss_bt_dev) *miss_bt_dev = s->d.miss_bt;
  if (n_miss_dev) *n_miss_dev = &s->d.ctl->n_miss;
  s->state = St::Stepped;
  return PA_OK;
}

pa_status pa_step(pa_solver* s, int* n_miss, const float** batch_x_dev, const int32_t** miss_bt_dev) {
  if (!s) return arg_fail("pa_step: solver is NULL");
  if (!n_miss) return arg_fail("pa_step: n_miss is NULL");
  *n_miss = 0;
  if (s->state == St::Done) return PA_DONE;
  if (s->state != St::Ready) return state_fail("pa_step");
  pa_status r = pa_step_async(s, batch_x_dev, miss_bt_dev, nullptr);
  if (r != PA_OK) return r;
  r = sync_ctl(s, "pa_step");
  if (r != PA_OK) {
    s->state = St::Ready;
    return r;
  }
  if (s->host_ctl->n_active == 0) {
    s->state = St::Done;
    return PA_DONE;
  }
  *n_miss = s->host_ctl->n_miss;
  return PA_OK;
}

const int32_t* pa_n_miss_dev(const pa_solver* s) { return s ? &s->d.ctl->n_miss : nullptr; }

pa_status pa_submit_eps(pa_solver* s, const float* batch_eps_dev) {
  if (!s) return arg_fail("pa_submit_eps: solver is NULL");
  if (s->state != St::Stepped) return state_fail("pa_submit_eps");
  if (!batch_eps_dev) return arg_fail("pa_submit_eps: batch_eps is NULL");
  const int par = (int)(s->k & 1);
  cudaError_t e = cudaSuccess;
  if (s->timing) {
    if (s->ev_next * 2 + 2 > s->ev.size()) {
      for (int k = 0; k < 2 && e == cudaSuccess; ++k) {
        cudaEvent_t x;
        e = cudaEventCreate(&x);
        if (e == cudaSuccess) s->ev.push_back(x);
      }
    }
    if (e == cudaSuccess) e = record_timing_event(s->ev[2 * s->ev_next], s->st);
    if (e != cudaSuccess) return cuda_fail("pa_submit_eps: timing event", e);
  }
  bool done = false, planned = false;
  if (s->d.taa) {  // triangular Anderson mixing: the mixing update, then the mix kernel
    e = pa::launch_update_taa(s->d, batch_eps_dev, par, s->st);
    if (e == cudaErrorNotSupported) return arg_fail("pa_submit_eps: Anderson mixing needs a 16-byte aligned batch_eps");
    if (e == cudaSuccess) {
      s->launches++;
      e = pa::launch_taa_mix(s->d, par, s->st);
    }
    s->last_kind = 4;
    done = true;
  }
  if (!done && s->update_kind == 3) {
    e = pa::launch_step_fused(s->d, batch_eps_dev, par, s->lean_shape, s->st);
    if (e == cudaErrorNotSupported) {
      e = cudaSuccess;  // the grid is not resident in one wave: update and planning kernels
    } else {
      s->last_kind = 3;
      done = planned = true;
    }
  }
  if (!done && s->update_kind >= 2 && pa::update_lean_supported(s->d, batch_eps_dev)) {
    e = pa::launch_update_lean(s->d, batch_eps_dev, par, s->lean_shape, s->st);
    if (e == cudaErrorNotSupported) {
      e = cudaSuccess;  // this shape cannot hold the window: the bulk forms below
    } else {
      s->last_kind = 2;
      done = true;
    }
  }
  if (done) {
  } else if (s->update_kind >= 1 && pa::update_bulk_supported(s->d, batch_eps_dev)) {
    e = pa::launch_update_bulk(s->d, batch_eps_dev, par, s->st);
    s->last_kind = 1;
  } else {
    e = pa::launch_update_plain(s->d, batch_eps_dev, par, s->st);
    s->last_kind = 0;
  }
  s->launches++;
  if (e != cudaSuccess) return cuda_fail("pa_submit_eps: update", e);
  if (s->timing) {
    e = record_timing_event(s->ev[2 * s->ev_next + 1], s->st);
    if (e != cudaSuccess) return cuda_fail("pa_submit_eps: timing event", e);
    s->ev_next++;
  }
  if (!planned) {  // the fused step took the decision and gathered the next batch itself
    int nl = 0;
    e = pa::launch_plan(s->d, par, s->st, &nl);
    s->launches += nl;
    if (e != cudaSuccess) return cuda_fail("pa_submit_eps: plan", e);
  }
  s->k++;
  s->state = St::Ready;
  return PA_OK;
}

pa_status pa_poll(pa_solver* s, int* n_active) {
  if (!s) return arg_fail("pa_poll: solver is NULL");
  if (s->state == St::Created) return state_fail("pa_poll");
  const pa_status r = sync_ctl(s, "pa_poll");
  if (r != PA_OK) return r;
  if (n_active) *n_active = s->host_ctl->n_active;
  if (s->host_ctl->n_active == 0 && s->state == St::Ready) {
    s->state = St::Done;
  }
  return (s->host_ctl->n_active == 0) ? PA_DONE : PA_OK;
}

pa_status pa_result(pa_solver* s, float* x_out) {
  if (!s) return arg_fail("pa_result: solver is NULL");
  if (!x_out) return arg_fail("pa_result: x_out is NULL");
  if (s->state != St::Done) return state_fail("pa_result");
  const cudaError_t e = copy_xt(s, x_out);
  if (e != cudaSuccess) return cuda_fail("pa_result", e);
  return sync_ctl(s, "pa_result");
}

pa_status pa_poll_result(pa_solver* s, float* x_out, int* n_active) {
  if (!s) return arg_fail("pa_poll_result: solver is NULL");
  if (!x_out) return arg_fail("pa_poll_result: x_out is NULL");
  if (s->state != St::Ready && s->state != St::Done) return state_fail("pa_poll_result");
  cudaError_t e = copy_xt(s, x_out);
  if (e != cudaSuccess) return cuda_fail("pa_poll_result", e);
  const pa_status r = sync_ctl(s, "pa_poll_result");
  if (r != PA_OK) return r;
  if (n_active) *n_active = s->host_ctl->n_active;
  if (s->host_ctl->n_active != 0) return PA_OK;
  s->state = St::Done;
  return PA_DONE;
}

pa_status pa_poll_begin(pa_solver* s, float* x_out) {
  if (!s) return arg_fail("pa_poll_begin: solver is NULL");
  if (s->state != St::Ready && s->state != St::Done) return state_fail("pa_poll_begin");
  if (s->poll_count == 2) {
    pa::set_error("pa_poll_begin: two polls are pending (pa_poll_end first)");
    return PA_ERR_STATE;
  }
  cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
  cudaError_t e = cudaStreamIsCapturing(s->st, &cs);
  if (e != cudaSuccess) return cuda_fail("pa_poll_begin", e);
  if (cs != cudaStreamCaptureStatusNone) {
    pa::set_error("pa_poll_begin: the solver's stream is being captured");
    return PA_ERR_STATE;
  }
  const int slot = (s->poll_head + s->poll_count) & 1;
  if (x_out) e = copy_xt(s, x_out);
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(&s->host_ring[slot], s->d.ctl, sizeof(pa::Ctl), cudaMemcpyDeviceToHost, s->st);
  if (e == cudaSuccess) e = cudaEventRecord(s->poll_ev[slot], s->st);
  if (e != cudaSuccess) return cuda_fail("pa_poll_begin", e);
  s->poll_count++;
  return PA_OK;
}

pa_status pa_poll_end(pa_solver* s, int* n_active) {
  if (!s) return arg_fail("pa_poll_end: solver is NULL");
  if (s->poll_count == 0) {
    pa::set_error("pa_poll_end: no poll is pending");
    return PA_ERR_STATE;
  }
  const int slot = s->poll_head;
  s->poll_head ^= 1;
  s->poll_count--;
  const cudaError_t e = cudaEventSynchronize(s->poll_ev[slot]);
  if (e != cudaSuccess) return cuda_fail("pa_poll_end", e);
  const pa::Ctl& c = s->host_ring[slot];
  const pa_status r = check_ctl(c, "pa_poll_end");
  if (r != PA_OK) return r;
  if (n_active) *n_active = c.n_active;
  if (c.n_active != 0) return PA_OK;
  if (s->state == St::Ready) s->state = St::Done;
  return PA_DONE;
}

pa_status pa_loop_capture_begin(pa_solver* s) {
  if (!s) return arg_fail("pa_loop_capture_begin: solver is NULL");
  if (s->loop_capturing) {
    pa::set_error("pa_loop_capture_begin: a capture is already open");
    return PA_ERR_STATE;
  }
  if (s->state != St::Ready || s->looped || (s->k & 1)) return state_fail("pa_loop_capture_begin");
  if (s->timing) {
    pa::set_error("pa_loop_capture_begin: kernel timing records events, which a loop body cannot hold");
    return PA_ERR_STATE;
  }
  cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
  cudaError_t e = cudaStreamIsCapturing(s->st, &cs);
  if (e != cudaSuccess) return cuda_fail("pa_loop_capture_begin", e);
  if (cs != cudaStreamCaptureStatusNone) {
    pa::set_error("pa_loop_capture_begin: the solver's stream is already being captured");
    return PA_ERR_STATE;
  }
  drop_loop(s);
  cudaGraphNode_t loop = nullptr;
  cudaGraphNodeParams np = {};
  e = cudaGraphCreate(&s->loop_graph, 0);
  // the condition is 1 at every launch: the body runs at least once (the
  // pass counter is cleared by pa_init's kernel, which pa_loop_launch issues
  // before the graph)
  if (e == cudaSuccess) e = cudaGraphConditionalHandleCreate(&s->loop_cond, s->loop_graph, 1, cudaGraphCondAssignDefault);
  if (e == cudaSuccess) {
    np.type = cudaGraphNodeTypeConditional;
    np.conditional.handle = s->loop_cond;
    np.conditional.type = cudaGraphCondTypeWhile;
    np.conditional.size = 1;
    e = cudaGraphAddNode(&loop, s->loop_graph, nullptr, nullptr, 0, &np);
  }
  if (e == cudaSuccess)
    // relaxed: calls this thread makes meanwhile on other work (a finalizer
    // destroying another graph, say) must not invalidate the capture
    e = cudaStreamBeginCaptureToGraph(s->st, np.conditional.phGraph_out[0], nullptr, nullptr, 0,
                                      cudaStreamCaptureModeRelaxed);
  if (e != cudaSuccess) {
    drop_loop(s);
    return cuda_fail("pa_loop_capture_begin", e);
  }
  s->loop_capturing = true;
  s->loop_k0 = s->k;
  s->loop_launches0 = s->launches;
  return PA_OK;
}

pa_status pa_loop_capture_end(pa_solver* s) {
  if (!s) return arg_fail("pa_loop_capture_end: solver is NULL");
  if (!s->loop_capturing) {
    pa::set_error("pa_loop_capture_end: no capture is open");
    return PA_ERR_STATE;
  }
  const int64_t n_body = s->k - s->loop_k0;  // iterations in the body
  const bool two = s->state == St::Ready && n_body >= 2 && n_body % 2 == 0;
  cudaError_t e = cudaSuccess;
  // at most T iterations reach t = T (the window advances by at least one
  // step in each): T / n_body + 2 passes cover them
  if (two) e = pa::launch_loop_cond(s->loop_cond, s->d.ctl, (int32_t)(s->d.T / n_body + 2), s->st);
  cudaGraph_t body = nullptr;
  const cudaError_t e2 = cudaStreamEndCapture(s->st, &body);
  if (e == cudaSuccess) e = e2;
  s->loop_capturing = false;
  if (e2 != cudaSuccess) {  // the runtime invalidated the capture: keep nothing, destroy nothing
    (void)cudaGetLastError();
    forget_loop(s);
    s->k = s->loop_k0;
    s->launches = s->loop_launches0;
    if (s->state == St::Stepped) s->state = St::Ready;
    return cuda_fail("pa_loop_capture_end", e2);
  }
  s->k = s->loop_k0;  // nothing ran: the host state is the one before the capture
  s->launches = s->loop_launches0;
  if (s->state == St::Stepped) s->state = St::Ready;
  if (e == cudaSuccess && !two) {
    drop_loop(s);
    pa::set_error("pa_loop_capture_end: the body must hold an even number of iterations, at least two "
                  "(pa_step_async, the denoiser, pa_submit_eps each)");
    return PA_ERR_STATE;
  }
  if (e == cudaSuccess) e = cudaGraphInstantiate(&s->loop_exec, s->loop_graph, 0);
  if (e != cudaSuccess) {
    (void)cudaGetLastError();
    drop_loop(s);
    return cuda_fail("pa_loop_capture_end", e);
  }
  return PA_OK;
}

pa_status pa_loop_launch(pa_solver* s, const float* x_init) {
  if (!s) return arg_fail("pa_loop_launch: solver is NULL");
  if (!x_init) return arg_fail("pa_loop_launch: x_init is NULL");
  if (!s->loop_exec) {
    pa::set_error("pa_loop_launch: no generation loop has been captured");
    return PA_ERR_STATE;
  }
  if (s->state == St::Stepped || s->loop_capturing) return state_fail("pa_loop_launch");
  cudaError_t e = copy_x_init(s, x_init);
  if (e == cudaSuccess) e = pa::launch_init(s->d, s->st);  // also clears the loop's pass counter
  if (e == cudaSuccess) e = cudaGraphLaunch(s->loop_exec, s->st);
  if (e != cudaSuccess) return cuda_fail("pa_loop_launch", e);
  s->k = 0;
  s->looped = true;
  s->state = St::Ready;
  return PA_OK;
}

int64_t pa_nfe(pa_solver* s) {
  if (!s || s->state == St::Created) return -1;
  if (sync_ctl(s, "pa_nfe") != PA_OK) return -1;
  return s->host_ctl->nfe;
}

pa_status pa_stats(pa_solver* s, pa_stats_t* out) {
  if (!s || !out) return arg_fail("pa_stats: NULL argument");
  std::memset(out, 0, sizeof(*out));
  out->launches = s->launches;
  out->update_kernel = s->last_kind;
  if (s->state == St::Created) return PA_OK;
  const pa_status r = sync_ctl(s, "pa_stats");
  const pa::Ctl& c = *s->host_ctl;
  out->iters = c.iter;
  out->nfe = c.nfe;
  out->hits = c.hits;
  out->n_active = c.n_active;
  out->n_miss = c.n_miss;
  out->device_status = c.status;
  return r;
}

pa_status pa_iter_log(pa_solver* s, int32_t* out, int max_iters, int* n_iters) {
  if (!s || !out || !n_iters || max_iters < 0) return arg_fail("pa_iter_log: bad argument");
  *n_iters = 0;
  if (s->state == St::Created) return state_fail("pa_iter_log");
  const pa_status r = sync_ctl(s, "pa_iter_log");
  if (r != PA_OK) return r;
  const int n = s->host_ctl->iter < max_iters ? s->host_ctl->iter : max_iters;
  if (n > 0) {
    const cudaError_t e = cudaMemcpy(out, s->d.iter_log,
                                     (size_t)n * s->d.B * pa::kLogFields * sizeof(int32_t),
                                     cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_fail("pa_iter_log", e);
  }
  *n_iters = n;
  return PA_OK;
}

pa_status pa_last_reductions(pa_solver* s, float* err_out, float* delta_out) {
  if (!s) return arg_fail("pa_last_reductions: solver is NULL");
  if (s->state == St::Created) return state_fail("pa_last_reductions");
  cudaError_t e = cudaStreamSynchronize(s->st);
  const size_t bytes = (size_t)s->d.B * s->d.P * sizeof(float);
  if (e == cudaSuccess && err_out) e = cudaMemcpy(err_out, s->d.red_err, bytes, cudaMemcpyDeviceToHost);
  if (e == cudaSuccess && delta_out) e = cudaMemcpy(delta_out, s->d.red_del, bytes, cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail("pa_last_reductions", e);
  return PA_OK;
}

pa_status pa_set_update_kernel(pa_solver* s, int kind) {
  if (!s) return arg_fail("pa_set_update_kernel: solver is NULL");
  if (loop_busy(s, "pa_set_update_kernel")) return PA_ERR_STATE;
  if (kind == 0 || kind == 1 || kind == 2 || kind == 3) {
    s->update_kind = kind;
    s->lean_shape = 0;
    s->d.bulk_cfg = 0;
  } else if (kind >= 100 && kind < 100 + pa::kBulkConfigs) {
    s->update_kind = 1;
    s->d.bulk_cfg = kind - 100;
  } else if (kind >= 200 && kind < 200 + pa::kLeanConfigs && (kind - 200) % 10 <= 6) {
    s->update_kind = 2;
    s->lean_shape = kind - 200;
    s->d.bulk_cfg = 0;
  } else if (kind >= 300 && kind <= 306) {
    s->update_kind = 3;
    s->lean_shape = kind - 300;
    s->d.bulk_cfg = 0;
  } else {
    return arg_fail("pa_set_update_kernel: kind must be 0, 1, 2, 3, 100 + bulk launch shape, "
                    "200 + lean launch shape or 300 + fused-step launch shape");
  }
  return PA_OK;
}

pa_status pa_set_cache_adaptation(pa_solver* s, double rate, double target, double tau_min, double tau_max) {
  if (!s) return arg_fail("pa_set_cache_adaptation: solver is NULL");
  if (loop_busy(s, "pa_set_cache_adaptation")) return PA_ERR_STATE;
  if (s->state == St::Stepped) return state_fail("pa_set_cache_adaptation");
  if (!(rate >= 0.0) || !std::isfinite(rate) || !(target >= 0.0 && target <= 1.0) || !(tau_min >= 0.0) ||
      !std::isfinite(tau_min) || std::isnan(tau_max) || !(tau_max >= tau_min))
    return arg_fail("pa_set_cache_adaptation: need rate >= 0, 0 <= target <= 1, 0 <= tau_min <= tau_max");
  pa::Dev& d = s->d;
  if (rate > 0.0 && d.B * d.P > 32 * 32)
    return arg_fail("pa_set_cache_adaptation: batch * window must be at most 1024");
  d.adapt = rate > 0.0 ? 1 : 0;
  d.adapt_up = 1.0 + rate;
  d.adapt_target = target;
  d.tau_min = tau_min;
  d.tau_max = tau_max;
  s->state = St::Created;  // pa_init restarts from tau_cache
  return PA_OK;
}

pa_status pa_cache_thresholds(pa_solver* s, double* tau_out) {
  if (!s || !tau_out) return arg_fail("pa_cache_thresholds: NULL argument");
  if (s->state == St::Created) return state_fail("pa_cache_thresholds");
  const pa::Dev& d = s->d;
  if (!d.adapt) {
    for (int b = 0; b < d.B; ++b) tau_out[b] = d.cache_thresh;
    return PA_OK;
  }
  cudaError_t e = cudaMemcpyAsync(tau_out, d.tau + (s->k & 1) * d.B, (size_t)d.B * sizeof(double),
                                  cudaMemcpyDeviceToHost, s->st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s->st);
  if (e != cudaSuccess) return cuda_fail("pa_cache_thresholds", e);
  return PA_OK;
}

size_t pa_anderson_workspace_bytes(int T, int window, int64_t D, int batch) {
  if (!sizes_ok(T, window, D, batch)) return 0;
  const int P = window < T ? window : T;
  size_t o_r = 0, o_acc = 0, o_xe = 0;
  return pa::taa_layout(P, D, batch, &o_r, &o_acc, &o_xe);
}

pa_status pa_set_anderson(pa_solver* s, int depth, void* workspace_dev, size_t workspace_bytes) {
  if (!s) return arg_fail("pa_set_anderson: solver is NULL");
  if (loop_busy(s, "pa_set_anderson")) return PA_ERR_STATE;
  if (depth != 0 && depth != 1) return arg_fail("pa_set_anderson: depth must be 0 or 1");
  if (s->state == St::Stepped) return state_fail("pa_set_anderson");
  pa::Dev& d = s->d;
  if (depth == 0) {
    d.taa = 0;
    d.taa_g = d.taa_r = d.taa_xe = nullptr;
    d.taa_acc = nullptr;
    s->state = St::Created;  // the iterates change meaning: pa_init starts over
    return PA_OK;
  }
  if (d.D % 4 != 0 || d.P > 16 * 7 || d.cache_bf16)
    return arg_fail("pa_set_anderson: needs D % 4 == 0, a window of at most 112 points and fp32 cache entries");
  size_t o_r = 0, o_acc = 0, o_xe = 0;
  const size_t need = pa::taa_layout(d.P, d.D, d.B, &o_r, &o_acc, &o_xe);
  if (!workspace_dev || (reinterpret_cast<uintptr_t>(workspace_dev) % pa::kAlign) != 0 || workspace_bytes < need) {
    pa::set_error("pa_set_anderson: workspace NULL, not 256-byte aligned, or smaller than pa_anderson_workspace_bytes()");
    return PA_ERR_WORKSPACE;
  }
  char* w = static_cast<char*>(workspace_dev);
  d.taa_g = reinterpret_cast<float*>(w);
  d.taa_r = reinterpret_cast<float*>(w + o_r);
  d.taa_acc = reinterpret_cast<double*>(w + o_acc);
  d.taa_xe = reinterpret_cast<float*>(w + o_xe);
  d.taa = 1;
  s->state = St::Created;
  return PA_OK;
}

pa_status pa_set_cache_precision(pa_solver* s, int bits) {
  if (!s) return arg_fail("pa_set_cache_precision: solver is NULL");
  if (loop_busy(s, "pa_set_cache_precision")) return PA_ERR_STATE;
  if (bits != 16 && bits != 32) return arg_fail("pa_set_cache_precision: bits must be 16 or 32");
  if (s->state == St::Stepped) return state_fail("pa_set_cache_precision");
  if (bits == 16 && s->d.taa) return arg_fail("pa_set_cache_precision: Anderson mixing keeps fp32 cache entries");
  s->d.cache_bf16 = bits == 16 ? 1 : 0;
  s->state = St::Created;  // the entries change meaning: pa_init starts over
  return PA_OK;
}

pa_status pa_debug_set_wait_limit(pa_solver* s, uint32_t polls) {
  if (!s) return arg_fail("pa_debug_set_wait_limit: solver is NULL");
  if (loop_busy(s, "pa_debug_set_wait_limit")) return PA_ERR_STATE;
  s->d.wait_limit = polls ? polls : 0u;
  return PA_OK;
}

pa_status pa_set_kernel_timing(pa_solver* s, int enable) {
  if (!s) return arg_fail("pa_set_kernel_timing: solver is NULL");
  if (loop_busy(s, "pa_set_kernel_timing")) return PA_ERR_STATE;
  s->timing = (enable != 0);
  return PA_OK;
}

pa_status pa_kernel_timing(pa_solver* s, double* update_ms, int64_t* n_launches, int reset) {
  if (!s || !update_ms || !n_launches) return arg_fail("pa_kernel_timing: NULL argument");
  *update_ms = 0.0;
  *n_launches = 0;
  cudaError_t e = cudaStreamSynchronize(s->st);
  if (e != cudaSuccess) return cuda_fail("pa_kernel_timing", e);
  double tot = 0.0;
  for (size_t k = 0; k < s->ev_next; ++k) {
    float ms = 0.f;
    e = cudaEventElapsedTime(&ms, s->ev[2 * k], s->ev[2 * k + 1]);
    if (e != cudaSuccess) return cuda_fail("pa_kernel_timing: elapsed", e);
    tot += ms;
  }
  *update_ms = tot;
  *n_launches = (int64_t)s->ev_next;
  if (reset) s->ev_next = 0;
  return PA_OK;
}

pa_status pa_debug_gap(void* stream) {
  const cudaError_t e = pa::launch_gap(static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail("pa_debug_gap", e);
  return PA_OK;
}

void pa_destroy(pa_solver* s) {
  if (!s) return;
  cudaStreamSynchronize(s->st);
  for (cudaEvent_t x : s->ev) cudaEventDestroy(x);
  for (cudaEvent_t x : s->poll_ev)
    if (x) cudaEventDestroy(x);
  if (s->loop_capturing) {  // close the capture so that the stream stays usable
    cudaGraph_t g = nullptr;
    if (cudaStreamEndCapture(s->st, &g) != cudaSuccess) forget_loop(s);
    (void)cudaGetLastError();
  }
  drop_loop(s);
  if (s->host_ctl) cudaFreeHost(s->host_ctl);
  delete s;
}

}  // extern "C"
