// Loader of libalr_cluster.so (the cluster kernel forms): dlopen from this library's own
// directory, once per process, skipped in a process that is one rank of several.
#include <dlfcn.h>

#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <string>

#include "cluster_forms.h"

namespace alr {
namespace {

struct Loaded {
  ClusterForms forms{};
  bool ok = false;
  char why[1024] = "";
};

template <typename Fn>
bool resolve(void* h, const char* name, Fn& fn, Loaded& L) {
  fn = reinterpret_cast<Fn>(dlsym(h, name));
  if (fn == nullptr) snprintf(L.why, sizeof(L.why), "libalr_cluster.so lacks %s", name);
  return fn != nullptr;
}

Loaded load() {
  Loaded L;
  if (multi_rank_process()) {
    snprintf(L.why, sizeof(L.why),
             "not loaded in a process that is one rank of several (WORLD_SIZE > 1)");
    return L;
  }
  Dl_info info{};
  if (dladdr(reinterpret_cast<void*>(&cluster_forms), &info) == 0 || info.dli_fname == nullptr) {
    snprintf(L.why, sizeof(L.why), "cannot locate libalr.so on disk");
    return L;
  }
  std::string path(info.dli_fname);
  const size_t slash = path.rfind('/');
  path = (slash == std::string::npos ? std::string("./") : path.substr(0, slash + 1)) +
         "libalr_cluster.so";
  void* h = dlopen(path.c_str(), RTLD_NOW | RTLD_LOCAL);
  if (h == nullptr) {
    const char* e = dlerror();
    snprintf(L.why, sizeof(L.why), "%s", e != nullptr ? e : path.c_str());
    return L;
  }
  decltype(&alr_cluster_args_size) args_size = nullptr;
  if (!resolve(h, "alr_cluster_args_size", args_size, L) ||
      !resolve(h, "alr_cluster_launch_loss", L.forms.launch_loss, L) ||
      !resolve(h, "alr_cluster_launch_gemm", L.forms.launch_gemm, L) ||
      !resolve(h, "alr_cluster_gemm_max_clusters", L.forms.gemm_max_clusters, L) ||
      !resolve(h, "alr_cluster_launch_pair_gemm", L.forms.launch_pair_gemm, L) ||
      !resolve(h, "alr_cluster_pair_gemm_max_pairs", L.forms.pair_gemm_max_pairs, L))
    return L;
  if (args_size(0) != sizeof(LossArgs) || args_size(1) != sizeof(GemmArgs)) {
    snprintf(L.why, sizeof(L.why),
             "libalr_cluster.so was built with other argument records (%zu / %zu bytes against "
             "%zu / %zu): rebuild both libraries together",
             args_size(0), args_size(1), sizeof(LossArgs), sizeof(GemmArgs));
    return L;
  }
  L.ok = true;
  return L;
}

const Loaded& loaded() {
  static const Loaded L = load();   // initialised once, thread-safe
  return L;
}

}  // namespace

bool multi_rank_process() {
  const char* w = getenv("WORLD_SIZE");
  return w != nullptr && atoi(w) > 1;
}

const ClusterForms* cluster_forms() {
  const Loaded& L = loaded();
  return L.ok ? &L.forms : nullptr;
}

const char* cluster_forms_error() { return loaded().why; }

}  // namespace alr
