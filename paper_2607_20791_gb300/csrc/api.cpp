// Error reporting shared by all entry points.
#include <cstring>

#include "common.h"

namespace rgd {

static thread_local char g_error[512] = "";

int set_error(int code, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_error, sizeof(g_error), fmt, ap);
  va_end(ap);
  return code;
}

void clear_error() { g_error[0] = '\0'; }

}  // namespace rgd

extern "C" const char* rgd_last_error_string(void) { return rgd::g_error; }

extern "C" const char* rgd_version(void) { return "rgd 0.1 (sm_103a)"; }
