// Small helpers shared by the host-side translation units of the library.
#pragma once

#include <string>

namespace t2i {
// Last error of a failed create call on this thread (no handle to hold it).
void set_thread_error(const std::string& e);
const char* thread_error();
}  // namespace t2i
